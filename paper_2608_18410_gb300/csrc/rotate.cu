// rotate.cu -- orthogonal value decomposition and packing (Sec. 3.2).
//
// For every stored token (segments with k > 0) and head h:
//   z = R_h^T v                      (row form: z^T = v^T R_h)
//   packed[seg][h][i][j][:] = z[idx_j * d_s : (idx_j + 1) * d_s]
// Segments with k = S keep every group and get indices 0..S-1 written here;
// routed segments read the indices the router wrote.
#include "common.cuh"
#include "internal.h"

namespace rs {

constexpr int kRotRows = 32;  // tokens per block

template <class T, int DH>
__global__ void __launch_bounds__(256)
k_rotate_pack_simt(const T *__restrict__ v, const T *__restrict__ R, PlanDev plan, int64_t Ms,
                   int64_t rows, int H, int G, T *__restrict__ packed, int64_t packed_per_layer,
                   uint8_t *__restrict__ idx, int64_t idx_per_layer, int32_t *status)
{
    extern __shared__ float sm[];
    float *Rs = sm;                   // [DH][DH]
    float *Vs = Rs + DH * DH;         // [kRotRows][DH]
    float *Zs = Vs + kRotRows * DH;   // [kRotRows][DH]
    const int h = blockIdx.y, l = blockIdx.z;
    const int64_t m0 = (int64_t)blockIdx.x * kRotRows;
    const int d = H * DH;
    const T *Rh = R + ((size_t)l * H + h) * DH * DH;
    for (int i = threadIdx.x; i < DH * DH; i += blockDim.x) Rs[i] = to_f(Rh[i]);
    for (int i = threadIdx.x; i < kRotRows * DH; i += blockDim.x) {
        const int r = i / DH, t = i % DH;
        const int64_t m = m0 + r;
        Vs[i] = m < Ms ? to_f(v[((size_t)l * rows + plan.stored[m]) * d + (size_t)h * DH + t]) : 0.f;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kRotRows * DH; i += blockDim.x) {
        const int r = i / DH, n = i % DH;
        float acc = 0.f;
#pragma unroll 8
        for (int m = 0; m < DH; ++m) acc = fmaf(Vs[r * DH + m], Rs[m * DH + n], acc);
        Zs[i] = acc;
    }
    __syncthreads();
    const int ds = DH / G;
    for (int i = threadIdx.x; i < kRotRows * G; i += blockDim.x) {
        const int r = i / G, j = i % G;
        const int64_t m = m0 + r;
        if (m >= Ms) continue;
        const int row = plan.stored[m];
        const rolesub_segment sg = plan.segs[plan.row_seg[row]];
        const int k = sg.k;
        if (j >= k) continue;
        const int64_t ti = row - sg.token_row;
        uint8_t *ix = idx + (size_t)l * idx_per_layer + sg.idx_off + ti * k;
        int g;
        if (k == G) {
            g = j;
            if (h == 0) ix[j] = (uint8_t)j;
        } else {
            g = ix[j];
            if (g >= G) {
                report(status, ROLESUB_EDEVICE, row);
                continue;
            }
        }
        T *dst = packed + (size_t)l * packed_per_layer + sg.packed_off +
                 (((int64_t)h * sg.n_tokens + ti) * k + j) * ds;
        for (int e = 0; e < ds; ++e) dst[e] = from_f<T>(Zs[r * DH + g * ds + e]);
    }
}

bool rotate_supported(const rolesub_shape *s) { return s->head_dim == 64 || s->head_dim == 128; }

template <class T, int DH>
static cudaError_t launch_rot_t(const CompressArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    const int64_t Ms = P.stored_rows_per_layer;
    if (Ms == 0) return cudaSuccess;
    const size_t smem = (size_t)(DH * DH + 2 * kRotRows * DH) * sizeof(float);
    cudaError_t err = cudaFuncSetAttribute(k_rotate_pack_simt<T, DH>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev,
               a.plan.stored_dev};
    k_rotate_pack_simt<T, DH><<<dim3((unsigned)((Ms + kRotRows - 1) / kRotRows), S.num_heads,
                                     S.num_layers), 256, smem, a.stream>>>(
        (const T *)a.v, (const T *)a.R, pd, Ms, P.rows_per_layer, S.num_heads, S.num_groups,
        (T *)a.packed, P.packed_elems_per_layer, a.idx, P.idx_bytes_per_layer, a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_rotate_pack(const CompressArgs &a)
{
    if (rotate_tc_supported(a.shape)) return launch_rotate_tc(a);
    const bool bf = a.shape->dtype == ROLESUB_BF16;
    if (a.shape->head_dim == 128)
        return bf ? launch_rot_t<__nv_bfloat16, 128>(a) : launch_rot_t<float, 128>(a);
    return bf ? launch_rot_t<__nv_bfloat16, 64>(a) : launch_rot_t<float, 64>(a);
}

}  // namespace rs
