// dense.cu -- the dense-rotation geometry of Sec. 4.1: one d x d orthonormal
// R per layer, the rotated vector z = R^T v (all d = H d_h dims) split into S
// contiguous groups of g = d / S dims.
//
// Compress: the router's indices (as for the per-head path), Z = V R on the
// tensor core (gemm_tc.cu), then k_pack_dense keeps each token's groups:
// segment (n tokens, k) holds [n][k][g] values, token i's groups in index
// order at packed_off + (i k + j) g.
// Attend: every head's output needs all d rotated dims of the routed values,
// so the routed values are brought back to the original space first,
//   v~_j = R (M_j z_j)        (k_unpack_dense scatters M_j z_j, then one GEMM)
// and attention then reads v~ as plain per-head values (head h's d_h slice),
// through store records that keep every group with an identity rotation.
#include "common.cuh"
#include "internal.h"

namespace rs {

namespace {

typedef __nv_bfloat16 bf16;

// One warp per (stored row, layer): copies the row's kept groups of Z
// (g bf16 each, 16 bytes per lane) to their packed slots.
__global__ void __launch_bounds__(256)
k_pack_dense(PlanDev plan, int64_t rows, int d, int G, const bf16 *__restrict__ Z, const uint8_t *__restrict__ idx,
             int64_t idx_per_layer, bf16 *__restrict__ packed, int64_t packed_per_layer, int32_t *status)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, l = blockIdx.y;
    const int64_t r = (int64_t)blockIdx.x * 8 + warp;
    if (r >= rows) return;
    const rolesub_segment sg = plan.segs[plan.row_seg[r]];
    const int k = sg.k;
    if (k == 0) return;
    const int g = d / G, v16 = g / 8;
    const int64_t i = r - sg.token_row;
    const uint8_t *ix = idx + (int64_t)l * idx_per_layer + sg.idx_off + i * k;
    const uint4 *src = reinterpret_cast<const uint4 *>(Z + ((int64_t)l * rows + r) * d);
    uint4 *dst = reinterpret_cast<uint4 *>(packed + (int64_t)l * packed_per_layer + sg.packed_off + i * k * g);
    for (int j = 0; j < k; ++j) {
        const int grp = ix[j];
        if (grp >= G) {
            if (lane == 0) report(status, ROLESUB_EDEVICE, (int)r);
            continue;
        }
        for (int c = lane; c < v16; c += 32) dst[j * v16 + c] = src[grp * v16 + c];
    }
}

// One warp per (row, layer): Zm row = M z, the kept groups from the packed
// cache and zeros elsewhere.
__global__ void __launch_bounds__(256)
k_unpack_dense(PlanDev plan, int64_t rows, int d, int G, const bf16 *__restrict__ packed, int64_t packed_per_layer,
               const uint8_t *__restrict__ idx, int64_t idx_per_layer, bf16 *__restrict__ Zm, int32_t *status)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, l = blockIdx.y;
    const int64_t r = (int64_t)blockIdx.x * 8 + warp;
    if (r >= rows) return;
    const rolesub_segment sg = plan.segs[plan.row_seg[r]];
    const int k = sg.k;
    const int g = d / G, v16 = g / 8;
    const int64_t i = r - sg.token_row;
    const uint8_t *ix = idx + (int64_t)l * idx_per_layer + sg.idx_off + i * k;
    const uint4 *src = reinterpret_cast<const uint4 *>(packed + (int64_t)l * packed_per_layer + sg.packed_off +
                                                       i * k * g);
    uint4 *dst = reinterpret_cast<uint4 *>(Zm + ((int64_t)l * rows + r) * d);
    uint32_t kept = 0;
    int pos[ROLESUB_MAX_GROUPS];
    for (int s = 0; s < G; ++s) pos[s] = -1;
    for (int j = 0; j < k; ++j) {
        const int grp = ix[j];
        if (grp >= G) {
            if (lane == 0) report(status, ROLESUB_EDEVICE, (int)r);
            continue;
        }
        pos[grp] = j;
        kept |= 1u << grp;
    }
    const uint4 zero = make_uint4(0, 0, 0, 0);
    for (int s = 0; s < G; ++s) {
        const bool on = (kept >> s) & 1u;
        const int j = pos[s];
        for (int c = lane; c < v16; c += 32) dst[s * v16 + c] = on ? src[j * v16 + c] : zero;
    }
}

// Store records for attention over v~ [rows][d] of each layer: every group of
// every head kept (identity ids), the row's first group for head 0 at
// r d / 8 and a per-head stride of d_h / 8 groups.
__global__ void __launch_bounds__(256)
k_records_dense(int64_t rows, int d, int dh, int L, uint4 *__restrict__ recs)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= (int64_t)L * rows) return;
    const int64_t r = t % rows;
    const uint32_t stride = (uint32_t)(dh / 8);
    recs[t] = make_uint4(0x76543210u, 0xFEDCBA98u, (uint32_t)(r * (d / 8)), (16u << 27) | stride);
}

// Identity R_h of every (layer, head), bf16.
__global__ void __launch_bounds__(256)
k_identity(int64_t n_mats, int dh, bf16 *__restrict__ R)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t per = (int64_t)dh * dh;
    if (t >= n_mats * per) return;
    const int64_t e = t % per;
    R[t] = __float2bfloat16_rn((e / dh) == (e % dh) ? 1.f : 0.f);
}

}  // namespace

cudaError_t launch_pack_dense(const CompressArgs &a, const void *Z)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.rows_per_layer == 0) return cudaSuccess;
    const PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev,
                     a.plan.route_tiles_dev};
    k_pack_dense<<<dim3((unsigned)((P.rows_per_layer + 7) / 8), S.num_layers), 256, 0, a.stream>>>(
        pd, P.rows_per_layer, S.num_heads * S.head_dim, S.num_groups, (const bf16 *)Z, a.idx, P.idx_bytes_per_layer,
        (bf16 *)a.packed, P.packed_elems_per_layer, a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_unpack_dense(const AttendArgs &a, void *Zm)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.rows_per_layer == 0) return cudaSuccess;
    const PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev,
                     a.plan.route_tiles_dev};
    k_unpack_dense<<<dim3((unsigned)((P.rows_per_layer + 7) / 8), S.num_layers), 256, 0, a.stream>>>(
        pd, P.rows_per_layer, S.num_heads * S.head_dim, S.num_groups, (const bf16 *)a.packed,
        P.packed_elems_per_layer, a.idx, P.idx_bytes_per_layer, (bf16 *)Zm, a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_dense_attend_prep(const AttendArgs &a, void *R_identity)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    const int L = S.num_layers, d = S.num_heads * S.head_dim;
    const int64_t nrec = (int64_t)L * P.rows_per_layer;
    if (nrec > 0) {
        k_records_dense<<<(unsigned)((nrec + 255) / 256), 256, 0, a.stream>>>(P.rows_per_layer, d, S.head_dim, L,
                                                                              reinterpret_cast<uint4 *>(a.ws.row_store));
        count_launches(1);
    }
    const int64_t nm = (int64_t)L * S.num_heads, ne = nm * S.head_dim * S.head_dim;
    k_identity<<<(unsigned)((ne + 255) / 256), 256, 0, a.stream>>>(nm, S.head_dim, (bf16 *)R_identity);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
