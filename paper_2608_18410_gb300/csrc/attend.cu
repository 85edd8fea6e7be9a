// attend.cu -- attention over the routed value cache (SIMT, fp32 arithmetic).
//
// Per (layer, episode, head, query tile):
//   s_j = (q . k_j) * scale over every cache token j of the episode
//   p   = softmax_j(s)            (online, in chunks of kKvTile tokens)
//   y   = sum_j p_j M_j z_j       (rotated space; unkept groups are zero)
//   o   = R_h y                   (R_h and the sum commute, Sec. 3.2)
// Keys are read in full (Sec. 3: keys and queries stay unchanged); values
// are read only as the packed kept groups.
#include "common.cuh"
#include "internal.h"

namespace rs {

constexpr int kQTile = 32;
constexpr int kKvTile = 64;

template <class T, int DH>
__global__ void __launch_bounds__(256)
k_attend_simt(const T *__restrict__ q, int64_t q_ls, int64_t q_rs, int64_t q_hs,
              const T *__restrict__ K, int64_t k_ls, int64_t k_rs, int64_t k_hs,
              const T *__restrict__ packed, int64_t packed_per_layer,
              const uint8_t *__restrict__ idx, int64_t idx_per_layer, const T *__restrict__ R,
              PlanDev plan, int H, int G, int qtiles, int64_t q_rows, float scale,
              T *__restrict__ o, int32_t *status)
{
    constexpr int QP = DH + 1;      // padded row pitch (bank spread)
    constexpr int SP = kKvTile + 1;
    constexpr int CPT = DH / 8;     // output columns per thread
    extern __shared__ float sm[];
    float *Qs = sm;                          // [kQTile][QP]
    float *Ks = Qs + kQTile * QP;            // [kKvTile][QP]
    float *Zs = Ks + kKvTile * QP;           // [kKvTile][DH]
    float *Ss = Zs + kKvTile * DH;           // [kQTile][SP]
    float *Rt = Ks;                          // [DH][DH] transposed R, reuses Ks+Zs
    __shared__ rolesub_segment sg[ROLESUB_NUM_KINDS];
    __shared__ int row0[ROLESUB_NUM_KINDS + 1];

    const int h = blockIdx.x, l = blockIdx.z;
    const int e = blockIdx.y / qtiles, qt = blockIdx.y % qtiles;
    const rolesub_episode ep = plan.eps[e];
    const int qb = qt * kQTile;
    if (qb >= ep.n_query) return;
    const int nq = min(kQTile, ep.n_query - qb);
    const int nc = ep.n_cache;
    const int tid = threadIdx.x;
    if (tid < ROLESUB_NUM_KINDS) sg[tid] = plan.segs[ep.seg_begin + tid];
    if (tid == 0) {
        int r = 0;
        for (int m = 0; m < ROLESUB_NUM_KINDS; ++m) {
            row0[m] = r;
            r += plan.segs[ep.seg_begin + m].n_tokens;
        }
        row0[ROLESUB_NUM_KINDS] = r;
    }
    for (int i = tid; i < kQTile * DH; i += 256) {
        const int r = i / DH, t = i % DH;
        float x = 0.f;
        if (r < nq) x = to_f(q[(size_t)l * q_ls + (ep.q_row_begin + qb + r) * q_rs + (int64_t)h * q_hs + t]);
        Qs[r * QP + t] = x;
    }
    const int my_q = tid >> 3;      // 0..31: query row owned by this thread
    const int my_c = tid & 7;       // column phase
    float y[CPT];
#pragma unroll
    for (int c = 0; c < CPT; ++c) y[c] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    const int ds = DH / G;

    for (int j0 = 0; j0 < nc; j0 += kKvTile) {
        const int nk = min(kKvTile, nc - j0);
        __syncthreads();
        for (int i = tid; i < kKvTile * DH; i += 256) {
            const int r = i / DH, t = i % DH;
            float x = 0.f;
            if (r < nk) x = to_f(K[(size_t)l * k_ls + (ep.row_begin + j0 + r) * k_rs + (int64_t)h * k_hs + t]);
            Ks[r * QP + t] = x;
            Zs[i] = 0.f;
        }
        __syncthreads();
        // expand the kept groups of this chunk into the zero-filled tile
        for (int i = tid; i < kKvTile * G; i += 256) {
            const int r = i / G, s = i % G;
            if (r >= nk) continue;
            const int j = j0 + r;
            int m = 0;
            while (m < ROLESUB_NUM_KINDS - 1 && j >= row0[m + 1]) ++m;
            const int k = sg[m].k;
            if (s >= k) continue;
            const int64_t ti = j - row0[m];
            const int g = idx[(size_t)l * idx_per_layer + sg[m].idx_off + ti * k + s];
            if (g >= G) {
                report(status, ROLESUB_EDEVICE, (int)(ep.row_begin + j));
                continue;
            }
            const T *src = packed + (size_t)l * packed_per_layer + sg[m].packed_off +
                           (((int64_t)h * sg[m].n_tokens + ti) * k + s) * ds;
            for (int t = 0; t < ds; ++t) Zs[r * DH + g * ds + t] = to_f(src[t]);
        }
        // scores: thread (my_q, my_c) computes columns my_c + 8*c
        float sv[kKvTile / 8];
        float cmax = -INFINITY;
#pragma unroll
        for (int c = 0; c < kKvTile / 8; ++c) {
            const int r = my_c + 8 * c;
            float acc = 0.f;
#pragma unroll 8
            for (int t = 0; t < DH; ++t) acc = fmaf(Qs[my_q * QP + t], Ks[r * QP + t], acc);
            sv[c] = r < nk ? acc * scale : -INFINITY;
            cmax = fmaxf(cmax, sv[c]);
        }
#pragma unroll
        for (int off = 4; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
        const float m_new = fmaxf(m_run, cmax);
        const float alpha = expf(m_run - m_new);
        float psum = 0.f;
#pragma unroll
        for (int c = 0; c < kKvTile / 8; ++c) {
            const float p = expf(sv[c] - m_new);
            psum += p;
            Ss[my_q * SP + my_c + 8 * c] = p;
        }
#pragma unroll
        for (int off = 4; off > 0; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
        l_run = l_run * alpha + psum;
        m_run = m_new;
#pragma unroll
        for (int c = 0; c < CPT; ++c) y[c] *= alpha;
        __syncthreads();
        for (int r = 0; r < nk; ++r) {
            const float p = Ss[my_q * SP + r];
#pragma unroll
            for (int c = 0; c < CPT; ++c) y[c] = fmaf(p, Zs[r * DH + my_c + 8 * c], y[c]);
        }
    }
    __syncthreads();
    // y / l into Qs (queries are no longer needed), R_h^T into Rt
    const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
#pragma unroll
    for (int c = 0; c < CPT; ++c) Qs[my_q * QP + my_c + 8 * c] = y[c] * inv;
    const T *Rh = R + ((size_t)l * H + h) * DH * DH;
    for (int i = tid; i < DH * DH; i += 256) {
        const int m = i / DH, t = i % DH;
        Rt[t * DH + m] = to_f(Rh[i]);
    }
    __syncthreads();
    if (my_q < nq) {
        T *orow = o + ((size_t)l * q_rows + ep.q_row_begin + qb + my_q) * (size_t)(H * DH) + (size_t)h * DH;
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
            const int mcol = my_c + 8 * c;
            float acc = 0.f;
#pragma unroll 8
            for (int t = 0; t < DH; ++t) acc = fmaf(Rt[t * DH + mcol], Qs[my_q * QP + t], acc);
            orow[mcol] = from_f<T>(acc);
        }
    }
}

bool attend_supported(const rolesub_shape *s) { return s->head_dim == 64 || s->head_dim == 128; }

template <class T, int DH>
static cudaError_t launch_attend_t(const AttendArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.max_query_tokens == 0 || P.num_episodes == 0) return cudaSuccess;
    constexpr int QP = DH + 1;
    const size_t smem = (size_t)(kQTile * QP + kKvTile * QP + kKvTile * DH + kQTile * (kKvTile + 1)) *
                        sizeof(float);
    static_assert((kKvTile * QP + kKvTile * DH) >= DH * DH, "R tile must fit in K+Z buffers");
    cudaError_t err = cudaFuncSetAttribute(k_attend_simt<T, DH>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    const int qtiles = (P.max_query_tokens + kQTile - 1) / kQTile;
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev,
               a.plan.stored_dev};
    const float scale = a.scale > 0.f ? a.scale : 1.0f / sqrtf((float)DH);
    k_attend_simt<T, DH><<<dim3(S.num_heads, P.num_episodes * qtiles, S.num_layers), 256, smem,
                           a.stream>>>(
        (const T *)a.q, a.q_ls, a.q_rs, a.q_hs, (const T *)a.K, a.k_ls, a.k_rs, a.k_hs,
        (const T *)a.packed, P.packed_elems_per_layer, a.idx, P.idx_bytes_per_layer,
        (const T *)a.R, pd, S.num_heads, S.num_groups, qtiles, P.q_rows_per_layer, scale,
        (T *)a.o, a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_attend(const AttendArgs &a)
{
    if (attend_tc_supported(a.shape)) return launch_attend_tc(a);
    const bool bf = a.shape->dtype == ROLESUB_BF16;
    if (a.shape->head_dim == 128)
        return bf ? launch_attend_t<__nv_bfloat16, 128>(a) : launch_attend_t<float, 128>(a);
    return bf ? launch_attend_t<__nv_bfloat16, 64>(a) : launch_attend_t<float, 64>(a);
}

}  // namespace rs
