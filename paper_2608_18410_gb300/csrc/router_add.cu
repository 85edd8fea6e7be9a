// router_add.cu -- the routing score in the additive form the paper prints
// (Sec. 3.4, Eq. routingscore), with linear token and language heads:
//   gamma_i = (W_v h_i + b_v) + alpha_role W_role a_i + alpha_lang (W_l c_e + b_l)
//   a_i = softmax(W_re h_i + b_re)                      Eq. (latentrole)
//   c_e = mean of episode e's retained language hidden states (Sec. 3.4 Pool)
// then the K_i largest scores are kept (ties: lower group index), written
// ascending -- the same selector as the concatenation router.
//
// Kernels, in order:
//   language pool      the concatenation router's pooling kernels
//   k_lang_term_add4   beta_e = alpha_lang (W_l c_e + b_l), fp32: a block
//                      per (layer, 4 episodes), S <= 16 (k_lang_term_add, a
//                      warp per (layer, episode, group), above that)
//   k_router_add_tc    bf16, S = 16: one CTA per (128-row router tile,
//                      layer); a single tcgen05 product [W_v ; W_re] h over
//                      d (N = S + C rounded up to 16, zero rows padding it)
//                      fed by a TMA ring; the epilogue (a thread per row /
//                      TMEM lane) takes the role softmax online over 32-column
//                      TMEM chunks, adds the role and language terms and
//                      selects the top k.
//   k_router_add_simt  every other shape (and float32): a warp per routed row.
// Token scores and role logits are products of the stored inputs with fp32
// accumulation; the role softmax, W_role a and the language term are fp32.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

// beta[l][e][s] = alpha_lang * (b_l[l][s] + W_l[l][s] . c[l][e])
template <class T>
__global__ void __launch_bounds__(256)
k_lang_term_add(const T *__restrict__ W_l, const float *__restrict__ b_l, const float *ctx, int E,
                int d, int G, float alpha_lang, float *__restrict__ beta)
{
    const int l = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int item = blockIdx.x * 8 + warp;
    pdl_trigger();
    pdl_wait();   // ctx comes from the pooling kernel
    if (item >= E * G) return;
    const int e = item / G, s = item % G;
    const T *w = W_l + ((size_t)l * G + s) * d;
    const float *c = ctx + ((size_t)l * E + e) * d;
    float acc = 0.f;
    for (int t = lane; t < d; t += 32) acc = fmaf(to_f(w[t]), ld_dep(c + t), acc);
    acc = warp_sum(acc);
    if (lane == 0) beta[((size_t)l * E + e) * G + s] = alpha_lang * (b_l[(size_t)l * G + s] + acc);
}

// The same for S <= 16: a block of 256 threads per (layer, 4 episodes);
// thread t takes columns t, t + 256, ... of the four contexts and all S rows
// of W_l (each W_l element read once per block), then the block sums.
constexpr int kTermEp = 4, kTermMaxG = 16;

template <class T>
__global__ void __launch_bounds__(256)
k_lang_term_add4(const T *__restrict__ W_l, const float *__restrict__ b_l, const float *ctx, int E,
                 int d, int G, float alpha_lang, float *__restrict__ beta)
{
    __shared__ float part[8][kTermEp * kTermMaxG];
    const int l = blockIdx.y, e0 = blockIdx.x * kTermEp, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    pdl_trigger();
    pdl_wait();   // ctx comes from the pooling kernel
    float acc[kTermEp][kTermMaxG];
#pragma unroll
    for (int i = 0; i < kTermEp; ++i)
#pragma unroll
        for (int s = 0; s < kTermMaxG; ++s) acc[i][s] = 0.f;
    const T *w = W_l + (size_t)l * G * d;
    const float *c = ctx + ((size_t)l * E + e0) * d;
    for (int t = threadIdx.x; t < d; t += 256) {
        float cv[kTermEp];
#pragma unroll
        for (int i = 0; i < kTermEp; ++i) cv[i] = e0 + i < E ? ld_dep(c + (size_t)i * d + t) : 0.f;
#pragma unroll
        for (int s = 0; s < kTermMaxG; ++s) {
            if (s < G) {
                const float wv = to_f(w[(size_t)s * d + t]);
#pragma unroll
                for (int i = 0; i < kTermEp; ++i) acc[i][s] = fmaf(wv, cv[i], acc[i][s]);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < kTermEp; ++i)
#pragma unroll
        for (int s = 0; s < kTermMaxG; ++s) {
            const float v = warp_sum(acc[i][s]);
            if (lane == 0) part[warp][i * kTermMaxG + s] = v;
        }
    __syncthreads();
    if (threadIdx.x < kTermEp * kTermMaxG) {
        const int i = threadIdx.x / kTermMaxG, s = threadIdx.x % kTermMaxG;
        if (s < G && e0 + i < E) {
            float v = 0.f;
#pragma unroll
            for (int q = 0; q < 8; ++q) v += part[q][threadIdx.x];
            beta[((size_t)l * E + e0 + i) * G + s] = alpha_lang * (b_l[(size_t)l * G + s] + v);
        }
    }
}

// One warp per routed row: the S + C dot products over d, the role softmax
// across lanes, lane s forms gamma_s, ranks by shuffles.
template <class T>
__global__ void __launch_bounds__(256)
k_router_add_simt(const T *__restrict__ h, PlanDev plan, int64_t M, int64_t rows, int d, int C, int G, int E,
                  const T *__restrict__ W_v, const T *__restrict__ W_re, const float *__restrict__ b_v,
                  const float *__restrict__ b_re, const T *__restrict__ W_role, const float *__restrict__ beta,
                  float alpha_role, uint8_t *__restrict__ idx, int64_t idx_per_layer)
{
    extern __shared__ float sl[];   // [8 warps][S + C]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, l = blockIdx.y;
    const int64_t m = (int64_t)blockIdx.x * 8 + warp;
    if (m >= M) return;   // uniform per warp
    float *sc = sl + warp * (G + C);
    float *a = sc + G;
    const int r = plan.routed[m];
    const rolesub_segment sg = plan.segs[plan.row_seg[r]];
    const T *hr = h + ((size_t)l * rows + r) * d;
    for (int j = 0; j < G + C; ++j) {
        const T *w = j < G ? W_v + ((size_t)l * G + j) * d : W_re + ((size_t)l * C + (j - G)) * d;
        float s = 0.f;
        for (int t = lane; t < d; t += 32) s = fmaf(to_f(w[t]), to_f(hr[t]), s);
        s = warp_sum(s);
        if (lane == 0) sc[j] = s;
    }
    __syncwarp();
    // a = softmax(logits + b_re), max-subtracted
    float mx = -INFINITY;
    for (int c = lane; c < C; c += 32) {
        a[c] += b_re[(size_t)l * C + c];
        mx = fmaxf(mx, a[c]);
    }
    mx = warp_max(mx);
    float z = 0.f;
    for (int c = lane; c < C; c += 32) {
        const float e = expf(a[c] - mx);
        a[c] = e;
        z += e;
    }
    z = warp_sum(z);
    __syncwarp();
    const float inv = 1.f / z;
    float gam = -INFINITY;
    if (lane < G) {
        const T *wr = W_role + ((size_t)l * G + lane) * C;
        float role = 0.f;
        for (int c = 0; c < C; ++c) role = fmaf(to_f(wr[c]), a[c], role);
        gam = sc[lane] + b_v[(size_t)l * G + lane] + alpha_role * (role * inv) +
              beta[((size_t)l * E + sg.episode) * G + lane];
    }
    int rank = 0;
    for (int g = 0; g < G; ++g) {
        const float o = __shfl_sync(0xffffffffu, gam, g);
        if (o > gam || (o == gam && g < lane)) ++rank;
    }
    const int k = sg.k;
    const bool keep = lane < G && rank < k;
    const unsigned ball = __ballot_sync(0xffffffffu, keep);
    const int pos = __popc(ball & ((1u << lane) - 1u));
    if (keep && pos < k) {   // pos < k: NaN scores rank 0 and must not overflow the row
        idx[(size_t)l * idx_per_layer + sg.idx_off + (int64_t)(r - sg.token_row) * k + pos] = (uint8_t)lane;
    }
}

// ------------------------------------------------------------ tensor core
constexpr int kTThreads = 192;
constexpr int kTRows = 128;
constexpr int kTG = 16;              // groups on this path
constexpr int kTMaxStages = 6;
constexpr uint32_t kTileA = 16384;   // 128 rows x 64 bf16
constexpr uint32_t kRingBudget = 96u * 1024u;   // two CTAs per SM

__host__ __device__ constexpr uint32_t tmem_cols_for(int nb)
{
    return nb <= 32 ? 32u : nb <= 64 ? 64u : nb <= 128 ? 128u : 256u;
}

// Shared memory (1024-aligned): stages x {A 16K | B nb rows x 128 B}, then
// W_role [S][C] as fp32, then the barriers.
__global__ void __launch_bounds__(kTThreads, 2)
k_router_add_tc(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_wv,
                const __grid_constant__ CUtensorMap tm_wre, PlanDev plan, int64_t rows, int d, int C, int E,
                int nb, int stages, const float *__restrict__ b_v, const float *__restrict__ b_re,
                const bf16 *__restrict__ W_role, const float *beta, float alpha_role,
                uint8_t *__restrict__ idx, int64_t idx_per_layer, const float *__restrict__ u_pri,
                float *__restrict__ scores, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int l = blockIdx.y;
    const int row0 = plan.route_tiles[blockIdx.x];
    const int nkb = d / 64;
    const uint32_t stage_bytes = kTileA + (uint32_t)nb * 128u;
    const uint32_t off_role = (uint32_t)stages * stage_bytes;
    const uint32_t off_bar = (off_role + 4u * (kTG + 1) * (uint32_t)C + 7u) & ~7u;
    const uint32_t bar_full = sb + off_bar, bar_empty = bar_full + 8u * kTMaxStages,
                   bar_acc = bar_empty + 8u * kTMaxStages;
    const uint32_t ncols = tmem_cols_for(nb);
    pdl_trigger();

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < stages; ++i) {
            mbar_init(bar_full + 8 * i, 1);
            mbar_init(bar_empty + 8 * i, 1);
        }
        mbar_init(bar_acc, 1);
        fence_mbar_init();
    }
    // rows S + C .. nb of every B tile stay zero (no load writes them); W_role
    // of this layer as fp32 for the epilogue
    const int pad_words = (nb - kTG - C) * 32;
    for (int s = 0; s < stages; ++s)
        for (int i = tid; i < pad_words; i += kTThreads)
            reinterpret_cast<uint32_t *>(sp + s * stage_bytes + kTileA + (kTG + C) * 128)[i] = 0u;
    float *wr = reinterpret_cast<float *>(sp + off_role);
    for (int i = tid; i < kTG * C; i += kTThreads) wr[i] = __bfloat162float(W_role[(size_t)l * kTG * C + i]);
    float *wu = wr + kTG * C;   // priority vector u (score mode), else zeros
    for (int i = tid; i < C; i += kTThreads) wu[i] = scores ? u_pri[(size_t)l * C + i] : 0.f;
    fence_async_smem();
    __syncthreads();
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), ncols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_h);
            prefetch_tmap(&tm_wv);
            prefetch_tmap(&tm_wre);
            const uint32_t tx = kTileA + 128u * (uint32_t)(kTG + C);
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % stages;
                if (kb >= stages && !mbar_wait(bar_empty + 8 * s, ((kb / stages) - 1) & 1, status, &abort_flag, 40))
                    break;
                const uint32_t st = sb + stage_bytes * s;
                mbar_expect_tx(bar_full + 8 * s, tx);
                tma_load_3d(st, &tm_h, 64 * kb, row0, l, bar_full + 8 * s);
                tma_load_3d(st + kTileA, &tm_wv, 64 * kb, 0, l, bar_full + 8 * s);
                tma_load_3d(st + kTileA + 128u * kTG, &tm_wre, 64 * kb, 0, l, bar_full + 8 * s);
            }
        }
    } else if (warp == 5) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(kTRows, nb, false);
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % stages;
                if (!mbar_wait(bar_full + 8 * s, (kb / stages) & 1, status, &abort_flag, 41)) break;
                tc_fence_after();
                const uint32_t st = sb + stage_bytes * s;
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_bf16(tmem, sdesc_sw128(st + 32u * kk, 16, 1024), sdesc_sw128(st + kTileA + 32u * kk, 16, 1024),
                             idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                mma_commit(bar_empty + 8 * s);
            }
            mma_commit(bar_acc);
        }
    } else {
        // ------------------------------------------------ epilogue warps 0-3
        const int64_t r = (int64_t)row0 + tid;
        bool routed = false;
        rolesub_segment sg{};
        if (r < rows) {
            sg = plan.segs[plan.row_seg[r]];
            routed = sg.k > 0 && sg.k < kTG;
        }
        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
        const float *bre = b_re + (size_t)l * C;
        // the language term comes from the kernel before this one, which may
        // still run while the products do
        pdl_wait();
        mbar_wait(bar_acc, 0, status, &abort_flag, 42);
        tc_fence_after();
        __syncwarp();
        // columns [0, S): token scores; [S, S + C): role logits. The role
        // softmax runs online over 32-column chunks: a running max mx, the
        // running sum z of exp(logit - mx) and acc_s = sum_c W_role[s][c]
        // exp(logit_c - mx), all rescaled when mx grows (accp: the same sum
        // with the priority vector u, pi = u . a, Sec. 3.5).
        float gam[kTG], acc[kTG];
#pragma unroll
        for (int s = 0; s < kTG; ++s) acc[s] = 0.f;
        float mx = -INFINITY, z = 0.f, accp = 0.f;
#pragma unroll 1
        for (int c0 = 0; c0 < kTG + C; c0 += 32) {
            uint32_t sr[32];
            tmem_ld32(lane_base + (uint32_t)c0, sr);
            tmem_wait_ld();
            if (!routed) continue;
            if (c0 == 0) {
#pragma unroll
                for (int j = 0; j < kTG; ++j) gam[j] = __uint_as_float(sr[j]) + __ldg(b_v + (size_t)l * kTG + j);
            }
            float lg[32];
            float cm = -INFINITY;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const int c = c0 + j - kTG;
                lg[j] = (c >= 0 && c < C) ? __uint_as_float(sr[j]) + __ldg(bre + c) : -INFINITY;
                cm = fmaxf(cm, lg[j]);
            }
            // every chunk holds at least one role logit, so nm is finite
            const float nm = fmaxf(mx, cm);
            const float rescale = expf(mx - nm);
            z *= rescale;
            accp *= rescale;
#pragma unroll
            for (int s = 0; s < kTG; ++s) acc[s] *= rescale;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const int c = c0 + j - kTG;
                if (c >= 0 && c < C) {
                    const float e = expf(lg[j] - nm);
                    z += e;
                    accp = fmaf(wu[c], e, accp);
#pragma unroll
                    for (int s = 0; s < kTG; ++s) acc[s] = fmaf(wr[s * C + c], e, acc[s]);
                }
            }
            mx = nm;
        }
        if (routed && !abort_flag) {
            const float *be = beta + ((size_t)l * E + sg.episode) * kTG;
            const float inv = 1.f / z;
#pragma unroll
            for (int s = 0; s < kTG; ++s) gam[s] += alpha_role * (acc[s] * inv) + ld_dep(be + s);
            if (scores) {
                // score mode (per-token budgets): gamma and pi to the
                // workspace, the selection runs once the segment's counts
                // are known
                float4 *dst = reinterpret_cast<float4 *>(scores + ((int64_t)l * rows + r) * kScoreStride);
#pragma unroll
                for (int q = 0; q < kTG / 4; ++q)
                    dst[q] = make_float4(gam[4 * q], gam[4 * q + 1], gam[4 * q + 2], gam[4 * q + 3]);
                dst[kTG / 4] = make_float4(accp * inv, 0.f, 0.f, 0.f);
            } else {
                const int k = sg.k;
                uint8_t *dst = idx + (int64_t)l * idx_per_layer + sg.idx_off + (r - sg.token_row) * k;
                int pos = 0;
#pragma unroll
                for (int g = 0; g < kTG; ++g) {
                    int rank = 0;
#pragma unroll
                    for (int g2 = 0; g2 < kTG; ++g2)
                        rank += (gam[g2] > gam[g] || (gam[g2] == gam[g] && g2 < g)) ? 1 : 0;
                    if (rank < k && pos < k) dst[pos++] = (uint8_t)g;   // pos < k: NaN-safe
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, ncols);
    }
}

}  // namespace

bool additive_tc_supported(const rolesub_shape *s)
{
    const int d = s->num_heads * s->head_dim;
    return s->dtype == ROLESUB_BF16 && s->num_groups == kTG && s->role_dim <= 256 - kTG && d % 64 == 0;
}

namespace {

template <class T>
cudaError_t launch_additive_t(const CompressArgs &a, const AdditiveWeights &w)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    const int L = S.num_layers, E = P.num_episodes, d = S.num_heads * S.head_dim;
    const int C = S.role_dim, G = S.num_groups;
    const int64_t M = P.routed_rows_per_layer;
    if (M == 0) return cudaSuccess;
    cudaError_t err = launch_lang_pool(a);
    if (err != cudaSuccess) return err;
    if (G <= kTermMaxG)
        err = launch_pdl(k_lang_term_add4<T>, dim3((unsigned)((E + kTermEp - 1) / kTermEp), L), dim3(256), 0,
                         a.stream, (const T *)w.W_l, w.b_l, (const float *)a.ws.lang_ctx, E, d, G, a.alpha_lang,
                         a.ws.lang_bias);
    else
        err = launch_pdl(k_lang_term_add<T>, dim3((unsigned)((E * G + 7) / 8), L), dim3(256), 0, a.stream,
                         (const T *)w.W_l, w.b_l, (const float *)a.ws.lang_ctx, E, d, G, a.alpha_lang,
                         a.ws.lang_bias);
    count_launches(1);
    if (err != cudaSuccess) return err;
    const PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev,
                     a.plan.route_tiles_dev};
    if (sizeof(T) == 2 && additive_tc_supported(a.shape)) {
        if (P.num_route_tiles == 0) return cudaSuccess;
        const int nb = (G + C + 15) / 16 * 16;
        const uint32_t stage_bytes = kTileA + 128u * (uint32_t)nb;
        const int stages = std::min<int>(kTMaxStages, (int)(kRingBudget / stage_bytes));
        const uint32_t smem = (uint32_t)stages * stage_bytes + 4u * (kTG + 1) * (uint32_t)C + 8u +
                              8u * (2 * kTMaxStages + 1) + 1024u;
        const int64_t rows = P.rows_per_layer;
        CUtensorMap th, twv, twre;
        {
            const uint64_t dims[3] = {(uint64_t)d, (uint64_t)rows, (uint64_t)L};
            const uint64_t str[2] = {(uint64_t)d * 2, (uint64_t)(rows * d * 2)};
            const uint32_t box[3] = {64, (uint32_t)kTRows, 1};
            if (!make_bf16_map(&th, a.h, 3, dims, str, box)) return cudaErrorInvalidValue;
        }
        {
            const uint64_t dims[3] = {(uint64_t)d, (uint64_t)kTG, (uint64_t)L};
            const uint64_t str[2] = {(uint64_t)d * 2, (uint64_t)d * kTG * 2};
            const uint32_t box[3] = {64, (uint32_t)kTG, 1};
            if (!make_bf16_map(&twv, w.W_v, 3, dims, str, box)) return cudaErrorInvalidValue;
        }
        {
            const uint64_t dims[3] = {(uint64_t)d, (uint64_t)C, (uint64_t)L};
            const uint64_t str[2] = {(uint64_t)d * 2, (uint64_t)d * C * 2};
            const uint32_t box[3] = {64, (uint32_t)C, 1};
            if (!make_bf16_map(&twre, a.W_re, 3, dims, str, box)) return cudaErrorInvalidValue;
        }
        err = cudaFuncSetAttribute(k_router_add_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        err = launch_pdl(k_router_add_tc, dim3((unsigned)P.num_route_tiles, L), dim3(kTThreads), smem, a.stream, th,
                         twv, twre, pd, rows, d, C, E, nb, stages, w.b_v, a.b_re, (const bf16 *)w.W_role,
                         (const float *)a.ws.lang_bias, a.alpha_role, a.idx, (int64_t)P.idx_bytes_per_layer, w.u,
                         w.scores, a.ws.status);
        count_launches(1);
        return err;
    }
    if (w.scores) return cudaErrorInvalidValue;   // score mode: tensor-core path only
    const size_t smem = (size_t)8 * (G + C) * sizeof(float);
    if (smem > 48 * 1024) {
        err = cudaFuncSetAttribute(k_router_add_simt<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
    }
    k_router_add_simt<T><<<dim3((unsigned)((M + 7) / 8), L), 256, smem, a.stream>>>(
        (const T *)a.h, pd, M, P.rows_per_layer, d, C, G, E, (const T *)w.W_v, (const T *)a.W_re, w.b_v, a.b_re,
        (const T *)w.W_role, a.ws.lang_bias, a.alpha_role, a.idx, P.idx_bytes_per_layer);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace

// S <= 32 (lane-per-group ranking); C bounded so the per-warp scratch of
// the fallback fits in shared memory
bool router_additive_supported(const rolesub_shape *s) { return s->num_groups <= 32 && s->role_dim <= 4096; }

cudaError_t launch_router_additive(const CompressArgs &a, const AdditiveWeights &w)
{
    if (a.shape->dtype == ROLESUB_BF16) return launch_additive_t<bf16>(a, w);
    return launch_additive_t<float>(a, w);
}

}  // namespace rs
