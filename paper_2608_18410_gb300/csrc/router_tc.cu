// router_tc.cu -- role-conditioned group scores and top-k on the
// 5th-generation tensor core (Sec. 3.3-3.4), bf16 inputs.
//
// Persistent: one CTA per SM walks the (layer, 128-row router tile) items,
// 320 threads:
//   warp 4  TMA producer, warp 5  MMA issuer, warps 0-3 and 6-9  epilogue:
//   two threads per tile row / TMEM lane (warp w reads lane quadrant w % 4),
//   each taking half of the row's role and hidden columns.
// Mainloop over the hidden size d in 64-column blocks (4-stage TMA ring of
// 56 KB stages; the epilogue's weights W1_a and W2 are loaded into stage 0
// as soon as its last products have read it, three blocks before the end,
// and the epilogue's operands go into stages 1-3 once the mainloop is done;
// the next item's loads start as soon as the output products have read the
// ring, so its first blocks and products overlap this item's top-k):
//   TMEM[0,256)   += h W1_h^T      (first d input columns of W1)
//   TMEM[256,320) += h W_re^T      (role logits)
// Epilogue, per routed row i:
//   a   = softmax(W_re h + b_re)                      Eq. (latentrole)
//   TMEM[0,256) += (alpha_role a) W1_a^T              tensor core, with
//         alpha_role a split into bf16 hi + lo parts (two MMAs) so the
//         product keeps ~16 mantissa bits
//   u   = ReLU(TMEM[0,256) + beta_e)                  beta_e = W1_c (alpha_lang
//         c_e) + b1 from the per-episode kernel
//   gamma = u W2^T + b2                               again hi + lo MMAs
//   keep the k largest gamma (ties: lower index), indices ascending.
// The scores that decide the top-k are thus computed with fp32
// accumulation and near-fp32 operands; no fp32 intermediate is rounded to
// plain bf16.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 320;
constexpr int kRows = 128;
constexpr int kF = 256;      // router hidden
constexpr int kC = 64;       // role dim
constexpr int kG = 16;       // groups
constexpr int kStages = 4;

constexpr uint32_t kStageBytes = 16384 + 32768 + 8192;       // A | W1_h | W_re
constexpr uint32_t kOffBar = kStages * kStageBytes;          // 224K
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;
// epilogue weights in stage 0: W1_a [256][64], W2 [16][256]
constexpr uint32_t kOffW1A = 0, kOffW2 = 32768;
static_assert(kOffW2 + 8192 <= kStageBytes, "epilogue weights inside stage 0");
// epilogue operands in stages 1-3 (1024-byte aligned for the 128-byte
// swizzle): alpha_role a hi / lo [128][64], u hi / lo [128][256]
constexpr uint32_t kOffARhi = kStageBytes, kOffARlo = kOffARhi + 16384, kOffUhi = kOffARlo + 16384,
                   kOffUlo = kOffUhi + 65536;
// role-softmax partial max / sum of each half row: [2][2][128] floats
constexpr uint32_t kOffXch = kOffUlo + 65536;
static_assert(kOffXch + 2048 <= kOffBar, "epilogue operands inside stages 1-3");

constexpr uint32_t kIdescH = idesc_bf16(128, 256, false);
constexpr uint32_t kIdescR = idesc_bf16(128, 64, false);
constexpr uint32_t kIdescG = idesc_bf16(128, 16, false);

// x0, x1 -> bf16 pairs hi = rn(x), lo = rn(x - hi) (x0 in the low halves)
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t &hi, uint32_t &lo)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    const float h0 = __uint_as_float(hi << 16), h1 = __uint_as_float(hi & 0xffff0000u);
    const __nv_bfloat162 l2 = __floats2bfloat162_rn(x0 - h0, x1 - h1);
    lo = *reinterpret_cast<const uint32_t *>(&l2);
}

__global__ void __launch_bounds__(kThreads, 1)
k_router_tc(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w1,
            const __grid_constant__ CUtensorMap tm_wre, const __grid_constant__ CUtensorMap tm_w2,
            PlanDev plan, int tiles, int L, int64_t rows, int d, int E, int G, const float *__restrict__ b_re,
            const float *beta, const float *__restrict__ b2, float alpha_role,
            uint8_t *__restrict__ idx, int64_t idx_per_layer, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nkb = d / 64;
    const int total = tiles * L;   // work items (layer, tile), layer-major
    pdl_trigger();

    const uint32_t bar_full = sb + kOffBar;                  // [kStages]
    const uint32_t bar_empty = bar_full + 8 * kStages;       // [kStages]
    const uint32_t bar_acc = bar_empty + 8 * kStages, bar_w = bar_acc + 8, bar_ar = bar_acc + 16,
                   bar_h = bar_acc + 24, bar_g = bar_acc + 32, bar_s = bar_acc + 40;
    const uint32_t bar_u = bar_acc + 48;   // [4]: u staged for K columns [32q, 32q + 32) of both halves

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < 2 * kStages; ++i) mbar_init(bar_full + 8 * i, 1);
        mbar_init(bar_acc, 1);
        mbar_init(bar_w, 1);
        mbar_init(bar_ar, 256);
        mbar_init(bar_h, 1);
        for (int q = 0; q < 4; ++q) mbar_init(bar_u + 8 * q, 256);
        mbar_init(bar_g, 1);
        mbar_init(bar_s, 128);
        fence_mbar_init();
    }
    __syncthreads();
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_h);
            prefetch_tmap(&tm_w1);
            prefetch_tmap(&tm_wre);
            prefetch_tmap(&tm_w2);
            bool ok = true;
            uint32_t g = 0;   // K blocks issued so far (ring position)
            for (int t = blockIdx.x, it = 0; t < total && ok; t += gridDim.x, ++it) {
                const int l = t / tiles, row0 = plan.route_tiles[t - l * tiles];
                // the previous item's epilogue operands and weights live in
                // the ring until its output products are done
                if (it > 0 && !mbar_wait(bar_g, (it - 1) & 1, status, &abort_flag, 29)) break;
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const uint32_t s = g % kStages;
                    if (g >= kStages && !mbar_wait(bar_empty + 8 * s, ((g / kStages) - 1) & 1, status, &abort_flag, 20)) {
                        ok = false;
                        break;
                    }
                    const uint32_t st = sb + kStageBytes * s;
                    mbar_expect_tx(bar_full + 8 * s, kStageBytes);
                    tma_load_3d(st, &tm_h, 64 * kb, row0, l, bar_full + 8 * s);
                    tma_load_3d(st + 16384, &tm_w1, 64 * kb, 0, l, bar_full + 8 * s);
                    tma_load_3d(st + 49152, &tm_wre, 64 * kb, 0, l, bar_full + 8 * s);
                }
                // the next item's first token blocks into L2 while this
                // item's last products and epilogue run
                {
                    const int tn = t + (int)gridDim.x;
                    if (ok && tn < total) {
                        const int ln = tn / tiles, rn = plan.route_tiles[tn - ln * tiles];
                        for (int kb = 0; kb < kStages && kb < nkb; ++kb) tma_prefetch_l2_3d(&tm_h, 64 * kb, rn, ln);
                    }
                }
                // epilogue weights of this layer, W1_a (input columns d..d+C)
                // and W2, into stage 0 once its last products are done
                if (ok && g > 0) {
                    const uint32_t last = kStages * ((g - 1) / kStages);
                    ok = mbar_wait(bar_empty, (last / kStages) & 1, status, &abort_flag, 28);
                }
                if (ok) {
                    mbar_expect_tx(bar_w, 32768 + 8192);
                    tma_load_3d(sb + kOffW1A, &tm_w1, d, 0, l, bar_w);
                    for (int kb = 0; kb < 4; ++kb) tma_load_3d(sb + kOffW2 + 2048 * kb, &tm_w2, 64 * kb, 0, l, bar_w);
                }
            }
        }
    } else if (warp == 5) {
        if (lane == 0) {
            bool ok = true;
            uint32_t g = 0;
            for (int t = blockIdx.x, it = 0; t < total && ok; t += gridDim.x, ++it) {
                const uint32_t ph = (uint32_t)it & 1u;
                // TMEM [0, 320) is free again: the previous item's epilogue
                // read it before arriving at bar_u[3], waited for below
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const uint32_t s = g % kStages;
                    if (!mbar_wait(bar_full + 8 * s, (g / kStages) & 1, status, &abort_flag, 21)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t st = sb + kStageBytes * s;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t a = sdesc_sw128(st + 32u * kk, 16, 1024);
                        const uint32_t acc = (kb > 0 || kk > 0) ? 1u : 0u;
                        mma_bf16(tmem, a, sdesc_sw128(st + 16384 + 32u * kk, 16, 1024), kIdescH, acc);
                        mma_bf16(tmem + 256, a, sdesc_sw128(st + 49152 + 32u * kk, 16, 1024), kIdescR, acc);
                    }
                    mma_commit(bar_empty + 8 * s);
                }
                if (!ok) break;
                mma_commit(bar_acc);
                // hidden += (alpha_role a) W1_a^T, hi and lo parts
                if (!mbar_wait(bar_ar, ph, status, &abort_flag, 22) || !mbar_wait(bar_w, ph, status, &abort_flag, 23))
                    break;
                tc_fence_after();
#pragma unroll
                for (int part = 0; part < 2; ++part)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_bf16(tmem, sdesc_sw128(sb + (part ? kOffARlo : kOffARhi) + 32u * kk, 16, 1024),
                                 sdesc_sw128(sb + kOffW1A + 32u * kk, 16, 1024), kIdescH, 1u);
                mma_commit(bar_h);
                // gamma = u W2^T, hi and lo parts, a quarter of K at a time
                // as the epilogue stages u, once the previous item's scores
                // have been read
                if (it > 0 && !mbar_wait(bar_s, ph ^ 1u, status, &abort_flag, 30)) break;
                for (int q = 0; q < 4 && ok; ++q) {
                    if (!mbar_wait(bar_u + 8 * q, ph, status, &abort_flag, 24)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int kk = 2 * q + (i & 1) + 8 * (i >> 1);   // K16 steps of quarter q, both halves
#pragma unroll
                        for (int part = 0; part < 2; ++part) {
                            const uint32_t ao = (part ? kOffUlo : kOffUhi) + (kk >> 2) * 16384u + (kk & 3) * 32u;
                            const uint32_t bo = kOffW2 + (kk >> 2) * 2048u + (kk & 3) * 32u;
                            mma_bf16(tmem + 320, sdesc_sw128(sb + ao, 16, 1024), sdesc_sw128(sb + bo, 16, 1024),
                                     kIdescG, (q > 0 || i > 0 || part > 0) ? 1u : 0u);
                        }
                    }
                }
                if (!ok) break;
                mma_commit(bar_g);
            }
        }
    } else {
        // ------------------------------------------- epilogue warps 0-3, 6-9
        const int quad = warp & 3, half = warp >= 6 ? 1 : 0;
        const int row = 32 * quad + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * quad) << 16);
        const uint32_t swz = (uint32_t)(row & 7);
        float *xch = reinterpret_cast<float *>(sp + kOffXch);
        // beta comes from the language-bias kernel, which may still run
        // while the first products do
        pdl_wait();
        // every epilogue thread walks all of its CTA's items (a wait that
        // gives up returns at once afterwards), so the pairs' named barriers
        // always match
        for (int t = blockIdx.x, it = 0; t < total; t += gridDim.x, ++it) {
            const uint32_t ph = (uint32_t)it & 1u;
            const int l = t / tiles;
            const int64_t r = (int64_t)plan.route_tiles[t - l * tiles] + row;
            bool routed = false;
            rolesub_segment sg{};
            if (r < rows) {
                sg = plan.segs[plan.row_seg[r]];
                routed = sg.k > 0 && sg.k < G;
            }
            // this row's bias lines into L1 while the products run: beta_e
            // (this half's 128 columns), b_re (32), b2
            {
                const float *be = beta + ((int64_t)l * E + sg.episode) * kF + 128 * half;
#pragma unroll
                for (int i = 0; i < 4; ++i) prefetch_l1(be + 32 * i);
                prefetch_l1(b_re + (int64_t)l * kC + 32 * half);
                prefetch_l1(b2 + (int64_t)l * kG);
            }
            mbar_wait(bar_acc, ph, status, &abort_flag, 25);
            tc_fence_after();
            __syncwarp();
            // role softmax over the two halves (max and sum exchanged
            // through shared memory, the halves' sums added in order) ->
            // alpha_role * a as bf16 hi / lo operand rows
            {
                uint32_t sr[32];
                tmem_ld32(lane_base + 256 + 32 * half, sr);
                tmem_wait_ld();
                const float4 *bre = reinterpret_cast<const float4 *>(b_re + (int64_t)l * kC + 32 * half);
                float lg[32];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float4 bb = __ldg(bre + q);
                    lg[4 * q] = __uint_as_float(sr[4 * q]) + bb.x;
                    lg[4 * q + 1] = __uint_as_float(sr[4 * q + 1]) + bb.y;
                    lg[4 * q + 2] = __uint_as_float(sr[4 * q + 2]) + bb.z;
                    lg[4 * q + 3] = __uint_as_float(sr[4 * q + 3]) + bb.w;
                }
                float mx = -INFINITY;
#pragma unroll
                for (int c = 0; c < 32; ++c) mx = fmaxf(mx, lg[c]);
                xch[128 * half + row] = mx;
                named_bar(1 + quad, 64);
                mx = fmaxf(xch[row], xch[128 + row]);
                float sum = 0.f;
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    lg[c] = expf(lg[c] - mx);
                    sum += lg[c];
                }
                xch[256 + 128 * half + row] = sum;
                named_bar(1 + quad, 64);
                const float sc = alpha_role / (xch[256 + row] + xch[384 + row]);
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    uint32_t hw[4], lw[4];
#pragma unroll
                    for (int p = 0; p < 4; ++p)
                        split_pair(lg[8 * cc + 2 * p] * sc, lg[8 * cc + 2 * p + 1] * sc, hw[p], lw[p]);
                    const uint32_t off = (uint32_t)row * 128u + (((uint32_t)(4 * half + cc) ^ swz) << 4);
                    st_shared_v4(sb + kOffARhi + off, hw[0], hw[1], hw[2], hw[3]);
                    st_shared_v4(sb + kOffARlo + off, lw[0], lw[1], lw[2], lw[3]);
                }
            }
            fence_async_smem();
            mbar_arrive(bar_ar);
            // u = ReLU(hidden + beta_e) on this half's 128 columns, split
            // into bf16 hi / lo operand rows
            mbar_wait(bar_h, ph, status, &abort_flag, 26);
            tc_fence_after();
            __syncwarp();
            {
                const float4 *be =
                    reinterpret_cast<const float4 *>(beta + ((int64_t)l * E + sg.episode) * kF + 128 * half);
#pragma unroll 1
                for (int q = 0; q < 4; ++q) {
                    uint32_t sr[32];
                    tmem_ld32(lane_base + 128 * half + 32 * q, sr);
                    tmem_wait_ld();
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc) {
                        const float4 b0 = ld_dep(be + 8 * q + 2 * cc), b1 = ld_dep(be + 8 * q + 2 * cc + 1);
                        const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
                        uint32_t hw[4], lw[4];
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            const int j = 8 * cc + 2 * p;
                            split_pair(fmaxf(__uint_as_float(sr[j]) + bb[2 * p], 0.f),
                                       fmaxf(__uint_as_float(sr[j + 1]) + bb[2 * p + 1], 0.f), hw[p], lw[p]);
                        }
                        const int chunk = 16 * half + 4 * q + cc;   // 16-byte chunk of the 256-column row
                        const uint32_t off = (uint32_t)(chunk >> 3) * 16384u + (uint32_t)row * 128u +
                                             (((uint32_t)(chunk & 7) ^ swz) << 4);
                        st_shared_v4(sb + kOffUhi + off, hw[0], hw[1], hw[2], hw[3]);
                        st_shared_v4(sb + kOffUlo + off, lw[0], lw[1], lw[2], lw[3]);
                    }
                    // quarter q staged; after the last one TMEM [0, 320)
                    // has been read and the next item's products may
                    // overwrite it
                    tc_fence_before();
                    fence_async_smem();
                    mbar_arrive(bar_u + 8 * q);
                }
            }
            // gamma + b2 -> top-k (first half)
            if (half == 0) {
                mbar_wait(bar_g, ph, status, &abort_flag, 27);
                tc_fence_after();
                __syncwarp();
                uint32_t sr[32];
                tmem_ld32(lane_base + 320, sr);
                tmem_wait_ld();
                tc_fence_before();
                mbar_arrive(bar_s);
                if (routed && !abort_flag) {
                    const float4 *b24 = reinterpret_cast<const float4 *>(b2 + (int64_t)l * kG);
                    float gam[kG];
#pragma unroll
                    for (int q = 0; q < kG / 4; ++q) {
                        const float4 bb = __ldg(b24 + q);
                        gam[4 * q] = __uint_as_float(sr[4 * q]) + bb.x;
                        gam[4 * q + 1] = __uint_as_float(sr[4 * q + 1]) + bb.y;
                        gam[4 * q + 2] = __uint_as_float(sr[4 * q + 2]) + bb.z;
                        gam[4 * q + 3] = __uint_as_float(sr[4 * q + 3]) + bb.w;
                    }
                    const int k = sg.k;
                    uint8_t *dst = idx + (int64_t)l * idx_per_layer + sg.idx_off + (r - sg.token_row) * k;
                    int pos = 0;
#pragma unroll
                    for (int g = 0; g < kG; ++g) {
                        int rank = 0;
#pragma unroll
                        for (int g2 = 0; g2 < kG; ++g2)
                            rank += (gam[g2] > gam[g] || (gam[g2] == gam[g] && g2 < g)) ? 1 : 0;
                        if (rank < k && pos < k) dst[pos++] = (uint8_t)g;   // pos < k: NaN-safe
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

bool router_tc_supported(const rolesub_shape *s)
{
    const int d = s->num_heads * s->head_dim;
    return s->dtype == ROLESUB_BF16 && s->router_hidden == kF && s->role_dim == kC && s->num_groups == kG &&
           d % 64 == 0;
}

cudaError_t launch_router_tc(const CompressArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.num_route_tiles == 0) return cudaSuccess;
    const int L = S.num_layers, d = S.num_heads * S.head_dim;
    const int64_t rows = P.rows_per_layer;
    const int64_t w1cols = 2 * (int64_t)d + kC;
    CUtensorMap th, tw1, twre, tw2;
    {
        const uint64_t dims[3] = {(uint64_t)d, (uint64_t)rows, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)d * 2, (uint64_t)(rows * d * 2)};
        const uint32_t box[3] = {64, (uint32_t)kRows, 1};
        if (!make_bf16_map(&th, a.h, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)w1cols, (uint64_t)kF, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)w1cols * 2, (uint64_t)(w1cols * kF * 2)};
        const uint32_t box[3] = {64, (uint32_t)kF, 1};
        if (!make_bf16_map(&tw1, a.W1, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)d, (uint64_t)kC, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)d * 2, (uint64_t)d * kC * 2};
        const uint32_t box[3] = {64, (uint32_t)kC, 1};
        if (!make_bf16_map(&twre, a.W_re, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)kF, (uint64_t)kG, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)kF * 2, (uint64_t)kF * kG * 2};
        const uint32_t box[3] = {64, (uint32_t)kG, 1};
        if (!make_bf16_map(&tw2, a.W2, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    cudaError_t err = cudaFuncSetAttribute(k_router_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (err != cudaSuccess) return err;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        sms = 152;
    // persistent: one CTA per SM walks the (layer, tile) items with a stride
    // of the grid size
    const int64_t total = (int64_t)P.num_route_tiles * L;
    const unsigned grid = (unsigned)(total < sms ? total : sms);
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev,
               a.plan.route_tiles_dev};
    // launched as a dependent of the language-bias kernel: the mainloop
    // reads only caller inputs, the epilogue waits for beta
    err = launch_pdl(k_router_tc, dim3(grid), dim3(kThreads), kSmemBytes, a.stream, th, tw1, twre, tw2, pd,
                     (int)P.num_route_tiles, L, rows, d, (int)P.num_episodes, (int)S.num_groups, (const float *)a.b_re,
                     (const float *)a.ws.lang_bias, (const float *)a.b2, a.alpha_role, a.idx,
                     (int64_t)P.idx_bytes_per_layer, a.ws.status);
    count_launches(1);
    return err;
}

}  // namespace rs
