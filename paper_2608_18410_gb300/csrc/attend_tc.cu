// attend_tc.cu -- attention over the routed value cache on the 5th-generation
// tensor core (tcgen05 + TMA), bf16 inputs, fp32 accumulation.
//
// One CTA per (layer, episode, head, tile of 64 queries); 128 threads.
// Per chunk c of 64 cache tokens:
//   S_c = Q K_c^T                 tcgen05 MMA, M=128 (rows >= 64 unused),
//                                 N=64, K=128; K_c staged by TMA (double
//                                 buffered) straight from the caller's cache
//   online softmax (warps 0-1, one query row per thread, exp2 domain):
//     m_c = max(m_{c-1}, rowmax S_c), P_c = exp(S_c - m_c) (bf16, smem)
//   Z_c = the chunk's packed kept groups scattered by their indices into a
//         zero-filled 64 x 128 tile (warps 2-3; MN-major, 16-byte stores:
//         one group of d_s = 8 bf16 is exactly one swizzle chunk)
//   Y_c = P_c Z_c                  tcgen05 MMA into TMEM; accumulated into
//                                 registers as y = y * exp(m_{c-1} - m_c) + Y_c
// Finally y /= l, O = Y R_h^T on the tensor core (o_q = R_h y_q, Sec. 3.2),
// and each thread stores its 256-byte output row.
//
// Shared memory (1024-aligned, 72 KB, two CTAs per SM):
//   [0,16K)    Q (two 64-column K-blocks at +0, +8K), later Y (bf16)
//   [16K,48K)  K chunk buffers 2 x 16K; after the last S MMA, R_h (32K)
//   [48K,56K)  P chunk (64 rows x 64 kv)
//   [56K,72K)  Z chunk (two 64-column MN-blocks of 64 kv rows)
// M=128 MMAs read 128 A rows; rows 64..127 of Q/Y/P fall on the next
// region and only produce output rows that are never read.
// TMEM (256 columns): S buffers at 0 and 64, Y_c at 128, O at 0.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 128;
constexpr int kChunk = 64;   // cache tokens per chunk
constexpr int kQRows = 64;   // query rows per CTA
constexpr int kDh = 128;
constexpr int kG = 16;       // groups per head (d_s = 8: one 16-byte chunk)

constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = 16384;
constexpr uint32_t kOffP = 49152;
constexpr uint32_t kOffZ = 57344;
constexpr uint32_t kOffBar = 73728;
constexpr uint32_t kSmemBytes = kOffBar + 128 + 1024;  // + alignment slack
constexpr uint32_t kTmemCols = 256;

constexpr uint32_t kIdescS = idesc_bf16(128, 64, false);
constexpr uint32_t kIdescPV = idesc_bf16(128, 128, true);
constexpr uint32_t kIdescO = idesc_bf16(128, 128, false);

__device__ __forceinline__ uint32_t tm_lane(uint32_t tmem, int warp, int col)
{
    return tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)col;
}

__global__ void __launch_bounds__(kThreads, 2)
k_attend_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
            const __grid_constant__ CUtensorMap tm_r, const bf16 *__restrict__ packed,
            int64_t packed_per_layer, const uint8_t *__restrict__ idx, int64_t idx_per_layer,
            PlanDev plan, int H, int qtiles, int64_t q_rows, float scale_log2,
            bf16 *__restrict__ o, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ rolesub_segment sg[ROLESUB_NUM_KINDS];
    __shared__ int row0[ROLESUB_NUM_KINDS + 1];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;

    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;   // 1024-aligned base (swizzle atoms)
    const int h = blockIdx.x, l = blockIdx.z;
    const int e = blockIdx.y / qtiles, qt = blockIdx.y % qtiles;
    const rolesub_episode ep = plan.eps[e];
    const int qb = qt * kQRows;
    if (qb >= ep.n_query) return;
    const int nq = min(kQRows, ep.n_query - qb);
    const int nc = ep.n_cache;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int64_t d = (int64_t)H * kDh;

    if (nc == 0) {  // no cache tokens: o = 0
        for (int i = tid; i < nq * (kDh / 8); i += kThreads) {
            const int r = i / (kDh / 8), c8 = i % (kDh / 8);
            uint4 *dst = reinterpret_cast<uint4 *>(o + ((int64_t)l * q_rows + ep.q_row_begin + qb + r) * d +
                                                   (int64_t)h * kDh) + c8;
            *dst = make_uint4(0, 0, 0, 0);
        }
        return;
    }
    const int nchunks = (nc + kChunk - 1) / kChunk;
    const uint32_t bar_q = sb + kOffBar, bar_k0 = bar_q + 8, bar_s0 = bar_q + 24, bar_pv = bar_q + 40,
                   bar_r = bar_q + 48, bar_o = bar_q + 56;
    const int krow0 = (int)ep.row_begin, qrow0 = (int)(ep.q_row_begin + qb);

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < 8; ++i) mbar_init(bar_q + 8 * i, 1);
        fence_mbar_init();
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_r);
        mbar_expect_tx(bar_q, 16384);
        tma_load_4d(sb + kOffQ, &tm_q, 0, h, qrow0, l, bar_q);
        tma_load_4d(sb + kOffQ + 8192, &tm_q, 64, h, qrow0, l, bar_q);
        for (int c = 0; c < 2 && c < nchunks; ++c) {
            mbar_expect_tx(bar_k0 + 8 * c, 16384);
            tma_load_4d(sb + kOffK + 16384 * c, &tm_k, 0, h, krow0 + kChunk * c, l, bar_k0 + 8 * c);
            tma_load_4d(sb + kOffK + 16384 * c + 8192, &tm_k, 64, h, krow0 + kChunk * c, l, bar_k0 + 8 * c);
        }
    }
    if (tid < ROLESUB_NUM_KINDS) sg[tid] = plan.segs[ep.seg_begin + tid];
    if (tid == 0) {
        int r = 0;
        for (int m = 0; m < ROLESUB_NUM_KINDS; ++m) {
            row0[m] = r;
            r += plan.segs[ep.seg_begin + m].n_tokens;
        }
        row0[ROLESUB_NUM_KINDS] = r;
    }
    __syncthreads();
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    // S_c = Q K_c^T into TMEM columns 64 * (c & 1)
    auto issue_s = [&](int c) {
        const uint32_t kb = sb + kOffK + 16384u * (c & 1);
        if (!mbar_wait(bar_k0 + 8 * (c & 1), (c >> 1) & 1, status, &abort_flag, 1)) return;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            const uint32_t koff = (kk >> 2) * 8192u + (kk & 3) * 32u;
            mma_bf16(tmem + 64u * (c & 1), sdesc_sw128(sb + kOffQ + koff, 16, 1024),
                     sdesc_sw128(kb + koff, 16, 1024), kIdescS, kk > 0);
        }
        mma_commit(bar_s0 + 8 * (c & 1));
    };
    if (tid == 0) {
        if (mbar_wait(bar_q, 0, status, &abort_flag, 0)) {
            issue_s(0);
            if (nchunks > 1) issue_s(1);
        }
    }

    float m_run = -INFINITY, l_run = 0.f;

    for (int c = 0; c < nchunks; ++c) {
        const int buf = c & 1;
        const int nk = min(kChunk, nc - c * kChunk);
        if (warp < 2) {
            mbar_wait(bar_s0 + 8 * buf, (c >> 1) & 1, status, &abort_flag, 2);
            tc_fence_after();
            if (tid == 0 && !abort_flag) {
                // K buffer `buf` is free once S_c completed
                if (c + 2 < nchunks) {
                    mbar_expect_tx(bar_k0 + 8 * buf, 16384);
                    tma_load_4d(sb + kOffK + 16384 * buf, &tm_k, 0, h, krow0 + kChunk * (c + 2), l, bar_k0 + 8 * buf);
                    tma_load_4d(sb + kOffK + 16384 * buf + 8192, &tm_k, 64, h, krow0 + kChunk * (c + 2), l,
                                bar_k0 + 8 * buf);
                }
                if (c == nchunks - 1) {  // every S MMA is done: R_h replaces both K buffers
                    mbar_expect_tx(bar_r, 32768);
                    tma_load_3d(sb + kOffK, &tm_r, 0, 0, l * H + h, bar_r);
                    tma_load_3d(sb + kOffK + 16384, &tm_r, 64, 0, l * H + h, bar_r);
                }
            }
            __syncwarp();
            // row max of this chunk (scores in the exp2 domain)
            uint32_t sr[32];
            float mx = -INFINITY;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                tmem_ld32(tm_lane(tmem, warp, 64 * buf + 32 * half), sr);
                tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (32 * half + j < nk) mx = fmaxf(mx, __uint_as_float(sr[j]) * scale_log2);
            }
            const float m_new = fmaxf(m_run, mx);
            const float alpha_c = exp2f(m_run - m_new);
            float psum = 0.f;
            uint32_t pk[32];
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                tmem_ld32(tm_lane(tmem, warp, 64 * buf + 32 * half), sr);
                tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                    const int jj = 32 * half + j;
                    const float p0 = jj < nk ? exp2f(__uint_as_float(sr[j]) * scale_log2 - m_new) : 0.f;
                    const float p1 = jj + 1 < nk ? exp2f(__uint_as_float(sr[j + 1]) * scale_log2 - m_new) : 0.f;
                    psum += p0 + p1;
                    pk[16 * half + j / 2] = pack_bf16(p0, p1);
                }
            }
            l_run = l_run * alpha_c + psum;
            m_run = m_new;
            if (c > 0) {
                // PV_{c-1} is complete (P and Z buffers free); bring the TMEM
                // accumulator to the new row max before PV_c adds to it
                mbar_wait(bar_pv, (c - 1) & 1, status, &abort_flag, 3);
                tc_fence_after();
                __syncwarp();
                if (__any_sync(0xffffffffu, alpha_c != 1.f)) {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        tmem_ld32(tm_lane(tmem, warp, 128 + 32 * q4), sr);
                        tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) sr[j] = __float_as_uint(__uint_as_float(sr[j]) * alpha_c);
                        tmem_st32(tm_lane(tmem, warp, 128 + 32 * q4), sr);
                    }
                    tmem_wait_st();
                }
            }
            // P_c row `tid`: 64 kv = 128 bytes = 8 swizzled 16-byte chunks
            const uint32_t prow = sb + kOffP + (uint32_t)tid * 128u;
#pragma unroll
            for (int cc = 0; cc < 8; ++cc)
                st_shared_v4(prow + ((uint32_t)(cc ^ (tid & 7)) << 4), pk[4 * cc], pk[4 * cc + 1], pk[4 * cc + 2],
                             pk[4 * cc + 3]);
        } else {
            // Z_c: kv row jl of the chunk, MN-major (two 64-column blocks)
            if (c > 0) mbar_wait(bar_pv, (c - 1) & 1, status, &abort_flag, 4);
            const int jl = tid - 64;
            const int j = c * kChunk + jl;
            const uint32_t zrow = sb + kOffZ + (uint32_t)jl * 128u;
            const uint32_t sw = (uint32_t)(jl & 7);
            uint32_t kept = 0;
            if (j < nc) {
                int m = 0;
                while (m < ROLESUB_NUM_KINDS - 1 && j >= row0[m + 1]) ++m;
                const int k = sg[m].k;
                const int64_t ti = j - row0[m];
                const uint8_t *ix = idx + (int64_t)l * idx_per_layer + sg[m].idx_off + ti * k;
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    packed + (int64_t)l * packed_per_layer + sg[m].packed_off + ((int64_t)h * sg[m].n_tokens + ti) * k * 8);
                int gid[kG];
#pragma unroll
                for (int s = 0; s < kG; ++s)
                    if (s < k) gid[s] = ix[s];
#pragma unroll
                for (int s = 0; s < kG; ++s) {
                    if (s < k) {
                        const int g = gid[s];
                        if (g >= kG) {
                            report(status, ROLESUB_EDEVICE, (int)(ep.row_begin + j));
                            continue;
                        }
                        if ((kept >> g) & 1u) continue;   // repeated index: keep the first
                        kept |= 1u << g;
                        cp_async16(zrow + (uint32_t)(g >> 3) * 8192u + (((uint32_t)(g & 7) ^ sw) << 4), src + s);
                    }
                }
            }
#pragma unroll
            for (int g = 0; g < kG; ++g)
                if (!((kept >> g) & 1u))
                    st_shared_v4(zrow + (uint32_t)(g >> 3) * 8192u + (((uint32_t)(g & 7) ^ sw) << 4), 0, 0, 0, 0);
            cp_async_wait_all();
        }
        fence_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0 && !abort_flag) {
            // Y_c = P_c Z_c (fresh accumulator), then the next S on this buffer
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                mma_bf16(tmem + 128, sdesc_sw128(sb + kOffP + 32u * kk, 16, 1024),
                         sdesc_sw128(sb + kOffZ + 2048u * kk, 8192, 1024), kIdescPV, (c > 0 || kk > 0) ? 1u : 0u);
            mma_commit(bar_pv);
            if (c + 2 < nchunks) issue_s(c + 2);
        }
    }

    if (warp < 2) {
        mbar_wait(bar_pv, (nchunks - 1) & 1, status, &abort_flag, 5);
        tc_fence_after();
        __syncwarp();
        uint32_t sr[32];
        const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
        // y / l as the bf16 A operand (Q region: K-blocks of 64 columns at +0, +8K)
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            tmem_ld32(tm_lane(tmem, warp, 128 + 32 * q4), sr);
            tmem_wait_ld();
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
                const int cc = 4 * q4 + c4;   // 16-byte chunk (8 columns) of the 128-column row
                const uint32_t addr = sb + kOffQ + (uint32_t)(cc >> 3) * 8192u + (uint32_t)tid * 128u +
                                      ((uint32_t)((cc & 7) ^ (tid & 7)) << 4);
                const float *f = reinterpret_cast<const float *>(sr) + 8 * c4;
                st_shared_v4(addr, pack_bf16(f[0] * inv, f[1] * inv), pack_bf16(f[2] * inv, f[3] * inv),
                             pack_bf16(f[4] * inv, f[5] * inv), pack_bf16(f[6] * inv, f[7] * inv));
            }
        }
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0 && !abort_flag) {
        // O = Y R_h^T: B = R_h rows (output dim) x K-major columns
        if (mbar_wait(bar_r, 0, status, &abort_flag, 6)) {
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const uint32_t aoff = (kk >> 2) * 8192u + (kk & 3) * 32u;
                const uint32_t boff = (kk >> 2) * 16384u + (kk & 3) * 32u;
                mma_bf16(tmem, sdesc_sw128(sb + kOffQ + aoff, 16, 1024), sdesc_sw128(sb + kOffK + boff, 16, 1024),
                         kIdescO, kk > 0);
            }
            mma_commit(bar_o);
        }
    }
    if (warp < 2) {
        const bool ok = mbar_wait(bar_o, 0, status, &abort_flag, 7);
        tc_fence_after();
        __syncwarp();
        bf16 *orow = o + ((int64_t)l * q_rows + ep.q_row_begin + qb + tid) * d + (int64_t)h * kDh;
        uint32_t sr[32];
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            tmem_ld32(tm_lane(tmem, warp, 32 * q4), sr);
            tmem_wait_ld();
            if (ok && tid < nq) {
                uint4 *dst = reinterpret_cast<uint4 *>(orow + 32 * q4);
#pragma unroll
                for (int v4 = 0; v4 < 4; ++v4)
                    dst[v4] = make_uint4(pack_bf16(__uint_as_float(sr[8 * v4]), __uint_as_float(sr[8 * v4 + 1])),
                                         pack_bf16(__uint_as_float(sr[8 * v4 + 2]), __uint_as_float(sr[8 * v4 + 3])),
                                         pack_bf16(__uint_as_float(sr[8 * v4 + 4]), __uint_as_float(sr[8 * v4 + 5])),
                                         pack_bf16(__uint_as_float(sr[8 * v4 + 6]), __uint_as_float(sr[8 * v4 + 7])));
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

bool attend_tc_supported(const rolesub_shape *s)
{
    return s->dtype == ROLESUB_BF16 && s->head_dim == kDh && s->num_groups == kG;
}

cudaError_t launch_attend_tc(const AttendArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.max_query_tokens == 0 || P.num_episodes == 0) return cudaSuccess;
    const int H = S.num_heads, L = S.num_layers;
    CUtensorMap tq, tk, tr;
    {
        const uint64_t dims[4] = {(uint64_t)kDh, (uint64_t)H, (uint64_t)P.q_rows_per_layer, (uint64_t)L};
        const uint64_t str[3] = {(uint64_t)a.q_hs * 2, (uint64_t)a.q_rs * 2, (uint64_t)a.q_ls * 2};
        const uint32_t box[4] = {64, 1, (uint32_t)kQRows, 1};
        if (!make_bf16_map(&tq, a.q, 4, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[4] = {(uint64_t)kDh, (uint64_t)H, (uint64_t)P.rows_per_layer, (uint64_t)L};
        const uint64_t str[3] = {(uint64_t)a.k_hs * 2, (uint64_t)a.k_rs * 2, (uint64_t)a.k_ls * 2};
        const uint32_t box[4] = {64, 1, (uint32_t)kChunk, 1};
        if (!make_bf16_map(&tk, a.K, 4, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)kDh, (uint64_t)kDh, (uint64_t)L * H};
        const uint64_t str[2] = {(uint64_t)kDh * 2, (uint64_t)kDh * kDh * 2};
        const uint32_t box[3] = {64, (uint32_t)kDh, 1};
        if (!make_bf16_map(&tr, a.R, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    cudaError_t err = cudaFuncSetAttribute(k_attend_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (err != cudaSuccess) return err;
    const int qtiles = (P.max_query_tokens + kQRows - 1) / kQRows;
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev};
    const float scale = a.scale > 0.f ? a.scale : 1.0f / sqrtf((float)kDh);
    k_attend_tc<<<dim3(H, P.num_episodes * qtiles, L), kThreads, kSmemBytes, a.stream>>>(
        tq, tk, tr, (const bf16 *)a.packed, P.packed_elems_per_layer, a.idx, P.idx_bytes_per_layer, pd, H, qtiles,
        P.q_rows_per_layer, scale * 1.4426950408889634f, (bf16 *)a.o, a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
