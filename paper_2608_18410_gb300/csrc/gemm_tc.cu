// gemm_tc.cu -- the two rotations of the dense geometry (one d x d orthonormal
// R per layer, S = 16 contiguous groups of g = d / S rotated dims, Sec. 4.1)
// as bf16 GEMMs on the 5th-generation tensor core that touch only the kept
// groups (fp32 accumulation in TMEM, one rounding to bf16).
//
// Compress (z_s = R_s^T v for every kept (row, group s) pair, R_s the g
// columns of group s): the pairs of a 4096-row chunk are listed per group
// (dense.cu), so a 128-pair tile shares one group and is a plain GEMM
//   C[128 x g] = V[rows of the pairs] . R[:, s g : s g + g]
// with K = d. A is gathered row by row from V; B is R's column block (N
// contiguous in memory: MN-major) by TMA. The epilogue writes each pair's g
// values straight to its packed slot -- no [rows][d] z is ever stored.
//
// Attend (v~_j = R M_j z_j = sum over kept s of R_s z_{j,s}): rows are
// bucketed by their kept-group set (dense.cu), and a 128-row tile runs the
// K blocks of the union of its rows' groups only. A is gathered from the
// packed cache itself (each row's slot of group s; rows that did not keep s
// load nothing), and the MMA's disable-output-lane mask leaves the
// accumulator of those rows untouched, so no M z is ever scattered to
// memory. B is R's rows (K contiguous: K-major) by TMA. The accumulator is
// zeroed with tcgen05.st first.
//
// One CTA per tile, 192 threads: warps 0-3 set the tile up, gather A with
// 16-byte cp.async into the 128-byte-swizzled K-major layout (a TMA
// tile::gather4 per four rows ran at about a quarter of the MMA rate), and
// run the epilogue (a TMEM lane and a tile row per thread); warp 4 loads B by
// TMA; warp 5 issues the MMAs. K runs in 64-wide blocks through a 2-stage
// ring of 48 KB stages. The gatherers form one team per stage (warps 0-1 the
// even K blocks, warps 2-3 the odd ones); a team waits for its own copies,
// fences them to the tensor core's proxy and arrives, so both stages are in
// flight at once. Two CTAs share an SM (about 106 KB of shared memory and 256
// TMEM columns each), so that one CTA's set-up and epilogue overlap the
// other's main loop. The epilogue stages the bf16 tile in the drained ring
// and stores one tile row (up to 512 bytes) per warp instruction.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kGThreads = 192;
constexpr int kBM = 128, kBN = 256, kBK = 64;
constexpr int kGStages = 2;
constexpr int kMaxGroups = 16;
constexpr uint32_t kGTileA = kBM * kBK * 2;          // 16 KB
constexpr uint32_t kGTileB = kBN * kBK * 2;          // 32 KB
constexpr uint32_t kGStage = kGTileA + kGTileB;      // 48 KB
constexpr uint32_t kGOffBar = kGStages * kGStage;    // 96 KB
constexpr uint32_t kGOffTab = kGOffBar + 128;
// The gatherers are warps 0-3 as kGStages teams of 128 / kGStages threads;
// team q fills the stages kb with kb % kGStages == q, waits for its own
// copies and arrives at once, so every stage of the ring is in flight.
constexpr int kTeam = 128 / kGStages;                 // threads per gather team
constexpr int kRowsPerThread = kBM * 8 / kTeam;       // 16-byte chunks per thread and stage
constexpr uint32_t kFullCount = kTeam + 1;            // the team's threads + the B loader
static_assert(kRowsPerThread * kTeam == kBM * 8, "a team covers the A tile");
// attend: slot table [16][128] int32, the lane masks [16][4] uint32, kept
// groups per row [128] uint32; compress: A row per tile row [128] int32,
// then packed offsets [128] int64
constexpr uint32_t kGTabBytes = kMaxGroups * kBM * 4 + kMaxGroups * 4 * 4 + kBM * 4;
constexpr uint32_t kGSmem = kGOffTab + kGTabBytes + 1024;
constexpr uint32_t kGPitch = kBN * 2 + 16;           // staged C row: 512 B + 16 B pad
static_assert(kBM * kGPitch <= kGOffBar, "C staging fits the ring");
static_assert(kBM * 4 + kBM * 8 <= kGTabBytes, "compress tables fit");

// This thread's copies of the stage have landed: made visible to the tensor
// core's proxy, then the stage barrier arrives.
__device__ __forceinline__ void gather_done(uint32_t full)
{
    cp_async_wait_group<0>();
    fence_async_smem();
    mbar_arrive(full);
}

// D[tmem] += A . B^T on the lanes whose bit in dis[] is clear (bit i of
// dis[w] disables TMEM lane 32 w + i, i.e. tile row 32 w + i).
__device__ __forceinline__ void mma_bf16_masked(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                                uint32_t m0, uint32_t m1, uint32_t m2, uint32_t m3,
                                                uint32_t accumulate)
{
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %8, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, {%4, %5, %6, %7}, p;\n}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(m0), "r"(m1), "r"(m2), "r"(m3), "r"(accumulate)
        : "memory");
}

// The fp32 accumulator columns [0, ncols) of this thread's TMEM lane to bf16
// in the staging row srow.
__device__ __forceinline__ void stage_row(uint32_t lane_base, int ncols, uint8_t *srow)
{
#pragma unroll 1
    for (int c = 0; c < ncols / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(lane_base + 32u * c, r);
        tmem_wait_ld();
        uint4 *dst = reinterpret_cast<uint4 *>(srow + 64 * c);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            dst[q] = make_uint4(pack_bf16(__uint_as_float(r[8 * q]), __uint_as_float(r[8 * q + 1])),
                                pack_bf16(__uint_as_float(r[8 * q + 2]), __uint_as_float(r[8 * q + 3])),
                                pack_bf16(__uint_as_float(r[8 * q + 4]), __uint_as_float(r[8 * q + 5])),
                                pack_bf16(__uint_as_float(r[8 * q + 6]), __uint_as_float(r[8 * q + 7])));
    }
}

// ------------------------------------------------------------- compress
// grid (tile bound x N-tiles per pair tile, chunks, L). Tile t of chunk c
// belongs to the group s whose 128-pair tiles cover t (groups in order);
// CTAs past the chunk's last tile return at once.
__global__ void __launch_bounds__(kGThreads, 2)
k_dense_compress_tc(const __grid_constant__ CUtensorMap tm_r, const bf16 *__restrict__ v, DenseCompressGemm p)
{
    const int x = blockIdx.x, c = blockIdx.y, l = blockIdx.z;
    const int ntn = p.g / p.nt;
    const int t = x / ntn, jn = x % ntn;
    const int32_t *mt = p.meta + ((int64_t)l * p.chunks + c) * kDenseMetaStride;
    int s = -1, m = 0, cnt = 0, start = 0, poff = 0, pstart = 0;
    for (int q = 0; q < kMaxGroups; ++q) {
        const int n = mt[q], nt = (n + kBM - 1) / kBM;
        if (s < 0 && t < start + nt) {
            s = q;
            m = t - start;
            cnt = n;
            pstart = poff;
        }
        start += nt;
        poff += n;
    }
    if (s < 0) return;  // the same decision in every thread of the CTA

    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    int32_t *arow = reinterpret_cast<int32_t *>(sp + kGOffTab);
    int64_t *dsto = reinterpret_cast<int64_t *>(sp + kGOffTab + kBM * 4);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nkb = p.d / kBK, NT = p.nt;
    const int n0 = s * p.g + NT * jn;
    const int nvalid = min(kBM, cnt - kBM * m);
    const uint32_t bar_full = sb + kGOffBar, bar_empty = bar_full + 8 * kGStages, bar_acc = bar_empty + 8 * kGStages;

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < kGStages; ++i) {
            mbar_init(bar_full + 8 * i, kFullCount);
            mbar_init(bar_empty + 8 * i, 1);
        }
        mbar_init(bar_acc, 1);
        fence_mbar_init();
    }
    if (tid < kBM) {
        // this tile row's pair: its V row (layer-global) and packed offset
        const int2 *pl = p.pairs + (int64_t)l * p.pairs_per_layer + mt[kMaxGroups] + pstart + (int64_t)kBM * m;
        const int2 pr = pl[tid < nvalid ? tid : 0];
        arow[tid] = (int32_t)((int64_t)l * p.rows + pr.x);
        dsto[tid] = tid < nvalid ? (int64_t)l * p.packed_per_layer + (int64_t)pr.y * p.g + NT * jn : -1;
    }
    __syncthreads();
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp < 4) {
        // ------------------------------------- A gather, then the epilogue
        // thread: team q, the 16-byte column cc of rows rq + 8 i
        const int q = tid / kTeam, tt = tid % kTeam, cc = tt & 7, rq = tt >> 3;
        const bf16 *src[kRowsPerThread];
        uint32_t doff[kRowsPerThread], valid = 0;
#pragma unroll
        for (int i = 0; i < kRowsPerThread; ++i) {
            const int row = rq + (kTeam / 8) * i;
            src[i] = v + (int64_t)arow[row] * p.d + 8 * cc;
            doff[i] = (uint32_t)row * 128u + ((uint32_t)(cc ^ (row & 7)) << 4);
            if (row < nvalid) valid |= 1u << i;
        }
        for (int kb = q; kb < nkb; kb += kGStages) {
            if (kb >= kGStages &&
                !mbar_wait(bar_empty + 8 * q, ((kb / kGStages) - 1) & 1, p.status, &abort_flag, 95))
                break;
            const uint32_t st = sb + kGStage * q;
#pragma unroll
            for (int i = 0; i < kRowsPerThread; ++i)
                if ((valid >> i) & 1u) cp_async16(st + doff[i], src[i] + kBK * kb);
            cp_async_commit();
            gather_done(bar_full + 8 * q);
        }

        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
        const bool ok = mbar_wait(bar_acc, 0, p.status, &abort_flag, 97);
        tc_fence_after();
        __syncwarp();
        stage_row(lane_base, NT, sp + (uint32_t)tid * kGPitch);
        __syncwarp();
        // the warp's 32 rows, one row of NT values per instruction, each to
        // its pair's packed slot
        if (ok && !abort_flag && 8 * lane < NT) {
#pragma unroll 1
            for (int i = 0; i < 32; ++i) {
                const int row = 32 * warp + i;
                const int64_t o = dsto[row];
                if (o < 0) break;
                const uint4 val = *reinterpret_cast<const uint4 *>(sp + (uint32_t)row * kGPitch + 16u * lane);
                *reinterpret_cast<uint4 *>(p.packed + o + 8 * lane) = val;
            }
        }
    } else if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_r);
            const uint32_t bytes = (uint32_t)NT * kBK * 2;
            for (int kb = 0; kb < nkb; ++kb) {
                const int st_i = kb % kGStages;
                if (kb >= kGStages &&
                    !mbar_wait(bar_empty + 8 * st_i, ((kb / kGStages) - 1) & 1, p.status, &abort_flag, 98))
                    break;
                const uint32_t st = sb + kGStage * st_i, full = bar_full + 8 * st_i;
                mbar_expect_tx(full, bytes);
                // NT / 64 column blocks of 64 K rows each (8 KB apart)
                for (int nb = 0; nb < NT / 64; ++nb)
                    tma_load_3d(st + kGTileA + 8192u * nb, &tm_r, n0 + 64 * nb, kBK * kb, l, full);
            }
        }
    } else {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(kBM, NT, true);
            for (int kb = 0; kb < nkb; ++kb) {
                const int st_i = kb % kGStages;
                if (!mbar_wait(bar_full + 8 * st_i, (kb / kGStages) & 1, p.status, &abort_flag, 96)) break;
                tc_fence_after();
                const uint32_t st = sb + kGStage * st_i;
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t a = sdesc_sw128(st + 32u * kk, 16, 1024);
                    // MN-major B: +16 K rows (2 KB) per K16 step, 64-column blocks 8 KB apart
                    const uint64_t b = sdesc_sw128(st + kGTileA + 2048u * kk, 8192, 1024);
                    mma_bf16(tmem, a, b, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(bar_empty + 8 * st_i);
            }
            mma_commit(bar_acc);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

// --------------------------------------------------------------- attend
// grid (d / 256, ceil(rows / 128), L): output columns n0.., sorted rows m0..
__global__ void __launch_bounds__(kGThreads, 2)
k_dense_attend_tc(const __grid_constant__ CUtensorMap tm_r, const bf16 *__restrict__ packed, DenseAttendGemm p)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    int32_t *slot = reinterpret_cast<int32_t *>(sp + kGOffTab);                         // [16][128]
    uint32_t *dis = reinterpret_cast<uint32_t *>(sp + kGOffTab + kMaxGroups * kBM * 4);  // [16][4]
    uint32_t *keeps = dis + kMaxGroups * 4;                                              // [128]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n0 = blockIdx.x * kBN, m0 = blockIdx.y * kBM, l = blockIdx.z;
    const int G = p.G, g = p.g;
    const uint32_t bar_full = sb + kGOffBar, bar_empty = bar_full + 8 * kGStages, bar_acc = bar_empty + 8 * kGStages;

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < kGStages; ++i) {
            mbar_init(bar_full + 8 * i, kFullCount);
            mbar_init(bar_empty + 8 * i, 1);
        }
        mbar_init(bar_acc, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp < 4) {
        // tile row tid = sorted row m0 + tid: its slot of every kept group
        uint32_t keep = 0;
        const int64_t q = m0 + tid;
        if (q < p.rows) {
            const int r = p.perm[(int64_t)l * p.rows + q];
            const rolesub_segment sg = p.segs[p.row_seg[r]];
            const int k = sg.k;
            const int64_t i = r - sg.token_row;
            const int32_t base = (int32_t)((int64_t)l * p.slots_per_layer + sg.packed_off / g + i * k);
            const uint8_t *ix = p.idx + (int64_t)l * p.idx_per_layer + sg.idx_off + i * k;
            for (int j = 0; j < k; ++j) {
                const int grp = ix[j];
                if (grp >= G) {
                    report(p.status, ROLESUB_EDEVICE, r);
                    continue;
                }
                keep |= 1u << grp;
                slot[grp * kBM + tid] = base + j;
            }
        }
        keeps[tid] = keep;
        for (int s = 0; s < kMaxGroups; ++s) {
            const uint32_t b = __ballot_sync(0xffffffffu, (keep >> s) & 1u);
            if (lane == 0) dis[4 * s + warp] = ~b;
        }
        // zero this warp's 32 accumulator lanes: every MMA accumulates
        const uint32_t zero[32] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u,
                                   0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) tmem_st32(lane_base + 32u * c, zero);
        tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    // groups kept by at least one row of the tile, each g / 64 K blocks
    uint32_t un = 0;
    for (int s = 0; s < G; ++s)
        if ((dis[4 * s] & dis[4 * s + 1] & dis[4 * s + 2] & dis[4 * s + 3]) != 0xffffffffu) un |= 1u << s;
    const int kpg = g / kBK;
    const int nkb = __popc(un) * kpg;

    if (warp < 4) {
        // ------------------------------------- A gather, then the epilogue
        // thread: team q, the 16-byte column cc of rows rq + 8 i
        const int q = tid / kTeam, tt = tid % kTeam, cc = tt & 7, rq = tt >> 3;
        uint32_t kp[kRowsPerThread], doff[kRowsPerThread];
#pragma unroll
        for (int i = 0; i < kRowsPerThread; ++i) {
            const int row = rq + (kTeam / 8) * i;
            kp[i] = keeps[row];
            doff[i] = (uint32_t)row * 128u + ((uint32_t)(cc ^ (row & 7)) << 4);
        }
        uint32_t rest = un;
        int s = -1, sub = kpg;
        uint32_t on = 0;                  // rows of this thread that kept s
        const bf16 *src[kRowsPerThread];  // their slots of group s
        for (int kb = 0; kb < nkb; ++kb) {
            if (sub == kpg) {
                s = __ffs(rest) - 1;
                rest &= rest - 1;
                sub = 0;
                on = 0;
#pragma unroll
                for (int i = 0; i < kRowsPerThread; ++i) {
                    on |= ((kp[i] >> s) & 1u) << i;
                    src[i] = packed + (int64_t)slot[s * kBM + rq + (kTeam / 8) * i] * g + 8 * cc;
                }
            }
            if (kb % kGStages == q) {
                if (kb >= kGStages &&
                    !mbar_wait(bar_empty + 8 * q, ((kb / kGStages) - 1) & 1, p.status, &abort_flag, 99))
                    break;
                const uint32_t st = sb + kGStage * q;
                // rows that did not keep s load nothing: their lanes are masked
#pragma unroll
                for (int i = 0; i < kRowsPerThread; ++i)
                    if ((on >> i) & 1u) cp_async16(st + doff[i], src[i] + kBK * sub);
                cp_async_commit();
                gather_done(bar_full + 8 * q);
            }
            ++sub;
        }

        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
        const bool ok = mbar_wait(bar_acc, 0, p.status, &abort_flag, 100);
        tc_fence_after();
        __syncwarp();
        stage_row(lane_base, kBN, sp + (uint32_t)tid * kGPitch);
        __syncwarp();
        if (ok && !abort_flag) {
            bf16 *cbase = p.vt + (int64_t)l * p.rows * p.d + n0;
#pragma unroll 1
            for (int i = 0; i < 32; ++i) {
                const int row = 32 * warp + i;
                const int64_t q = m0 + row;
                if (q >= p.rows) break;
                const uint4 val = *reinterpret_cast<const uint4 *>(sp + (uint32_t)row * kGPitch + 16u * lane);
                *reinterpret_cast<uint4 *>(cbase + q * p.d + 8 * lane) = val;
            }
        }
    } else if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_r);
            uint32_t rest = un;
            int s = -1, sub = kpg;
            for (int kb = 0; kb < nkb; ++kb) {
                if (sub == kpg) {
                    s = __ffs(rest) - 1;
                    rest &= rest - 1;
                    sub = 0;
                }
                const int st_i = kb % kGStages;
                if (kb >= kGStages &&
                    !mbar_wait(bar_empty + 8 * st_i, ((kb / kGStages) - 1) & 1, p.status, &abort_flag, 101))
                    break;
                const uint32_t st = sb + kGStage * st_i, full = bar_full + 8 * st_i;
                mbar_expect_tx(full, kGTileB);
                tma_load_3d(st + kGTileA, &tm_r, s * g + kBK * sub, n0, l, full);
                ++sub;
            }
        }
    } else {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(kBM, kBN, false);
            uint32_t rest = un;
            int s = -1, sub = kpg;
            for (int kb = 0; kb < nkb; ++kb) {
                if (sub == kpg) {
                    s = __ffs(rest) - 1;
                    rest &= rest - 1;
                    sub = 0;
                }
                ++sub;
                const int st_i = kb % kGStages;
                if (!mbar_wait(bar_full + 8 * st_i, (kb / kGStages) & 1, p.status, &abort_flag, 102)) break;
                tc_fence_after();
                const uint32_t st = sb + kGStage * st_i;
                const uint32_t d0 = dis[4 * s], d1 = dis[4 * s + 1], d2 = dis[4 * s + 2], d3 = dis[4 * s + 3];
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t a = sdesc_sw128(st + 32u * kk, 16, 1024);
                    const uint64_t b = sdesc_sw128(st + kGTileA + 32u * kk, 16, 1024);
                    mma_bf16_masked(tmem, a, b, idesc, d0, d1, d2, d3, 1u);
                }
                mma_commit(bar_empty + 8 * st_i);
            }
            mma_commit(bar_acc);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

}  // namespace

cudaError_t launch_dense_compress_gemm(const DenseCompressGemm &p, const void *v, const void *R, int L,
                                       int tiles_per_chunk, cudaStream_t stream)
{
    if (L == 0 || p.chunks == 0 || tiles_per_chunk == 0) return cudaSuccess;
    if (p.d % kBK != 0 || p.g % p.nt != 0 || p.nt % 64 != 0 || p.nt > kBN) return cudaErrorInvalidValue;
    CUtensorMap tr;
    {
        // R [L][d (K)][d (N)], N contiguous: boxes of 64 N x 64 K
        const uint64_t dims[3] = {(uint64_t)p.d, (uint64_t)p.d, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)p.d * 2, (uint64_t)p.d * p.d * 2};
        const uint32_t box[3] = {64, kBK, 1};
        if (!make_bf16_map(&tr, R, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    cudaError_t err = cudaFuncSetAttribute(k_dense_compress_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kGSmem);
    if (err != cudaSuccess) return err;
    const dim3 grid((unsigned)(tiles_per_chunk * (p.g / p.nt)), (unsigned)p.chunks, (unsigned)L);
    k_dense_compress_tc<<<grid, kGThreads, kGSmem, stream>>>(tr, static_cast<const bf16 *>(v), p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_dense_attend_gemm(const DenseAttendGemm &p, const void *packed, const void *R, int L,
                                     cudaStream_t stream)
{
    if (L == 0 || p.rows == 0) return cudaSuccess;
    if (p.d % kBN != 0 || p.g % kBK != 0 || p.G > kMaxGroups) return cudaErrorInvalidValue;
    CUtensorMap tr;
    {
        // R [L][d (N)][d (K)], K contiguous: boxes of 64 K x 256 N
        const uint64_t dims[3] = {(uint64_t)p.d, (uint64_t)p.d, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)p.d * 2, (uint64_t)p.d * p.d * 2};
        const uint32_t box[3] = {kBK, kBN, 1};
        if (!make_bf16_map(&tr, R, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    cudaError_t err = cudaFuncSetAttribute(k_dense_attend_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kGSmem);
    if (err != cudaSuccess) return err;
    const dim3 grid((unsigned)(p.d / kBN), (unsigned)((p.rows + kBM - 1) / kBM), (unsigned)L);
    k_dense_attend_tc<<<grid, kGThreads, kGSmem, stream>>>(tr, static_cast<const bf16 *>(packed), p);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
