// attend_tc.cuh -- attention over the routed value cache on the 5th-generation
// tensor core (tcgen05 + TMA), bf16 inputs, fp32 accumulation.
//
// Work unit = (layer, head, episode, tile of 64 queries). A persistent CTA
// per SM walks a contiguous range of units (episode fastest), so R_h stays
// in shared memory while (layer, head) is unchanged.
//
// All products are M = 64 (the 64 query rows of a unit): their TMEM
// accumulators put rows 16q..16q+15 in lanes 32q..32q+15, so each of the
// four lane quadrants -- one per SM sub-partition -- holds 16 complete rows
// and one warp per quadrant does that quadrant's softmax with row maxima
// reduced by shuffles inside the warp (16x256b TMEM loads: thread t holds
// rows t/4 and t/4 + 8, column pairs 8j + 2(t%4)).
//
// Per chunk c of 64 cache tokens of a unit:
//   S_c = Q K_c^T                 tcgen05, M=64, N=64, K=128; K_c by TMA
//                                 straight from the caller's cache
//   softmax, exp2 domain:         P_c = exp(S_c - m) -> bf16 smem, with a
//                                 reference max m per row that is raised
//                                 (and the TMEM accumulator Y rescaled) only
//                                 when a chunk's row max exceeds it by more
//                                 than 2^8; Y and the row sum l always share
//                                 the same m, so y / l is exact
//   Z_c = the chunk's kept groups scattered by index into a zero-filled
//         64 x 128 MN-major tile. One group of d_s = 8 bf16 is one 16-byte
//         swizzle chunk, copied by cp.async from the packed cache straight
//         to its slot; per-row records (kept ids, packed offset) are loaded
//         into registers two chunks ahead.
//   Y += P_c Z_c                   tcgen05, M=64, N=128 (rotated space)
// Unit tail: Y / l -> bf16 smem (a staging tile of its own, so that a Q
// slot is free as soon as its unit's last S is issued),
// O = Y R_h^T (o_q = R_h y_q, Sec. 3.2) into the unit's Y buffer; O as
// bf16 back into the (now free) staging tile, each tail warp its own 16
// rows, then read back and stored 16 bytes per lane, two full rows per warp
// instruction.
//
// Warp roles (544 threads), all hand-offs through mbarriers. Warp w runs on
// sub-partition w % 4.
//   warps 0-3   softmax, one per TMEM lane quadrant
//   warps 4-5, 12-13  value gather, one kv row per thread: warps 4-5 the
//               even chunks, warps 12-13 the odd ones (budget caches: 608
//               threads, warps 17-18 a third gatherer, chunks g % 3)
//   warp 6      issues S = Q K^T, chunk by chunk
//   warp 14     issues Y += P Z, chunk by chunk
//   warp 15     issues O = Y R_h^T, unit by unit
//   warp 7      TMA producer of K (3-slot ring), chunk by chunk
//   warp 16     TMA producer of Q (2 slots) and R_h, unit by unit (apart
//               from the K producer, so that neither's waits hold up the other)
//   warps 8-11  unit tail, one per lane quadrant, overlapping the next
//               unit's chunks (Y is double buffered in TMEM)
// S and P have three buffers and Z four slots: a chunk's S product waits for
// the softmax three chunks back, its softmax for the P.Z product three chunks
// back, its gatherer for the one four chunks back, and a gatherer publishes a
// chunk when it starts its next one.
//
// Shared memory (1024-aligned):
//   0K   Q[2]   16K each (two 64-column K-blocks of 64 rows)
//   32K  K[3]   16K each (64-row chunks)
//   80K  Y      16K, Y / l of the unit in its tail (A of the output product)
//   96K  R_h    32K (two 64-column K-blocks of 128 rows)
//   128K P[3]   8K each (64 rows x 64 kv)
//   152K Z[4]   16K each (two 64-column MN-blocks of 64 kv rows)
//   216K row sums 2 x 64 fp32 (softmax -> unit tail)
//   217K the unit list (up to 512 units per CTA and launch), the barriers
// TMEM (448 of 512 columns): S[3] at 0, 64 and 128, Y[2] at 192 and 320
// (each later holding its unit's O).
#pragma once

#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 544;
constexpr int kThreadsBudget = 608;   // budget caches: a third gatherer (warps 17-18)
constexpr int kChunk = 64;   // cache tokens per chunk
constexpr int kQRows = 64;   // query rows per unit
constexpr int kDh = 128;
constexpr int kG = 16;       // groups per head (d_s = 8)
constexpr int kMaxUnits = 512;   // units per CTA and launch (unit list in smem)
constexpr int kKSlots = 3;
constexpr float kRescaleLog2 = 8.f;   // raise the reference max beyond 2^8 growth

constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = 32768;
constexpr uint32_t kOffY = kOffK + kKSlots * 16384;   // normalised Y of the unit in its tail
constexpr uint32_t kOffR = 98304;
constexpr int kSBufs = 3;                             // S (TMEM) and P (smem) buffers
constexpr uint32_t kOffP = 131072;                    // 3 x 8K
constexpr uint32_t kOffZ = kOffP + kSBufs * 8192;     // 4 x 16K ring
constexpr int kZSlots = 4;
constexpr uint32_t kOffL = kOffZ + kZSlots * 16384;   // 2 x 64 fp32 row sums
constexpr uint32_t kOffUnits = kOffL + 1024;         // kMaxUnits x 16 B unit records
constexpr uint32_t kOffBar = kOffUnits + 16 * kMaxUnits;
constexpr uint32_t kSmemBytes = kOffBar + 512 + 1024;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0, kColY = 192;   // S[b] at 64b, Y[b] at kColY + 128b

constexpr uint32_t kIdescS = idesc_bf16(64, 64, false);
constexpr uint32_t kIdescPV = idesc_bf16(64, 128, true);
constexpr uint32_t kIdescO = idesc_bf16(64, 128, false);

// barrier slots (8 bytes each); [2] / [4] entries are per buffer
enum {
    B_QF = 0, B_QE = 2, B_KF = 4, B_KE = 8, B_RF = 12, B_RE = 13, B_SF = 14, B_PF = 17, B_ZF = 20, B_PV = 24,
    B_YR = 28, B_YF = 30, B_OF = 31, B_OE = 32, B_LF = 34, B_COUNT = 36
};

struct Unit {
    int l, h, nq, nc, nch, krow, qrow;
};

// A CTA's units with queries and cache tokens, in processing order, as
// 16-byte records {first cache row, first query row, n_cache,
// n_q | h << 8 | l << 18} built once at kernel start; every role walks the
// same list.
__device__ __forceinline__ Unit load_unit(const uint8_t *sp, int k)
{
    const uint4 v = *reinterpret_cast<const uint4 *>(sp + kOffUnits + 16u * (uint32_t)k);
    Unit t;
    t.krow = (int)v.x;
    t.qrow = (int)v.y;
    t.nc = (int)v.z;
    t.nch = (t.nc + kChunk - 1) / kChunk;
    t.nq = (int)(v.w & 255u);
    t.h = (int)((v.w >> 8) & 1023u);
    t.l = (int)(v.w >> 18);
    return t;
}

// Iterator over the units of the list and the chunks of each unit.
struct ChunkIt {
    int k, c;   // unit (nu = done), chunk within unit
    Unit t;
};

__device__ __forceinline__ void it_first(const uint8_t *sp, ChunkIt &it, int nu)
{
    it.k = 0;
    it.c = 0;
    if (nu > 0) it.t = load_unit(sp, 0);
}

// advances one chunk; returns true when it moved to another unit
__device__ __forceinline__ bool it_next(const uint8_t *sp, ChunkIt &it, int nu)
{
    if (it.k >= nu) return false;
    if (++it.c < it.t.nch) return false;
    it.c = 0;
    if (++it.k < nu) it.t = load_unit(sp, it.k);
    return true;
}

__device__ __forceinline__ void next_unit(const uint8_t *sp, ChunkIt &it, int nu)
{
    it.c = 0;
    if (++it.k < nu) it.t = load_unit(sp, it.k);
}

__device__ __forceinline__ float quad_sum(float v)
{
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

__device__ __forceinline__ float quad_max(float v)
{
    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
    return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}

template <bool kBudget>
__global__ void __launch_bounds__(kBudget ? kThreadsBudget : kThreads, 1)
k_attend_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
            const __grid_constant__ CUtensorMap tm_r, const bf16 *__restrict__ packed,
            int64_t packed_per_layer, const uint4 *rec, int64_t rows,
            const rolesub_episode *__restrict__ eps, int E, int H, int qtiles, int64_t u0, int64_t u1, int64_t q_rows,
            float scale_log2, bf16 *__restrict__ o, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t d = (int64_t)H * kDh;

    // ---- this CTA's share of units [u0, u1) -------------------------------
    const int64_t span = u1 - u0;
    const int64_t ub = u0 + span * blockIdx.x / gridDim.x;
    const int cnt = (int)(u0 + span * (blockIdx.x + 1) / gridDim.x - ub);   // <= kMaxUnits
    const uint32_t bar = sb + kOffBar;
    auto B = [&](int i) { return bar + 8u * (uint32_t)i; };
    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < B_COUNT; ++i) {
            uint32_t cnt = 1;
            if ((i >= B_PF && i < B_PF + kSBufs) || i == B_YF || i == B_OE || i == B_OE + 1 || i == B_LF ||
                i == B_LF + 1)
                cnt = 128;
            if (i >= B_ZF && i < B_ZF + kZSlots) cnt = 64;
            mbar_init(B(i), cnt);
        }
        fence_mbar_init();
    }
    __syncthreads();

    // unit list: units with queries and cache tokens, in order; units with
    // queries but no cache tokens get o = 0 here
    constexpr int kNT = kBudget ? kThreadsBudget : kThreads;
    __shared__ int warp_cnt[kNT / 32];
    int nu = 0;
    for (int base = 0; base < cnt; base += kNT) {
        const int i = base + tid;
        bool keep = false;
        uint4 rec4 = make_uint4(0, 0, 0, 0);
        if (i < cnt) {
            const int64_t u = ub + i;
            const int qt = (int)(u % qtiles);
            int64_t r = u / qtiles;
            const int e = (int)(r % E);
            r /= E;
            const int h = (int)(r % H), l = (int)(r / H);
            const rolesub_episode ep = eps[e];
            const int nq = max(0, min(kQRows, ep.n_query - qt * kQRows));
            const int qrow = (int)ep.q_row_begin + qt * kQRows;
            keep = nq > 0 && ep.n_cache > 0;
            rec4 = make_uint4((uint32_t)ep.row_begin, (uint32_t)qrow, (uint32_t)ep.n_cache,
                              (uint32_t)nq | ((uint32_t)h << 8) | ((uint32_t)l << 18));
            if (nq > 0 && ep.n_cache == 0)
                for (int j = 0; j < nq * (kDh / 8); ++j) {
                    uint4 *dst = reinterpret_cast<uint4 *>(o + ((int64_t)l * q_rows + qrow + j / (kDh / 8)) * d +
                                                           (int64_t)h * kDh) + j % (kDh / 8);
                    *dst = make_uint4(0, 0, 0, 0);
                }
        }
        const uint32_t bal = __ballot_sync(0xffffffffu, keep);
        if (lane == 0) warp_cnt[warp] = __popc(bal);
        __syncthreads();
        int off = nu, tot = 0;
        for (int w = 0; w < kNT / 32; ++w) {
            off += w < warp ? warp_cnt[w] : 0;
            tot += warp_cnt[w];
        }
        if (keep)
            *reinterpret_cast<uint4 *>(sp + kOffUnits + 16u * (uint32_t)(off + __popc(bal & ((1u << lane) - 1u)))) = rec4;
        nu += tot;
        __syncthreads();
    }
    if (nu == 0) return;   // uniform across the CTA
    ChunkIt first;
    it_first(sp, first, nu);

    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 7) {
        // ================= TMA producer: keys =============================
        if (lane == 0) {
            prefetch_tmap(&tm_q);
            prefetch_tmap(&tm_k);
            prefetch_tmap(&tm_r);
            ChunkIt it = first;
            uint32_t g = 0;
            auto load_k = [&](const Unit &t, int c) -> bool {
                const uint32_t ks = g % kKSlots;
                if (g >= kKSlots && !mbar_wait(B(B_KE + ks), ((g / kKSlots) - 1) & 1, status, &abort_flag, 41))
                    return false;
                const uint32_t dst = sb + kOffK + 16384 * ks;
                mbar_expect_tx(B(B_KF + ks), 16384);
                tma_load_4d(dst, &tm_k, 0, t.h, t.krow + kChunk * c, t.l, B(B_KF + ks));
                tma_load_4d(dst + 8192, &tm_k, 64, t.h, t.krow + kChunk * c, t.l, B(B_KF + ks));
                ++g;
                return true;
            };
            while (it.k < nu) {
                if (!load_k(it.t, it.c)) break;
                it_next(sp, it, nu);
            }
        }
    } else if (warp == 16) {
        // ================= TMA producer: Q and R_h ======================
        // Q of unit n waits for its slot (unit n - 2's last S product); R_h
        // of a new (layer, head) for the previous run's last output product
        if (lane == 0) {
            ChunkIt it = first;
            uint32_t n = 0;
            int run = -1, pl = -1, ph = -1;
            while (it.k < nu) {
                const Unit t = it.t;
                const uint32_t qs = n & 1;
                if (n >= 2 && !mbar_wait(B(B_QE + qs), ((n >> 1) - 1) & 1, status, &abort_flag, 40)) break;
                mbar_expect_tx(B(B_QF + qs), 16384);
                tma_load_4d(sb + kOffQ + 16384 * qs, &tm_q, 0, t.h, t.qrow, t.l, B(B_QF + qs));
                tma_load_4d(sb + kOffQ + 16384 * qs + 8192, &tm_q, 64, t.h, t.qrow, t.l, B(B_QF + qs));
                if (t.l != pl || t.h != ph) {
                    ++run;
                    if (run >= 1 && !mbar_wait(B(B_RE), (run - 1) & 1, status, &abort_flag, 42)) break;
                    mbar_expect_tx(B(B_RF), 32768);
                    tma_load_3d(sb + kOffR, &tm_r, 0, 0, t.l * H + t.h, B(B_RF));
                    tma_load_3d(sb + kOffR + 16384, &tm_r, 64, 0, t.l * H + t.h, B(B_RF));
                    pl = t.l;
                    ph = t.h;
                }
                next_unit(sp, it, nu);
                ++n;
            }
        }
    } else if (warp == 6 || warp == 14 || warp == 15) {
        // ================= MMA issuers =====================================
        // Three threads in three warps, one per product, each walking its
        // chunks or units in order with blocking waits; the tensor pipe
        // interleaves what they issue. tcgen05.mma issue stalls while the
        // pipe is busy, so the work between products is kept minimal: every
        // shared-memory descriptor is a base plus a constant (offset / 16 in
        // the start address field, which cannot carry out of its 14 bits
        // below 256 KB). A commit tracks the issuing thread's own products.
        if (lane == 0 && warp == 6) {
            // S_g = Q K_g^T into S buffer g % 3
            const uint64_t dq = sdesc_sw128(sb + kOffQ, 16, 1024), dk = sdesc_sw128(sb + kOffK, 16, 1024);
            ChunkIt cs = first;
            uint32_t gs = 0, ns = 0;   // chunk counter, unit counter
            while (cs.k < nu) {
                const uint32_t ks = gs % kKSlots;
                // S buffer gs % 3 was read by the softmax of chunk gs - 3
                const uint32_t sbuf = gs % kSBufs;
                if (gs >= kSBufs && !mbar_wait(B(B_PF + sbuf), ((gs / kSBufs) - 1) & 1, status, &abort_flag, 50))
                    break;
                if (cs.c == 0 && !mbar_wait(B(B_QF + (ns & 1)), (ns >> 1) & 1, status, &abort_flag, 51)) break;
                if (!mbar_wait(B(B_KF + ks), (gs / kKSlots) & 1, status, &abort_flag, 52)) break;
                tc_fence_after();
                const uint64_t qd = dq + 1024u * (ns & 1), kd = dk + 1024u * ks;
                const uint32_t sc = tmem + kColS + 64u * sbuf;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t o16 = (kk >> 2) * 512u + (kk & 3) * 2u;   // (kk/4) * 8K + (kk%4) * 32 bytes
                    mma_bf16(sc, qd + o16, kd + o16, kIdescS, kk > 0);
                }
                mma_commit(B(B_SF + sbuf));
                mma_commit(B(B_KE + ks));
                if (it_next(sp, cs, nu)) {
                    mma_commit(B(B_QE + (ns & 1)));   // the unit's last S: its Q slot is free
                    ++ns;
                }
                ++gs;
            }
        } else if (lane == 0 && warp == 14) {
            // Y += P_g Z_g; a unit's first product starts its Y buffer afresh,
            // once the unit two back has had its output read from it
            const uint64_t dp = sdesc_sw128(sb + kOffP, 16, 1024), dz = sdesc_sw128(sb + kOffZ, 8192, 1024);
            ChunkIt cp = first;
            uint32_t gp = 0, np = 0;
            while (cp.k < nu) {
                const uint32_t yb = np & 1, b = gp % kSBufs, zs = gp & 3;
                if (cp.c == 0 && np >= 2 && !mbar_wait(B(B_OE + yb), ((np - 2) >> 1) & 1, status, &abort_flag, 53))
                    break;
                if (!mbar_wait(B(B_PF + b), (gp / kSBufs) & 1, status, &abort_flag, 54)) break;
                if (!mbar_wait(B(B_ZF + zs), (gp >> 2) & 1, status, &abort_flag, 55)) break;
                tc_fence_after();
                const uint64_t pd = dp + 512u * b, zd = dz + 1024u * zs;
                const uint32_t yc = tmem + kColY + 128u * yb;
                mma_bf16(yc, pd, zd, kIdescPV, cp.c > 0 ? 1u : 0u);
#pragma unroll
                for (int kk = 1; kk < 4; ++kk)   // P: +32 bytes, Z: +16 kv rows (2 KB) per step
                    mma_bf16(yc, pd + 2u * kk, zd + 128u * kk, kIdescPV, 1u);
                mma_commit(B(B_PV + zs));
                if (it_next(sp, cp, nu)) {
                    mma_commit(B(B_YR + yb));   // the unit's Y is complete
                    ++np;
                }
                ++gp;
            }
        } else if (lane == 0) {
            // O = Y R_h^T of each unit, from its normalised Y in shared memory,
            // written over that unit's Y buffer
            const uint64_t dr = sdesc_sw128(sb + kOffR, 16, 1024), yd = sdesc_sw128(sb + kOffY, 16, 1024);
            ChunkIt co = first;
            uint32_t no = 0;
            int run_o = 0;
            while (co.k < nu) {
                if (!mbar_wait(B(B_YF), no & 1, status, &abort_flag, 56)) break;
                if (!mbar_wait(B(B_RF), run_o & 1, status, &abort_flag, 57)) break;
                tc_fence_after();
                const uint32_t oc = tmem + kColY + 128u * (no & 1);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t a16 = (kk >> 2) * 512u + (kk & 3) * 2u;    // Y: 8K K-blocks
                    const uint32_t b16 = (kk >> 2) * 1024u + (kk & 3) * 2u;   // R_h: 16K K-blocks
                    mma_bf16(oc, yd + a16, dr + b16, kIdescO, kk > 0);
                }
                mma_commit(B(B_OF));
                ChunkIt nx = co;
                next_unit(sp, nx, nu);
                if (nx.k >= nu || nx.t.l != co.t.l || nx.t.h != co.t.h) {
                    mma_commit(B(B_RE));
                    ++run_o;
                }
                co = nx;
                ++no;
            }
        }
    } else if (kBudget && (warp == 4 || warp == 5 || warp == 12 || warp == 13 || warp == 17 || warp == 18)) {
        // ================= value gather of a budget cache =================
        // Per-token counts K_i differ within a chunk, so a thread that owns
        // a row would hold its warp for the largest K_i; instead every row
        // is written whole (its K_i kept groups copied, the other 16 - K_i
        // zeroed: 16 stores per row whatever K_i) and three gatherers of 64
        // threads (warps 4-5, 12-13, 17-18) take the chunks g % 3. A gatherer
        // publishes a chunk as soon as its own copies have landed, so up to
        // three chunks are in flight; Z slot g % 4 is reused once the product
        // of chunk g - 4 has read it.
        constexpr int kGath = 3;
        const int gi = (warp == 4 || warp == 5) ? 0 : (warp == 12 || warp == 13) ? 1 : 2;
        const int jl = ((warp == 5 || warp == 13 || warp == 18) ? 32 : 0) + lane;
        const uint32_t sw = (uint32_t)(jl & 7);
        pdl_wait();   // the row records come from the kernel before this one
        ChunkIt it = first;
        for (int i = 0; i < gi; ++i) it_next(sp, it, nu);
        uint32_t g = (uint32_t)gi;
        ChunkIt ahead = it;
        uint4 mnext = make_uint4(0, 0, 0, 0);
        auto fetch_rec = [&]() {   // record of chunk `ahead`, then ahead += 3
            mnext = make_uint4(0, 0, 0, 0);
            if (ahead.k < nu) {
                const int r = ahead.c * kChunk + jl;
                if (r < ahead.t.nc) mnext = ld_dep(rec + (int64_t)ahead.t.l * rows + ahead.t.krow + r);
            }
            for (int i = 0; i < kGath; ++i) it_next(sp, ahead, nu);
        };
        fetch_rec();
        for (; it.k < nu && !abort_flag; g += kGath) {
            const uint4 m = mnext;
            fetch_rec();
            if (g >= 4 && !mbar_wait(B(B_PV + (g & 3u)), ((g - 4) >> 2) & 1, status, &abort_flag, 61)) break;
            const int nk = min(kChunk, it.t.nc - it.c * kChunk);
            uint32_t kept = 0;
            const uint32_t zrow = sb + kOffZ + 16384u * (g & 3u) + (uint32_t)jl * 128u;
            if (jl < nk) {
                const int k = (int)(m.w >> 27);
                const uint64_t gid = (uint64_t)m.x | ((uint64_t)m.y << 32);
                const bf16 *src = packed + (int64_t)it.t.l * packed_per_layer +
                                  ((int64_t)m.z + (int64_t)it.t.h * (int64_t)(m.w & 0x7FFFFFFu)) * 8;
                for (int s = 0; s < k; ++s) {
                    const uint32_t gg = (uint32_t)(gid >> (4 * s)) & 15u;
                    kept |= 1u << gg;
                    cp_async16(zrow + (gg >> 3) * 8192u + (((gg & 7u) ^ sw) << 4), src + 8 * s);
                }
            }
            for (uint32_t zm = 0xFFFFu & ~kept; zm; zm &= zm - 1) {
                const uint32_t gg = (uint32_t)(__ffs(zm) - 1);
                st_shared_v4(zrow + (gg >> 3) * 8192u + (((gg & 7u) ^ sw) << 4), 0, 0, 0, 0);
            }
            cp_async_commit();
            cp_async_wait_group<0>();
            fence_async_smem();
            mbar_arrive(B(B_ZF + (g & 3u)));
            for (int i = 0; i < kGath; ++i) it_next(sp, it, nu);
        }
    } else if (!kBudget && (warp == 4 || warp == 5 || warp == 12 || warp == 13)) {
        // ================= value gather (one kv row per thread) ===========
        // Two gatherers of 64 threads (warps 4-5 and 12-13) take the even and
        // the odd chunks. Chunk g goes to Z slot g % 4; its row record is
        // loaded into registers one own chunk (two chunks) ahead. At chunk g
        // a gatherer publishes its previous chunk g - 2 (copies complete),
        // waits for the product of chunk g - 4 to free the slot, copies the
        // kept groups of chunk g by cp.async straight into their swizzled
        // slots of the tile and zeroes the groups left over from the slot's
        // previous chunk.
        const int par = (warp == 4 || warp == 5) ? 0 : 1;
        const int jl = ((warp & 1) ? 32 : 0) + lane;
        const uint32_t sw = (uint32_t)(jl & 7);
        // groups of this thread's row that may be non-zero, per Z slot (16 bits
        // each); a slot's first use clears everything
        uint64_t dirty = ~0ull;
        pdl_wait();   // the row records come from the kernel before this one
        ChunkIt it = first;
        uint32_t g = (uint32_t)par;
        if (par) it_next(sp, it, nu);
        ChunkIt ahead = it;
        uint4 mnext = make_uint4(0, 0, 0, 0);
        auto fetch_rec = [&]() {   // record of chunk `ahead`, then ahead += 2
            mnext = make_uint4(0, 0, 0, 0);
            if (ahead.k < nu) {
                const int r = ahead.c * kChunk + jl;
                if (r < ahead.t.nc) mnext = ld_dep(rec + (int64_t)ahead.t.l * rows + ahead.t.krow + r);
            }
            it_next(sp, ahead, nu);
            it_next(sp, ahead, nu);
        };
        fetch_rec();
        for (; it.k < nu && !abort_flag; g += 2) {
            const uint4 m = mnext;
            fetch_rec();
            cp_async_wait_group<0>();   // the copies of chunk g - 2 have landed
            if (g >= 2) {
                fence_async_smem();
                mbar_arrive(B(B_ZF + ((g - 2) & 3u)));
            }
            // Z slot g % 4 was last read by the product of chunk g - 4
            if (g >= 4) mbar_wait(B(B_PV + (g & 3u)), ((g - 4) >> 2) & 1, status, &abort_flag, 60);
            const int nk = min(kChunk, it.t.nc - it.c * kChunk);
            uint32_t kept = 0;
            const uint32_t zrow = sb + kOffZ + 16384u * (g & 3u) + (uint32_t)jl * 128u;
            if (jl < nk) {
                const int k = (int)(m.w >> 27);
                const uint64_t gid = (uint64_t)m.x | ((uint64_t)m.y << 32);
                const bf16 *src = packed + (int64_t)it.t.l * packed_per_layer +
                                  ((int64_t)m.z + (int64_t)it.t.h * (int64_t)(m.w & 0x7FFFFFFu)) * 8;
                for (int s = 0; s < k; ++s) {
                    const uint32_t gg = (uint32_t)(gid >> (4 * s)) & 15u;
                    kept |= 1u << gg;
                    cp_async16(zrow + (gg >> 3) * 8192u + (((gg & 7u) ^ sw) << 4), src + 8 * s);
                }
            }
            const uint32_t sh = 16u * (g & 3u);
            for (uint32_t zm = (uint32_t)(dirty >> sh) & 0xFFFFu & ~kept; zm; zm &= zm - 1) {
                const uint32_t gg = (uint32_t)(__ffs(zm) - 1);
                st_shared_v4(zrow + (gg >> 3) * 8192u + (((gg & 7u) ^ sw) << 4), 0, 0, 0, 0);
            }
            dirty = (dirty & ~(0xFFFFull << sh)) | ((uint64_t)kept << sh);
            cp_async_commit();
            it_next(sp, it, nu);
            it_next(sp, it, nu);
        }
        cp_async_wait_group<0>();
        fence_async_smem();
        if (g >= 2 + (uint32_t)par) mbar_arrive(B(B_ZF + ((g - 2) & 3u)));
    } else if (warp < 4) {
        // ================= softmax (warps 0-3) ============================
        // rows ra = 16w + lane/4 and rb = ra + 8 of the unit; column pairs
        // 8j + 2(lane%4) + {0,1}
        const int cq = lane & 3;
        const int ra = 16 * warp + (lane >> 2), rb = ra + 8;
        const uint32_t lbase = tmem + ((uint32_t)(32 * warp) << 16);
        ChunkIt it = first;
        uint32_t n = 0, g = 0;
        while (it.k < nu && !abort_flag) {
            const Unit t = it.t;
            const uint32_t ycol = kColY + 128u * (n & 1);
            float ma = -INFINITY, mb = -INFINITY;   // reference maxima (exp2 domain)
            float la = 0.f, lb = 0.f;               // this thread's share of the row sums
            for (int c = 0; c < t.nch; ++c, ++g) {
                const int nk = min(kChunk, t.nc - c * kChunk);
                const uint32_t sbuf = g % kSBufs;
                mbar_wait(B(B_SF + sbuf), (g / kSBufs) & 1, status, &abort_flag, 70);
                tc_fence_after();
                __syncwarp();
                uint32_t sr[32];
                tmem_ld16x256_x8(lbase + kColS + 64u * sbuf, sr);
                tmem_wait_ld();
                if (nk < kChunk) {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
#pragma unroll
                        for (int e = 0; e < 2; ++e)
                            if (8 * j + 2 * cq + e >= nk) {
                                sr[4 * j + e] = __float_as_uint(-INFINITY);
                                sr[4 * j + 2 + e] = __float_as_uint(-INFINITY);
                            }
                }
                float xa = -INFINITY, xb = -INFINITY;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    xa = fmaxf(xa, fmaxf(__uint_as_float(sr[4 * j]), __uint_as_float(sr[4 * j + 1])));
                    xb = fmaxf(xb, fmaxf(__uint_as_float(sr[4 * j + 2]), __uint_as_float(sr[4 * j + 3])));
                }
                xa = quad_max(xa) * scale_log2;
                xb = quad_max(xb) * scale_log2;
                // raise the reference max (first chunk, or growth beyond 2^8)
                const bool raise_a = c == 0 || xa > ma + kRescaleLog2;
                const bool raise_b = c == 0 || xb > mb + kRescaleLog2;
                const float na = raise_a ? xa : ma, nb = raise_b ? xb : mb;
                if (c > 0 && __any_sync(0xffffffffu, raise_a || raise_b)) {
                    const float alpha_a = ex2(ma - na), alpha_b = ex2(mb - nb);
                    // Y holds chunks up to c-1: wait for the last of them, then rescale
                    mbar_wait(B(B_PV + ((g - 1) & 3u)), ((g - 1) >> 2) & 1, status, &abort_flag, 71);
                    tc_fence_after();
                    __syncwarp();
                    uint32_t yr[32];
#pragma unroll 1
                    for (int h2 = 0; h2 < 2; ++h2) {
                        const uint32_t ya = lbase + ycol + 64u * h2;
                        tmem_ld16x256_x8(ya, yr);
                        tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            yr[4 * j] = __float_as_uint(__uint_as_float(yr[4 * j]) * alpha_a);
                            yr[4 * j + 1] = __float_as_uint(__uint_as_float(yr[4 * j + 1]) * alpha_a);
                            yr[4 * j + 2] = __float_as_uint(__uint_as_float(yr[4 * j + 2]) * alpha_b);
                            yr[4 * j + 3] = __float_as_uint(__uint_as_float(yr[4 * j + 3]) * alpha_b);
                        }
                        tmem_st16x256_x8(ya, yr);
                    }
                    tmem_wait_st();
                    la *= alpha_a;
                    lb *= alpha_b;
                }
                ma = na;
                mb = nb;
                uint32_t pa[8], pb[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {   // p = 2^(s * scale - m); masked -inf -> 0
                    const float a0 = ex2(fmaf(__uint_as_float(sr[4 * j]), scale_log2, -ma));
                    const float a1 = ex2(fmaf(__uint_as_float(sr[4 * j + 1]), scale_log2, -ma));
                    const float b0 = ex2(fmaf(__uint_as_float(sr[4 * j + 2]), scale_log2, -mb));
                    const float b1 = ex2(fmaf(__uint_as_float(sr[4 * j + 3]), scale_log2, -mb));
                    la += a0 + a1;
                    lb += b0 + b1;
                    pa[j] = pack_bf16(a0, a1);
                    pb[j] = pack_bf16(b0, b1);
                }
                // P buffer g % 3 was last read by the product of chunk g - 3
                if (g >= (uint32_t)kSBufs) {
                    mbar_wait(B(B_PV + ((g - kSBufs) & 3u)), ((g - kSBufs) >> 2) & 1, status, &abort_flag, 72);
                    tc_fence_after();
                }
                // 8x8 blocks (rows of ra / rb, 8 columns = one swizzle chunk each):
                // lane t addresses row t%8 of block t/8
                const uint32_t prow = sb + kOffP + 8192u * sbuf + (uint32_t)(16 * warp + (lane & 7)) * 128u;
                const uint32_t c0 = ((uint32_t)(lane >> 3) ^ (uint32_t)(lane & 7)) << 4;
                const uint32_t c1 = ((uint32_t)((lane >> 3) + 4) ^ (uint32_t)(lane & 7)) << 4;
                stmatrix_x4(prow + c0, pa[0], pa[1], pa[2], pa[3]);
                stmatrix_x4(prow + c1, pa[4], pa[5], pa[6], pa[7]);
                stmatrix_x4(prow + 1024u + c0, pb[0], pb[1], pb[2], pb[3]);
                stmatrix_x4(prow + 1024u + c1, pb[4], pb[5], pb[6], pb[7]);
                fence_async_smem();
                tc_fence_before();
                mbar_arrive(B(B_PF + sbuf));
            }
            // row sums to the unit tail; buffer n & 1 was last read by the tail
            // of unit n - 2 before it released that unit's output
            const float lta = quad_sum(la), ltb = quad_sum(lb);
            if (n >= 2) mbar_wait(B(B_OE + (n & 1)), ((n - 2) >> 1) & 1, status, &abort_flag, 75);
            if (cq == 0) {
                float *lbuf = reinterpret_cast<float *>(sp + kOffL) + 64 * (n & 1);
                lbuf[ra] = lta;
                lbuf[rb] = ltb;
            }
            mbar_arrive(B(B_LF + (n & 1)));
            next_unit(sp, it, nu);
            ++n;
        }
    } else if (warp >= 8 && warp < 12) {
        // ================= unit tail (warps 8-11) =========================
        // y / l -> bf16 operand in the staging tile; after O = Y R_h^T, the
        // output rows through the same tile. Lane quadrant w = warp % 4, same
        // row mapping as softmax.
        const int w = warp & 3;
        const int ra = 16 * w + (lane >> 2), rb = ra + 8;
        const uint32_t lbase = tmem + ((uint32_t)(32 * w) << 16);
        ChunkIt it = first;
        uint32_t n = 0;
        while (it.k < nu) {
            const Unit t = it.t;
            const uint32_t yb = n & 1, ycol = kColY + 128u * yb;
            mbar_wait(B(B_LF + yb), (n >> 1) & 1, status, &abort_flag, 76);
            const float *lbuf = reinterpret_cast<const float *>(sp + kOffL) + 64 * yb;
            const float lta = lbuf[ra], ltb = lbuf[rb];
            mbar_wait(B(B_YR + yb), (n >> 1) & 1, status, &abort_flag, 73);
            tc_fence_after();
            __syncwarp();
            const float ia = lta > 0.f ? 1.f / lta : 0.f, ib = ltb > 0.f ? 1.f / ltb : 0.f;
            const uint32_t yrow = sb + kOffY + (uint32_t)(16 * w + (lane & 7)) * 128u;
            const uint32_t c0 = ((uint32_t)(lane >> 3) ^ (uint32_t)(lane & 7)) << 4;
            const uint32_t c1 = ((uint32_t)((lane >> 3) + 4) ^ (uint32_t)(lane & 7)) << 4;
#pragma unroll 1
            for (int h2 = 0; h2 < 2; ++h2) {
                uint32_t yr[32];
                tmem_ld16x256_x8(lbase + ycol + 64u * h2, yr);
                tmem_wait_ld();
                uint32_t ya[8], yb8[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    ya[j] = pack_bf16(__uint_as_float(yr[4 * j]) * ia, __uint_as_float(yr[4 * j + 1]) * ia);
                    yb8[j] = pack_bf16(__uint_as_float(yr[4 * j + 2]) * ib, __uint_as_float(yr[4 * j + 3]) * ib);
                }
                const uint32_t kb = yrow + 8192u * (uint32_t)h2;   // K-block of these 64 columns
                stmatrix_x4(kb + c0, ya[0], ya[1], ya[2], ya[3]);
                stmatrix_x4(kb + c1, ya[4], ya[5], ya[6], ya[7]);
                stmatrix_x4(kb + 1024u + c0, yb8[0], yb8[1], yb8[2], yb8[3]);
                stmatrix_x4(kb + 1024u + c1, yb8[4], yb8[5], yb8[6], yb8[7]);
            }
            fence_async_smem();
            tc_fence_before();
            mbar_arrive(B(B_YF));
            const bool ok = mbar_wait(B(B_OF), n & 1, status, &abort_flag, 74);
            tc_fence_after();
            __syncwarp();
#pragma unroll 1
            for (int h2 = 0; h2 < 2; ++h2) {
                uint32_t orr[32];
                tmem_ld16x256_x8(lbase + ycol + 64u * h2, orr);
                tmem_wait_ld();
                uint32_t oa8[8], ob8[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    oa8[j] = pack_bf16(__uint_as_float(orr[4 * j]), __uint_as_float(orr[4 * j + 1]));
                    ob8[j] = pack_bf16(__uint_as_float(orr[4 * j + 2]), __uint_as_float(orr[4 * j + 3]));
                }
                const uint32_t kb = yrow + 8192u * (uint32_t)h2;
                stmatrix_x4(kb + c0, oa8[0], oa8[1], oa8[2], oa8[3]);
                stmatrix_x4(kb + c1, oa8[4], oa8[5], oa8[6], oa8[7]);
                stmatrix_x4(kb + 1024u + c0, ob8[0], ob8[1], ob8[2], ob8[3]);
                stmatrix_x4(kb + 1024u + c1, ob8[4], ob8[5], ob8[6], ob8[7]);
            }
            tc_fence_before();
            mbar_arrive(B(B_OE + yb));
            __syncwarp();
            // this warp's 16 output rows, 16 bytes per lane and store
            if (ok) {
                bf16 *obase = o + ((int64_t)t.l * q_rows + t.qrow) * d + (int64_t)t.h * kDh;
#pragma unroll 1
                for (int it2 = 0; it2 < 8; ++it2) {
                    const int i = it2 * 32 + lane, row = 16 * w + (i >> 4), c = i & 15;
                    if (row < t.nq) {
                        const uint4 v = ld_shared_v4(sb + kOffY + 8192u * (uint32_t)(c >> 3) + (uint32_t)row * 128u +
                                                     ((((uint32_t)c & 7u) ^ ((uint32_t)row & 7u)) << 4));
                        *reinterpret_cast<uint4 *>(obase + (int64_t)row * d + 8 * c) = v;
                    }
                }
            }
            __syncwarp();
            next_unit(sp, it, nu);
            ++n;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}


// The launches of one instance (fixed-k or budget cache): records, maps,
// grid. Each instance is instantiated in a translation unit of its own
// (attend_tc.cu, attend_budget_tc.cu): with both in one module the fixed-k
// kernel measured 10 % slower on the c4 cache, same code.
template <bool kBudget>
cudaError_t launch_attend_impl(const AttendArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.max_query_tokens == 0 || P.num_episodes == 0) return cudaSuccess;
    const int H = S.num_heads, L = S.num_layers;
    const int64_t rows = P.rows_per_layer;
    CUtensorMap tq, tk, tr;
    {
        const uint64_t dims[4] = {(uint64_t)kDh, (uint64_t)H, (uint64_t)P.q_rows_per_layer, (uint64_t)L};
        const uint64_t str[3] = {(uint64_t)a.q_hs * 2, (uint64_t)a.q_rs * 2, (uint64_t)a.q_ls * 2};
        const uint32_t box[4] = {64, 1, (uint32_t)kQRows, 1};
        if (!make_bf16_map(&tq, a.q, 4, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[4] = {(uint64_t)kDh, (uint64_t)H, (uint64_t)rows, (uint64_t)L};
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
    auto kern = k_attend_tc<kBudget>;
    const int nthreads = kBudget ? kThreadsBudget : kThreads;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (err != cudaSuccess) return err;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        sms = 152;
    // per-row records (kept groups, packed offset) from the caller's indices
    uint4 *recs = reinterpret_cast<uint4 *>(a.ws.row_store);
    if (!a.records_ready)
        err = a.k_tok ? launch_row_store_budget(a.plan, L, a.idx, P.idx_bytes_per_layer, a.k_tok, recs, a.ws.status,
                                            a.stream)
                  : launch_row_store(a.plan, L, const_cast<uint8_t *>(a.idx), P.idx_bytes_per_layer, false, recs,
                                     a.ws.status, a.stream);
    if (err != cudaSuccess) return err;
    const int qtiles = (P.max_query_tokens + kQRows - 1) / kQRows;
    const float scale = a.scale > 0.f ? a.scale : 1.0f / sqrtf((float)kDh);
    // units (layer, head, episode, query tile); a launch gives each CTA at
    // most kMaxUnits of them
    const int E = P.num_episodes;
    const int64_t U = (int64_t)L * H * E * qtiles, per_launch = (int64_t)kMaxUnits * sms;
    for (int64_t u0 = 0; u0 < U; u0 += per_launch) {
        const int64_t u1 = std::min(U, u0 + per_launch);
        const int grid = (int)std::min<int64_t>(u1 - u0, sms);
        const int64_t ppl = a.packed_per_layer ? a.packed_per_layer : P.packed_elems_per_layer;
        if (!a.records_ready) {
            // a dependent of the record kernel: queries, keys and R_h are the
            // caller's, only the gather waits for the records
            err = launch_pdl(kern, dim3(grid), dim3(nthreads), kSmemBytes, a.stream, tq, tk, tr,
                             (const bf16 *)a.packed, ppl, (const uint4 *)recs, rows, a.plan.eps_dev, E, H, qtiles,
                             u0, u1, (int64_t)P.q_rows_per_layer, scale * 1.4426950408889634f, (bf16 *)a.o,
                             a.ws.status);
        } else {
            kern<<<grid, nthreads, kSmemBytes, a.stream>>>(
                tq, tk, tr, (const bf16 *)a.packed, ppl, recs, rows, a.plan.eps_dev, E, H, qtiles, u0, u1,
                P.q_rows_per_layer, scale * 1.4426950408889634f, (bf16 *)a.o, a.ws.status);
            err = cudaGetLastError();
        }
        count_launches(1);
        if (err != cudaSuccess) return err;
    }
    return cudaSuccess;
}

}  // namespace

}  // namespace rs
