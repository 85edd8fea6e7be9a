// rotate_tc.cu -- orthogonal value decomposition and packing (Sec. 3.2) on
// the 5th-generation tensor core, bf16 inputs, fp32 accumulation.
//
// z = R_h^T v for every cache row and head, in row form Z = V_h R_h:
//   A = 128 value rows of head h (K-major, TMA from v),
//   B = R_h with B[n][k] = R_h[k][n]: R_h is row-major in k, so it is the
//       MN-major operand (two 64-column blocks loaded by TMA),
//   D = 128 x 128 fp32 in TMEM.
// The epilogue (one row per thread) keeps only the row's kept groups: each
// group of d_s = 8 values becomes one 16-byte bf16 store into
// packed[seg][h][i][j][:]. Segments with k = S also get indices 0..S-1.
//
// Persistent: one CTA per SM walks the items (head, layer, range of 128-row
// tiles), 192 threads:
//   warp 4  TMA producer: R_h of each item into one of two buffers (the
//           next item's while this one's tiles are multiplied), value tiles
//           into a 4-stage ring that runs on across items
//   warp 5  MMA issuer: one 128x128x128 MMA per tile, TMEM double-buffered
//   warps 0-3 epilogue: TMEM -> bf16 group stores; the row metadata
//           (segment, kept groups) is fetched two tiles ahead, across items
// R_h is read from L2 once per item instead of once per tile.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 192;
constexpr int kRows = 128;
constexpr int kDh = 128;
constexpr int kG = 16;
constexpr int kStages = 4;

constexpr uint32_t kOffR = 0;                       // R_h: 2 buffers x (2 x 16K MN-blocks)
constexpr uint32_t kOffV = 65536;                   // V ring: 4 x 32K
constexpr uint32_t kVBytes = 32768;
constexpr uint32_t kOffZ = kOffV + kStages * kVBytes;   // bf16 z rows: 128 x 256 B
constexpr uint32_t kOffBar = kOffZ + 32768;
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kIdesc = idesc_bf16(128, 128, true);

// Per-row store record, built once per (layer, row) by k_row_store:
//   x, y: kept group ids, 4 bits each in storage order (64 bits)
//   z:    (packed_off + i * k * d_s) / 8, the row's first group for head 0
//   w:    k << 27 | n * k, i.e. kept groups and the per-head stride / 8
// k = 0 means nothing is stored for the row (or its indices were corrupt).
// write_identity: also write indices 0..S-1 of k = S rows (compress only).
__global__ void __launch_bounds__(256)
k_row_store(PlanDev plan, int64_t rows, uint8_t *idx, int64_t idx_per_layer, bool write_identity,
            uint4 *__restrict__ meta, int32_t *status)
{
    pdl_trigger();
    pdl_wait();   // idx may come from the kernel just before
    const int l = blockIdx.y;
    const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= rows) return;
    const rolesub_segment sg = plan.segs[plan.row_seg[r]];
    const int k = sg.k;
    const int64_t ti = r - sg.token_row;
    uint8_t *ix = idx + (int64_t)l * idx_per_layer + sg.idx_off + ti * k;
    uint64_t gid = 0;
    int kk = k;
    if (k == kG) {
        gid = 0xFEDCBA9876543210ull;
        if (write_identity)
            for (int s = 0; s < kG; ++s) ix[s] = (uint8_t)s;   // byte stores: no alignment needed
    } else {
        for (int s = 0; s < k; ++s) {
            const uint32_t g = ld_dep(ix + s);
            if (g >= kG) {
                report(status, ROLESUB_EDEVICE, (int)r);
                kk = 0;
                break;
            }
            gid |= (uint64_t)g << (4 * s);
        }
    }
    const int64_t base8 = sg.packed_off / 8 + ti * k;
    meta[(int64_t)l * rows + r] = make_uint4((uint32_t)gid, (uint32_t)(gid >> 32), (uint32_t)base8,
                                             ((uint32_t)kk << 27) | (uint32_t)((int64_t)sg.n_tokens * k));
}

struct RotItem {
    int h, l, t0, nt;
};

__device__ __forceinline__ RotItem rot_item(int it, int H, int L, int per, int ntiles)
{
    RotItem r;
    r.h = it % H;
    r.l = (it / H) % L;
    r.t0 = (it / (H * L)) * per;
    r.nt = min(per, ntiles - r.t0);
    return r;
}

__global__ void __launch_bounds__(kThreads, 1)
k_rotate_tc(const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_r,
            const uint4 *meta, int64_t rows, int H, int L, int per, int ntiles, int nitems,
            bf16 *__restrict__ packed, int64_t packed_per_layer, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    const uint32_t bar_rfull = sb + kOffBar;             // [2]
    const uint32_t bar_rempty = bar_rfull + 16;          // [2]
    const uint32_t bar_full = bar_rempty + 16;           // [4]
    const uint32_t bar_empty = bar_full + 32;            // [4]
    const uint32_t bar_tfull = bar_empty + 32;           // [2]
    const uint32_t bar_tempty = bar_tfull + 16;          // [2]

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_rfull + 8 * i, 1);
            mbar_init(bar_rempty + 8 * i, 1);
        }
        for (int i = 0; i < kStages; ++i) {
            mbar_init(bar_full + 8 * i, 1);
            mbar_init(bar_empty + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_tfull + 8 * i, 1);
            mbar_init(bar_tempty + 8 * i, 128);
        }
        fence_mbar_init();
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

    if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_v);
            prefetch_tmap(&tm_r);
            bool ok = true;
            uint32_t gt = 0;   // tiles issued so far (ring position)
            for (int it = blockIdx.x, n = 0; it < nitems && ok; it += gridDim.x, ++n) {
                const RotItem w = rot_item(it, H, L, per, ntiles);
                const uint32_t rb = (uint32_t)n & 1u;
                // R buffer rb is free once the products of item n - 2 are done
                if (n >= 2 && !mbar_wait(bar_rempty + 8 * rb, ((uint32_t)(n - 2) >> 1) & 1u, status, &abort_flag, 35))
                    break;
                mbar_expect_tx(bar_rfull + 8 * rb, 32768);
                tma_load_3d(sb + kOffR + 32768u * rb, &tm_r, 0, 0, w.l * H + w.h, bar_rfull + 8 * rb);
                tma_load_3d(sb + kOffR + 32768u * rb + 16384u, &tm_r, 64, 0, w.l * H + w.h, bar_rfull + 8 * rb);
                for (int t = 0; t < w.nt; ++t, ++gt) {
                    const uint32_t s = gt % kStages;
                    if (gt >= kStages &&
                        !mbar_wait(bar_empty + 8 * s, ((gt / kStages) - 1) & 1, status, &abort_flag, 30)) {
                        ok = false;
                        break;
                    }
                    const uint32_t st = sb + kOffV + kVBytes * s;
                    const int r0 = (w.t0 + t) * kRows;
                    mbar_expect_tx(bar_full + 8 * s, kVBytes);
                    tma_load_4d(st, &tm_v, 0, w.h, r0, w.l, bar_full + 8 * s);
                    tma_load_4d(st + 16384, &tm_v, 64, w.h, r0, w.l, bar_full + 8 * s);
                }
            }
        }
    } else if (warp == 5) {
        if (lane == 0) {
            bool ok = true;
            uint32_t gt = 0;
            for (int it = blockIdx.x, n = 0; it < nitems && ok; it += gridDim.x, ++n) {
                const RotItem w = rot_item(it, H, L, per, ntiles);
                const uint32_t rb = (uint32_t)n & 1u;
                if (!mbar_wait(bar_rfull + 8 * rb, ((uint32_t)n >> 1) & 1u, status, &abort_flag, 31)) break;
                for (int t = 0; t < w.nt; ++t, ++gt) {
                    const uint32_t s = gt % kStages, b = gt & 1u;
                    if (!mbar_wait(bar_full + 8 * s, (gt / kStages) & 1, status, &abort_flag, 32) ||
                        (gt >= 2 && !mbar_wait(bar_tempty + 8 * b, ((gt >> 1) - 1) & 1, status, &abort_flag, 33))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t st = sb + kOffV + kVBytes * s;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const uint64_t a = sdesc_sw128(st + (kk >> 2) * 16384u + (kk & 3) * 32u, 16, 1024);
                        const uint64_t bd = sdesc_sw128(sb + kOffR + 32768u * rb + 2048u * kk, 16384, 1024);
                        mma_bf16(tmem + 128u * b, a, bd, kIdesc, kk > 0);
                    }
                    mma_commit(bar_empty + 8 * s);
                    mma_commit(bar_tfull + 8 * b);
                }
                mma_commit(bar_rempty + 8 * rb);
            }
        }
    } else {
        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
        // the records (and the indices behind them) come from the kernels
        // before this one, which may still run while the first products do
        pdl_wait();
        // row record of this thread's row in the tile two ahead, across items
        const uint4 zero4 = make_uint4(0, 0, 0, 0);
        int ai = blockIdx.x, at = 0;   // lookahead cursor (item, tile)
        RotItem aw = ai < nitems ? rot_item(ai, H, L, per, ntiles) : RotItem{0, 0, 0, 0};
        auto fetch_adv = [&]() -> uint4 {
            uint4 m = zero4;
            if (ai < nitems) {
                const int64_t r = (int64_t)(aw.t0 + at) * kRows + tid;
                if (r < rows) m = ld_dep(meta + (int64_t)aw.l * rows + r);
                if (++at >= aw.nt) {
                    at = 0;
                    ai += gridDim.x;
                    if (ai < nitems) aw = rot_item(ai, H, L, per, ntiles);
                }
            }
            return m;
        };
        uint4 m0 = fetch_adv();
        uint4 m1 = fetch_adv();
        const uint32_t zrow = sb + kOffZ + (uint32_t)tid * 256u;
        const uint32_t sw = (uint32_t)(tid & 15);
        uint32_t gt = 0;
        for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
            const RotItem w = rot_item(it, H, L, per, ntiles);
            bf16 *pl = packed + (int64_t)w.l * packed_per_layer;
            for (int t = 0; t < w.nt; ++t, ++gt) {
                const uint32_t b = gt & 1u;
                const uint4 m2 = fetch_adv();
                mbar_wait(bar_tfull + 8 * b, (gt >> 1) & 1, status, &abort_flag, 34);
                tc_fence_after();
                __syncwarp();
                const uint64_t gid = (uint64_t)m0.x | ((uint64_t)m0.y << 32);
                const int k = abort_flag ? 0 : (int)(m0.w >> 27);
                uint4 *dst =
                    reinterpret_cast<uint4 *>(pl + ((int64_t)m0.z + (int64_t)w.h * (int64_t)(m0.w & 0x7FFFFFFu)) * 8);
                // the row's z as 16 bf16 chunks (one per group) in shared
                // memory, chunk c at position c ^ (row & 15) to spread banks
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    uint32_t sa[32], sc[32];
                    tmem_ld32(lane_base + 128u * b + 64u * half, sa);
                    tmem_ld32(lane_base + 128u * b + 64u * half + 32u, sc);
                    tmem_wait_ld();
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const uint32_t(&src)[32] = c < 4 ? sa : sc;
                        const int o = 8 * (c & 3);
                        st_shared_v4(zrow + ((((uint32_t)(8 * half + c)) ^ sw) << 4),
                                     pack_bf16(__uint_as_float(src[o]), __uint_as_float(src[o + 1])),
                                     pack_bf16(__uint_as_float(src[o + 2]), __uint_as_float(src[o + 3])),
                                     pack_bf16(__uint_as_float(src[o + 4]), __uint_as_float(src[o + 5])),
                                     pack_bf16(__uint_as_float(src[o + 6]), __uint_as_float(src[o + 7])));
                    }
                }
                tc_fence_before();
                mbar_arrive(bar_tempty + 8 * b);   // TMEM buffer b is free for the tile two on
                // kept groups in storage order: same-thread shared-memory round trip
                for (int s2 = 0; s2 < k; ++s2) {
                    const uint32_t g = (uint32_t)(gid >> (4 * s2)) & 15u;
                    dst[s2] = ld_shared_v4(zrow + ((g ^ sw) << 4));
                }
                m0 = m1;
                m1 = m2;
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

bool rotate_tc_supported(const rolesub_shape *s)
{
    return s->dtype == ROLESUB_BF16 && s->head_dim == kDh && s->num_groups == kG;
}

cudaError_t launch_rotate_tc(const CompressArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    if (P.stored_rows_per_layer == 0) return cudaSuccess;
    const int H = S.num_heads, L = S.num_layers;
    const int64_t rows = P.rows_per_layer, d = (int64_t)H * kDh;
    CUtensorMap tv, tr;
    {
        const uint64_t dims[4] = {(uint64_t)kDh, (uint64_t)H, (uint64_t)rows, (uint64_t)L};
        const uint64_t str[3] = {(uint64_t)kDh * 2, (uint64_t)d * 2, (uint64_t)(rows * d * 2)};
        const uint32_t box[4] = {64, 1, (uint32_t)kRows, 1};
        if (!make_bf16_map(&tv, a.v, 4, dims, str, box)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)kDh, (uint64_t)kDh, (uint64_t)L * H};
        const uint64_t str[2] = {(uint64_t)kDh * 2, (uint64_t)kDh * kDh * 2};
        const uint32_t box[3] = {64, (uint32_t)kDh, 1};
        if (!make_bf16_map(&tr, a.R, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    cudaError_t err = cudaFuncSetAttribute(k_rotate_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (err != cudaSuccess) return err;
    const int ntiles = (int)((rows + kRows - 1) / kRows);
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        sms = 152;
    // split each (head, layer) tile list until there are at least eight
    // items per persistent CTA, so that the last round of items is short
    int splits = 1;
    while ((int64_t)H * L * splits < 8 * (int64_t)sms && splits < ntiles) ++splits;
    const int per = (ntiles + splits - 1) / splits;
    splits = (ntiles + per - 1) / per;
    const int nitems = H * L * splits;
    const unsigned grid = (unsigned)(nitems < sms ? nitems : sms);
    uint4 *meta = reinterpret_cast<uint4 *>(a.ws.row_store);
    // the records (when built here) and then the products start while the
    // router's tail still runs; both wait for their predecessor before
    // reading its output
    if (!a.records_ready) {
        err = launch_row_store(a.plan, L, a.idx, P.idx_bytes_per_layer, true, meta, a.ws.status, a.stream, true);
        if (err != cudaSuccess) return err;
    }
    err = launch_pdl(k_rotate_tc, dim3(grid), dim3(kThreads), kSmemBytes, a.stream, tv, tr, (const uint4 *)meta, rows,
                     H, L, per, ntiles, nitems, (bf16 *)a.packed, (int64_t)P.packed_elems_per_layer, a.ws.status);
    count_launches(1);
    return err;
}

cudaError_t launch_row_store(const PlanView &pv, int L, uint8_t *idx, int64_t idx_per_layer, bool write_identity,
                             uint4 *recs, int32_t *status, cudaStream_t stream, bool pdl)
{
    const int64_t rows = pv.hdr->rows_per_layer;
    if (rows == 0) return cudaSuccess;
    PlanDev pd{pv.segs_dev, pv.eps_dev, pv.row_seg_dev, pv.routed_dev, pv.stored_dev, pv.route_tiles_dev};
    const dim3 grid((unsigned)((rows + 255) / 256), L);
    cudaError_t err;
    if (pdl) {
        err = launch_pdl(k_row_store, grid, dim3(256), 0, stream, pd, rows, idx, idx_per_layer, write_identity, recs,
                         status);
    } else {
        k_row_store<<<grid, 256, 0, stream>>>(pd, rows, idx, idx_per_layer, write_identity, recs, status);
        err = cudaGetLastError();
    }
    count_launches(1);
    return err;
}

}  // namespace rs
