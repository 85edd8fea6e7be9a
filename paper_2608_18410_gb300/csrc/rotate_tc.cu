// rotate_tc.cu -- orthogonal value decomposition and packing (Sec. 3.2) on
// the 5th-generation tensor core, bf16 inputs, fp32 accumulation.
//
// z = R_h^T v for every cache row and head, in row form Z_h = V_h R_h:
//   A = 128 value rows of head h (K-major, TMA from v),
//   B = R_h with B[n][k] = R_h[k][n]: R_h is row-major in k, so it is the
//       MN-major operand, loaded by TMA as two 64-column blocks,
//   D = 128 x 128 fp32 in TMEM (double buffered across heads).
// The epilogue (one row per thread) keeps only the row's kept groups: each
// group of d_s = 8 values becomes one 16-byte bf16 store into
// packed[seg][h][i][j][:]. Segments with k = S also get indices 0..S-1.
//
// Grid: (128-row tiles of the layer, head groups, layers); each CTA loops
// over `hpb` heads with a two-stage TMA/MMA pipeline so that loading and
// multiplying head h+1 overlaps the epilogue of head h.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace rs {

namespace {

using namespace sm100;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 128;
constexpr int kRows = 128;
constexpr int kDh = 128;
constexpr int kG = 16;

constexpr uint32_t kStage = 65536;           // V tile (32K) + R_h (32K)
constexpr uint32_t kOffBar = 2 * kStage;
constexpr uint32_t kSmemBytes = kOffBar + 128 + 1024;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kIdesc = idesc_bf16(128, 128, true);

__device__ __forceinline__ void store_group(bf16 *dst, const uint32_t (&sr)[32], int w)
{
    // columns 8w .. 8w+7 of this 32-column slice
    uint32_t a, b, c, d;
#define RS_PACK(o)                                                                   \
    a = pack_bf16(__uint_as_float(sr[o + 0]), __uint_as_float(sr[o + 1]));           \
    b = pack_bf16(__uint_as_float(sr[o + 2]), __uint_as_float(sr[o + 3]));           \
    c = pack_bf16(__uint_as_float(sr[o + 4]), __uint_as_float(sr[o + 5]));           \
    d = pack_bf16(__uint_as_float(sr[o + 6]), __uint_as_float(sr[o + 7]));
    switch (w) {
    case 0: RS_PACK(0); break;
    case 1: RS_PACK(8); break;
    case 2: RS_PACK(16); break;
    default: RS_PACK(24); break;
    }
#undef RS_PACK
    *reinterpret_cast<uint4 *>(dst) = make_uint4(a, b, c, d);
}

__global__ void __launch_bounds__(kThreads, 1)
k_rotate_tc(const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_r, PlanDev plan,
            int64_t rows, int H, int hpb, bf16 *__restrict__ packed, int64_t packed_per_layer,
            uint8_t *__restrict__ idx, int64_t idx_per_layer, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int l = blockIdx.z;
    const int64_t r0 = (int64_t)blockIdx.x * kRows;
    const int h0 = blockIdx.y * hpb;
    const int nh = min(hpb, H - h0);
    if (nh <= 0) return;
    const uint32_t bar_full = sb + kOffBar, bar_done = bar_full + 16;

    auto load_head = [&](int i) {  // stage i & 1 <- V tile and R of head h0 + i
        const uint32_t st = sb + kStage * (uint32_t)(i & 1);
        const int h = h0 + i;
        mbar_expect_tx(bar_full + 8 * (i & 1), 65536);
        tma_load_4d(st, &tm_v, 0, h, (int)r0, l, bar_full + 8 * (i & 1));
        tma_load_4d(st + 16384, &tm_v, 64, h, (int)r0, l, bar_full + 8 * (i & 1));
        tma_load_3d(st + 32768, &tm_r, 0, 0, l * H + h, bar_full + 8 * (i & 1));
        tma_load_3d(st + 49152, &tm_r, 64, 0, l * H + h, bar_full + 8 * (i & 1));
    };
    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < 4; ++i) mbar_init(bar_full + 8 * i, 1);
        fence_mbar_init();
        prefetch_tmap(&tm_v);
        prefetch_tmap(&tm_r);
        load_head(0);
        if (nh > 1) load_head(1);
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

    auto issue_mma = [&](int i) {
        const uint32_t st = sb + kStage * (uint32_t)(i & 1);
        if (!mbar_wait(bar_full + 8 * (i & 1), (i >> 1) & 1, status, &abort_flag, 10)) return;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            const uint64_t a = sdesc_sw128(st + (kk >> 2) * 16384u + (kk & 3) * 32u, 16, 1024);
            const uint64_t b = sdesc_sw128(st + 32768u + 2048u * kk, 16384, 1024);
            mma_bf16(tmem + 128u * (i & 1), a, b, kIdesc, kk > 0);
        }
        mma_commit(bar_done + 8 * (i & 1));
    };
    if (tid == 0) issue_mma(0);

    // this thread's row: segment, kept groups
    const int64_t r = r0 + tid;
    int k = 0;
    rolesub_segment sg{};
    int gid[kG];
    if (r < rows) {
        sg = plan.segs[plan.row_seg[r]];
        k = sg.k;
    }
    const int64_t ti = r - sg.token_row;
    uint8_t *ix = idx + (int64_t)l * idx_per_layer + sg.idx_off + ti * k;
#pragma unroll
    for (int s = 0; s < kG; ++s) gid[s] = s;
    if (k > 0 && k < kG) {
#pragma unroll
        for (int s = 0; s < kG; ++s)
            if (s < k) gid[s] = ix[s];
    }
    if (k == kG && blockIdx.y == 0) {   // byte stores: idx offsets need no alignment
#pragma unroll
        for (int s = 0; s < kG; ++s) ix[s] = (uint8_t)s;
    }
    bool bad = false;
#pragma unroll
    for (int s = 0; s < kG; ++s)
        if (s < k && gid[s] >= kG) bad = true;
    if (bad) report(status, ROLESUB_EDEVICE, (int)r);

    for (int i = 0; i < nh; ++i) {
        const int h = h0 + i;
        if (tid == 0 && !abort_flag && i + 1 < nh) issue_mma(i + 1);  // overlaps this head's epilogue
        mbar_wait(bar_done + 8 * (i & 1), (i >> 1) & 1, status, &abort_flag, 11);
        tc_fence_after();
        if (tid == 0 && !abort_flag && i + 2 < nh) load_head(i + 2);   // stage i & 1 is free
        __syncwarp();
        bf16 *dst = packed + (int64_t)l * packed_per_layer + sg.packed_off + ((int64_t)h * sg.n_tokens + ti) * k * 8;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            uint32_t sr[32];
            tmem_ld32(tmem + ((uint32_t)(32 * warp) << 16) + 128u * (i & 1) + 32u * q4, sr);
            tmem_wait_ld();
            if (bad || abort_flag) continue;
#pragma unroll
            for (int s = 0; s < kG; ++s)
                if (s < k && (gid[s] >> 2) == q4) store_group(dst + 8 * s, sr, gid[s] & 3);
        }
        tc_fence_before();
        __syncthreads();   // TMEM buffer i & 1 may be overwritten by head i + 2
        tc_fence_after();
    }
    if (warp == 0) tmem_dealloc(tmem, kTmemCols);
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
    const int64_t tiles = (rows + kRows - 1) / kRows;
    // heads per CTA: enough CTAs to fill the GPU twice over, otherwise all heads
    int hpb = H;
    const int64_t units = tiles * L;
    while (hpb > 1 && units * ((H + hpb - 1) / hpb) < 2 * 152) hpb = (hpb + 1) / 2;
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev};
    k_rotate_tc<<<dim3((unsigned)tiles, (H + hpb - 1) / hpb, L), kThreads, kSmemBytes, a.stream>>>(
        tv, tr, pd, rows, H, hpb, (bf16 *)a.packed, P.packed_elems_per_layer, a.idx, P.idx_bytes_per_layer,
        a.ws.status);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
