// gemm_tc.cu -- bf16 GEMM on the 5th-generation tensor core for the
// dense-rotation geometry (one d x d orthonormal R per layer, Sec. 4.1):
//   C[l] = A[l] . B[l]^T   (B given as [N][K], K contiguous)      kBMN = false
//   C[l] = A[l] . B[l]     (B given as [K][N], N contiguous)      kBMN = true
// A [M][K] row-major, C [M][N] row-major bf16 (fp32 accumulation, one
// rounding). Used for z = R^T v over all d dims (A = V, B = R as [K][N]) and
// for the routed values v~ = R (M z) (A = M Z, B = R as [N][K]).
//
// One CTA per (128-row tile, 256-column tile, layer), 192 threads: warp 4
// TMA producer, warp 5 MMA issuer, warps 0-3 epilogue (a TMEM lane and a
// tile row per thread). K runs in 64-wide blocks through a 4-stage ring of
// 48 KB stages. The epilogue stages the bf16 tile in the drained ring and
// stores it with 16-byte lanes, one tile row per warp instruction.
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
constexpr int kGStages = 4;
constexpr uint32_t kGTileA = kBM * kBK * 2;          // 16 KB
constexpr uint32_t kGTileB = kBN * kBK * 2;          // 32 KB
constexpr uint32_t kGStage = kGTileA + kGTileB;      // 48 KB
constexpr uint32_t kGOffBar = kGStages * kGStage;    // 192 KB
constexpr uint32_t kGSmem = kGOffBar + 128 + 1024;
constexpr uint32_t kGPitch = kBN * 2 + 16;           // staged C row: 512 B + 16 B pad
static_assert(kBM * kGPitch <= kGOffBar, "C staging fits the ring");

template <bool kBMN>
__global__ void __launch_bounds__(kGThreads, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b, int M, int N, int K,
          bf16 *__restrict__ C, int64_t c_layer_stride, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    const uint32_t sraw = smem_u32(smem_raw);
    const uint32_t sb = (sraw + 1023u) & ~1023u;
    uint8_t *sp = smem_raw + (sb - sraw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n0 = blockIdx.x * kBN, m0 = blockIdx.y * kBM, l = blockIdx.z;
    const int nkb = K / kBK;
    const uint32_t bar_full = sb + kGOffBar, bar_empty = bar_full + 8 * kGStages, bar_acc = bar_empty + 8 * kGStages;

    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < 2 * kGStages; ++i) mbar_init(bar_full + 8 * i, 1);
        mbar_init(bar_acc, 1);
        fence_mbar_init();
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

    if (warp == 4) {
        if (lane == 0) {
            prefetch_tmap(&tm_a);
            prefetch_tmap(&tm_b);
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kGStages;
                if (kb >= kGStages &&
                    !mbar_wait(bar_empty + 8 * s, ((kb / kGStages) - 1) & 1, status, &abort_flag, 90))
                    break;
                const uint32_t st = sb + kGStage * s;
                mbar_expect_tx(bar_full + 8 * s, kGStage);
                tma_load_3d(st, &tm_a, kBK * kb, m0, l, bar_full + 8 * s);
                if (kBMN) {
                    // four 64-column blocks of 64 K rows each (8 KB apart)
                    for (int nb = 0; nb < kBN / 64; ++nb)
                        tma_load_3d(st + kGTileA + 8192u * nb, &tm_b, n0 + 64 * nb, kBK * kb, l, bar_full + 8 * s);
                } else {
                    tma_load_3d(st + kGTileA, &tm_b, kBK * kb, n0, l, bar_full + 8 * s);
                }
            }
        }
    } else if (warp == 5) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(kBM, kBN, kBMN);
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kGStages;
                if (!mbar_wait(bar_full + 8 * s, (kb / kGStages) & 1, status, &abort_flag, 91)) break;
                tc_fence_after();
                const uint32_t st = sb + kGStage * s;
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t a = sdesc_sw128(st + 32u * kk, 16, 1024);
                    // K-major B: +32 bytes per K16 step; MN-major B: +16 K rows
                    // (2 KB) per step, 64-column blocks 8 KB apart
                    const uint64_t b = kBMN ? sdesc_sw128(st + kGTileA + 2048u * kk, 8192, 1024)
                                            : sdesc_sw128(st + kGTileA + 32u * kk, 16, 1024);
                    mma_bf16(tmem, a, b, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(bar_empty + 8 * s);
            }
            mma_commit(bar_acc);
        }
    } else {
        // ------------------------------------------------ epilogue warps 0-3
        const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
        const bool ok = mbar_wait(bar_acc, 0, status, &abort_flag, 92);
        tc_fence_after();
        __syncwarp();
        // this thread's row (warp * 32 + lane) into the staging tile
        uint8_t *srow = sp + (uint32_t)tid * kGPitch;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
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
        __syncwarp();
        // the warp's 32 rows, one 512-byte row per instruction
        if (ok && !abort_flag) {
            bf16 *cbase = C + (int64_t)l * c_layer_stride + n0;
#pragma unroll 1
            for (int i = 0; i < 32; ++i) {
                const int row = 32 * warp + i, m = m0 + row;
                if (m >= M) break;
                const uint4 v = *reinterpret_cast<const uint4 *>(sp + (uint32_t)row * kGPitch + 16u * lane);
                *reinterpret_cast<uint4 *>(cbase + (int64_t)m * N + 8 * lane) = v;
            }
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

// M rows of A per layer, K = inner size, N = output columns; K % 64 == 0,
// N % 256 == 0; pointers and strides in elements.
cudaError_t launch_gemm_tc(bool b_mn_major, int L, int M, int N, int K, const void *A, int64_t a_layer_stride,
                           const void *B, int64_t b_layer_stride, void *C, int64_t c_layer_stride, int32_t *status,
                           cudaStream_t stream)
{
    if (M == 0 || L == 0) return cudaSuccess;
    if (K % kBK != 0 || N % kBN != 0) return cudaErrorInvalidValue;
    CUtensorMap ta, tb;
    {
        // A [L][M][K] with its own layer stride
        const uint64_t dims[3] = {(uint64_t)K, (uint64_t)M, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)K * 2, (uint64_t)a_layer_stride * 2};
        const uint32_t box[3] = {kBK, kBM, 1};
        if (!make_bf16_map(&ta, A, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    if (b_mn_major) {
        const uint64_t dims[3] = {(uint64_t)N, (uint64_t)K, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)N * 2, (uint64_t)b_layer_stride * 2};
        const uint32_t box[3] = {64, kBK, 1};
        if (!make_bf16_map(&tb, B, 3, dims, str, box)) return cudaErrorInvalidValue;
    } else {
        const uint64_t dims[3] = {(uint64_t)K, (uint64_t)N, (uint64_t)L};
        const uint64_t str[2] = {(uint64_t)K * 2, (uint64_t)b_layer_stride * 2};
        const uint32_t box[3] = {kBK, kBN, 1};
        if (!make_bf16_map(&tb, B, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    const dim3 grid((unsigned)(N / kBN), (unsigned)((M + kBM - 1) / kBM), (unsigned)L);
    cudaError_t err;
    if (b_mn_major) {
        err = cudaFuncSetAttribute(k_gemm_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGSmem);
        if (err != cudaSuccess) return err;
        k_gemm_tc<true><<<grid, kGThreads, kGSmem, stream>>>(ta, tb, M, N, K, (bf16 *)C, c_layer_stride, status);
    } else {
        err = cudaFuncSetAttribute(k_gemm_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGSmem);
        if (err != cudaSuccess) return err;
        k_gemm_tc<false><<<grid, kGThreads, kGSmem, stream>>>(ta, tb, M, N, K, (bf16 *)C, c_layer_stride, status);
    }
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
