// select.cu -- token-level reduction (Sec. 3.1), the step before the value
// path: for every episode and camera view, keep the ceil(r n) visual tokens
// with the highest importance scores (ties: lower token index), in their
// original order, and gather their rows.
//
// k_select_tokens  one block per (episode, view): scores to order keys in
//                  shared memory, a rank per token by counting, kept tokens'
//                  output slots by a block scan of the keep flags, the index
//                  list, then the kept rows copied 16 bytes per lane.
#include "common.cuh"
#include "internal.h"

namespace rs {

namespace {

constexpr int kST = 256;

__device__ __forceinline__ uint32_t score_key(float x)
{
    if (x != x) return 0u;   // NaN ranks lowest
    if (x == 0.f) x = 0.f;   // -0 == +0
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Shared memory: keys [n] u32 | slot [n] i32
__global__ void __launch_bounds__(kST)
k_select_tokens(int n, int k, const float *__restrict__ scores, const uint8_t *__restrict__ x, int64_t row_bytes,
                int32_t *__restrict__ keep_idx, uint8_t *__restrict__ x_keep)
{
    extern __shared__ __align__(16) uint32_t sk[];
    __shared__ int part[kST];
    int *slot = reinterpret_cast<int *>(sk + n);
    const int tid = threadIdx.x;
    const int64_t ev = blockIdx.x;   // (episode, view)
    const float *sc = scores + ev * n;
    for (int i = tid; i < n; i += kST) sk[i] = score_key(sc[i]);
    __syncthreads();
    // keep flags in token order, each thread a contiguous run of tokens
    const int per = (n + kST - 1) / kST;
    const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
    int cnt = 0;
    for (int i = i0; i < i1; ++i) {
        const uint32_t p = sk[i];
        int rank = 0;
        for (int j = 0; j < n; ++j) {
            const uint32_t q = sk[j];
            rank += (q > p || (q == p && j < i)) ? 1 : 0;
        }
        slot[i] = rank < k ? 1 : 0;
        cnt += slot[i];
    }
    part[tid] = cnt;
    __syncthreads();
    for (int off = 1; off < kST; off <<= 1) {
        const int v = tid >= off ? part[tid - off] : 0;
        __syncthreads();
        part[tid] += v;
        __syncthreads();
    }
    int run = tid > 0 ? part[tid - 1] : 0;
    for (int i = i0; i < i1; ++i) {
        if (slot[i]) {
            keep_idx[ev * k + run] = i;
            slot[i] = run++;
        } else {
            slot[i] = -1;
        }
    }
    __syncthreads();
    // rows: one warp per kept row, 16 bytes per lane
    const int warp = tid >> 5, lane = tid & 31;
    const int64_t v16 = row_bytes / 16;
    for (int i = warp; i < n; i += kST / 32) {
        const int s = slot[i];
        if (s < 0) continue;
        const uint4 *src = reinterpret_cast<const uint4 *>(x + (ev * n + i) * row_bytes);
        uint4 *dst = reinterpret_cast<uint4 *>(x_keep + (ev * k + s) * row_bytes);
        for (int64_t c = lane; c < v16; c += 32) dst[c] = __ldg(src + c);
    }
}

}  // namespace

cudaError_t launch_select_tokens(int64_t groups, int n, int k, const float *scores, const void *x, int64_t row_bytes,
                                 int32_t *keep_idx, void *x_keep, cudaStream_t stream)
{
    if (groups == 0 || n == 0) return cudaSuccess;
    const size_t smem = (size_t)n * 8 + 16;
    cudaError_t err = cudaFuncSetAttribute(k_select_tokens, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    k_select_tokens<<<(unsigned)groups, kST, smem, stream>>>(n, k, scores, (const uint8_t *)x, row_bytes, keep_idx,
                                                             (uint8_t *)x_keep);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
