// dense.cu -- bookkeeping of the dense-rotation geometry of Sec. 4.1: one
// d x d orthonormal R per layer, the rotated vector z = R^T v split into S
// contiguous groups of g = d / S dims. Only kept groups are ever computed:
//
// Compress: the router's indices give every stored row's k kept groups.
// k_dense_pairs lists, per 4096-row chunk and per group s, the (row, packed
// slot) pairs that keep s; the tensor-core kernel (gemm_tc.cu) then forms
// z_s = R_s^T v for 128 such pairs at a time and writes them to their slots
// (segment (n tokens, k) holds [n][k][g] values, token i's groups in index
// order at packed_off + (i k + j) g).
//
// Attend: every head's output needs all d rotated dims of the routed values,
// so they are brought back to the original space, v~_j = R (M_j z_j) =
// sum over kept s of R_s z_{j,s}. k_dense_sort orders each layer's rows by
// their kept-group set (k, then the two lowest kept groups), so that a
// 128-row tile of the tensor-core kernel needs the K blocks of few groups;
// it also writes the attention's store records (every group of every head
// kept, identity ids) pointing at each row's sorted position in v~, and
// k_identity the identity R_h, so that the attention kernel reads v~ as
// plain per-head values.
#include "common.cuh"
#include "internal.h"

namespace rs {

namespace {

typedef __nv_bfloat16 bf16;

constexpr int kPairThreads = 512;                              // 16 warps: one per group in the scan
constexpr int kPairRowsPerThread = kDenseChunk / kPairThreads;  // 8 consecutive rows per thread
static_assert(kPairThreads / 32 == 16, "one scanning warp per group");

// One CTA per (chunk, layer). Pairs of group s come out in row order:
// thread t owns rows [c0 + 8 t, c0 + 8 t + 8), counts its pairs per group,
// and a per-group exclusive scan over the threads gives each thread its
// first position, so the listing is deterministic.
__global__ void __launch_bounds__(kPairThreads)
k_dense_pairs(const rolesub_segment *__restrict__ segs, const int32_t *__restrict__ row_seg, int64_t rows, int G,
              int g, const uint8_t *__restrict__ idx, int64_t idx_per_layer, int2 *__restrict__ pairs,
              int32_t *__restrict__ meta, int chunks, int32_t *status)
{
    __shared__ int hist[16][kPairThreads];
    __shared__ int tot[16], gbase[16];
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31, c = blockIdx.x, l = blockIdx.y;
    const int64_t c0 = (int64_t)c * kDenseChunk, c1 = min(rows, c0 + kDenseChunk);
    const int64_t r0 = c0 + (int64_t)t * kPairRowsPerThread, r1 = min(c1, r0 + kPairRowsPerThread);
    const uint8_t *ixl = idx + (int64_t)l * idx_per_layer;
    for (int s = 0; s < 16; ++s) hist[s][t] = 0;
    for (int64_t r = r0; r < r1; ++r) {
        const rolesub_segment sg = segs[row_seg[r]];
        const int k = sg.k;
        const uint8_t *ix = ixl + sg.idx_off + (r - sg.token_row) * k;
        for (int j = 0; j < k; ++j) {
            const int grp = ix[j];
            if (grp < G)
                ++hist[grp][t];
            else
                report(status, ROLESUB_EDEVICE, (int)r);
        }
    }
    __syncthreads();
    {
        // warp w: exclusive scan of hist[w][0..511], 16 entries per lane
        int v[16], run = 0;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            v[e] = run;
            run += hist[warp][16 * lane + e];
        }
        int incl = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        const int excl = incl - run;
#pragma unroll
        for (int e = 0; e < 16; ++e) hist[warp][16 * lane + e] = excl + v[e];
        if (lane == 31) tot[warp] = incl;
    }
    __syncthreads();
    // the chunk's pairs start at the idx position of its first row (rows,
    // indices and packed slots are laid out in the same order)
    const rolesub_segment s0 = segs[row_seg[c0]];
    const int64_t pbase = s0.idx_off + (c0 - s0.token_row) * s0.k;
    if (t == 0) {
        int b = 0;
        int32_t *mt = meta + ((int64_t)l * chunks + c) * kDenseMetaStride;
        for (int s = 0; s < 16; ++s) {
            gbase[s] = b;
            b += tot[s];
            mt[s] = tot[s];
        }
        mt[16] = (int32_t)pbase;
    }
    __syncthreads();
    int2 *out = pairs + (int64_t)l * idx_per_layer + pbase;
    for (int64_t r = r0; r < r1; ++r) {
        const rolesub_segment sg = segs[row_seg[r]];
        const int k = sg.k;
        const int64_t i = r - sg.token_row;
        const uint8_t *ix = ixl + sg.idx_off + i * k;
        const int64_t slot0 = sg.packed_off / g + i * k;
        for (int j = 0; j < k; ++j) {
            const int grp = ix[j];
            if (grp >= G) continue;
            const int pos = gbase[grp] + hist[grp][t]++;
            out[pos] = make_int2((int)r, (int)(slot0 + j));
        }
    }
}

constexpr int kSortThreads = 1024;
constexpr int kSortBins = 1 + 16 * 256;  // k = 0, then (k - 1, lowest, second lowest kept group)
constexpr int kSortPer = (kSortBins + kSortThreads - 1) / kSortThreads;

__device__ __forceinline__ int dense_key(const rolesub_segment *segs, const int32_t *row_seg, const uint8_t *ixl,
                                         int64_t r, int G)
{
    const rolesub_segment sg = segs[row_seg[r]];
    const int k = sg.k;
    if (k == 0) return 0;
    const uint8_t *ix = ixl + sg.idx_off + (r - sg.token_row) * k;
    int f1 = 255, f2 = 255;
    for (int j = 0; j < k; ++j) {
        const int x = min((int)ix[j], G - 1);  // a bad index is reported by the GEMM
        if (x < f1) {
            f2 = f1;
            f1 = x;
        } else if (x < f2) {
            f2 = x;
        }
    }
    if (f2 == 255) f2 = f1;
    return 1 + (k - 1) * 256 + f1 * 16 + f2;
}

// One CTA per layer: counting sort of the rows by key (order within a key
// is whatever the shared-memory atomics give; each row's v~ does not depend
// on which rows share its tile), perm[p] = row, and the row's record.
__global__ void __launch_bounds__(kSortThreads)
k_dense_sort(const rolesub_segment *__restrict__ segs, const int32_t *__restrict__ row_seg, int64_t rows, int G,
             int d, int dh, const uint8_t *__restrict__ idx, int64_t idx_per_layer, int32_t *__restrict__ perm,
             uint4 *__restrict__ recs)
{
    __shared__ int hist[kSortBins];
    __shared__ int wsum[32];
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31, l = blockIdx.x;
    const uint8_t *ixl = idx + (int64_t)l * idx_per_layer;
    for (int b = t; b < kSortBins; b += kSortThreads) hist[b] = 0;
    __syncthreads();
    for (int64_t r = t; r < rows; r += kSortThreads) atomicAdd(&hist[dense_key(segs, row_seg, ixl, r, G)], 1);
    __syncthreads();
    {
        int loc[kSortPer], sum = 0;
#pragma unroll
        for (int e = 0; e < kSortPer; ++e) {
            const int b = t * kSortPer + e;
            loc[e] = sum;
            sum += b < kSortBins ? hist[b] : 0;
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const int w = wsum[lane];
            int wi = w;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, wi, o);
                if (lane >= o) wi += y;
            }
            wsum[lane] = wi - w;
        }
        __syncthreads();
        const int excl = wsum[warp] + incl - sum;
#pragma unroll
        for (int e = 0; e < kSortPer; ++e) {
            const int b = t * kSortPer + e;
            if (b < kSortBins) hist[b] = excl + loc[e];
        }
    }
    __syncthreads();
    const uint32_t w3 = (16u << 27) | (uint32_t)(dh / 8);
    for (int64_t r = t; r < rows; r += kSortThreads) {
        const int pos = atomicAdd(&hist[dense_key(segs, row_seg, ixl, r, G)], 1);
        perm[(int64_t)l * rows + pos] = (int32_t)r;
        recs[(int64_t)l * rows + r] = make_uint4(0x76543210u, 0xFEDCBA98u, (uint32_t)((int64_t)pos * (d / 8)), w3);
    }
}

// Identity R_h of every (layer, head), bf16.
__global__ void __launch_bounds__(256)
k_identity(int64_t n_mats, int dh, bf16 *__restrict__ R)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t per = (int64_t)dh * dh;
    if (t >= n_mats * per) return;
    const int64_t e = t % per;
    R[t] = __float2bfloat16_rn((e / dh) == (e % dh) ? 1.f : 0.f);
}

}  // namespace

cudaError_t launch_dense_pairs(const PlanView &pv, int L, int g, const uint8_t *idx, int2 *pairs, int32_t *meta,
                               int chunks, int32_t *status, cudaStream_t stream)
{
    const rolesub_plan &P = *pv.hdr;
    if (P.rows_per_layer == 0 || L == 0 || chunks == 0) return cudaSuccess;
    k_dense_pairs<<<dim3((unsigned)chunks, (unsigned)L), kPairThreads, 0, stream>>>(
        pv.segs_dev, pv.row_seg_dev, P.rows_per_layer, P.num_groups, g, idx, P.idx_bytes_per_layer, pairs, meta,
        chunks, status);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_dense_sort(const PlanView &pv, int L, int d, int dh, const uint8_t *idx, int32_t *perm,
                              uint4 *recs, int32_t *status, cudaStream_t stream)
{
    (void)status;
    const rolesub_plan &P = *pv.hdr;
    if (P.rows_per_layer == 0 || L == 0) return cudaSuccess;
    k_dense_sort<<<(unsigned)L, kSortThreads, 0, stream>>>(pv.segs_dev, pv.row_seg_dev, P.rows_per_layer,
                                                            P.num_groups, d, dh, idx, P.idx_bytes_per_layer, perm,
                                                            recs);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_dense_identity(int L, int H, int dh, void *R_identity, cudaStream_t stream)
{
    const int64_t nm = (int64_t)L * H, ne = nm * dh * dh;
    if (ne == 0) return cudaSuccess;
    k_identity<<<(unsigned)((ne + 255) / 256), 256, 0, stream>>>(nm, dh, (bf16 *)R_identity);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
