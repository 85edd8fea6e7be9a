// budget.cu -- per-token value budgets (Sec. 3.5).
//
// Within one token type of one episode (a segment of n tokens with target
// K_m), the tokens share B_m = K_m n value groups: 0 <= K_i <= S and
// sum_i K_i = B_m, more for tokens of higher role-derived priority. The
// paper gives no formula for the allocator; the reading built here:
//   pi_i = u . a_i (a_i the latent role of Eq. latentrole, u per layer);
//   rank the tokens by (pi descending, token index ascending);
//   rank r gets the real share x_r = min(S, lambda (n - r)), lambda such that
//   sum x = B_m (the best ranks saturate at S first): with c saturated ranks,
//   x_r = rest (n - r) / W for r >= c, rest = B_m - cS, W = sum_{r>=c} (n - r);
//   K is x rounded by largest remainders (floor, plus one for the
//   rest - sum floor ranks with the largest remainder rest (n - r) mod W;
//   ties: the better rank) -- integer arithmetic once the ranks are known.
// Token i keeps its K_i highest-scoring groups (ties: lower index), stored
// ascending at the segment's index offset + sum_{j<i} K_j; its values at
// packed_off + (h B_m + sum_{j<i} K_j) d_s for head h.
//
// k_budget_select   one block per (segment, layer): ranks, counts, prefix
//                   offsets, top-K_i of the router's scores, indices, k_tok
//                   and the 16-byte store records the rotation and the
//                   attention kernels read.
// k_row_store_budget  the store records again from (idx, k_tok), for the
//                   attention call; counts or indices out of range are
//                   reported in the status word and that row stores nothing.
#include "common.cuh"
#include "internal.h"

namespace rs {

namespace {

constexpr int kBT = 256;   // threads per segment block
constexpr int kG = 16;     // groups (the tensor-core path's S)
constexpr uint64_t kIdentityIds = 0xFEDCBA9876543210ull;

// A total order on scores for the selectors, so that every ranking is a
// permutation whatever the data: NaN lowest, -0 equal to +0, otherwise the
// float order.
__device__ __forceinline__ uint32_t order_key(float x)
{
    if (x != x) return 0u;
    if (x == 0.f) x = 0.f;
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive prefix sums pre[0..n) of v[0..n) by the block; returns the
// total. part: kBT ints of shared scratch.
__device__ int block_scan(const uint8_t *v, int *pre, int n, int *part)
{
    const int tid = threadIdx.x;
    const int per = (n + kBT - 1) / kBT;
    const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
    int s = 0;
    for (int i = i0; i < i1; ++i) s += v[i];
    part[tid] = s;
    __syncthreads();
    for (int off = 1; off < kBT; off <<= 1) {
        const int x = tid >= off ? part[tid - off] : 0;
        __syncthreads();
        part[tid] += x;
        __syncthreads();
    }
    int run = tid > 0 ? part[tid - 1] : 0;
    for (int i = i0; i < i1; ++i) {
        pre[i] = run;
        run += v[i];
    }
    const int total = part[kBT - 1];
    __syncthreads();
    return total;
}

__device__ __forceinline__ uint4 record(uint64_t gid, int64_t base8, int k, int64_t stride)
{
    return make_uint4((uint32_t)gid, (uint32_t)(gid >> 32), (uint32_t)base8,
                      ((uint32_t)k << 27) | (uint32_t)stride);
}

// Shared memory: pri [n] order keys | rem [n] u32 | pre [n] i32 | kk [n] u8
__global__ void __launch_bounds__(kBT)
k_budget_select(PlanDev plan, int64_t rows, const float *scores, uint8_t *__restrict__ idx,
                int64_t idx_per_layer, uint8_t *__restrict__ k_tok, uint4 *__restrict__ recs)
{
    extern __shared__ __align__(16) uint8_t smb[];
    __shared__ int part[kBT];
    __shared__ int sh_c;
    __shared__ long long sh_left;
    pdl_trigger();
    pdl_wait();   // the scores come from the router kernel just before
    const int tid = threadIdx.x, l = blockIdx.y;
    const rolesub_segment sg = plan.segs[blockIdx.x];
    const int n = sg.n_tokens, km = sg.k;
    if (n == 0) return;
    uint32_t *pri = reinterpret_cast<uint32_t *>(smb);
    uint32_t *rem = reinterpret_cast<uint32_t *>(pri + n);
    int *pre = reinterpret_cast<int *>(rem + n);
    uint8_t *kk = reinterpret_cast<uint8_t *>(pre + n);
    const int64_t row0 = sg.token_row, lrow = (int64_t)l * rows;
    const int64_t B = (int64_t)km * n;
    uint8_t *ixl = idx + (int64_t)l * idx_per_layer + sg.idx_off;
    if (km == 0 || km == kG) {
        for (int i = tid; i < n; i += kBT) {
            const int64_t r = row0 + i;
            k_tok[lrow + r] = (uint8_t)km;
            if (km == kG)
                for (int s = 0; s < kG; ++s) ixl[(int64_t)i * kG + s] = (uint8_t)s;
            recs[lrow + r] = record(km ? kIdentityIds : 0, sg.packed_off / 8 + (int64_t)i * km, km, B);
        }
        return;
    }
    for (int i = tid; i < n; i += kBT) pri[i] = order_key(ld_dep(scores + (lrow + row0 + i) * kScoreStride + kG));
    if (tid == 0) {
        int c = 0;   // saturated ranks: the first c whose largest unsaturated share is <= S
        for (; c < n; ++c) {
            const long long rest = B - (long long)c * kG, W = (long long)(n - c) * (n - c + 1) / 2;
            if (rest * (long long)(n - c) <= (long long)kG * W) break;
        }
        sh_c = c;
    }
    __syncthreads();
    const int c = sh_c;
    const long long rest = B - (long long)c * kG, W = (long long)(n - c) * (n - c + 1) / 2;
    // remainders of the unsaturated ranks and the sum of their floors
    long long fl = 0;
    for (int r = c + tid; r < n; r += kBT) {
        const long long num = rest * (long long)(n - r);
        fl += num / W;
        rem[r] = (uint32_t)(num % W);
    }
    for (int o = 16; o > 0; o >>= 1) fl += __shfl_xor_sync(0xffffffffu, fl, o);
    if ((tid & 31) == 0) part[tid >> 5] = (int)fl;
    __syncthreads();
    if (tid == 0) {
        long long t = 0;
        for (int w = 0; w < kBT / 32; ++w) t += part[w];
        sh_left = c < n ? rest - t : 0;
    }
    __syncthreads();
    const long long left = sh_left;
    // counts: rank by priority, then the share of that rank
    for (int i = tid; i < n; i += kBT) {
        const uint32_t p = pri[i];
        int rank = 0;
        for (int j = 0; j < n; ++j) {
            const uint32_t q = pri[j];
            rank += (q > p || (q == p && j < i)) ? 1 : 0;
        }
        int K;
        if (rank < c) {
            K = kG;
        } else {
            K = (int)(rest * (long long)(n - rank) / W);
            const uint32_t rr = rem[rank];
            long long before = 0;
            for (int r2 = c; r2 < n; ++r2) before += (rem[r2] > rr || (rem[r2] == rr && r2 < rank)) ? 1 : 0;
            if (before < left) ++K;
        }
        kk[i] = (uint8_t)K;
    }
    __syncthreads();
    block_scan(kk, pre, n, part);
    // top-K_i of the token's scores, indices ascending at its prefix offset
    for (int i = tid; i < n; i += kBT) {
        const int64_t r = row0 + i;
        const int K = kk[i];
        const float4 *sp = reinterpret_cast<const float4 *>(scores + (lrow + r) * kScoreStride);
        uint32_t gam[kG];
#pragma unroll
        for (int q = 0; q < kG / 4; ++q) {
            const float4 v = ld_dep(sp + q);
            gam[4 * q] = order_key(v.x);
            gam[4 * q + 1] = order_key(v.y);
            gam[4 * q + 2] = order_key(v.z);
            gam[4 * q + 3] = order_key(v.w);
        }
        uint8_t *dst = ixl + pre[i];
        uint64_t gid = 0;
        int pos = 0;
#pragma unroll
        for (int g = 0; g < kG; ++g) {
            int rk = 0;
#pragma unroll
            for (int g2 = 0; g2 < kG; ++g2) rk += (gam[g2] > gam[g] || (gam[g2] == gam[g] && g2 < g)) ? 1 : 0;
            if (rk < K) {
                dst[pos] = (uint8_t)g;
                gid |= (uint64_t)g << (4 * pos);
                ++pos;
            }
        }
        k_tok[lrow + r] = (uint8_t)K;
        recs[lrow + r] = record(gid, sg.packed_off / 8 + pre[i], K, B);
    }
}

// Store records from a budget cache's indices and counts (attention side).
__global__ void __launch_bounds__(kBT)
k_row_store_budget(PlanDev plan, int64_t rows, const uint8_t *__restrict__ idx, int64_t idx_per_layer,
                   const uint8_t *__restrict__ k_tok, uint4 *__restrict__ recs, int32_t *status)
{
    extern __shared__ __align__(16) uint8_t smb[];
    __shared__ int part[kBT];
    pdl_trigger();
    const int tid = threadIdx.x, l = blockIdx.y;
    const rolesub_segment sg = plan.segs[blockIdx.x];
    const int n = sg.n_tokens;
    if (n == 0) return;
    int *pre = reinterpret_cast<int *>(smb);
    uint8_t *kk = reinterpret_cast<uint8_t *>(pre + n);
    const int64_t row0 = sg.token_row, lrow = (int64_t)l * rows;
    const int64_t B = (int64_t)sg.k * n;
    for (int i = tid; i < n; i += kBT) {
        int K = k_tok[lrow + row0 + i];
        if (K > kG) {
            report(status, ROLESUB_EDEVICE, (int)(row0 + i));
            K = 0;
        }
        kk[i] = (uint8_t)K;
    }
    __syncthreads();
    block_scan(kk, pre, n, part);
    const uint8_t *ixl = idx + (int64_t)l * idx_per_layer + sg.idx_off;
    for (int i = tid; i < n; i += kBT) {
        const int64_t r = row0 + i;
        int K = kk[i];
        if (pre[i] + K > B) {   // counts beyond the segment's budget
            report(status, ROLESUB_EDEVICE, (int)r);
            K = 0;
        }
        uint64_t gid = 0;
        for (int s = 0; s < K; ++s) {
            const uint32_t g = ixl[pre[i] + s];
            if (g >= (uint32_t)kG) {
                report(status, ROLESUB_EDEVICE, (int)r);
                K = 0;
                gid = 0;
                break;
            }
            gid |= (uint64_t)g << (4 * s);
        }
        recs[lrow + r] = record(gid, sg.packed_off / 8 + pre[i], K, B);
    }
}

int max_segment_tokens(const PlanView &pv)
{
    int m = 0;
    for (int s = 0; s < pv.hdr->num_segments; ++s) m = pv.segs[s].n_tokens > m ? pv.segs[s].n_tokens : m;
    return m;
}

}  // namespace

cudaError_t launch_budget_select(const CompressArgs &a, const float *scores, uint8_t *k_tok)
{
    const rolesub_plan &P = *a.plan.hdr;
    if (P.rows_per_layer == 0 || P.num_segments == 0) return cudaSuccess;
    const int nmax = max_segment_tokens(a.plan);
    const size_t smem = (size_t)nmax * (4 + 4 + 4 + 1) + 16;
    cudaError_t err = cudaFuncSetAttribute(k_budget_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    const PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev, a.plan.stored_dev,
                     a.plan.route_tiles_dev};
    err = launch_pdl(k_budget_select, dim3((unsigned)P.num_segments, a.shape->num_layers), dim3(kBT), smem, a.stream,
                     pd, (int64_t)P.rows_per_layer, scores, a.idx, (int64_t)P.idx_bytes_per_layer, k_tok,
                     reinterpret_cast<uint4 *>(a.ws.row_store));
    count_launches(1);
    return err;
}

cudaError_t launch_row_store_budget(const PlanView &pv, int L, const uint8_t *idx, int64_t idx_per_layer,
                                    const uint8_t *k_tok, uint4 *recs, int32_t *status, cudaStream_t stream)
{
    const rolesub_plan &P = *pv.hdr;
    if (P.rows_per_layer == 0 || P.num_segments == 0) return cudaSuccess;
    const int nmax = max_segment_tokens(pv);
    const size_t smem = (size_t)nmax * (4 + 1) + 16;
    cudaError_t err =
        cudaFuncSetAttribute(k_row_store_budget, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    const PlanDev pd{pv.segs_dev, pv.eps_dev, pv.row_seg_dev, pv.routed_dev, pv.stored_dev, pv.route_tiles_dev};
    k_row_store_budget<<<dim3((unsigned)P.num_segments, L), kBT, smem, stream>>>(pd, P.rows_per_layer, idx,
                                                                                idx_per_layer, k_tok, recs, status);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rs
