// router.cu -- role-conditioned value routing (Sec. 3.3-3.4).
//
// For every routed token i (segments with 0 < k < S) of layer l:
//   a_i   = softmax(W_re h_i + b_re)                       Eq. (latentrole)
//   u_i   = ReLU(W1_h h_i + W1_a (alpha_role a_i) + beta_e)
//   beta_e = W1_c (alpha_lang c_e) + b1, c_e = mean of the episode's
//            retained language hidden states                Sec. 3.4 Pool
//   gamma = W2 u_i + b2                                     Eq. (routingscore)
//   keep the k largest gamma (ties: lower index), written ascending.
// W1's input columns are [h (d) | role (C) | language (d)].
//
// Kernels: k_lang_pool -> k_lang_bias (per episode), then the token GEMM
// [W1_h ; W_re] h_i and the per-token epilogue with the top-k selector.
#include "common.cuh"
#include "internal.h"

namespace rs {

template <class T>
__global__ void k_lang_pool(const T *__restrict__ h, const rolesub_episode *__restrict__ eps,
                            int E, int64_t rows, int d, float *__restrict__ ctx)
{
    const int l = blockIdx.z, e = blockIdx.y;
    const int col = blockIdx.x * blockDim.x + threadIdx.x;
    if (col >= d) return;
    const rolesub_episode ep = eps[e];
    const T *base = h + ((size_t)l * rows + ep.lang_row_begin) * d + col;
    float s = 0.f;
    for (int j = 0; j < ep.n_lang; ++j) s += to_f(base[(size_t)j * d]);
    ctx[((size_t)l * E + e) * d + col] = ep.n_lang > 0 ? s / (float)ep.n_lang : 0.f;
}

// bf16, d % 8 == 0: a block covers 512 columns of one (layer, episode); a
// thread sums eight adjacent columns (one 16-byte load per row) over every
// fourth language row, four rows in flight, and the four row classes are
// added in a fixed order (0, 1, 2, 3) through shared memory, so the result
// does not depend on timing.
constexpr int kPoolParts = 4;

__global__ void __launch_bounds__(256)
k_lang_pool_v8(const __nv_bfloat16 *__restrict__ h, const rolesub_episode *__restrict__ eps, int E, int64_t rows,
               int d, float *__restrict__ ctx)
{
    __shared__ float part[kPoolParts - 1][64][9];
    pdl_trigger();
    const int l = blockIdx.z, e = blockIdx.y;
    const int cl = threadIdx.x & 63, p = threadIdx.x >> 6;
    const int c8 = blockIdx.x * 64 + cl;
    const bool live = 8 * c8 < d;
    const rolesub_episode ep = eps[e];
    const uint4 *base = reinterpret_cast<const uint4 *>(h + ((size_t)l * rows + ep.lang_row_begin) * d) + c8;
    const size_t stride = (size_t)d / 8;
    float s[8] = {};
    const int n = live ? ep.n_lang : 0;
    auto add = [&](const uint4 &v) {
        const __nv_bfloat162 *q2 = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(q2[i]);
            s[2 * i] += f.x;
            s[2 * i + 1] += f.y;
        }
    };
    int j = p;
    for (; j + 3 * kPoolParts < n; j += 4 * kPoolParts) {
        uint4 v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) v[q] = __ldg(base + (size_t)(j + kPoolParts * q) * stride);
#pragma unroll
        for (int q = 0; q < 4; ++q) add(v[q]);
    }
    for (; j < n; j += kPoolParts) add(__ldg(base + (size_t)j * stride));
    if (p > 0) {
#pragma unroll
        for (int i = 0; i < 8; ++i) part[p - 1][cl][i] = s[i];
    }
    __syncthreads();
    if (p > 0 || !live) return;
#pragma unroll
    for (int q = 0; q < kPoolParts - 1; ++q)
#pragma unroll
        for (int i = 0; i < 8; ++i) s[i] += part[q][cl][i];
    const float fn = (float)n;
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i] = n > 0 ? s[i] / fn : 0.f;
    float *out = ctx + ((size_t)l * E + e) * d + 8 * c8;
    *reinterpret_cast<float4 *>(out) = make_float4(s[0], s[1], s[2], s[3]);
    *reinterpret_cast<float4 *>(out + 4) = make_float4(s[4], s[5], s[6], s[7]);
}

// beta[l][e][f] = b1[f] + alpha_lang * W1[f][d+C : 2d+C] . ctx[l][e]
// A small GEMM per layer (episodes x F x d) in fp32. A cluster of four
// blocks shares one 64-episode x 32-output tile, each block a quarter of d;
// every thread holds 4 episodes x 2 outputs. d runs in 64-wide steps through
// shared memory, the next step's tiles loaded into registers meanwhile.
// Ranks 1-3 then add into rank 0 through distributed shared memory, in rank
// order, so the sum does not depend on timing.
constexpr int kBiasSplit = 4;

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <class T>
__global__ void __cluster_dims__(kBiasSplit, 1, 1) __launch_bounds__(256)
k_lang_bias(const T *__restrict__ W1, const float *__restrict__ b1, const float *__restrict__ ctx,
            int E, int d, int C, int F, float alpha_lang, float *__restrict__ beta)
{
    constexpr int BE = 64, BF = 32, BK = 64, PE = BE + 4, PF = BF + 4;   // padded pitches
    // Cs [t][e] and Ws [t][f]; afterwards the whole array holds the partial
    // sums of ranks 1-3 (3 x 256 x 8 floats)
    __shared__ __align__(16) float tiles[BK * PE + BK * PF];
    static_assert(BK * PE + BK * PF >= (kBiasSplit - 1) * 256 * 8, "reduction buffer");
    float(*Cs)[PE] = reinterpret_cast<float(*)[PE]>(tiles);
    float(*Ws)[PF] = reinterpret_cast<float(*)[PF]>(tiles + BK * PE);
    const int l = blockIdx.z, tid = threadIdx.x;
    const uint32_t rank = cluster_rank();
    const int f0 = (blockIdx.x / kBiasSplit) * BF, e0 = blockIdx.y * BE;
    const int kper = ((d + kBiasSplit * BK - 1) / (kBiasSplit * BK)) * BK;
    const int kb = (int)rank * kper, ke = min(d, kb + kper);
    const int te = tid & 15, tf = tid >> 4;       // episodes e0 + 4te + i, outputs f0 + 2tf + j
    const size_t wstride = (size_t)(2 * d + C);
    const T *wbase = W1 + (size_t)l * F * wstride + d + C;
    const float *cbase = ctx + (size_t)l * E * d;
    // loaders, t fastest across a warp so that global reads are coalesced:
    // ctx 64 episodes x 64 t (16 per thread), W 32 outputs x 64 t (8 per thread)
    const int lt = tid & 63, lr = tid >> 6;
    float cr[16], wr[8];
    auto fetch = [&](int k0) {
        const int t = k0 + lt;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int e = e0 + lr + 4 * i;
            cr[i] = (e < E && t < ke) ? cbase[(size_t)e * d + t] : 0.f;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int f = f0 + lr + 4 * i;
            wr[i] = (f < F && t < ke) ? to_f(wbase[(size_t)f * wstride + t]) : 0.f;
        }
    };
    float acc[8] = {};   // [i][j] = acc[2i + j]
    if (kb < ke) fetch(kb);
    for (int k0 = kb; k0 < ke; k0 += BK) {
        __syncthreads();   // previous step's tiles are consumed
#pragma unroll
        for (int i = 0; i < 16; ++i) Cs[lt][lr + 4 * i] = cr[i];
#pragma unroll
        for (int i = 0; i < 8; ++i) Ws[lt][lr + 4 * i] = wr[i];
        __syncthreads();
        if (k0 + BK < ke) fetch(k0 + BK);
#pragma unroll 16
        for (int t = 0; t < BK; ++t) {
            const float4 c = *reinterpret_cast<const float4 *>(&Cs[t][4 * te]);
            const float2 w = *reinterpret_cast<const float2 *>(&Ws[t][2 * tf]);
            acc[0] = fmaf(c.x, w.x, acc[0]);
            acc[1] = fmaf(c.x, w.y, acc[1]);
            acc[2] = fmaf(c.y, w.x, acc[2]);
            acc[3] = fmaf(c.y, w.y, acc[3]);
            acc[4] = fmaf(c.z, w.x, acc[4]);
            acc[5] = fmaf(c.z, w.y, acc[5]);
            acc[6] = fmaf(c.w, w.x, acc[6]);
            acc[7] = fmaf(c.w, w.y, acc[7]);
        }
    }
    // every block is done with its tiles; ranks 1-3 write their partial sums
    // into rank 0's tile array, thread-major
    __syncthreads();
    cluster_sync();
    if (rank != 0) {
        const uint32_t local = static_cast<uint32_t>(__cvta_generic_to_shared(tiles)) +
                               4u * (((rank - 1) * 256u + (uint32_t)tid) * 8u);
        uint32_t remote;
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(0u));
#pragma unroll
        for (int q = 0; q < 8; ++q)
            asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote + 4u * q), "f"(acc[q]) : "memory");
    }
    cluster_sync();
    if (rank != 0) return;
    const float *red = tiles;
#pragma unroll
    for (int r = 0; r < kBiasSplit - 1; ++r)
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] += red[(r * 256 + tid) * 8 + q];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int e = e0 + 4 * te + i;
        if (e >= E) continue;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const int f = f0 + 2 * tf + j;
            if (f < F) beta[((size_t)l * E + e) * F + f] = b1[(size_t)l * F + f] + alpha_lang * acc[2 * i + j];
        }
    }
}

// bf16 weights, at most kGemvEpisodes episodes (a single control step): the
// product is a matrix-vector one, bound by reading W1_c once. A warp per
// output f walks W1_c's row with 16-byte loads (eight weights per lane and
// step), multiplies by the episodes' ctx in fp32 and sums the lanes with a
// butterfly. The block's 8 warps share the layer's contexts, staged once in
// shared memory after the wait; each lane's first kGemvBatch weight loads are
// issued before it (W1 is a caller input), later ones a batch at a time, so
// that the weight stream keeps loads in flight. Needs d % 8 == 0 and
// C % 8 == 0 (16-byte weight rows).
constexpr int kGemvEpisodes = 4;
constexpr int kGemvBatch = 8;

__global__ void __launch_bounds__(256)
k_lang_bias_gemv(const __nv_bfloat16 *__restrict__ W1, const float *__restrict__ b1, const float *ctx,
                 int E, int d, int C, int F, float alpha_lang, float *__restrict__ beta)
{
    extern __shared__ float4 csm[];   // [E][d / 4]: the layer's contexts
    const int l = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int f = blockIdx.x * 8 + warp;
    const bool live = f < F;
    const uint4 *w =
        reinterpret_cast<const uint4 *>(W1 + ((size_t)l * F + (live ? f : 0)) * (size_t)(2 * d + C) + d + C);
    const int n8 = d / 8;
    pdl_trigger();
    uint4 wb[kGemvBatch];
#pragma unroll
    for (int j = 0; j < kGemvBatch; ++j) {
        const int k8 = lane + 32 * j;
        wb[j] = live && k8 < n8 ? __ldg(w + k8) : make_uint4(0, 0, 0, 0);
    }
    pdl_wait();   // ctx comes from the pooling kernel
    {
        const float4 *c4 = reinterpret_cast<const float4 *>(ctx + (size_t)l * E * d);
        const int nc = E * (d / 4);
        for (int i0 = threadIdx.x; i0 < nc; i0 += 4 * 256) {
            float4 t[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = i0 + 256 * q;
                t[q] = i < nc ? ld_dep(c4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (i0 + 256 * q < nc) csm[i0 + 256 * q] = t[q];
        }
    }
    __syncthreads();
    if (!live) return;
    float acc[kGemvEpisodes] = {};
    for (int j0 = 0; 32 * j0 < n8; j0 += kGemvBatch) {
        if (j0 > 0) {
#pragma unroll
            for (int j = 0; j < kGemvBatch; ++j) {
                const int k8 = lane + 32 * (j0 + j);
                wb[j] = k8 < n8 ? __ldg(w + k8) : make_uint4(0, 0, 0, 0);
            }
        }
#pragma unroll
        for (int j = 0; j < kGemvBatch; ++j) {
            const int k8 = lane + 32 * (j0 + j);
            if (k8 >= n8) break;
            const __nv_bfloat162 *wp = reinterpret_cast<const __nv_bfloat162 *>(&wb[j]);
            float wf[8];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 t = __bfloat1622float2(wp[i]);
                wf[2 * i] = t.x;
                wf[2 * i + 1] = t.y;
            }
#pragma unroll
            for (int e = 0; e < kGemvEpisodes; ++e) {
                if (e >= E) break;
                const float4 x0 = csm[e * (d / 4) + 2 * k8], x1 = csm[e * (d / 4) + 2 * k8 + 1];
                float a = acc[e];
                a = fmaf(wf[0], x0.x, a);
                a = fmaf(wf[1], x0.y, a);
                a = fmaf(wf[2], x0.z, a);
                a = fmaf(wf[3], x0.w, a);
                a = fmaf(wf[4], x1.x, a);
                a = fmaf(wf[5], x1.y, a);
                a = fmaf(wf[6], x1.z, a);
                a = fmaf(wf[7], x1.w, a);
                acc[e] = a;
            }
        }
    }
#pragma unroll
    for (int e = 0; e < kGemvEpisodes; ++e) {
        if (e >= E) break;
        const float v = warp_sum(acc[e]);
        if (lane == 0) beta[((size_t)l * E + e) * F + f] = b1[(size_t)l * F + f] + alpha_lang * v;
    }
}

// bf16 weights: the same product on the tensor cores (mma.sync m16n8k16,
// fp32 accumulation). ctx is split into bf16 parts hi + lo (together exact to
// about 2^-16 relative) and both are multiplied by the bf16 weights. Block:
// 64 episodes x 64 outputs x 1/kSplit of d, four warps of 16 episodes each;
// a cluster of kSplit blocks along d reduces through distributed shared
// memory: rank r owns 8/kSplit of the eight 8-output column tiles, receives
// every rank's partial sums for them and adds them in rank order, so the
// result does not depend on timing. kSplit = 8 (d % 512 == 0) keeps each
// block's walk over d short; kSplit = 2 needs d % 128 == 0. C % 8 == 0
// (16-byte weight rows) in both.

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1)
{
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
                 "{%8, %9}, {%0, %1, %2, %3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack2(float a, float b)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

template <int kSplit>
__global__ void __cluster_dims__(kSplit, 1, 1) __launch_bounds__(128)
k_lang_bias_mma(const __nv_bfloat16 *__restrict__ W1, const float *__restrict__ b1, const float *ctx,
                int E, int d, int C, int F, float alpha_lang, float *__restrict__ beta)
{
    constexpr int BE = 64, BF = 64, BK = 64;
    // rows of 64 bf16 (128 B) as 8 16-byte chunks, chunk c of row r stored at
    // position c ^ (r % 8) so that ldmatrix rows hit distinct banks
    __shared__ __align__(128) uint8_t sm[3 * BE * BK * 2];   // A hi, A lo, B; later rank 1's sums
    const uint32_t sA0 = static_cast<uint32_t>(__cvta_generic_to_shared(sm));
    const uint32_t sA1 = sA0 + BE * BK * 2, sBs = sA1 + BE * BK * 2;
    pdl_trigger();
    pdl_wait();   // ctx comes from the pooling kernel
    const int l = blockIdx.z, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_rank();
    const int f0 = (blockIdx.x / kSplit) * BF, e0 = blockIdx.y * BE;
    const int kper = d / kSplit;
    const int kb = (int)rank * kper, ke = kb + kper;
    const size_t wstride = (size_t)(2 * d + C);
    const __nv_bfloat16 *wbase = W1 + (size_t)l * F * wstride + d + C;
    const float *cbase = ctx + (size_t)l * E * d;
    float4 cr[8];
    uint4 wr[4];
    auto fetch = [&](int k0) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {   // ctx: row e, float4 kq of the 64-wide step
            const int idx = tid + 128 * j, e = e0 + (idx >> 4), kq = idx & 15;
            cr[j] = e < E ? ld_dep(reinterpret_cast<const float4 *>(cbase + (size_t)e * d + k0 + 4 * kq))
                          : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {   // W: row f, 16-byte chunk c
            const int idx = tid + 128 * j, f = f0 + (idx >> 3), c = idx & 7;
            wr[j] = f < F ? *reinterpret_cast<const uint4 *>(wbase + (size_t)f * wstride + k0 + 8 * c)
                          : make_uint4(0, 0, 0, 0);
        }
    };
    float acc[8][4] = {};
    fetch(kb);
    for (int k0 = kb; k0 < ke; k0 += BK) {
        __syncthreads();   // previous step's tiles are consumed
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int idx = tid + 128 * j, e = idx >> 4, kq = idx & 15;
            const float4 v = cr[j];
            const uint32_t h0 = pack2(v.x, v.y), h1 = pack2(v.z, v.w);
            const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
            const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
            const uint32_t l0 = pack2(v.x - __low2float(hb0), v.y - __high2float(hb0));
            const uint32_t l1 = pack2(v.z - __low2float(hb1), v.w - __high2float(hb1));
            const uint32_t off = (uint32_t)e * 128u + ((((uint32_t)kq >> 1) ^ ((uint32_t)e & 7u)) << 4) +
                                 ((uint32_t)kq & 1u) * 8u;
            asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(sA0 + off), "r"(h0), "r"(h1) : "memory");
            asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(sA1 + off), "r"(l0), "r"(l1) : "memory");
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int idx = tid + 128 * j, f = idx >> 3, c = idx & 7;
            const uint32_t off = (uint32_t)f * 128u + (((uint32_t)c ^ ((uint32_t)f & 7u)) << 4);
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(sBs + off), "r"(wr[j].x), "r"(wr[j].y),
                         "r"(wr[j].z), "r"(wr[j].w)
                         : "memory");
        }
        __syncthreads();
        if (k0 + BK < ke) fetch(k0 + BK);
#pragma unroll
        for (int s16 = 0; s16 < BK / 16; ++s16) {
            const uint32_t ar = (uint32_t)(16 * warp + (lane & 15));
            const uint32_t aoff = ar * 128u + ((((uint32_t)(2 * s16 + (lane >> 4))) ^ (ar & 7u)) << 4);
            uint32_t ah[4], al[4];
            ldsm_x4(sA0 + aoff, ah[0], ah[1], ah[2], ah[3]);
            ldsm_x4(sA1 + aoff, al[0], al[1], al[2], al[3]);
#pragma unroll
            for (int pr = 0; pr < 4; ++pr) {   // output tiles 2pr, 2pr + 1
                const uint32_t n = (uint32_t)(16 * pr + (lane & 7) + ((lane >> 4) << 3));
                const uint32_t boff = n * 128u + ((((uint32_t)(2 * s16 + ((lane >> 3) & 1))) ^ (n & 7u)) << 4);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(sBs + boff, b0, b1, b2, b3);
                mma_16816(acc[2 * pr], ah[0], ah[1], ah[2], ah[3], b0, b1);
                mma_16816(acc[2 * pr], al[0], al[1], al[2], al[3], b0, b1);
                mma_16816(acc[2 * pr + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
                mma_16816(acc[2 * pr + 1], al[0], al[1], al[2], al[3], b2, b3);
            }
        }
    }
    // every rank sends column tiles j of its sums to the rank that owns them:
    // slot ((q * 128 + tid) * J + jj) of rank r holds rank q's tile r J + jj
    constexpr int J = 8 / kSplit;
    static_assert(kSplit * 128 * J * 16 <= (int)sizeof(sm), "reduction buffer");
    __syncthreads();
    cluster_sync();
    {
        const uint32_t local = sA0 + 16u * ((rank * 128u + (uint32_t)tid) * (uint32_t)J);
#pragma unroll
        for (int r = 0; r < kSplit; ++r) {
            uint32_t remote;
            asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"((uint32_t)r));
#pragma unroll
            for (int jj = 0; jj < J; ++jj)
                asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote + 16u * jj),
                             "f"(acc[r * J + jj][0]), "f"(acc[r * J + jj][1]), "f"(acc[r * J + jj][2]),
                             "f"(acc[r * J + jj][3])
                             : "memory");
        }
    }
    cluster_sync();
    const float4 *red = reinterpret_cast<const float4 *>(sm);
    const int g = lane >> 2, t2 = 2 * (lane & 3);
#pragma unroll
    for (int jj = 0; jj < J; ++jj) {
        float4 v = red[tid * J + jj];
#pragma unroll
        for (int q = 1; q < kSplit; ++q) {
            const float4 w = red[(q * 128 + tid) * J + jj];
            v.x += w.x;
            v.y += w.y;
            v.z += w.z;
            v.w += w.w;
        }
        const float o[4] = {v.x, v.y, v.z, v.w};
        const int j = (int)rank * J + jj;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int e = e0 + 16 * warp + g + 8 * hh;
            if (e >= E) continue;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const int f = f0 + 8 * j + t2 + q;
                if (f < F) beta[((size_t)l * E + e) * F + f] = b1[(size_t)l * F + f] + alpha_lang * o[2 * hh + q];
            }
        }
    }
}

// logits[l][m][n] for routed token m: n < F -> W1_h[n] . h, n >= F -> W_re[n-F] . h + b_re.
template <class T>
__global__ void __launch_bounds__(256)
k_router_gemm_simt(const T *__restrict__ h, const int32_t *__restrict__ routed, int64_t M,
                   int64_t rows, int d, int C, int F, const T *__restrict__ W1,
                   const T *__restrict__ W_re, const float *__restrict__ b_re,
                   float *__restrict__ out)
{
    constexpr int BM = 64, BN = 64, BK = 32;
    __shared__ float As[BK][BM + 4];
    __shared__ float Bs[BK][BN + 4];
    const int l = blockIdx.z;
    const int64_t m0 = (int64_t)blockIdx.x * BM;
    const int n0 = blockIdx.y * BN;
    const int N = F + C;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < d; k0 += BK) {
        for (int i = threadIdx.x; i < BM * BK; i += 256) {
            const int mm = i / BK, kk = i % BK;
            const int64_t m = m0 + mm;
            float x = 0.f;
            if (m < M && k0 + kk < d) x = to_f(h[((size_t)l * rows + routed[m]) * d + k0 + kk]);
            As[kk][mm] = x;
        }
        for (int i = threadIdx.x; i < BN * BK; i += 256) {
            const int nn = i / BK, kk = i % BK;
            const int n = n0 + nn;
            float x = 0.f;
            if (n < N && k0 + kk < d) {
                x = n < F ? to_f(W1[((size_t)l * F + n) * (size_t)(2 * d + C) + k0 + kk])
                          : to_f(W_re[((size_t)l * C + (n - F)) * d + k0 + kk]);
            }
            Bs[kk][nn] = x;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < BK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (n >= N) continue;
            const float bias = n >= F ? b_re[(size_t)l * C + (n - F)] : 0.f;
            out[((size_t)l * M + m) * N + n] = acc[i][j] + bias;
        }
    }
}

// One warp per routed token: role softmax, hidden layer, output layer, top-k.
template <class T>
__global__ void __launch_bounds__(256)
k_router_epilogue(const float *__restrict__ logits, PlanDev plan, int64_t M, int d, int C, int F,
                  int G, int E, const T *__restrict__ W1, const float *__restrict__ beta,
                  const T *__restrict__ W2, const float *__restrict__ b2, float alpha_role,
                  uint8_t *__restrict__ idx, int64_t idx_per_layer)
{
    extern __shared__ float sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t m = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp;
    const int l = blockIdx.y;
    if (m >= M) return;
    float *a = sm + (size_t)warp * (C + F);
    float *u = a + C;
    const int N = F + C;
    const float *lg = logits + ((size_t)l * M + m) * N;
    const int row = plan.routed[m];
    const rolesub_segment sg = plan.segs[plan.row_seg[row]];

    float mx = -INFINITY;
    for (int c = lane; c < C; c += 32) mx = fmaxf(mx, lg[F + c]);
    mx = warp_max(mx);
    float s = 0.f;
    for (int c = lane; c < C; c += 32) {
        const float e = expf(lg[F + c] - mx);
        a[c] = e;
        s += e;
    }
    s = warp_sum(s);
    __syncwarp();
    const float sc = alpha_role / s;
    for (int c = lane; c < C; c += 32) a[c] *= sc;
    __syncwarp();

    const float *be = beta + ((size_t)l * E + sg.episode) * F;
    for (int f = lane; f < F; f += 32) {
        const T *w = W1 + ((size_t)l * F + f) * (size_t)(2 * d + C) + d;
        float acc = lg[f] + be[f];
        for (int c = 0; c < C; ++c) acc = fmaf(to_f(w[c]), a[c], acc);
        u[f] = fmaxf(acc, 0.f);
    }
    __syncwarp();

    float gam = -INFINITY;
    for (int g = 0; g < G; ++g) {
        const T *w = W2 + ((size_t)l * G + g) * F;
        float acc = 0.f;
        for (int f = lane; f < F; f += 32) acc = fmaf(to_f(w[f]), u[f], acc);
        acc = warp_sum(acc);
        if (lane == g) gam = acc + b2[(size_t)l * G + g];
    }
    // rank of every group under (gamma desc, index asc); keep rank < k
    int rank = 0;
    for (int g = 0; g < G; ++g) {
        const float o = __shfl_sync(0xffffffffu, gam, g);
        if (o > gam || (o == gam && g < lane)) ++rank;
    }
    const int k = sg.k;
    const bool keep = lane < G && rank < k;
    const unsigned ball = __ballot_sync(0xffffffffu, keep);
    const int pos = __popc(ball & ((1u << lane) - 1u));
    if (keep && pos < k) {   // pos < k: NaN scores rank 0 and must not overflow the row
        const int64_t ti = row - sg.token_row;
        idx[(size_t)l * idx_per_layer + sg.idx_off + ti * k + pos] = (uint8_t)lane;
    }
}

bool router_supported(const rolesub_shape *s)
{
    return s->role_dim + s->router_hidden <= 1536 && s->num_groups <= 32;
}

cudaError_t launch_lang_pool(const CompressArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    const int L = S.num_layers, E = P.num_episodes, d = S.num_heads * S.head_dim;
    if (S.dtype == ROLESUB_BF16 && d % 8 == 0 && ((uintptr_t)a.h & 15) == 0)
        k_lang_pool_v8<<<dim3((d / 8 + 63) / 64, E, L), 256, 0, a.stream>>>(
            (const __nv_bfloat16 *)a.h, a.plan.eps_dev, E, P.rows_per_layer, d, a.ws.lang_ctx);
    else if (S.dtype == ROLESUB_BF16)
        k_lang_pool<__nv_bfloat16><<<dim3((d + 255) / 256, E, L), 256, 0, a.stream>>>(
            (const __nv_bfloat16 *)a.h, a.plan.eps_dev, E, P.rows_per_layer, d, a.ws.lang_ctx);
    else
        k_lang_pool<float><<<dim3((d + 255) / 256, E, L), 256, 0, a.stream>>>(
            (const float *)a.h, a.plan.eps_dev, E, P.rows_per_layer, d, a.ws.lang_ctx);
    count_launches(1);
    return cudaGetLastError();
}

template <class T>
static cudaError_t launch_router_t(const CompressArgs &a)
{
    const rolesub_shape &S = *a.shape;
    const rolesub_plan &P = *a.plan.hdr;
    const int L = S.num_layers, E = P.num_episodes, d = S.num_heads * S.head_dim;
    const int C = S.role_dim, F = S.router_hidden, G = S.num_groups;
    const int64_t M = P.routed_rows_per_layer;
    if (M == 0) return cudaSuccess;
    const T *h = (const T *)a.h, *W1 = (const T *)a.W1, *Wre = (const T *)a.W_re,
            *W2 = (const T *)a.W2;
    cudaError_t err = launch_lang_pool(a);
    if (err != cudaSuccess) return err;
    const size_t gemv_smem = (size_t)E * d * sizeof(float);
    if (sizeof(T) == 2 && E <= kGemvEpisodes && d % 8 == 0 && C % 8 == 0 && ((uintptr_t)a.W1 & 15) == 0 &&
        gemv_smem <= 200 * 1024) {
        err = cudaFuncSetAttribute(k_lang_bias_gemv, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemv_smem);
        if (err == cudaSuccess)
            err = launch_pdl(k_lang_bias_gemv, dim3((F + 7) / 8, L), dim3(256), gemv_smem, a.stream,
                             (const __nv_bfloat16 *)a.W1, a.b1, (const float *)a.ws.lang_ctx, E, d, C, F,
                             a.alpha_lang, a.ws.lang_bias);
    }
    else if (sizeof(T) == 2 && d % 512 == 0 && C % 8 == 0 && ((uintptr_t)a.W1 & 15) == 0)
        err = launch_pdl(k_lang_bias_mma<8>, dim3((F + 63) / 64 * 8, (E + 63) / 64, L), dim3(128), 0, a.stream,
                         (const __nv_bfloat16 *)a.W1, a.b1, (const float *)a.ws.lang_ctx, E, d, C, F, a.alpha_lang,
                         a.ws.lang_bias);
    else if (sizeof(T) == 2 && d % 128 == 0 && C % 8 == 0 && ((uintptr_t)a.W1 & 15) == 0)
        err = launch_pdl(k_lang_bias_mma<2>, dim3((F + 63) / 64 * 2, (E + 63) / 64, L), dim3(128), 0, a.stream,
                         (const __nv_bfloat16 *)a.W1, a.b1, (const float *)a.ws.lang_ctx, E, d, C, F, a.alpha_lang,
                         a.ws.lang_bias);
    else
        k_lang_bias<T><<<dim3((F + 31) / 32 * kBiasSplit, (E + 63) / 64, L), 256, 0, a.stream>>>(
            W1, a.b1, a.ws.lang_ctx, E, d, C, F, a.alpha_lang, a.ws.lang_bias);
    if (err != cudaSuccess) return err;
    if (router_tc_supported(a.shape)) {
        count_launches(1);
        cudaError_t e = cudaGetLastError();
        return e != cudaSuccess ? e : launch_router_tc(a);
    }
    k_router_gemm_simt<T><<<dim3((unsigned)((M + 63) / 64), (F + C + 63) / 64, L), 256, 0, a.stream>>>(
        h, a.plan.routed_dev, M, P.rows_per_layer, d, C, F, W1, Wre, a.b_re, a.ws.logits);
    PlanDev pd{a.plan.segs_dev, a.plan.eps_dev, a.plan.row_seg_dev, a.plan.routed_dev,
               a.plan.stored_dev};
    const size_t smem = (size_t)8 * (C + F) * sizeof(float);
    k_router_epilogue<T><<<dim3((unsigned)((M + 7) / 8), L), 256, smem, a.stream>>>(
        a.ws.logits, pd, M, d, C, F, G, E, W1, a.ws.lang_bias, W2, a.b2, a.alpha_role, a.idx,
        P.idx_bytes_per_layer);
    count_launches(3);
    return cudaGetLastError();
}

cudaError_t launch_router(const CompressArgs &a)
{
    if (a.shape->dtype == ROLESUB_BF16) return launch_router_t<__nv_bfloat16>(a);
    return launch_router_t<float>(a);
}

}  // namespace rs
