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

// beta[l][e][f] = b1[f] + alpha_lang * W1[f][d+C : 2d+C] . ctx[l][e]
// A small GEMM per layer (episodes x F x d): 16 episodes x 64 outputs per
// block, the hidden dimension streamed through shared memory in 64-wide
// steps; every thread owns one episode and four outputs.
template <class T>
__global__ void __launch_bounds__(256)
k_lang_bias(const T *__restrict__ W1, const float *__restrict__ b1, const float *__restrict__ ctx,
            int E, int d, int C, int F, float alpha_lang, float *__restrict__ beta)
{
    constexpr int BE = 16, BF = 64, BK = 64, WP = BF + 4;   // WP: padded row pitch
    __shared__ __align__(16) float Ws[BK * WP];             // [t][f]
    __shared__ float Cs[BE][BK + 1];                        // [e][t]
    const int l = blockIdx.z;
    const int f0 = blockIdx.x * BF, e0 = blockIdx.y * BE;
    const int te = threadIdx.x >> 4, tf = threadIdx.x & 15;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    const size_t wstride = (size_t)(2 * d + C);
    for (int k0 = 0; k0 < d; k0 += BK) {
        for (int i = threadIdx.x; i < BF * BK; i += 256) {
            const int ff = i / BK, t = i % BK;
            const int f = f0 + ff;
            Ws[t * WP + ff] = (f < F && k0 + t < d)
                                   ? to_f(W1[((size_t)l * F + f) * wstride + d + C + k0 + t])
                                   : 0.f;
        }
        for (int i = threadIdx.x; i < BE * BK; i += 256) {
            const int ee = i / BK, t = i % BK;
            const int e = e0 + ee;
            Cs[ee][t] = (e < E && k0 + t < d) ? ctx[((size_t)l * E + e) * d + k0 + t] : 0.f;
        }
        __syncthreads();
#pragma unroll 16
        for (int t = 0; t < BK; ++t) {
            const float c = Cs[te][t];
            const float4 w = *reinterpret_cast<const float4 *>(&Ws[t * WP + 4 * tf]);
            acc[0] = fmaf(c, w.x, acc[0]);
            acc[1] = fmaf(c, w.y, acc[1]);
            acc[2] = fmaf(c, w.z, acc[2]);
            acc[3] = fmaf(c, w.w, acc[3]);
        }
        __syncthreads();
    }
    const int e = e0 + te;
    if (e >= E) return;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int f = f0 + 4 * tf + j;
        if (f < F) beta[((size_t)l * E + e) * F + f] = b1[(size_t)l * F + f] + alpha_lang * acc[j];
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
    if (keep) {
        const int pos = __popc(ball & ((1u << lane) - 1u));
        const int64_t ti = row - sg.token_row;
        idx[(size_t)l * idx_per_layer + sg.idx_off + ti * k + pos] = (uint8_t)lane;
    }
}

bool router_supported(const rolesub_shape *s)
{
    return s->role_dim + s->router_hidden <= 1536 && s->num_groups <= 32;
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
    k_lang_pool<T><<<dim3((d + 255) / 256, E, L), 256, 0, a.stream>>>(
        h, a.plan.eps_dev, E, P.rows_per_layer, d, a.ws.lang_ctx);
    k_lang_bias<T><<<dim3((F + 63) / 64, (E + 15) / 16, L), 256, 0, a.stream>>>(
        W1, a.b1, a.ws.lang_ctx, E, d, C, F, a.alpha_lang, a.ws.lang_bias);
    if (router_tc_supported(a.shape)) {
        count_launches(2);
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
    count_launches(4);
    return cudaGetLastError();
}

cudaError_t launch_router(const CompressArgs &a)
{
    if (a.shape->dtype == ROLESUB_BF16) return launch_router_t<__nv_bfloat16>(a);
    return launch_router_t<float>(a);
}

}  // namespace rs
