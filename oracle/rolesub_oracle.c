/*
 * rolesub_oracle.c -- fp64 CPU oracle for RoleSub's value routing and for
 * attention over the routed values.
 *
 * TEST INFRASTRUCTURE ONLY. It is called by the test-suite, by the smoke
 * check and by the CPU-baseline leg of the benchmark. The CUDA library never
 * links, loads or calls it, and the two share no code, header, table or
 * helper. Everything here is plain double-precision loops, written to be
 * checked against the paper by eye:
 *
 *   Sec. 3.2  z = R^T v; z split into S equal groups of d_s = d_v / S;
 *             a 0/1 mask m with sum_s m_s = K_i keeps K_i groups;
 *             the routed value is v~ = R M R^T v.
 *   Sec. 3.3  Eq. (latentrole): a = softmax(f_role(h)), f_role linear here.
 *   Sec. 3.4  Eq. (routingscore): the group score combines the token state h,
 *             the role vector a and the pooled language context; this file
 *             uses the concatenation form gamma = W2 ReLU(W1 [h; a_r a; a_l c]
 *             + b1) + b2 with c the mean of the episode's retained language
 *             hidden states; the K_i largest scores are kept (ties: lower
 *             group index first). oracle_router_score_linear is the
 *             additive form as printed (linear f_v and f_lang heads, W_role
 *             a, each term weighted as in the equation).
 *   Sec. 3.5  per-token budgets: within a token type, K_i of the S groups
 *             with sum_i K_i = K_m |I_m|, more for higher role-derived
 *             priority (oracle_budget_*: the allocator as read here);
 *             packed with each token's groups at the prefix sum of the
 *             counts before it.
 *   Attention (Sec. 3, keys and queries unchanged; values routed):
 *             s_j = q . k_j * scale, p = softmax_j(s) over every cache token
 *             of the episode (non-causal), o = sum_j p_j v~_j, evaluated as
 *             o = R_h sum_j p_j M_j z_j (R_h and the sum commute).
 *
 * The value space is per head: R = blockdiag(R_1 .. R_H) with group s of a
 * head holding head dims [s*d_s, (s+1)*d_s); one mask per token is shared by
 * all heads. Packed storage follows the cache layout documented with the
 * library (segments episode-major, kinds vis, lang, prop, act; a segment of n
 * tokens keeping k groups holds [H][n][k][d_s] values and [n][k] indices);
 * the offsets are recomputed here independently by oracle_layout().
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_KINDS 4

/* Segment offsets of one layer. Segment e*4+kind. Sizes: rows n, packed
 * H*n*k*d_s values, indices n*k bytes. Returns 0, or -1 on bad arguments. */
int oracle_layout(int E, int H, int dh, int G, const int *n_tok, const int *k,
                  long long *row_off, long long *packed_off, long long *idx_off,
                  long long *totals)
{
    if (E < 0 || H <= 0 || dh <= 0 || G <= 0 || dh % G != 0) return -1;
    long long ds = dh / G;
    long long r = 0, p = 0, x = 0;
    for (int e = 0; e < E; ++e) {
        for (int m = 0; m < OR_KINDS; ++m) {
            int s = e * OR_KINDS + m;
            int n = n_tok[s], kk = k[s];
            if (n < 0 || kk < 0 || kk > G) return -1;
            row_off[s] = r;
            packed_off[s] = p;
            idx_off[s] = x;
            r += n;
            p += (long long)H * n * kk * ds;
            x += (long long)n * kk;
        }
    }
    totals[0] = r;
    totals[1] = p;
    totals[2] = x;
    return 0;
}

/* Pool of Sec. 3.4: mean of the retained language hidden states; an empty
 * language set gives c = 0. */
void oracle_lang_pool(int d, int n_lang, const double *h_lang, double *c)
{
    for (int t = 0; t < d; ++t) c[t] = 0.0;
    if (n_lang <= 0) return;
    for (int j = 0; j < n_lang; ++j)
        for (int t = 0; t < d; ++t) c[t] += h_lang[(size_t)j * d + t];
    for (int t = 0; t < d; ++t) c[t] /= (double)n_lang;
}

/* Eq. (latentrole): a = softmax(W_re h + b_re), W_re is [C][d]. */
void oracle_role(int d, int C, const double *W_re, const double *b_re,
                 const double *h, double *a)
{
    double mx = -INFINITY;
    for (int r = 0; r < C; ++r) {
        double s = b_re[r];
        for (int t = 0; t < d; ++t) s += W_re[(size_t)r * d + t] * h[t];
        a[r] = s;
        if (s > mx) mx = s;
    }
    double z = 0.0;
    for (int r = 0; r < C; ++r) {
        a[r] = exp(a[r] - mx);
        z += a[r];
    }
    for (int r = 0; r < C; ++r) a[r] /= z;
}

/* Eq. (routingscore), concatenation reading:
 *   x = [h (d) ; alpha_role * a (C) ; alpha_lang * c (d)]
 *   u = max(0, W1 x + b1)        W1 is [F][2d + C]
 *   gamma = W2 u + b2            W2 is [G][F]                              */
void oracle_router_score(int d, int C, int F, int G,
                         const double *W1, const double *b1,
                         const double *W2, const double *b2,
                         const double *h, const double *a, const double *c,
                         double alpha_role, double alpha_lang, double *gamma)
{
    int in = 2 * d + C;
    double *x = (double *)malloc(sizeof(double) * (size_t)in);
    double *u = (double *)malloc(sizeof(double) * (size_t)F);
    for (int t = 0; t < d; ++t) x[t] = h[t];
    for (int r = 0; r < C; ++r) x[d + r] = alpha_role * a[r];
    for (int t = 0; t < d; ++t) x[d + C + t] = alpha_lang * c[t];
    for (int f = 0; f < F; ++f) {
        double s = b1[f];
        for (int t = 0; t < in; ++t) s += W1[(size_t)f * in + t] * x[t];
        u[f] = s > 0.0 ? s : 0.0;
    }
    for (int g = 0; g < G; ++g) {
        double s = b2[g];
        for (int f = 0; f < F; ++f) s += W2[(size_t)g * F + f] * u[f];
        gamma[g] = s;
    }
    free(x);
    free(u);
}

/* Eq. (routingscore) as printed, the additive form, with linear scoring
 * heads (the paper leaves f_v and f_lang as "learned scoring functions"):
 *   gamma_token = W_v h + b_v            W_v is [G][d]
 *   gamma_role  = W_role a               W_role is [G][C], no bias
 *   gamma_lang  = W_l c + b_l            W_l is [G][d], c the pooled context
 *   gamma = gamma_token + alpha_role gamma_role + alpha_lang gamma_lang      */
void oracle_router_score_linear(int d, int C, int G,
                                const double *W_v, const double *b_v,
                                const double *W_role,
                                const double *W_l, const double *b_l,
                                const double *h, const double *a, const double *c,
                                double alpha_role, double alpha_lang, double *gamma)
{
    for (int g = 0; g < G; ++g) {
        double tok = b_v[g];
        for (int t = 0; t < d; ++t) tok += W_v[(size_t)g * d + t] * h[t];
        double role = 0.0;
        for (int r = 0; r < C; ++r) role += W_role[(size_t)g * C + r] * a[r];
        double lang = b_l[g];
        for (int t = 0; t < d; ++t) lang += W_l[(size_t)g * d + t] * c[t];
        gamma[g] = tok + alpha_role * role + alpha_lang * lang;
    }
}

/* Top-K_i of Sec. 3.4. Groups are ranked by (gamma descending, index
 * ascending); the first k are kept and written in ascending index order.
 * margin = gamma_(k) - gamma_(k+1) (r-th largest); k = 0 or k = G gives
 * +infinity (nothing to decide). */
void oracle_topk(int G, int k, const double *gamma, unsigned char *idx,
                 double *margin)
{
    int order[64];
    for (int g = 0; g < G; ++g) order[g] = g;
    /* selection sort by the ranking rule */
    for (int i = 0; i < G; ++i) {
        int best = i;
        for (int j = i + 1; j < G; ++j) {
            int a = order[j], b = order[best];
            if (gamma[a] > gamma[b] || (gamma[a] == gamma[b] && a < b)) best = j;
        }
        int t = order[i];
        order[i] = order[best];
        order[best] = t;
    }
    int keep[64];
    for (int g = 0; g < G; ++g) keep[g] = 0;
    for (int i = 0; i < k; ++i) keep[order[i]] = 1;
    int w = 0;
    for (int g = 0; g < G; ++g)
        if (keep[g]) idx[w++] = (unsigned char)g;
    if (margin) {
        if (k <= 0 || k >= G) *margin = INFINITY;
        else *margin = gamma[order[k - 1]] - gamma[order[k]];
    }
}

/* Sec. 3.2: z = R^T v for one head, R is [dh][dh] row-major (R[m][n]). */
void oracle_rotate(int dh, const double *R, const double *v, double *z)
{
    for (int n = 0; n < dh; ++n) {
        double s = 0.0;
        for (int m = 0; m < dh; ++m) s += R[(size_t)m * dh + n] * v[m];
        z[n] = s;
    }
}

/*
 * Compress one episode of one layer.
 *   n_tok[4], k[4]          tokens and kept groups of the episode's segments
 *   packed_off[4], idx_off[4]  where those segments live in the layer
 *   h_ep, v_ep              [n_cache][d] rows of the episode (kind order)
 *   R                       [H][dh][dh] of the layer
 *   W_re [C][d], b_re [C], W1 [F][2d+C], b1 [F], W2 [G][F], b2 [G]
 *   idx_force               NULL, or the layer's index array to use instead
 *                           of the router (tests of arbitrary masks)
 * Outputs (layer arrays are indexed with the offsets above):
 *   packed_layer, idx_layer; optionally gamma_ep [n_cache][G] (NaN where the
 *   router does not run), margin_ep [n_cache], z_ep [n_cache][d].
 * Returns 0, or -1 on bad arguments / forced indices out of range.
 */
int oracle_compress_episode(int H, int dh, int G, int C, int F,
                            const int *n_tok, const int *k,
                            const long long *packed_off, const long long *idx_off,
                            const double *h_ep, const double *v_ep, const double *R,
                            const double *W_re, const double *b_re,
                            const double *W1, const double *b1,
                            const double *W2, const double *b2,
                            double alpha_role, double alpha_lang,
                            const unsigned char *idx_force,
                            double *packed_layer, unsigned char *idx_layer,
                            double *gamma_ep, double *margin_ep, double *z_ep)
{
    if (H <= 0 || dh <= 0 || G <= 0 || G > 64 || dh % G != 0) return -1;
    int d = H * dh, ds = dh / G;
    int row0[OR_KINDS];
    int nc = 0;
    for (int m = 0; m < OR_KINDS; ++m) {
        if (n_tok[m] < 0 || k[m] < 0 || k[m] > G) return -1;
        row0[m] = nc;
        nc += n_tok[m];
    }
    /* pooled language context of this episode and layer */
    double *c = (double *)malloc(sizeof(double) * (size_t)d);
    oracle_lang_pool(d, n_tok[1], h_ep + (size_t)row0[1] * d, c);

    double *a = (double *)malloc(sizeof(double) * (size_t)(C > 0 ? C : 1));
    double *gam = (double *)malloc(sizeof(double) * (size_t)G);
    double *z = (double *)malloc(sizeof(double) * (size_t)dh);
    int rc = 0;
    for (int m = 0; m < OR_KINDS && rc == 0; ++m) {
        int n = n_tok[m], kk = k[m];
        for (int i = 0; i < n; ++i) {
            int r = row0[m] + i;
            const double *h = h_ep + (size_t)r * d;
            const double *v = v_ep + (size_t)r * d;
            unsigned char *ix = idx_layer + idx_off[m] + (long long)i * kk;
            double mg = INFINITY;
            if (gamma_ep)
                for (int g = 0; g < G; ++g) gamma_ep[(size_t)r * G + g] = NAN;
            if (idx_force) {
                const unsigned char *fx = idx_force + idx_off[m] + (long long)i * kk;
                for (int j = 0; j < kk; ++j) {
                    if (fx[j] >= G || (j > 0 && fx[j] <= fx[j - 1])) { rc = -1; break; }
                    ix[j] = fx[j];
                }
                if (rc) break;
            } else if (kk == G) {
                for (int j = 0; j < G; ++j) ix[j] = (unsigned char)j;
            } else if (kk > 0) {
                oracle_role(d, C, W_re, b_re, h, a);
                oracle_router_score(d, C, F, G, W1, b1, W2, b2, h, a, c,
                                    alpha_role, alpha_lang, gam);
                oracle_topk(G, kk, gam, ix, &mg);
                if (gamma_ep)
                    for (int g = 0; g < G; ++g) gamma_ep[(size_t)r * G + g] = gam[g];
            }
            if (margin_ep) margin_ep[r] = mg;
            for (int hh = 0; hh < H; ++hh) {
                oracle_rotate(dh, R + (size_t)hh * dh * dh, v + (size_t)hh * dh, z);
                if (z_ep)
                    for (int t = 0; t < dh; ++t) z_ep[(size_t)r * d + (size_t)hh * dh + t] = z[t];
                /* packed[seg][h][i][j][:] = z[idx_j * ds : +ds] */
                double *dst = packed_layer + packed_off[m]
                            + (((long long)hh * n + i) * kk) * ds;
                for (int j = 0; j < kk; ++j)
                    for (int t = 0; t < ds; ++t) dst[(long long)j * ds + t] = z[ix[j] * ds + t];
            }
        }
    }
    free(c);
    free(a);
    free(gam);
    free(z);
    return rc;
}

/*
 * Routing of one episode of one layer with the additive router above:
 * c = pool of the language rows, then for every token of a segment with
 * 0 < k < G the top-k of gamma (Sec. 3.4); k = G keeps every group in order.
 * Writes the layer's index array at the segment offsets, and optionally
 * gamma_ep [n_cache][G] (NaN where the router does not run) and margin_ep.
 * The packing that follows is oracle_compress_episode with these indices.
 * Returns 0, or -1 on bad arguments.
 */
int oracle_route_episode_linear(int d, int G, int C, const int *n_tok, const int *k,
                                const long long *idx_off, const double *h_ep,
                                const double *W_re, const double *b_re,
                                const double *W_v, const double *b_v, const double *W_role,
                                const double *W_l, const double *b_l,
                                double alpha_role, double alpha_lang,
                                unsigned char *idx_layer, double *gamma_ep, double *margin_ep)
{
    if (d <= 0 || G <= 0 || G > 64 || C < 0) return -1;
    int row0[OR_KINDS];
    int nc = 0;
    for (int m = 0; m < OR_KINDS; ++m) {
        if (n_tok[m] < 0 || k[m] < 0 || k[m] > G) return -1;
        row0[m] = nc;
        nc += n_tok[m];
    }
    double *c = (double *)malloc(sizeof(double) * (size_t)d);
    oracle_lang_pool(d, n_tok[1], h_ep + (size_t)row0[1] * d, c);
    double *a = (double *)malloc(sizeof(double) * (size_t)(C > 0 ? C : 1));
    double *gam = (double *)malloc(sizeof(double) * (size_t)G);
    for (int m = 0; m < OR_KINDS; ++m) {
        int n = n_tok[m], kk = k[m];
        for (int i = 0; i < n; ++i) {
            int r = row0[m] + i;
            const double *h = h_ep + (size_t)r * d;
            unsigned char *ix = idx_layer + idx_off[m] + (long long)i * kk;
            double mg = INFINITY;
            if (gamma_ep)
                for (int g = 0; g < G; ++g) gamma_ep[(size_t)r * G + g] = NAN;
            if (kk == G) {
                for (int j = 0; j < G; ++j) ix[j] = (unsigned char)j;
            } else if (kk > 0) {
                oracle_role(d, C, W_re, b_re, h, a);
                oracle_router_score_linear(d, C, G, W_v, b_v, W_role, W_l, b_l, h, a, c,
                                           alpha_role, alpha_lang, gam);
                oracle_topk(G, kk, gam, ix, &mg);
                if (gamma_ep)
                    for (int g = 0; g < G; ++g) gamma_ep[(size_t)r * G + g] = gam[g];
            }
            if (margin_ep) margin_ep[r] = mg;
        }
    }
    free(c);
    free(a);
    free(gam);
    return 0;
}

/*
 * Attention of one episode's query tokens over its routed cache, heads
 * [head_begin, head_end) of one layer.
 *   q_ep [n_q][d], K_ep [n_cache][d] (kind order), packed_layer/idx_layer with
 *   the segment offsets, R [H][dh][dh], scale (<= 0 means 1/sqrt(dh)).
 *   o_ep [n_q][d]: only the selected heads are written.
 * Returns 0, or -1 on bad arguments or stored indices out of range.
 */
int oracle_attend_episode(int H, int dh, int G, const int *n_tok, const int *k,
                          const long long *packed_off, const long long *idx_off,
                          int n_q, const double *q_ep, const double *K_ep,
                          const double *packed_layer, const unsigned char *idx_layer,
                          const double *R, double scale,
                          int head_begin, int head_end, double *o_ep)
{
    if (H <= 0 || dh <= 0 || G <= 0 || G > 64 || dh % G != 0) return -1;
    int d = H * dh, ds = dh / G;
    if (scale <= 0.0) scale = 1.0 / sqrt((double)dh);
    int nc = 0;
    for (int m = 0; m < OR_KINDS; ++m) {
        if (n_tok[m] < 0 || k[m] < 0 || k[m] > G) return -1;
        nc += n_tok[m];
    }
    /* the routed value of every cache token in rotated space, zeros where a
     * group was not kept: ztil[j][h][:] = M_j z_{j,h} */
    for (int m = 0; m < OR_KINDS; ++m) {
        int n = n_tok[m], kk = k[m];
        const unsigned char *ix = idx_layer + idx_off[m];
        for (long long t = 0; t < (long long)n * kk; ++t)
            if (ix[t] >= G) return -1;
    }
    double *s = (double *)malloc(sizeof(double) * (size_t)(nc > 0 ? nc : 1));
    double *y = (double *)malloc(sizeof(double) * (size_t)dh);
    double *ztil = (double *)malloc(sizeof(double) * (size_t)dh);
    for (int hh = head_begin; hh < head_end; ++hh) {
        const double *Rh = R + (size_t)hh * dh * dh;
        for (int qi = 0; qi < n_q; ++qi) {
            const double *qv = q_ep + (size_t)qi * d + (size_t)hh * dh;
            double *o = o_ep + (size_t)qi * d + (size_t)hh * dh;
            for (int t = 0; t < dh; ++t) y[t] = 0.0;
            if (nc > 0) {
                double mx = -INFINITY;
                for (int j = 0; j < nc; ++j) {
                    const double *kv = K_ep + (size_t)j * d + (size_t)hh * dh;
                    double acc = 0.0;
                    for (int t = 0; t < dh; ++t) acc += qv[t] * kv[t];
                    s[j] = acc * scale;
                    if (s[j] > mx) mx = s[j];
                }
                double zsum = 0.0;
                for (int j = 0; j < nc; ++j) {
                    s[j] = exp(s[j] - mx);
                    zsum += s[j];
                }
                int j = 0;
                for (int m = 0; m < OR_KINDS; ++m) {
                    int n = n_tok[m], kk = k[m];
                    for (int i = 0; i < n; ++i, ++j) {
                        double p = s[j] / zsum;
                        for (int t = 0; t < dh; ++t) ztil[t] = 0.0;
                        const unsigned char *ix = idx_layer + idx_off[m] + (long long)i * kk;
                        const double *src = packed_layer + packed_off[m]
                                          + (((long long)hh * n + i) * kk) * ds;
                        for (int jj = 0; jj < kk; ++jj)
                            for (int t = 0; t < ds; ++t)
                                ztil[ix[jj] * ds + t] = src[(long long)jj * ds + t];
                        for (int t = 0; t < dh; ++t) y[t] += p * ztil[t];
                    }
                }
            }
            /* o = R_h y */
            for (int m = 0; m < dh; ++m) {
                double acc = 0.0;
                for (int t = 0; t < dh; ++t) acc += Rh[(size_t)m * dh + t] * y[t];
                o[m] = acc;
            }
        }
    }
    free(s);
    free(y);
    free(ztil);
    return 0;
}

/*
 * Role-driven budget allocation, Sec. 3.5 (the allocator B^(l)). The paper
 * fixes its constraints -- 0 <= K_i <= S and sum_i K_i = B_m = K_m |I_m| for
 * the tokens of one type -- and that tokens of higher role-derived priority
 * get more value groups; it gives no formula. Reading used here:
 *   - rank the n tokens by priority (higher first, ties: lower token index);
 *   - rank r (0-based) has weight n - r;
 *   - real shares x_r = min(S, lambda (n - r)), lambda chosen so that
 *     sum_r x_r = B (the best ranks saturate at S first);
 *   - K is x rounded by largest remainders: floor(x_r), plus one for the
 *     B - sum floor(x_r) ranks with the largest fractional parts (ties: the
 *     better rank).
 * Once the ranks are fixed everything is integer arithmetic: with c ranks
 * saturated, x_r = (B - cS)(n - r) / W_c for r >= c, W_c = sum_{r>=c}(n - r).
 * K_by_rank[r] receives the count of rank r. Returns 0, or -1 on bad
 * arguments (B outside [0, nS]).
 */
int oracle_budget_shares(int n, long long B, int S, int *K_by_rank)
{
    if (n < 0 || S < 0 || B < 0 || B > (long long)n * S) return -1;
    if (n == 0) return 0;
    /* number of saturated ranks: the first c whose largest unsaturated share
     * (rank c) does not exceed S */
    int c = 0;
    for (; c < n; ++c) {
        long long rest = B - (long long)c * S;
        long long W = (long long)(n - c) * (n - c + 1) / 2;
        if (rest * (long long)(n - c) <= (long long)S * W) break;
    }
    for (int r = 0; r < c; ++r) K_by_rank[r] = S;
    if (c == n) return 0;
    long long rest = B - (long long)c * S;
    long long W = (long long)(n - c) * (n - c + 1) / 2;
    long long assigned = 0;
    long long *rem = (long long *)malloc(sizeof(long long) * (size_t)n);
    for (int r = c; r < n; ++r) {
        long long num = rest * (long long)(n - r);
        K_by_rank[r] = (int)(num / W);
        rem[r] = num % W;
        assigned += K_by_rank[r];
    }
    /* the left-over groups, one each, to the largest remainders */
    long long left = rest - assigned;
    for (long long t = 0; t < left; ++t) {
        int best = -1;
        for (int r = c; r < n; ++r)
            if (rem[r] >= 0 && (best < 0 || rem[r] > rem[best])) best = r;
        K_by_rank[best] += 1;
        rem[best] = -1; /* taken */
    }
    free(rem);
    return 0;
}

/* The allocation of one token type: ranks the n priorities (higher first,
 * ties: lower index) and gives token i the count of its rank.
 * Returns 0, or -1 on bad arguments. */
int oracle_budget_allocate(int n, long long B, int S, const double *pri, int *K)
{
    if (n < 0) return -1;
    if (n == 0) return 0;
    int *byrank = (int *)malloc(sizeof(int) * (size_t)n);
    if (oracle_budget_shares(n, B, S, byrank) != 0) {
        free(byrank);
        return -1;
    }
    for (int i = 0; i < n; ++i) {
        int rank = 0;
        for (int j = 0; j < n; ++j)
            if (pri[j] > pri[i] || (pri[j] == pri[i] && j < i)) ++rank;
        K[i] = byrank[rank];
    }
    free(byrank);
    return 0;
}

/*
 * Routing of one episode of one layer with per-token budgets (Sec. 3.4 and
 * Sec. 3.5): the additive score of oracle_router_score_linear, the latent
 * role a_i of Eq. (latentrole) and the priority pi_i = u . a_i. For a segment
 * of n tokens with target K_m (k[m]):
 *   0 < K_m < G  K_i from oracle_budget_allocate(pi, B = K_m n), unless
 *                k_force_ep gives them ([n_cache], summing to B); the
 *                K_i largest scores are kept (oracle_topk) and written at
 *                idx_off[m] + sum_{j<i} K_j;
 *   K_m = G      every token keeps every group (indices 0..G-1);
 *   K_m = 0      nothing is kept.
 * Outputs: idx_layer at the segment offsets; ktok_ep [n_cache] = K_i; and
 * optionally gamma_ep [n_cache][G] and pri_ep [n_cache] (NaN where the
 * router does not run) and margin_ep [n_cache] (top-K_i margin).
 * Returns 0, or -1 on bad arguments or forced counts that break the budget.
 */
int oracle_route_episode_budget(int d, int G, int C, const int *n_tok, const int *k,
                                const long long *idx_off, const double *h_ep,
                                const double *W_re, const double *b_re,
                                const double *W_v, const double *b_v, const double *W_role,
                                const double *W_l, const double *b_l, const double *u,
                                double alpha_role, double alpha_lang, const int *k_force_ep,
                                unsigned char *idx_layer, int *ktok_ep, double *gamma_ep,
                                double *pri_ep, double *margin_ep)
{
    if (d <= 0 || G <= 0 || G > 64 || C < 1) return -1;
    int row0[OR_KINDS];
    int nc = 0;
    for (int m = 0; m < OR_KINDS; ++m) {
        if (n_tok[m] < 0 || k[m] < 0 || k[m] > G) return -1;
        row0[m] = nc;
        nc += n_tok[m];
    }
    double *c = (double *)malloc(sizeof(double) * (size_t)d);
    oracle_lang_pool(d, n_tok[1], h_ep + (size_t)row0[1] * d, c);
    double *a = (double *)malloc(sizeof(double) * (size_t)C);
    double *gam = (double *)malloc(sizeof(double) * (size_t)(nc > 0 ? nc : 1) * G);
    double *pri = (double *)malloc(sizeof(double) * (size_t)(nc > 0 ? nc : 1));
    int rc = 0;
    for (int m = 0; m < OR_KINDS && rc == 0; ++m) {
        int n = n_tok[m], km = k[m];
        for (int i = 0; i < n; ++i) {
            int r = row0[m] + i;
            pri[r] = NAN;
            for (int g = 0; g < G; ++g) gam[(size_t)r * G + g] = NAN;
            if (margin_ep) margin_ep[r] = INFINITY;
        }
        if (km == G) {
            for (int i = 0; i < n; ++i) {
                ktok_ep[row0[m] + i] = G;
                for (int g = 0; g < G; ++g) idx_layer[idx_off[m] + (long long)i * G + g] = (unsigned char)g;
            }
            continue;
        }
        if (km == 0) {
            for (int i = 0; i < n; ++i) ktok_ep[row0[m] + i] = 0;
            continue;
        }
        for (int i = 0; i < n; ++i) {
            int r = row0[m] + i;
            const double *h = h_ep + (size_t)r * d;
            oracle_role(d, C, W_re, b_re, h, a);
            double p = 0.0;
            for (int t = 0; t < C; ++t) p += u[t] * a[t];
            pri[r] = p;
            oracle_router_score_linear(d, C, G, W_v, b_v, W_role, W_l, b_l, h, a, c, alpha_role,
                                       alpha_lang, gam + (size_t)r * G);
        }
        long long B = (long long)km * n;
        if (k_force_ep) {
            long long s = 0;
            for (int i = 0; i < n; ++i) {
                int kk = k_force_ep[row0[m] + i];
                if (kk < 0 || kk > G) rc = -1;
                ktok_ep[row0[m] + i] = kk;
                s += kk;
            }
            if (s != B) rc = -1;
            if (rc != 0) break;
        } else if (oracle_budget_allocate(n, B, G, pri + row0[m], ktok_ep + row0[m]) != 0) {
            rc = -1;
            break;
        }
        long long off = idx_off[m];
        for (int i = 0; i < n; ++i) {
            int r = row0[m] + i, kk = ktok_ep[r];
            double mg;
            oracle_topk(G, kk, gam + (size_t)r * G, idx_layer + off, &mg);
            if (margin_ep) margin_ep[r] = mg;
            off += kk;
        }
    }
    if (gamma_ep)
        for (size_t t = 0; t < (size_t)nc * G; ++t) gamma_ep[t] = gam[t];
    if (pri_ep)
        for (int t = 0; t < nc; ++t) pri_ep[t] = pri[t];
    free(c);
    free(a);
    free(gam);
    free(pri);
    return rc;
}
