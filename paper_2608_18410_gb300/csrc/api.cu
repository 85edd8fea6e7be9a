// api.cu -- the C ABI of include/rolesub.h: plan construction, argument
// validation (always before any launch) and the launch sequences.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>

#include "common.cuh"
#include "internal.h"

namespace rs {
static std::atomic<uint64_t> g_launches{0};
void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }
}  // namespace rs

namespace {

using rs::PlanView;
using rs::Workspace;

constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

int elem_bytes(int dtype) { return dtype == ROLESUB_BF16 ? 2 : 4; }

bool shape_ok(const rolesub_shape *s)
{
    if (!s) return false;
    if (s->num_layers < 1 || s->num_heads < 1 || s->head_dim < 1) return false;
    if (s->num_groups < 1 || s->num_groups > ROLESUB_MAX_GROUPS) return false;
    if (s->head_dim % s->num_groups != 0) return false;
    if (s->role_dim < 1 || s->router_hidden < 1) return false;
    if (s->dtype != ROLESUB_F32 && s->dtype != ROLESUB_BF16) return false;
    if (s->reserved != 0) return false;
    if ((int64_t)s->num_heads * s->head_dim > (1 << 20)) return false;
    return true;
}

// The per-token budget path (Sec. 3.5): bf16, d_h = 128, S = 16 (the
// tensor-core rotation, attention and additive router), S + C <= 256,
// d % 64 == 0, and segments of at most 8192 tokens.
bool budget_supported(const rolesub_shape *s, const PlanView &pv);

struct Sizes {
    size_t header, segs, eps, row_seg, routed, stored, tiles, total;
};

Sizes plan_sizes(int32_t E, int64_t rows)
{
    Sizes z;
    z.header = align_up(sizeof(rolesub_plan), 16);
    z.segs = align_up(sizeof(rolesub_segment) * (size_t)E * ROLESUB_NUM_KINDS, 16);
    z.eps = align_up(sizeof(rolesub_episode) * (size_t)E, 16);
    z.row_seg = align_up(sizeof(int32_t) * (size_t)rows, 16);
    z.routed = z.row_seg;
    z.stored = z.row_seg;
    z.tiles = z.row_seg;   // at most one router tile per routed row
    z.total = z.header + z.segs + z.eps + z.row_seg + z.routed + z.stored + z.tiles;
    return z;
}

// Validates a plan blob against a shape and fills the host view.
rolesub_status view_plan(const rolesub_shape *s, const void *plan_host, const void *plan_dev,
                         PlanView *pv)
{
    if (!plan_host || !aligned16(plan_host)) return ROLESUB_EINVAL;
    const rolesub_plan *p = (const rolesub_plan *)plan_host;
    if (p->magic != ROLESUB_PLAN_MAGIC || p->version != ROLESUB_VERSION) return ROLESUB_EINVAL;
    if (p->num_heads != s->num_heads || p->head_dim != s->head_dim ||
        p->num_groups != s->num_groups)
        return ROLESUB_EINVAL;
    if (p->num_episodes < 0 || p->num_segments != p->num_episodes * ROLESUB_NUM_KINDS)
        return ROLESUB_EINVAL;
    if (p->rows_per_layer >= (int64_t)1 << 31) return ROLESUB_EUNSUPPORTED;
    if (plan_dev && !aligned16(plan_dev)) return ROLESUB_EINVAL;
    const char *b = (const char *)plan_host;
    pv->hdr = p;
    pv->segs = (const rolesub_segment *)(b + p->off_segments);
    pv->eps = (const rolesub_episode *)(b + p->off_episodes);
    const char *d = (const char *)plan_dev;
    pv->dev = d;
    pv->segs_dev = d ? (const rolesub_segment *)(d + p->off_segments) : nullptr;
    pv->eps_dev = d ? (const rolesub_episode *)(d + p->off_episodes) : nullptr;
    pv->row_seg_dev = d ? (const int32_t *)(d + p->off_row_seg) : nullptr;
    pv->routed_dev = d ? (const int32_t *)(d + p->off_routed_rows) : nullptr;
    pv->stored_dev = d ? (const int32_t *)(d + p->off_stored_rows) : nullptr;
    pv->route_tiles_dev = d ? (const int32_t *)(d + p->off_route_tiles) : nullptr;
    return ROLESUB_OK;
}

struct WsSizes {
    size_t status, ctx, bias, logits, rowst, total;
};

WsSizes ws_sizes(const rolesub_shape *s, const rolesub_plan *p)
{
    WsSizes w;
    const size_t L = s->num_layers, E = p->num_episodes;
    const size_t d = (size_t)s->num_heads * s->head_dim;
    w.status = rs::kStatusBytes;
    w.ctx = align_up(sizeof(float) * L * E * d, kAlign);
    // per-episode router terms: F wide for the concatenation router, S for
    // the additive one
    w.bias = align_up(sizeof(float) * L * E * (size_t)(s->router_hidden > s->num_groups ? s->router_hidden
                                                                                      : s->num_groups),
                      kAlign);
    // router logits are only staged in memory when the fused tensor-core
    // router does not apply
    w.logits = rs::router_tc_supported(s)
                   ? 0
                   : align_up(sizeof(float) * L * (size_t)p->routed_rows_per_layer *
                                  (size_t)(s->router_hidden + s->role_dim),
                              kAlign);
    w.rowst = rs::rotate_tc_supported(s) ? align_up((size_t)16 * L * (size_t)p->rows_per_layer, kAlign) : 0;
    w.total = w.status + w.ctx + w.bias + w.logits + w.rowst;
    return w;
}

Workspace carve(const WsSizes &w, void *base)
{
    Workspace ws;
    char *b = (char *)base;
    ws.status = (int32_t *)b;
    ws.lang_ctx = (float *)(b + w.status);
    ws.lang_bias = (float *)(b + w.status + w.ctx);
    ws.logits = (float *)(b + w.status + w.ctx + w.bias);
    ws.row_store = b + w.status + w.ctx + w.bias + w.logits;
    ws.bytes = w.total;
    return ws;
}

rolesub_status from_cuda(cudaError_t e) { return e == cudaSuccess ? ROLESUB_OK : ROLESUB_ECUDA; }

// The dense-rotation path: bf16, d_h = 128, S = 16 (the attention kernel
// reads v~ through store records), d % 256 == 0 (the v~ GEMM's column tile)
// and g = d / 16 either 64, 128 or a multiple of 256 (a group is a whole
// number of 64-wide K blocks, and a whole number of N tiles of the z GEMM).
bool dense_supported(const rolesub_shape *s)
{
    const int d = s->num_heads * s->head_dim, g = d / 16;
    return rs::rotate_tc_supported(s) && rs::attend_tc_supported(s) && d % 256 == 0 && d <= 65536 &&
           (g == 64 || g == 128 || g % 256 == 0);
}

int dense_chunks(const rolesub_plan *p) { return (int)((p->rows_per_layer + rs::kDenseChunk - 1) / rs::kDenseChunk); }

// After the common workspace: v~ [L][rows][d] bf16, perm [L][rows] int32,
// the identity rotations [L][H][d_h][d_h] bf16, the pair lists [L][idx
// bytes per layer] int2, and the chunk tables [L][chunks][32] int32.
struct DenseWs {
    size_t vt, perm, ident, pairs, meta, total;
};

DenseWs dense_ws(const rolesub_shape *s, const rolesub_plan *p)
{
    const size_t d = (size_t)s->num_heads * s->head_dim, L = s->num_layers, rows = (size_t)p->rows_per_layer;
    DenseWs w;
    w.vt = align_up(2 * L * rows * d, kAlign);
    w.perm = align_up(4 * L * rows, kAlign);
    w.ident = align_up(2 * L * s->num_heads * (size_t)s->head_dim * s->head_dim, kAlign);
    w.pairs = align_up(8 * L * (size_t)p->idx_bytes_per_layer, kAlign);
    w.meta = align_up(4 * L * (size_t)dense_chunks(p) * rs::kDenseMetaStride, kAlign);
    w.total = w.vt + w.perm + w.ident + w.pairs + w.meta;
    return w;
}

size_t dense_extra_bytes(const rolesub_shape *s, const rolesub_plan *p) { return dense_ws(s, p).total; }

// The layout the dense kernels rely on (the one rolesub_plan_build makes):
// segments in row order, indices and packed groups in the same order,
// packed_off = g * idx_off; and row / slot counts that fit the int32
// coordinates of the gather loads.
bool dense_plan_ok(const rolesub_shape *s, const PlanView &pv)
{
    const rolesub_plan &P = *pv.hdr;
    const int64_t g = (int64_t)s->num_heads * s->head_dim / 16;
    int64_t r = 0, ix = 0;
    for (int i = 0; i < P.num_segments; ++i) {
        const rolesub_segment &sg = pv.segs[i];
        if (sg.token_row != r || sg.idx_off != ix || sg.packed_off != g * ix) return false;
        r += sg.n_tokens;
        ix += (int64_t)sg.n_tokens * sg.k;
    }
    const int64_t L = s->num_layers;
    return r == P.rows_per_layer && ix == P.idx_bytes_per_layer && P.packed_elems_per_layer == g * ix &&
           L * P.rows_per_layer < ((int64_t)1 << 31) && L * ix < ((int64_t)1 << 31);
}

// Upper bound on the 128-pair tiles of any chunk: ceil(pairs / 128) plus one
// partial tile per group.
int dense_tiles_per_chunk(const PlanView &pv, int chunks)
{
    const rolesub_plan &P = *pv.hdr;
    int best = 0;
    int i = 0;
    for (int c = 0; c < chunks; ++c) {
        const int64_t c0 = (int64_t)c * rs::kDenseChunk, c1 = std::min(P.rows_per_layer, c0 + rs::kDenseChunk);
        int64_t pairs = 0;
        while (i < P.num_segments && pv.segs[i].token_row + pv.segs[i].n_tokens <= c0) ++i;
        for (int j = i; j < P.num_segments && pv.segs[j].token_row < c1; ++j) {
            const rolesub_segment &sg = pv.segs[j];
            const int64_t a = std::max(c0, sg.token_row), b = std::min(c1, sg.token_row + sg.n_tokens);
            if (b > a) pairs += (b - a) * sg.k;
        }
        best = std::max(best, (int)((pairs + 127) / 128) + 16);
    }
    return best;
}

bool budget_supported(const rolesub_shape *s, const PlanView &pv)
{
    if (!rs::rotate_tc_supported(s) || !rs::attend_tc_supported(s) || !rs::additive_tc_supported(s)) return false;
    for (int i = 0; i < pv.hdr->num_segments; ++i)
        if (pv.segs[i].n_tokens > 8192) return false;
    return true;
}

}  // namespace

extern "C" {

int32_t rolesub_version(void) { return ROLESUB_VERSION; }

uint64_t rolesub_launch_count(void) { return rs::g_launches.load(std::memory_order_relaxed); }

const char *rolesub_status_string(rolesub_status s)
{
    switch (s) {
    case ROLESUB_OK: return "ok";
    case ROLESUB_EINVAL: return "invalid argument";
    case ROLESUB_EUNSUPPORTED: return "unsupported geometry";
    case ROLESUB_ECUDA: return "CUDA error";
    case ROLESUB_EDEVICE: return "bad data found on the device";
    case ROLESUB_ETIMEOUT: return "in-kernel wait timed out";
    case ROLESUB_ETOOLARGE: return "problem needs more scratch than the library's static array";
    }
    return "unknown status";
}

rolesub_status rolesub_plan_size(int32_t num_episodes, const int32_t *n_tok, size_t *bytes)
{
    if (num_episodes < 0 || !bytes || (num_episodes > 0 && !n_tok)) return ROLESUB_EINVAL;
    int64_t rows = 0;
    for (int64_t i = 0; i < (int64_t)num_episodes * ROLESUB_NUM_KINDS; ++i) {
        if (n_tok[i] < 0) return ROLESUB_EINVAL;
        rows += n_tok[i];
    }
    *bytes = plan_sizes(num_episodes, rows).total;
    return ROLESUB_OK;
}

rolesub_status rolesub_layout_plan(const rolesub_shape *shape, int32_t E, const int32_t *n_tok,
                                   const int32_t *k, const int32_t *n_query, void *plan,
                                   size_t plan_bytes)
{
    if (!shape_ok(shape) || E < 0 || !plan || !aligned16(plan)) return ROLESUB_EINVAL;
    if (E > 0 && (!n_tok || !k || !n_query)) return ROLESUB_EINVAL;
    const int G = shape->num_groups, H = shape->num_heads;
    const int64_t ds = shape->head_dim / G;
    int64_t rows = 0, qrows = 0;
    for (int64_t i = 0; i < (int64_t)E * ROLESUB_NUM_KINDS; ++i) {
        if (n_tok[i] < 0 || k[i] < 0 || k[i] > G) return ROLESUB_EINVAL;
        rows += n_tok[i];
    }
    for (int e = 0; e < E; ++e) {
        if (n_query[e] < 0) return ROLESUB_EINVAL;
        qrows += n_query[e];
    }
    const Sizes z = plan_sizes(E, rows);
    if (plan_bytes < z.total) return ROLESUB_EINVAL;
    memset(plan, 0, z.total);
    char *b = (char *)plan;
    rolesub_plan *p = (rolesub_plan *)b;
    p->magic = ROLESUB_PLAN_MAGIC;
    p->version = ROLESUB_VERSION;
    p->num_episodes = E;
    p->num_segments = E * ROLESUB_NUM_KINDS;
    p->num_heads = H;
    p->head_dim = shape->head_dim;
    p->num_groups = G;
    p->off_segments = (int64_t)z.header;
    p->off_episodes = (int64_t)(z.header + z.segs);
    p->off_row_seg = (int64_t)(z.header + z.segs + z.eps);
    p->off_routed_rows = p->off_row_seg + (int64_t)z.row_seg;
    p->off_stored_rows = p->off_routed_rows + (int64_t)z.routed;
    p->off_route_tiles = p->off_stored_rows + (int64_t)z.stored;
    p->total_bytes = (int64_t)z.total;
    rolesub_segment *segs = (rolesub_segment *)(b + p->off_segments);
    rolesub_episode *eps = (rolesub_episode *)(b + p->off_episodes);
    int32_t *row_seg = (int32_t *)(b + p->off_row_seg);
    int32_t *routed = (int32_t *)(b + p->off_routed_rows);
    int32_t *stored = (int32_t *)(b + p->off_stored_rows);
    int64_t r = 0, qr = 0, pk = 0, ix = 0, nrouted = 0, nstored = 0;
    int32_t max_c = 0, max_q = 0;
    for (int e = 0; e < E; ++e) {
        rolesub_episode &ep = eps[e];
        ep.row_begin = r;
        ep.q_row_begin = qr;
        ep.n_query = n_query[e];
        ep.seg_begin = e * ROLESUB_NUM_KINDS;
        int32_t nc = 0;
        for (int m = 0; m < ROLESUB_NUM_KINDS; ++m) {
            const int s = e * ROLESUB_NUM_KINDS + m;
            rolesub_segment &sg = segs[s];
            sg.episode = e;
            sg.kind = m;
            sg.n_tokens = n_tok[s];
            sg.k = k[s];
            sg.token_row = r;
            sg.packed_off = pk;
            sg.idx_off = ix;
            if (m == ROLESUB_LANG) {
                ep.n_lang = n_tok[s];
                ep.lang_row_begin = r;
            }
            for (int i = 0; i < n_tok[s]; ++i) {
                row_seg[r + i] = s;
                if (k[s] > 0) stored[nstored++] = (int32_t)(r + i);
                if (k[s] > 0 && k[s] < G) routed[nrouted++] = (int32_t)(r + i);
            }
            r += n_tok[s];
            nc += n_tok[s];
            pk += (int64_t)H * n_tok[s] * k[s] * ds;
            ix += (int64_t)n_tok[s] * k[s];
        }
        ep.n_cache = nc;
        if (nc > max_c) max_c = nc;
        if (n_query[e] > max_q) max_q = n_query[e];
        qr += n_query[e];
    }
    p->rows_per_layer = r;
    p->q_rows_per_layer = qr;
    p->packed_elems_per_layer = pk;
    p->idx_bytes_per_layer = ix;
    p->routed_rows_per_layer = nrouted;
    p->stored_rows_per_layer = nstored;
    p->max_cache_tokens = max_c;
    p->max_query_tokens = max_q;
    // router tiles: 128-row windows, each starting at the first routed row
    // the previous windows left uncovered
    int32_t *tiles = (int32_t *)(b + p->off_route_tiles);
    int32_t nt = 0;
    int64_t covered = -1;
    for (int64_t i = 0; i < nrouted; ++i) {
        if (routed[i] > covered) {
            tiles[nt++] = routed[i];
            covered = (int64_t)routed[i] + 127;
        }
    }
    p->num_route_tiles = nt;
    return ROLESUB_OK;
}

rolesub_status rolesub_workspace_size(const rolesub_shape *shape, const void *plan_host,
                                      size_t *bytes)
{
    if (!shape_ok(shape) || !bytes) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, nullptr, &pv);
    if (st != ROLESUB_OK) return st;
    *bytes = ws_sizes(shape, pv.hdr).total;
    return ROLESUB_OK;
}

rolesub_status rolesub_compress(const rolesub_shape *shape, const void *plan_host,
                                const void *plan_dev, const void *h, const void *v,
                                const void *R, const void *W_re, const float *b_re,
                                const void *W1, const float *b1, const void *W2,
                                const float *b2, float alpha_role, float alpha_lang,
                                void *packed_v, uint8_t *idx, void *workspace, size_t ws_bytes,
                                void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const void *ptrs[] = {h, v, R, W_re, b_re, W1, b1, W2, b2, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && (!idx || !aligned16(idx))) return ROLESUB_EINVAL;
    if (!isfinite(alpha_role) || !isfinite(alpha_lang)) return ROLESUB_EINVAL;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (ws_bytes < w.total) return ROLESUB_EINVAL;
    if (!rs::router_supported(shape) || !rs::rotate_supported(shape)) return ROLESUB_EUNSUPPORTED;
    rs::CompressArgs a;
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.h = h;
    a.v = v;
    a.R = R;
    a.W_re = W_re;
    a.W1 = W1;
    a.W2 = W2;
    a.b_re = b_re;
    a.b1 = b1;
    a.b2 = b2;
    a.alpha_role = alpha_role;
    a.alpha_lang = alpha_lang;
    a.packed = packed_v;
    a.idx = idx;
    a.stream = (cudaStream_t)stream;
    cudaError_t e = rs::launch_router(a);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    return from_cuda(rs::launch_rotate_pack(a));
}

rolesub_status rolesub_compress_additive(const rolesub_shape *shape, const void *plan_host,
                                         const void *plan_dev, const void *h, const void *v,
                                         const void *R, const void *W_re, const float *b_re,
                                         const void *W_v, const float *b_v, const void *W_role,
                                         const void *W_l, const float *b_l, float alpha_role,
                                         float alpha_lang, void *packed_v, uint8_t *idx,
                                         void *workspace, size_t ws_bytes, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const void *ptrs[] = {h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && (!idx || !aligned16(idx))) return ROLESUB_EINVAL;
    if (!isfinite(alpha_role) || !isfinite(alpha_lang)) return ROLESUB_EINVAL;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (ws_bytes < w.total) return ROLESUB_EINVAL;
    if (!rs::router_additive_supported(shape) || !rs::rotate_supported(shape)) return ROLESUB_EUNSUPPORTED;
    rs::CompressArgs a{};
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.h = h;
    a.v = v;
    a.R = R;
    a.W_re = W_re;
    a.b_re = b_re;
    a.alpha_role = alpha_role;
    a.alpha_lang = alpha_lang;
    a.packed = packed_v;
    a.idx = idx;
    a.stream = (cudaStream_t)stream;
    const rs::AdditiveWeights wt{W_v, W_role, W_l, b_v, b_l};
    cudaError_t e = rs::launch_router_additive(a, wt);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    return from_cuda(rs::launch_rotate_pack(a));
}

}  // extern "C"

namespace {

// Scores and priorities of the budget path's router: [L][rows][20] fp32
// after the common workspace.
size_t budget_scores_bytes(const rolesub_shape *shape, const rolesub_plan *p)
{
    return align_up(sizeof(float) * rs::kScoreStride * (size_t)shape->num_layers * (size_t)p->rows_per_layer,
                    kAlign);
}

// Shared by rolesub_attend (k_tok = NULL: the plan's k per segment) and
// rolesub_attend_budget (per-token counts).
rolesub_status attend_common(const rolesub_shape *shape, const void *plan_host, const void *plan_dev,
                             const void *q, int64_t q_ls, int64_t q_rs, int64_t q_hs, const void *K, int64_t k_ls,
                             int64_t k_rs, int64_t k_hs, const void *packed_v, const uint8_t *idx,
                             const uint8_t *k_tok, bool budget, const void *R, float softmax_scale, void *o,
                             void *workspace, size_t ws_bytes, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    const void *ptrs[] = {q, K, R, o, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && !idx) return ROLESUB_EINVAL;
    if (budget && P.rows_per_layer > 0 && !k_tok) return ROLESUB_EINVAL;
    const int64_t sm = 16 / elem_bytes(shape->dtype);
    const int64_t strides[] = {q_ls, q_rs, q_hs, k_ls, k_rs, k_hs};
    for (int64_t x : strides)
        if (x < 0 || x % sm != 0) return ROLESUB_EINVAL;
    if (!isfinite(softmax_scale) || softmax_scale < 0.f) return ROLESUB_EINVAL;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (ws_bytes < w.total) return ROLESUB_EINVAL;
    if (!rs::attend_supported(shape)) return ROLESUB_EUNSUPPORTED;
    if (budget && !budget_supported(shape, pv)) return ROLESUB_EUNSUPPORTED;
    rs::AttendArgs a;
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.q = q;
    a.K = K;
    a.packed = packed_v;
    a.R = R;
    a.idx = idx;
    a.q_ls = q_ls;
    a.q_rs = q_rs;
    a.q_hs = q_hs;
    a.k_ls = k_ls;
    a.k_rs = k_rs;
    a.k_hs = k_hs;
    a.scale = softmax_scale;
    a.o = o;
    a.stream = (cudaStream_t)stream;
    if (budget) {
        a.k_tok = k_tok;
        return from_cuda(rs::launch_attend_tc(a));
    }
    return from_cuda(rs::launch_attend(a));
}

}  // namespace

extern "C" {

rolesub_status rolesub_attend(const rolesub_shape *shape, const void *plan_host,
                              const void *plan_dev, const void *q, int64_t q_ls, int64_t q_rs,
                              int64_t q_hs, const void *K, int64_t k_ls, int64_t k_rs,
                              int64_t k_hs, const void *packed_v, const uint8_t *idx,
                              const void *R, float softmax_scale, void *o, void *workspace,
                              size_t ws_bytes, void *stream)
{
    return attend_common(shape, plan_host, plan_dev, q, q_ls, q_rs, q_hs, K, k_ls, k_rs, k_hs, packed_v, idx,
                         nullptr, false, R, softmax_scale, o, workspace, ws_bytes, stream);
}

rolesub_status rolesub_attend_budget(const rolesub_shape *shape, const void *plan_host,
                                     const void *plan_dev, const void *q, int64_t q_ls, int64_t q_rs,
                                     int64_t q_hs, const void *K, int64_t k_ls, int64_t k_rs,
                                     int64_t k_hs, const void *packed_v, const uint8_t *idx,
                                     const uint8_t *k_tok, const void *R, float softmax_scale, void *o,
                                     void *workspace, size_t ws_bytes, void *stream)
{
    return attend_common(shape, plan_host, plan_dev, q, q_ls, q_rs, q_hs, K, k_ls, k_rs, k_hs, packed_v, idx,
                         k_tok, true, R, softmax_scale, o, workspace, ws_bytes, stream);
}

rolesub_status rolesub_budget_workspace_size(const rolesub_shape *shape, const void *plan_host, size_t *bytes)
{
    if (!shape_ok(shape) || !bytes) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, nullptr, &pv);
    if (st != ROLESUB_OK) return st;
    *bytes = ws_sizes(shape, pv.hdr).total + budget_scores_bytes(shape, pv.hdr);
    return ROLESUB_OK;
}

rolesub_status rolesub_compress_budget(const rolesub_shape *shape, const void *plan_host,
                                       const void *plan_dev, const void *h, const void *v,
                                       const void *R, const void *W_re, const float *b_re,
                                       const void *W_v, const float *b_v, const void *W_role,
                                       const void *W_l, const float *b_l, const float *u,
                                       float alpha_role, float alpha_lang, void *packed_v,
                                       uint8_t *idx, uint8_t *k_tok, void *workspace,
                                       size_t ws_bytes, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const void *ptrs[] = {h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, u, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && (!idx || !aligned16(idx))) return ROLESUB_EINVAL;
    if (P.rows_per_layer > 0 && !k_tok) return ROLESUB_EINVAL;
    if (!isfinite(alpha_role) || !isfinite(alpha_lang)) return ROLESUB_EINVAL;
    if (!budget_supported(shape, pv)) return ROLESUB_EUNSUPPORTED;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    const size_t sb = budget_scores_bytes(shape, pv.hdr);
    if (ws_bytes < w.total + sb) return ROLESUB_EINVAL;
    rs::CompressArgs a{};
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.h = h;
    a.v = v;
    a.R = R;
    a.W_re = W_re;
    a.b_re = b_re;
    a.alpha_role = alpha_role;
    a.alpha_lang = alpha_lang;
    a.packed = packed_v;
    a.idx = idx;
    a.stream = (cudaStream_t)stream;
    float *scores = reinterpret_cast<float *>(static_cast<char *>(workspace) + w.total);
    rs::AdditiveWeights wt{W_v, W_role, W_l, b_v, b_l};
    wt.u = u;
    wt.scores = scores;
    cudaError_t e = rs::launch_router_additive(a, wt);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    e = rs::launch_budget_select(a, scores, k_tok);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    a.records_ready = true;
    return from_cuda(rs::launch_rotate_pack(a));
}

int32_t rolesub_select_count(int32_t n_view, double ratio)
{
    if (n_view < 0 || !(ratio > 0.0) || ratio > 1.0) return -1;
    const double x = ratio * (double)n_view;
    int64_t k = (int64_t)x;
    if ((double)k < x) ++k;   // ceil
    return (int32_t)k;
}

rolesub_status rolesub_select_tokens(int32_t num_episodes, int32_t num_views, int32_t n_view, double ratio,
                                     const float *scores, const void *x, int32_t hidden, int32_t dtype,
                                     int32_t *keep_idx, void *x_keep, void *stream)
{
    if (num_episodes < 0 || num_views < 1 || n_view < 0 || n_view > 16384 || hidden < 1) return ROLESUB_EINVAL;
    if (dtype != ROLESUB_F32 && dtype != ROLESUB_BF16) return ROLESUB_EINVAL;
    const int32_t k = rolesub_select_count(n_view, ratio);
    if (k < 0) return ROLESUB_EINVAL;
    const int64_t row_bytes = (int64_t)hidden * elem_bytes(dtype);
    if (row_bytes % 16 != 0) return ROLESUB_EINVAL;
    const int64_t groups = (int64_t)num_episodes * num_views;
    if (groups == 0 || n_view == 0) return ROLESUB_OK;
    const void *ptrs[] = {scores, x, keep_idx, x_keep};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    return from_cuda(rs::launch_select_tokens(groups, n_view, k, scores, x, row_bytes, keep_idx, x_keep,
                                              (cudaStream_t)stream));
}

rolesub_status rolesub_dense_workspace_size(const rolesub_shape *shape, const void *plan_host, size_t *bytes)
{
    if (!shape_ok(shape) || !bytes) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, nullptr, &pv);
    if (st != ROLESUB_OK) return st;
    *bytes = ws_sizes(shape, pv.hdr).total + dense_extra_bytes(shape, pv.hdr);
    return ROLESUB_OK;
}

rolesub_status rolesub_compress_dense(const rolesub_shape *shape, const void *plan_host, const void *plan_dev,
                                      const void *h, const void *v, const void *R_dense, const void *W_re,
                                      const float *b_re, const void *W1, const float *b1, const void *W2,
                                      const float *b2, float alpha_role, float alpha_lang, void *packed_v,
                                      uint8_t *idx, void *workspace, size_t ws_bytes, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const void *ptrs[] = {h, v, R_dense, W_re, b_re, W1, b1, W2, b2, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && (!idx || !aligned16(idx))) return ROLESUB_EINVAL;
    if (!isfinite(alpha_role) || !isfinite(alpha_lang)) return ROLESUB_EINVAL;
    if (!dense_supported(shape) || !rs::router_supported(shape) || !dense_plan_ok(shape, pv))
        return ROLESUB_EUNSUPPORTED;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (ws_bytes < w.total + dense_extra_bytes(shape, pv.hdr)) return ROLESUB_EINVAL;
    rs::CompressArgs a{};
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.h = h;
    a.v = v;
    a.R = R_dense;
    a.W_re = W_re;
    a.W1 = W1;
    a.W2 = W2;
    a.b_re = b_re;
    a.b1 = b1;
    a.b2 = b2;
    a.alpha_role = alpha_role;
    a.alpha_lang = alpha_lang;
    a.packed = packed_v;
    a.idx = idx;
    a.stream = (cudaStream_t)stream;
    const int L = shape->num_layers, d = shape->num_heads * shape->head_dim, g = d / 16;
    const DenseWs dw = dense_ws(shape, pv.hdr);
    char *xb = static_cast<char *>(workspace) + w.total;
    int2 *pairs = reinterpret_cast<int2 *>(xb + dw.vt + dw.perm + dw.ident);
    int32_t *meta = reinterpret_cast<int32_t *>(xb + dw.vt + dw.perm + dw.ident + dw.pairs);
    cudaError_t e = rs::launch_router(a);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    // indices 0..S-1 of k = S rows (the records it also writes are not used)
    e = rs::launch_row_store(pv, L, idx, P.idx_bytes_per_layer, true, reinterpret_cast<uint4 *>(a.ws.row_store),
                             a.ws.status, a.stream);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    if (P.idx_bytes_per_layer == 0) return ROLESUB_OK;
    // the kept (row, group) pairs per chunk and group, then z_s = R_s^T v of
    // each pair straight to its packed slot
    const int chunks = dense_chunks(pv.hdr);
    e = rs::launch_dense_pairs(pv, L, g, idx, pairs, meta, chunks, a.ws.status, a.stream);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    rs::DenseCompressGemm gp{};
    gp.rows = P.rows_per_layer;
    gp.d = d;
    gp.g = g;
    gp.nt = std::min(g, 256);
    gp.chunks = chunks;
    gp.pairs = pairs;
    gp.pairs_per_layer = P.idx_bytes_per_layer;
    gp.meta = meta;
    gp.packed = static_cast<__nv_bfloat16 *>(packed_v);
    gp.packed_per_layer = P.packed_elems_per_layer;
    gp.status = a.ws.status;
    return from_cuda(rs::launch_dense_compress_gemm(gp, v, R_dense, L, dense_tiles_per_chunk(pv, chunks), a.stream));
}

rolesub_status rolesub_attend_dense(const rolesub_shape *shape, const void *plan_host, const void *plan_dev,
                                    const void *q, int64_t q_ls, int64_t q_rs, int64_t q_hs, const void *K,
                                    int64_t k_ls, int64_t k_rs, int64_t k_hs, const void *packed_v,
                                    const uint8_t *idx, const void *R_dense, float softmax_scale, void *o,
                                    void *workspace, size_t ws_bytes, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    const void *ptrs[] = {q, K, R_dense, o, workspace};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && !idx) return ROLESUB_EINVAL;
    const int64_t strides[] = {q_ls, q_rs, q_hs, k_ls, k_rs, k_hs};
    for (int64_t x : strides)
        if (x < 0 || x % 8 != 0) return ROLESUB_EINVAL;
    if (!isfinite(softmax_scale) || softmax_scale < 0.f) return ROLESUB_EINVAL;
    if (!dense_supported(shape) || !dense_plan_ok(shape, pv)) return ROLESUB_EUNSUPPORTED;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (ws_bytes < w.total + dense_extra_bytes(shape, pv.hdr)) return ROLESUB_EINVAL;
    const int L = shape->num_layers, d = shape->num_heads * shape->head_dim, g = d / 16;
    const int64_t rows = P.rows_per_layer;
    const DenseWs dw = dense_ws(shape, pv.hdr);
    char *Vt = static_cast<char *>(workspace) + w.total;
    int32_t *perm = reinterpret_cast<int32_t *>(Vt + dw.vt);
    char *Rid = Vt + dw.vt + dw.perm;
    rs::AttendArgs a;
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, workspace);
    a.q = q;
    a.K = K;
    a.packed = packed_v;
    a.idx = idx;
    a.q_ls = q_ls;
    a.q_rs = q_rs;
    a.q_hs = q_hs;
    a.k_ls = k_ls;
    a.k_rs = k_rs;
    a.k_hs = k_hs;
    a.scale = softmax_scale;
    a.o = o;
    a.stream = (cudaStream_t)stream;
    // rows bucketed by kept-group set (and the attention's records pointing
    // at their sorted positions), then v~ = R M z over the kept groups only
    cudaError_t e = rs::launch_dense_sort(pv, L, d, shape->head_dim, idx, perm,
                                          reinterpret_cast<uint4 *>(a.ws.row_store), a.ws.status, a.stream);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    if (P.idx_bytes_per_layer > 0) {
        rs::DenseAttendGemm gp{};
        gp.rows = rows;
        gp.d = d;
        gp.g = g;
        gp.G = shape->num_groups;
        gp.segs = pv.segs_dev;
        gp.row_seg = pv.row_seg_dev;
        gp.idx = idx;
        gp.idx_per_layer = P.idx_bytes_per_layer;
        gp.slots_per_layer = P.idx_bytes_per_layer;
        gp.perm = perm;
        gp.vt = reinterpret_cast<__nv_bfloat16 *>(Vt);
        gp.status = a.ws.status;
        e = rs::launch_dense_attend_gemm(gp, packed_v, R_dense, L, a.stream);
    } else if (rows > 0) {
        e = cudaMemsetAsync(Vt, 0, 2 * (size_t)L * rows * d, a.stream);   // nothing kept: v~ = 0
    }
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    e = rs::launch_dense_identity(L, shape->num_heads, shape->head_dim, Rid, a.stream);
    if (e != cudaSuccess) return ROLESUB_ECUDA;
    // attention over v~ as plain per-head values (every group kept, R_h = I)
    a.packed = Vt;
    a.packed_per_layer = rows * d;
    a.R = Rid;
    a.records_ready = true;
    return from_cuda(rs::launch_attend_tc(a));
}

rolesub_status rolesub_get_device_status(const void *workspace, void *stream, int32_t *code_out,
                                         int32_t *detail_out)
{
    if (!workspace || !code_out || !aligned16(workspace)) return ROLESUB_EINVAL;
    int32_t hs[2] = {0, 0};
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemcpyAsync(hs, workspace, sizeof(hs), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return ROLESUB_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return ROLESUB_ECUDA;
    *code_out = hs[0];
    if (detail_out) *detail_out = hs[1];
    return ROLESUB_OK;
}

rolesub_status rolesub_reset_device_status(void *workspace, void *stream)
{
    if (!workspace || !aligned16(workspace)) return ROLESUB_EINVAL;
    return from_cuda(cudaMemsetAsync(workspace, 0, rs::kStatusBytes, (cudaStream_t)stream));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// rolesub_compress_static: compress without any allocation by the caller or
// the library. Its scratch is this fixed array, one per GPU that loads the
// library, held until the process exits. The host only ever passes the
// array's device address, looked up once per device; host code never
// dereferences the symbol itself (on the host it names a stand-in, not
// device memory).
// ---------------------------------------------------------------------------
#include <mutex>

static __device__ __align__(256) unsigned char g_compress_scratch[ROLESUB_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void *g_scratch_addr[kMaxDevices];  // device address of g_compress_scratch per device

// Device address of the scratch array on the current device (set-up on the
// first call per device).
rolesub_status static_scratch(void **out)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return ROLESUB_ECUDA;
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_compress_scratch) != cudaSuccess || !p) return ROLESUB_ECUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return ROLESUB_OK;
}

}  // namespace

extern "C" rolesub_status rolesub_compress_static(
    const rolesub_shape *shape, const void *plan_host, const void *plan_dev, const void *h,
    const void *v, const void *R, const void *W_re, const float *b_re, const void *W1,
    const float *b1, const void *W2, const float *b2, float alpha_role, float alpha_lang,
    void *packed_v, uint8_t *idx, void *stream)
{
    if (!shape_ok(shape)) return ROLESUB_EINVAL;
    PlanView pv;
    rolesub_status st = view_plan(shape, plan_host, plan_dev, &pv);
    if (st != ROLESUB_OK) return st;
    if (!plan_dev) return ROLESUB_EINVAL;
    const void *ptrs[] = {h, v, R, W_re, b_re, W1, b1, W2, b2};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ROLESUB_EINVAL;
    const rolesub_plan &P = *pv.hdr;
    if (P.packed_elems_per_layer > 0 && (!packed_v || !aligned16(packed_v))) return ROLESUB_EINVAL;
    if (P.idx_bytes_per_layer > 0 && (!idx || !aligned16(idx))) return ROLESUB_EINVAL;
    if (!isfinite(alpha_role) || !isfinite(alpha_lang)) return ROLESUB_EINVAL;
    const WsSizes w = ws_sizes(shape, pv.hdr);
    if (w.total > (size_t)ROLESUB_STATIC_SCRATCH_BYTES) return ROLESUB_ETOOLARGE;
    if (!rs::router_supported(shape) || !rs::rotate_supported(shape)) return ROLESUB_EUNSUPPORTED;
    void *scratch = nullptr;
    st = static_scratch(&scratch);
    if (st != ROLESUB_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    // the previous call's status word is still in the array
    if (cudaMemsetAsync(scratch, 0, rs::kStatusBytes, s) != cudaSuccess) return ROLESUB_ECUDA;
    rs::CompressArgs a;
    a.shape = shape;
    a.plan = pv;
    a.ws = carve(w, scratch);
    a.h = h;
    a.v = v;
    a.R = R;
    a.W_re = W_re;
    a.W1 = W1;
    a.W2 = W2;
    a.b_re = b_re;
    a.b1 = b1;
    a.b2 = b2;
    a.alpha_role = alpha_role;
    a.alpha_lang = alpha_lang;
    a.packed = packed_v;
    a.idx = idx;
    a.stream = s;
    if (rs::launch_router(a) != cudaSuccess) return ROLESUB_ECUDA;
    return from_cuda(rs::launch_rotate_pack(a));
}

extern "C" rolesub_status rolesub_static_device_status(void *stream, int32_t *code_out, int32_t *detail_out)
{
    if (!code_out) return ROLESUB_EINVAL;
    void *scratch = nullptr;
    rolesub_status st = static_scratch(&scratch);
    if (st != ROLESUB_OK) return st;
    // the status word is the first 8 bytes of the array (code, detail)
    int32_t hs[2] = {0, 0};
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemcpyAsync(hs, scratch, sizeof(hs), cudaMemcpyDeviceToHost, s) != cudaSuccess) return ROLESUB_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return ROLESUB_ECUDA;
    *code_out = hs[0];
    if (detail_out) *detail_out = hs[1];
    return ROLESUB_OK;
}

extern "C" size_t rolesub_static_scratch_bytes(void) { return (size_t)ROLESUB_STATIC_SCRATCH_BYTES; }
