/*
 * rolesub.h -- C ABI of the RoleSub hot path on sm_103a (GB300).
 *
 * RoleSub (role-conditioned sub-token routing) keeps keys and queries as
 * they are and compresses the value vectors of retained tokens (Sec. 3):
 *
 *   compress (Sec. 3.2-3.4): per retained token i and layer l
 *     z_i   = R^T v_i                   rotation into the routing space
 *     a_i   = softmax(W_re h_i + b_re)   latent role, Eq. (latentrole)
 *     gamma = W2 ReLU(W1 [h_i ; alpha_role a_i ; alpha_lang c] + b1) + b2
 *             with c the mean hidden state of the episode's retained
 *             language tokens, Eq. (routingscore) in concatenation form
 *     keep the K_i groups with the largest gamma (ties: lower index) and
 *     store only those groups of z_i plus their indices.
 *   attend: query tokens read full keys and the routed values,
 *     o = sum_j softmax_j(q.k_j * scale) R M_j R^T v_j
 *       = R_h sum_j p_j M_j z_j        (accumulated in the rotated space)
 *
 * Geometry. d = H * d_h. The orthonormal value rotation is per head,
 * R = blockdiag(R_1..R_H); group s of head h holds head dims
 * [s*d_s, (s+1)*d_s), d_s = d_h / S. One group mask per token is shared by
 * all heads (one score vector gamma in R^S per token, Sec. 3.4).
 *
 * Conventions for every entry point:
 *  - All functions are synchronous on the host for validation and return a
 *    rolesub_status. Device work is enqueued on the caller's CUDA stream
 *    (cudaStream_t passed as void*; NULL = legacy default stream) and is
 *    asynchronous; no entry point synchronises except
 *    rolesub_get_device_status. The first kernel of a call starts after
 *    all earlier work on the stream; the later kernels of the same call are
 *    launched as programmatic dependents of the kernel before them (they
 *    may be scheduled while it finishes and wait for it before reading
 *    anything it writes), so a call's result is the same as with plain
 *    stream order.
 *  - The caller owns every buffer. The library allocates no memory and keeps
 *    no state between calls, apart from one-time per-process lookups, a
 *    diagnostic counter of kernel launches (rolesub_launch_count) and the
 *    fixed per-GPU scratch array of rolesub_compress_static, which that
 *    call alone uses and which keeps its contents from one call to the next.
 *  - Device pointers must be 16-byte aligned; ROLESUB_EINVAL otherwise.
 *  - Argument errors return ROLESUB_EINVAL (or ROLESUB_EUNSUPPORTED for a
 *    valid geometry this build does not implement) before anything is
 *    launched. A failed launch returns ROLESUB_ECUDA.
 *  - Bad data found on the device (a stored group index >= S, a bounded
 *    wait that ran out) is recorded in the workspace's status word; the
 *    kernel skips the offending item and never traps. Read it with
 *    rolesub_get_device_status.
 *  - Tensor element type: one dtype per call (shape.dtype) for h, v, R,
 *    W_re, W1, W2, q, K, packed values and o. Biases are float32.
 */
#ifndef ROLESUB_H
#define ROLESUB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ROLESUB_VERSION 1
#define ROLESUB_PLAN_MAGIC 0x42555352u /* "RSUB" */
#define ROLESUB_NUM_KINDS 4
#define ROLESUB_MAX_GROUPS 16

typedef enum {
    ROLESUB_OK = 0,
    ROLESUB_EINVAL = 1,        /* bad argument or plan; nothing launched      */
    ROLESUB_EUNSUPPORTED = 2,  /* geometry not implemented; nothing launched  */
    ROLESUB_ECUDA = 3,         /* CUDA runtime error or failed launch         */
    ROLESUB_EDEVICE = 4,       /* kernel found bad data (device status word)  */
    ROLESUB_ETIMEOUT = 5,      /* a bounded in-kernel wait gave up            */
    ROLESUB_ETOOLARGE = 6      /* needs more than the static scratch holds    */
} rolesub_status;

typedef enum { ROLESUB_F32 = 0, ROLESUB_BF16 = 1 } rolesub_dtype;

/* Token types of Sec. 3.1; every episode has one segment of each, in this
 * order (a segment may be empty). */
typedef enum { ROLESUB_VIS = 0, ROLESUB_LANG = 1, ROLESUB_PROP = 2, ROLESUB_ACT = 3 } rolesub_kind;

typedef struct {
    int32_t num_layers;    /* L                                               */
    int32_t num_heads;     /* H                                               */
    int32_t head_dim;      /* d_h (d = H * d_h)                               */
    int32_t num_groups;    /* S, 1..16, divides d_h (Sec. 3.2)                */
    int32_t role_dim;      /* C, latent role components (Sec. 3.3)            */
    int32_t router_hidden; /* F, width of the router's hidden layer           */
    int32_t dtype;         /* rolesub_dtype                                   */
    int32_t reserved;      /* must be 0                                       */
} rolesub_shape;

/* One (episode, kind) run of cache rows. Offsets are per layer; layer l's
 * arrays start at l * {rows,packed_elems,idx_bytes}_per_layer. */
typedef struct {
    int32_t episode;
    int32_t kind;          /* rolesub_kind                                    */
    int32_t n_tokens;      /* retained tokens of this type (|I_m^keep|)       */
    int32_t k;             /* kept groups per token K_m, 0..S                 */
    int64_t token_row;     /* first row of this segment in h / v / K          */
    int64_t packed_off;    /* element offset of its [H][n_tokens][k][d_s]     */
    int64_t idx_off;       /* byte offset of its [n_tokens][k] uint8 indices  */
} rolesub_segment;

typedef struct {
    int64_t row_begin;     /* first cache row of the episode                  */
    int64_t q_row_begin;   /* first query row of the episode                  */
    int32_t n_cache;       /* cache rows (all kinds)                          */
    int32_t n_query;       /* query rows                                      */
    int32_t seg_begin;     /* index of its first segment (= 4 * episode)      */
    int32_t n_lang;        /* retained language tokens                        */
    int64_t lang_row_begin;
} rolesub_episode;

/* A plan is one self-contained byte blob: this header followed by the
 * arrays it points to (byte offsets from the start of the blob). The same
 * bytes are used on the host (validation, grid sizes) and, copied verbatim
 * by the caller into device memory, by the kernels. */
typedef struct {
    uint32_t magic;                  /* ROLESUB_PLAN_MAGIC                     */
    uint32_t version;                /* ROLESUB_VERSION                        */
    int32_t num_episodes;
    int32_t num_segments;            /* 4 * num_episodes                       */
    int64_t rows_per_layer;          /* cache rows of every episode            */
    int64_t q_rows_per_layer;        /* query rows of every episode            */
    int64_t packed_elems_per_layer;  /* sum over segments of H*n*k*d_s         */
    int64_t idx_bytes_per_layer;     /* sum over segments of n*k               */
    int64_t routed_rows_per_layer;   /* rows of segments with 0 < k < S        */
    int64_t stored_rows_per_layer;   /* rows of segments with k > 0            */
    int32_t max_cache_tokens;        /* max n_cache over episodes              */
    int32_t max_query_tokens;        /* max n_query over episodes              */
    int32_t num_heads, head_dim, num_groups, reserved;  /* geometry checked at use */
    int64_t off_segments;            /* rolesub_segment[num_segments]          */
    int64_t off_episodes;            /* rolesub_episode[num_episodes]          */
    int64_t off_row_seg;             /* int32[rows_per_layer]: segment of row  */
    int64_t off_routed_rows;         /* int32[routed_rows]: ascending row ids  */
    int64_t off_stored_rows;         /* int32[stored_rows]: ascending row ids  */
    int64_t total_bytes;             /* size of the whole blob                 */
    int32_t num_route_tiles;         /* 128-row windows covering routed rows   */
    int32_t reserved2;
    int64_t off_route_tiles;         /* int32[num_route_tiles]: first row      */
} rolesub_plan;

/* Bytes needed for the plan of num_episodes episodes with n_tok[e*4+kind]
 * tokens. ROLESUB_EINVAL on negative counts. */
rolesub_status rolesub_plan_size(int32_t num_episodes, const int32_t *n_tok, size_t *bytes);

/*
 * Cache layout of Sec. 3.2's packed values (the paper fixes only the
 * accounting: keys full, K_i of S value groups per token; the layout is this
 * library's): segments ordered episode-major, kind-minor; segment
 * (n tokens, k groups) holds values [H][n][k][d_s] at packed_off and indices
 * [n][k] (ascending group ids, uint8) at idx_off. k = S stores every group
 * with indices 0..S-1; k = 0 stores nothing.
 *   n_tok[e*4+m], k[e*4+m]: tokens and kept groups of kind m in episode e
 *   n_query[e]: query tokens of episode e
 *   plan / plan_bytes: host output buffer (>= rolesub_plan_size), 16-byte
 *   aligned. Copy plan->total_bytes of it to a 16-byte-aligned device buffer
 *   to obtain plan_dev for the calls below.
 * ROLESUB_EINVAL on k outside 0..S, bad geometry or a short buffer.
 */
rolesub_status rolesub_layout_plan(const rolesub_shape *shape, int32_t num_episodes,
                                   const int32_t *n_tok, const int32_t *k,
                                   const int32_t *n_query, void *plan, size_t plan_bytes);

/* Scratch bytes a compress or attend call needs (the larger of the two).
 * The workspace also holds the device status word; zero it once (or call
 * rolesub_reset_device_status) before the first call that uses it. */
rolesub_status rolesub_workspace_size(const rolesub_shape *shape, const void *plan_host,
                                      size_t *bytes);

/*
 * Routing and packing of every routed token of every layer (Sec. 3.2-3.4).
 * Inputs (device, dtype = shape.dtype unless noted, row-major contiguous):
 *   h     [L][rows][d]          hidden states of the cache rows
 *   v     [L][rows][H][d_h]     value vectors
 *   R     [L][H][d_h][d_h]      per-head orthonormal rotation (R[m][n])
 *   W_re  [L][C][d], b_re [L][C] float32    role estimator
 *   W1    [L][F][2d+C], b1 [L][F] float32   router hidden layer; input
 *                                            columns [h | role | language]
 *   W2    [L][S][F],  b2 [L][S]  float32    router output layer
 *   alpha_role, alpha_lang                   Eq. (routingscore) weights
 * Outputs (device):
 *   packed_v [L][packed_elems_per_layer]  dtype; rotated kept groups
 *   idx      [L][idx_bytes_per_layer]     uint8; kept groups, ascending
 * workspace / ws_bytes: device scratch (>= rolesub_workspace_size).
 * Segments with k = 0 write nothing; k = S store every group without
 * running the router.
 */
rolesub_status rolesub_compress(const rolesub_shape *shape, const void *plan_host,
                                const void *plan_dev, const void *h, const void *v,
                                const void *R, const void *W_re, const float *b_re,
                                const void *W1, const float *b1, const void *W2,
                                const float *b2, float alpha_role, float alpha_lang,
                                void *packed_v, uint8_t *idx, void *workspace,
                                size_t ws_bytes, void *stream);

/*
 * rolesub_compress with the routing score in the additive form of Sec. 3.4
 * (Eq. routingscore), the token and language heads being linear maps:
 *   gamma_i = (W_v h_i + b_v) + alpha_role W_role a_i
 *             + alpha_lang (W_l c_e + b_l)
 *   a_i = softmax(W_re h_i + b_re)            Eq. (latentrole)
 *   c_e = mean of the episode's retained language hidden states (Sec. 3.4)
 * then the K_i largest gamma are kept (ties: lower group index) and the
 * rotation and packing run exactly as in rolesub_compress.
 * Inputs (device, dtype = shape.dtype unless noted, row-major contiguous):
 *   h, v, R, W_re, b_re     as rolesub_compress
 *   W_v    [L][S][d], b_v [L][S] float32     token head
 *   W_role [L][S][C]                          role head
 *   W_l    [L][S][d], b_l [L][S] float32     language head
 * shape.router_hidden is not used by this call (any value >= 1).
 * Outputs, workspace (rolesub_workspace_size of the same shape), stream and
 * errors: as rolesub_compress; ROLESUB_EUNSUPPORTED when S > 32 or C > 4096.
 */
rolesub_status rolesub_compress_additive(const rolesub_shape *shape, const void *plan_host,
                                         const void *plan_dev, const void *h, const void *v,
                                         const void *R, const void *W_re, const float *b_re,
                                         const void *W_v, const float *b_v, const void *W_role,
                                         const void *W_l, const float *b_l, float alpha_role,
                                         float alpha_lang, void *packed_v, uint8_t *idx,
                                         void *workspace, size_t ws_bytes, void *stream);

/*
 * Attention of every episode's query tokens over its own routed cache
 * (all cache tokens of the episode, non-causal), per layer and head:
 *   s_j = (q . k_j) * scale, p = softmax_j(s), y = sum_j p_j M_j z_j,
 *   o = R_h y.
 * Inputs (device, dtype = shape.dtype):
 *   q  [L][q_rows][H][d_h], element (l, r, h, t) at
 *      l*q_layer_stride + r*q_row_stride + h*q_head_stride + t
 *   K  [L][rows][H][d_h], same addressing with the k_* strides (the
 *      caller's key cache; read in place). Strides are in elements and must
 *      be multiples of 8 (16 bytes of bf16; 4 suffice for float32).
 *   packed_v, idx   as written by rolesub_compress
 *   R  [L][H][d_h][d_h]
 *   softmax_scale   0 means 1/sqrt(d_h)
 * Output: o [L][q_rows][H][d_h] contiguous, dtype.
 * A cache with no tokens gives o = 0. Stored indices >= S are skipped and
 * reported through the device status word.
 */
rolesub_status rolesub_attend(const rolesub_shape *shape, const void *plan_host,
                              const void *plan_dev, const void *q, int64_t q_layer_stride,
                              int64_t q_row_stride, int64_t q_head_stride, const void *K,
                              int64_t k_layer_stride, int64_t k_row_stride,
                              int64_t k_head_stride, const void *packed_v, const uint8_t *idx,
                              const void *R, float softmax_scale, void *o, void *workspace,
                              size_t ws_bytes, void *stream);

/*
 * Per-token value budgets (Sec. 3.5) with the additive routing score
 * (Sec. 3.4, as in rolesub_compress_additive).
 *
 * In a segment of n tokens whose plan entry has k = K_m with 0 < K_m < S,
 * the tokens share B_m = K_m n groups: token i keeps K_i groups,
 * 0 <= K_i <= S, sum_i K_i = B_m, more for higher role-derived priority.
 * The paper states those constraints but no formula; this library's
 * allocator:
 *   pi_i = u . a_i, a_i = softmax(W_re h_i + b_re)   (Eq. latentrole)
 *   rank the tokens by pi (higher first; ties: lower token index); rank r
 *   has weight n - r; real shares x_r = min(S, lambda (n - r)) with
 *   sum x = B_m; K = x rounded by largest remainders (ties: better rank).
 * Priorities and scores are fp32 on the device; tokens whose priorities lie
 * within rounding of each other may exchange ranks.
 * Token i keeps its K_i largest scores (ties: lower group index), indices
 * ascending. Segments with K_m = S keep everything, K_m = 0 nothing.
 *
 * Cache layout: the plan's segment regions are unchanged (B_m groups per
 * head, B_m index bytes); inside a segment token i's indices start at
 * idx_off + sum_{j<i} K_j and head h's values at
 * packed_off + (h B_m + sum_{j<i} K_j) d_s.
 *
 * Inputs: as rolesub_compress_additive, plus
 *   u      [L][C] float32   priority vector of each layer's allocator
 * Outputs: packed_v, idx as above and
 *   k_tok  [L][rows_per_layer] uint8   K_i of every cache row (the attention
 *          call needs it)
 * workspace: at least rolesub_budget_workspace_size bytes (the common
 * workspace followed by the router's scores and priorities).
 * Supported geometry: bf16, d_h = 128, S = 16, S + C <= 256, d % 64 == 0,
 * segments of at most 8192 tokens; otherwise ROLESUB_EUNSUPPORTED.
 * Other errors: as rolesub_compress.
 */
rolesub_status rolesub_budget_workspace_size(const rolesub_shape *shape, const void *plan_host,
                                             size_t *bytes);
rolesub_status rolesub_compress_budget(const rolesub_shape *shape, const void *plan_host,
                                       const void *plan_dev, const void *h, const void *v,
                                       const void *R, const void *W_re, const float *b_re,
                                       const void *W_v, const float *b_v, const void *W_role,
                                       const void *W_l, const float *b_l, const float *u,
                                       float alpha_role, float alpha_lang, void *packed_v,
                                       uint8_t *idx, uint8_t *k_tok, void *workspace,
                                       size_t ws_bytes, void *stream);

/*
 * rolesub_attend over a cache written by rolesub_compress_budget: the same
 * arguments plus its k_tok. Counts above S, counts that overrun a segment's
 * B_m and stored indices >= S are reported through the device status word
 * (ROLESUB_EDEVICE) and that row contributes no values. workspace:
 * rolesub_workspace_size bytes. Geometry: as rolesub_compress_budget.
 */
rolesub_status rolesub_attend_budget(const rolesub_shape *shape, const void *plan_host,
                                     const void *plan_dev, const void *q, int64_t q_layer_stride,
                                     int64_t q_row_stride, int64_t q_head_stride, const void *K,
                                     int64_t k_layer_stride, int64_t k_row_stride,
                                     int64_t k_head_stride, const void *packed_v,
                                     const uint8_t *idx, const uint8_t *k_tok, const void *R,
                                     float softmax_scale, void *o, void *workspace,
                                     size_t ws_bytes, void *stream);

/*
 * Token-level reduction (Sec. 3.1), the step before the value path: a
 * selector scores every visual token (u_i = psi(h_i, X); the paper takes
 * the scores from a separate method, so they are an input here) and the
 * ceil(r |I|) highest-scoring tokens are retained, the budget divided
 * evenly between the camera views (Sec. 4.1).
 *
 * rolesub_select_count: tokens kept per view, ceil(ratio * n_view) in double
 * precision; -1 unless 0 < ratio <= 1 and n_view >= 0.
 *
 * rolesub_select_tokens: for each of num_episodes x num_views groups of
 * n_view tokens (episode-major, then view; row-major rows of `hidden`
 * elements of `dtype`), keeps the k = rolesub_select_count(n_view, ratio)
 * tokens with the highest score (ties: lower token index; NaN scores rank
 * lowest) in their original order.
 *   scores   [E][V][n_view] float32 (device)
 *   x        [E][V][n_view][hidden] (device), hidden * element size a
 *            multiple of 16 bytes
 * Outputs (device):
 *   keep_idx [E][V][k] int32, the kept tokens' indices within their view,
 *            ascending
 *   x_keep   [E][V][k][hidden], their rows
 * All pointers 16-byte aligned. n_view <= 16384. Errors: ROLESUB_EINVAL on
 * bad arguments (nothing launched), ROLESUB_ECUDA on a failed launch.
 */
int32_t rolesub_select_count(int32_t n_view, double ratio);
rolesub_status rolesub_select_tokens(int32_t num_episodes, int32_t num_views, int32_t n_view, double ratio,
                                     const float *scores, const void *x, int32_t hidden, int32_t dtype,
                                     int32_t *keep_idx, void *x_keep, void *stream);

/*
 * The dense-rotation geometry of the paper's setup (Sec. 4.1): one d x d
 * orthonormal R per layer (d = H d_h) and S contiguous groups of g = d / S
 * rotated dims, in place of the per-head R_h of rolesub_compress.
 *
 * rolesub_compress_dense: routing as rolesub_compress (same router, same
 * indices), then z_i = R^T v_i over all d dims and the kept groups packed:
 * segment (n tokens, k) holds [n][k][g] values, token i's groups in index
 * order at packed_off + (i k + j) g (the plan's segment sizes are the same:
 * n k H d_s = n k g).
 *   R_dense [L][d][d] (R[m][n], dtype); other arguments as rolesub_compress.
 * Only the kept groups are computed: z_s = R_s^T v (R_s the g columns of
 * group s) for each kept (token, group) pair, written to its packed slot.
 * rolesub_attend_dense: attention over such a cache; every head's output
 * needs all d rotated dims (o_{q,h} = R_h sum_j p_j M_j z_j with R_h the d_h
 * rows of head h), so the call first forms the routed values
 * v~_j = R M_j z_j = sum over kept s of R_s z_{j,s} of every cache row on
 * the tensor core (reading the packed groups in place) and then attends
 * over them; arguments as rolesub_attend plus R_dense.
 * workspace: at least rolesub_dense_workspace_size bytes for either call
 * (the common workspace, then L rows d + L H d_h^2 bf16 elements, L rows
 * int32, 2 L idx_bytes_per_layer int32 and 32 L ceil(rows / 4096) int32).
 * Supported geometry: bf16, d_h = 128, S = 16, d a multiple of 256 with
 * g = d / 16 equal to 64, 128 or a multiple of 256, and a plan laid out by
 * rolesub_plan_build; otherwise ROLESUB_EUNSUPPORTED.
 */
rolesub_status rolesub_dense_workspace_size(const rolesub_shape *shape, const void *plan_host,
                                            size_t *bytes);
rolesub_status rolesub_compress_dense(const rolesub_shape *shape, const void *plan_host,
                                      const void *plan_dev, const void *h, const void *v,
                                      const void *R_dense, const void *W_re, const float *b_re,
                                      const void *W1, const float *b1, const void *W2,
                                      const float *b2, float alpha_role, float alpha_lang,
                                      void *packed_v, uint8_t *idx, void *workspace,
                                      size_t ws_bytes, void *stream);
rolesub_status rolesub_attend_dense(const rolesub_shape *shape, const void *plan_host,
                                    const void *plan_dev, const void *q, int64_t q_layer_stride,
                                    int64_t q_row_stride, int64_t q_head_stride, const void *K,
                                    int64_t k_layer_stride, int64_t k_row_stride,
                                    int64_t k_head_stride, const void *packed_v,
                                    const uint8_t *idx, const void *R_dense, float softmax_scale,
                                    void *o, void *workspace, size_t ws_bytes, void *stream);

/* Waits for the stream, then reads the workspace's status word:
 * *code_out = 0 when no kernel reported bad data, else a ROLESUB_E* code.
 * *detail_out (may be NULL) receives the first reported item. */
rolesub_status rolesub_get_device_status(const void *workspace, void *stream, int32_t *code_out,
                                         int32_t *detail_out);

/*
 * Self-test of the bounded in-kernel waits (the library's failure handling;
 * the paper has no counterpart). Launches one small kernel in which one
 * thread waits on an mbarrier that nothing arrives on, through the same wait
 * loop the tensor-core kernels use but with a limit of limit_ns, and a
 * second thread waits on it with the production limit (about 2 s). The
 * first wait runs out: it records ROLESUB_ETIMEOUT with site 900 in the
 * workspace's status word and raises the CTA's abort flag, which ends the
 * second wait at once (it records nothing). No copy or tensor-core work is
 * in flight; the kernel then returns and the context stays usable.
 *   limit_ns   1e3 .. 2e9
 *   workspace  device, 16-byte aligned, at least 256 bytes; its status word
 *              should be clear before the call
 *   out        device int64[4], 16-byte aligned: {first wait completed (0/1),
 *              its duration in ns, second wait completed (0/1), its duration}
 * ROLESUB_EINVAL (nothing launched) on bad arguments, ROLESUB_ECUDA on a
 * failed launch.
 */
rolesub_status rolesub_wait_selftest(int64_t limit_ns, void *workspace, int64_t *out, void *stream);

/* Enqueues a clear of the status word on the stream. */
rolesub_status rolesub_reset_device_status(void *workspace, void *stream);

/* Static description of a status code. */
const char *rolesub_status_string(rolesub_status s);

/* ROLESUB_VERSION of the library actually loaded. */
int32_t rolesub_version(void);

/*
 * rolesub_compress_static -- rolesub_compress for callers that cannot
 * allocate device memory. (The paper has no counterpart: this is a
 * deployment variant of the compress call.)
 *
 * Some callers cannot call cudaMalloc at the point where they compress: a
 * serving engine or robot-control loop that reserves all of its device
 * memory up front and forbids allocation afterwards, or a plug-in whose
 * host framework hands it inputs and outputs but no scratch buffer. This
 * entry point takes the same inputs and outputs as rolesub_compress, minus
 * the workspace: its scratch (language contexts, per-episode biases,
 * router logits, status word) lives in a fixed array compiled into the
 * library, ROLESUB_STATIC_SCRATCH_BYTES per GPU, which every GPU that loads
 * the library holds until the process exits. It calls no allocator.
 *
 * Limits and behaviour:
 *  - Problems whose scratch (rolesub_workspace_size) exceeds
 *    ROLESUB_STATIC_SCRATCH_BYTES return ROLESUB_ETOOLARGE; nothing runs.
 *  - The first call on a device looks up the array's device address (once
 *    per device, with that device current); make that first call before
 *    any stream capture.
 *  - Every call shares the one array and leaves its contents behind; the
 *    call clears what must start at zero itself. Calls whose work overlaps
 *    on the GPU (different streams, or different host threads on one
 *    device) race on the array: serialise them.
 *  - The device status word (a wait in the router or rotation kernel that
 *    ran out, ROLESUB_ETIMEOUT, with the site in the detail) is kept at the
 *    start of the array. Each call clears it when it starts; read the
 *    status of the latest call with rolesub_static_device_status.
 * Other arguments, errors and results: as rolesub_compress.
 */
#define ROLESUB_STATIC_SCRATCH_BYTES (8u << 20)
rolesub_status rolesub_compress_static(const rolesub_shape *shape, const void *plan_host,
                                       const void *plan_dev, const void *h, const void *v,
                                       const void *R, const void *W_re, const float *b_re,
                                       const void *W1, const float *b1, const void *W2,
                                       const float *b2, float alpha_role, float alpha_lang,
                                       void *packed_v, uint8_t *idx, void *stream);

/* Waits for the stream, then reads the status word that the latest
 * rolesub_compress_static call on the current device left in the fixed
 * array: *code_out = 0 when no kernel reported a problem, else a ROLESUB_E*
 * code; *detail_out (may be NULL) receives the reported site or item. No
 * counterpart in the paper. Allocates nothing; like the static call, its
 * first use on a device looks up the array's address. */
rolesub_status rolesub_static_device_status(void *stream, int32_t *code_out, int32_t *detail_out);

/* ROLESUB_STATIC_SCRATCH_BYTES as compiled into the loaded library. */
size_t rolesub_static_scratch_bytes(void);

/* Number of kernels this process has launched through the library so far
 * (all threads, all devices). Diagnostic only: a caller takes the
 * difference around a region to count its launches. */
uint64_t rolesub_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* ROLESUB_H */
