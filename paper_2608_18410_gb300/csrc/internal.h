// internal.h -- host-side launchers shared between the C-ABI layer and the
// kernel translation units. Not part of the public ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "rolesub.h"

struct CUtensorMap_st;

namespace rs {

struct PlanView {  // host view of a validated plan + device copy
    const rolesub_plan *hdr;
    const rolesub_segment *segs;     // host
    const rolesub_episode *eps;      // host
    const char *dev;                 // device copy base
    const rolesub_segment *segs_dev;
    const rolesub_episode *eps_dev;
    const int32_t *row_seg_dev;
    const int32_t *routed_dev;
    const int32_t *stored_dev;
    const int32_t *route_tiles_dev;
};

struct Workspace {  // carve-up of the caller's workspace
    int32_t *status;
    float *lang_ctx;   // [L][E][d]
    float *lang_bias;  // [L][E][F]
    float *logits;     // [L][routed][F + C]   (router GEMM output)
    void *row_store;   // [L][rows] 16-byte store records (tensor-core rotation)
    size_t bytes;
};

struct CompressArgs {
    const rolesub_shape *shape;
    PlanView plan;
    Workspace ws;
    const void *h, *v, *R, *W_re, *W1, *W2;
    const float *b_re, *b1, *b2;
    float alpha_role, alpha_lang;
    void *packed;
    uint8_t *idx;
    cudaStream_t stream;
    bool records_ready = false;   // ws.row_store already holds the store records
};

// Weights of the additive routing score (Sec. 3.4, Eq. routingscore):
// W_v, W_l [L][S][d] and W_role [L][S][C] in the shape's dtype, b_v, b_l
// [L][S] float32.
struct AdditiveWeights {
    const void *W_v, *W_role, *W_l;
    const float *b_v, *b_l;
    // score mode (per-token budgets, Sec. 3.5): u [L][C] float32 gives the
    // priority pi = u . a; gamma and pi of every routed row go to scores
    // [L][rows][kScoreStride] (gamma at 0..S-1, pi at S) instead of a top-k
    const float *u = nullptr;
    float *scores = nullptr;
};
constexpr int kScoreStride = 20;   // floats per row: 16 scores, pi, padding to 16 bytes

struct AttendArgs {
    const rolesub_shape *shape;
    PlanView plan;
    Workspace ws;
    const void *q, *K, *packed, *R;
    const uint8_t *idx;
    int64_t q_ls, q_rs, q_hs, k_ls, k_rs, k_hs;
    float scale;
    void *o;
    cudaStream_t stream;
    const uint8_t *k_tok = nullptr;   // per-token kept counts (budget cache), or fixed k
    bool records_ready = false;       // ws.row_store already holds the store records
    int64_t packed_per_layer = 0;     // values per layer of `packed`; 0: the plan's
};

// Router: language pool + per-episode bias, router GEMM, epilogue/top-k.
cudaError_t launch_router(const CompressArgs &a);
// Language pool c_e of every (layer, episode) into ws.lang_ctx.
cudaError_t launch_lang_pool(const CompressArgs &a);
// Additive router: language term per episode, then scores and top-k per
// routed row (tcgen05 for bf16, S = 16, S + C <= 256, d % 64 == 0).
bool router_additive_supported(const rolesub_shape *s);
bool additive_tc_supported(const rolesub_shape *s);
cudaError_t launch_router_additive(const CompressArgs &a, const AdditiveWeights &w);
// Rotation z = R_h^T v and packing of the kept groups.
cudaError_t launch_rotate_pack(const CompressArgs &a);
// Fused router GEMM + epilogue + top-k on tcgen05/TMA (bf16, F = 256,
// C = 64, S = 16); needs the per-episode biases in the workspace.
bool router_tc_supported(const rolesub_shape *s);
cudaError_t launch_router_tc(const CompressArgs &a);
// 16-byte per-(layer, row) store records (kept group ids, packed offset, k)
// from the group indices; write_identity also fills indices of k = S rows.
// pdl: launched as a programmatic dependent of the kernel before it.
cudaError_t launch_row_store(const PlanView &pv, int L, uint8_t *idx, int64_t idx_per_layer,
                             bool write_identity, uint4 *recs, int32_t *status, cudaStream_t stream,
                             bool pdl = false);
// Rotation and packing on tcgen05/TMA (bf16, d_h = 128, S = 16).
bool rotate_tc_supported(const rolesub_shape *s);
cudaError_t launch_rotate_tc(const CompressArgs &a);
// Routed attention.
cudaError_t launch_attend(const AttendArgs &a);
// Routed attention on tcgen05/TMA (bf16, d_h = 128, S = 16).
bool attend_tc_supported(const rolesub_shape *s);
cudaError_t launch_attend_tc(const AttendArgs &a);
// The same for a budget cache (a.k_tok set); launch_attend_tc dispatches.
cudaError_t launch_attend_tc_budget(const AttendArgs &a);

// Per-token budgets (Sec. 3.5): from the scores and priorities of score
// mode, the counts K_i of every routed segment, the kept groups at prefix
// offsets, k_tok and the store records (also for k = 0 and k = S segments).
cudaError_t launch_budget_select(const CompressArgs &a, const float *scores, uint8_t *k_tok);
// Store records of a budget cache from its indices and per-token counts.
cudaError_t launch_row_store_budget(const PlanView &pv, int L, const uint8_t *idx, int64_t idx_per_layer,
                                    const uint8_t *k_tok, uint4 *recs, int32_t *status, cudaStream_t stream);

// Token-level reduction: per group of n scores keep the k best (ties: lower
// index) in order, their indices and rows (row_bytes each).
cudaError_t launch_select_tokens(int64_t groups, int n, int k, const float *scores, const void *x, int64_t row_bytes,
                                 int32_t *keep_idx, void *x_keep, cudaStream_t stream);

// Dense rotation (one d x d R per layer, S = 16 groups of g = d / S rotated
// dims). Compress: the kept (row, group) pairs of every 4096-row chunk,
// listed per group (dense.cu), then z of each pair on the tensor core,
// written to its packed slot (gemm_tc.cu). Attend: the rows of every layer
// bucketed by kept-group set, with attention records pointing at the sorted
// rows of v~ (dense.cu), then v~ = R M z on the tensor core over the kept
// groups only, read from the packed cache (gemm_tc.cu).
constexpr int kDenseChunk = 4096;       // rows per pair-list chunk
constexpr int kDenseMetaStride = 32;    // int32 per (layer, chunk): 16 counts, pair base
struct DenseCompressGemm {
    int64_t rows;                // cache rows per layer
    int d, g, nt;                // d = H d_h; g = d / 16; N tile min(g, 256)
    int chunks;                  // ceil(rows / kDenseChunk)
    const int2 *pairs;           // [L][pairs_per_layer] {row, packed slot}
    int64_t pairs_per_layer;     // = idx bytes per layer
    const int32_t *meta;         // [L][chunks][kDenseMetaStride]
    __nv_bfloat16 *packed;
    int64_t packed_per_layer;
    int32_t *status;
};
struct DenseAttendGemm {
    int64_t rows;
    int d, g, G;
    const rolesub_segment *segs;  // device plan
    const int32_t *row_seg;
    const uint8_t *idx;
    int64_t idx_per_layer;
    int64_t slots_per_layer;      // packed elements per layer / g
    const int32_t *perm;          // [L][rows]: sorted position -> row
    __nv_bfloat16 *vt;            // [L][rows][d]: v~ in sorted row order
    int32_t *status;
};
cudaError_t launch_dense_pairs(const PlanView &pv, int L, int g, const uint8_t *idx, int2 *pairs, int32_t *meta,
                               int chunks, int32_t *status, cudaStream_t stream);
cudaError_t launch_dense_compress_gemm(const DenseCompressGemm &p, const void *v, const void *R, int L,
                                       int tiles_per_chunk, cudaStream_t stream);
cudaError_t launch_dense_sort(const PlanView &pv, int L, int d, int dh, const uint8_t *idx, int32_t *perm,
                              uint4 *recs, int32_t *status, cudaStream_t stream);
cudaError_t launch_dense_attend_gemm(const DenseAttendGemm &p, const void *packed, const void *R, int L,
                                     cudaStream_t stream);
// Identity R_h of every (layer, head), so that the attention kernel reads
// v~ as plain per-head values.
cudaError_t launch_dense_identity(int L, int H, int dh, void *R_identity, cudaStream_t stream);

// Adds n to the process-wide launch counter (rolesub_launch_count).
void count_launches(int n);

// bf16 TMA descriptor with 128-byte swizzle (dims and strides innermost first).
bool make_bf16_map(CUtensorMap_st *m, const void *base, int rank, const uint64_t *dims,
                   const uint64_t *strides_bytes, const uint32_t *box);

// Limits of this build (checked before any launch).
bool router_supported(const rolesub_shape *s);
bool rotate_supported(const rolesub_shape *s);
bool attend_supported(const rolesub_shape *s);

}  // namespace rs
