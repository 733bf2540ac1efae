// Host-side launchers of the Fusion kernels (one translation unit each).
#pragma once

#include <cuda_runtime.h>

#include "common.cuh"
#include "plan.cuh"

namespace fz {

// ---- exit check (+ optional plan for the fused stage) ----------------------
struct ExitParams {
    Ragged in;
    const void *x;
    int dim;
    Head head;
    uint8_t *exit_mask;
    float *logits;
    float *max_prob;
    int *counters;   // workspace: [n_btile + 1], zero on entry, zero on exit
    float2 *partials;
    float *lg_tmp;   // workspace [n_btile * kExitBT][classes]: logits tiles of the general kernel (its
                     // last CTA per sample tile writes the rows of the samples that exit); NULL when
                     // no logits are requested or the cluster kernel runs
    int n_ctile;
    int n_btile;
    int do_plan;     // run the compaction plan in the last CTA
    PlanArgs plan;
    int *status;
    // the layers of an MLP exit head (zero for the linear head of the ragged CLS rows)
    int in_mode;     // 0: CLS rows of the ragged batch x; 1: dense rows x[s] of [B, dim]; 2: dense float32 rows u_in[s]
    int skip_ln;     // 1: the rows enter the product as they are (no LayerNorm)
    int out_mode;    // 0: softmax maximum and exit rule; 1: GELU(W u + b) rounded to the dtype into hidden_out
    const float *u_in;   // [max_batch, dim] for in_mode 2 (float-float high parts)
    const float *u_in_lo;   // [max_batch, dim] their low parts
    void *hidden_out;    // [max_batch, classes] for out_mode 1
};
cudaError_t launch_exit(int dtype, const ExitParams &p, cudaStream_t s);
size_t exit_smem_bytes(int dtype, int dim);

// ---- merge router with profile scaling ----------------------------------------------
struct RouterParams {
    Ragged in;
    const void *x;
    int dim;
    const void *w;    // router weight [dim], the tokens' dtype
    float beta, tau_tgt, tau_ref;
    int *r_out;       // [max_batch] merge counts by original id
    float *m_out;     // [max_batch] scaled merge ratios by original id, or NULL
    int *status;
};
cudaError_t launch_router(int dtype, const RouterParams &p, cudaStream_t s);

// ---- exit-head pooling: the CLS row or the size-weighted mean of the patch rows ----------
struct PoolParams {
    Ragged in;
    const void *x;
    int dim;
    const float *sizes;
    int pool;        // FUSION_POOL_CLS or FUSION_POOL_SPATIAL
    float *u_out;    // [max_batch, dim]: the pooled rows, float-float high parts
    float *u_lo;     // [max_batch, dim]: their low parts
    int *status;
};
cudaError_t launch_head_pool(int dtype, const PoolParams &p, cudaStream_t s);

// ---- size-aware attention over a ragged batch ---------------------------------------------------
struct AttnParams {
    Ragged in;
    const void *qkv;       // [max_rows, 3, heads, 64] bf16
    int heads;
    const float *sizes;    // [max_rows] or NULL (plain attention)
    void *out;             // [max_rows, heads, 64] bf16
    int *status;
};
size_t attn_smem_bytes(int max_tokens);
cudaError_t launch_attention(const AttnParams &p, cudaStream_t s);

// ---- pruning router: linear token scores ------------------------------------------------
struct ScoreParams {
    Ragged in;
    const void *x;
    int dim;
    const void *w;      // scoring head weight [dim], the tokens' dtype
    float b;            // scoring head bias
    float *scores_out;  // [max_rows]
    int group;          // lanes per row (set by the launcher)
    int *status;
};
struct ScoreLayout {
    int group;    // lanes per row
    int chunks;   // 16-byte chunks per lane
};
ScoreLayout score_layout(int dtype, int dim);
cudaError_t launch_token_scores(int dtype, const ScoreParams &p, cudaStream_t s);

// ---- stand-alone plan ----------------------------------------------------------
cudaError_t launch_plan(const PlanArgs &a, cudaStream_t s);

// ---- per-sample merge / prune / gather -----------------------------------------
// Batches of at most this many samples plan inside the per-sample kernel (every CTA
// scans the batch), larger ones run the plan kernel first.
constexpr int kFusedPlanMaxBatch = FUSION_FUSED_PLAN_MAX_BATCH;

struct ImageParams {
    Ragged in;
    const void *x;
    const void *keys;
    int dim;
    int kdim;
    int keys_alias;
    const float *sizes;
    const float *scores;
    const int *r;
    const float *rho;
    int do_merge;
    int do_prune;
    int need_match;      // compute matches even when no token merges (a_match requested)
    const int *slot;     // workspace: output sample of every input sample (-1: gone)
    const int *plan;     // workspace: plan[0] = batch valid
    const int *offsets_out;
    void *x_out;
    float *sizes_out;
    float *scores_out;
    int *keep_idx;
    const int *gate;        // NULL, or a device flag to wait for (bounded) before reading any input
    unsigned gate_spins;    // polls of that wait
    const int *keep_map;   // NULL, or the input row of every row of x (keep_idx = keep_map[row])
    int *dst_map;
    int *a_match;
    int *status;
    // fused_plan: no plan kernel ran; every CTA derives its sample's slot and output
    // offset from plan_args (which also receives the plan's outputs)
    int fused_plan;
    PlanArgs plan_args;
    // staging geometry, fixed by the host from max_tokens and the key width
    int resident;        // every key dim staged at once
    int kc;              // key dims staged per chunk (multiple of 16)
    int ra, rb;          // rows per chunk column of the A and B staging regions
};

struct ImageGeometry {
    int ok;              // fits in shared memory
    int resident;
    int kc;
    int ra, rb;
    size_t smem;         // dynamic shared memory bytes
};
ImageGeometry image_geometry(int dtype, int max_tokens, int kdim, int do_merge);
cudaError_t launch_image(int dtype, const ImageParams &p, size_t smem, cudaStream_t s);

// ---- per-sample kernel on TMA + tcgen05 (bf16, |A|, |B| <= 128, key width % 64 == 0) ----
struct TcGeometry {
    int ok;
    int tiled;         // halves beyond one tile: k_image_tc_tiled (M-tiles of 128 A rows, one CTA per SM)
    int grouped;       // samples that fit in shared memory load in 8-row groups of all K-blocks (one 3-D box
                       // per group) instead of through the ring
    int n_kb;          // key K-blocks of 64 dims
    int stages;        // K-block stages of a sample of max_tokens tokens (more for smaller samples)
    int tmem_cols;     // tensor-memory columns allocated per CTA
    uint32_t kb_a, kb_b;             // bytes of one K-block of half A / half B at max_tokens
    uint32_t stage_region;           // bytes of the K-block ring, from offset 0
    uint32_t meta_base;              // offset of the per-sample metadata
    uint32_t cls_base;               // offset of the staged CLS row (0: read from global memory)
    uint32_t usable;                 // bytes addressable after the 1 KB alignment
    size_t smem;                     // dynamic shared memory bytes (usable + 1 KB alignment slack)
};
TcGeometry image_tc_geometry(int dtype, int max_tokens, int kdim, int dim, long long max_rows, int do_merge,
                             int stage_budget_kb);
// pdl: launched as a programmatic dependent of the kernel before it on the stream (the exit
// check of a fused stage); the kernel waits for that grid before it reads any input
cudaError_t launch_image_tc(const ImageParams &p, const TcGeometry &g, cudaStream_t s, bool pdl = false);

}  // namespace fz
