/*
 * fusion.h: C ABI of the GB300 (sm_103a) library for the Fusion staged
 * token-adaptation step of Vision Transformers (arXiv 2607.02612):
 *
 *     merge  ->  exit-check  ->  prune  ->  compact
 *
 * run over a batch of ViT token tensors after a transformer block
 * (Sec. III-B: tokens are merged first, the exit check reads merged but
 * unpruned tokens, and only samples that continue are pruned; Algorithm 1).
 *
 * Conventions shared by every call
 * --------------------------------
 * Memory.   Every pointer argument is DEVICE memory owned by the caller, except
 *           where a comment says otherwise.  The library never allocates or
 *           frees; scratch space is the caller's `workspace` of
 *           fusion_workspace_size() bytes (see there).
 * Ragged batches.   A batch of samples is packed row-major: sample i owns the
 *           rows offsets[i] .. offsets[i+1]-1 of every per-token array, its
 *           first row is the CLS token (position 0) and rows 1..P_i are its patch
 *           tokens (positions 1..P_i, N_i = P_i + 1 rows).  Offsets must be
 *           non-decreasing with N_i >= 1.
 * Halves.   Inside a sample, half B is the odd positions 1,3,5,... (ceil(P/2)
 *           tokens) and half A the even positions 2,4,6,... (floor(P/2)
 *           tokens).  CLS is in neither half and is never merged or pruned.
 * Order.    Surviving tokens keep ascending position, CLS first; surviving
 *           samples keep ascending sample order.
 * Ties.     Lowest index wins everywhere: argmax -> lowest B position; top-r ->
 *           lowest A position; top-k pruning -> lowest position.
 * Types.    `dtype` (FUSION_F32 / FUSION_BF16) is the storage type of token
 *           rows (x, keys, x_out) and of the exit head's LayerNorm gamma/beta and
 *           weight.  Token sizes, scores, keep ratios, biases, logits and
 *           probabilities are float32; indices and counts are int32.
 *           bf16 rounding points: keys enter the dot products as stored; the
 *           LayerNorm output is rounded to bf16 before the head; a merged token
 *           is rounded to bf16 once, from the exact size-weighted mean.
 * Shapes.   dim and key_dim must be multiples of 16 and at most FUSION_MAX_DIM;
 *           every sample must have 1 <= N_i <= max_tokens <= FUSION_MAX_TOKENS.
 *           Token-row pointers (x, keys, x_out) must be 16-byte aligned.
 * Streams.  `stream` is a cudaStream_t passed as void*.  Every call only
 *           enqueues work on it and returns; nothing synchronises.  Device-side
 *           counts (survivor count, offsets) stay on the device.
 * Errors.   A negative return code means an argument failed a host-side check
 *           (or a launch failed) and NOTHING was enqueued (FUSION_ERR_CUDA: some
 *           work may have been enqueued before the failing launch).
 *           Problems only visible on the device (malformed offsets, a batch count
 *           out of range, NaN/Inf in a decision input) are OR-ed as
 *           FUSION_DEV_* bits into *dev_status, which the caller zeroes and
 *           reads after synchronising.  Kernels that detect such a problem write
 *           no token outputs for the affected samples (or for the whole call,
 *           for malformed offsets) and never access memory out of bounds.
 * Router outputs.  Per-sample merge counts r and keep ratios rho hold
 *           max_batch entries and are indexed by the sample's original id:
 *           r[ids[i]] when the batch carries ids, r[i] otherwise (so arrays drawn
 *           once per image stay valid after compaction).
 */
#ifndef FUSION_H
#define FUSION_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes -------------------------------------------------------- */
#define FUSION_OK 0
#define FUSION_ERR_INVALID_ARG -1 /* NULL where a pointer is required, bad flags, misalignment */
#define FUSION_ERR_SHAPE -2       /* dim / key_dim / max_tokens / classes out of range */
#define FUSION_ERR_DTYPE -3       /* dtype is neither FUSION_F32 nor FUSION_BF16 */
#define FUSION_ERR_WORKSPACE -4   /* workspace NULL or smaller than fusion_workspace_size() */
#define FUSION_ERR_CUDA -5        /* a CUDA call failed (launch configuration, device) */

/* ---- device status bits (OR-ed into *dev_status) -------------------------- */
#define FUSION_DEV_BAD_OFFSETS 1 /* offsets decreasing, N_i < 1, N_i > max_tokens or rows > max_rows */
#define FUSION_DEV_BAD_BATCH 2   /* *batch outside [0, max_batch] */
#define FUSION_DEV_NONFINITE 4   /* NaN/Inf in keys, scores, rho or a CLS row */
#define FUSION_DEV_INTERNAL 8    /* an internal consistency check failed (a library bug) */
#define FUSION_DEV_BAD_IDS 16    /* a sample id outside [0, max_batch) */
#define FUSION_DEV_TIMEOUT 32    /* a bounded wait inside a kernel gave up (outputs of that sample skipped) */

/* ---- storage types and stage flags --------------------------------------- */
#define FUSION_F32 0
#define FUSION_BF16 1

#define FUSION_STAGE_MERGE 1 /* merge (Sec. III-C) */
#define FUSION_STAGE_EXIT 2  /* exit check (Sec. III-D); exited samples leave the batch */
#define FUSION_STAGE_PRUNE 4 /* prune the samples that continue (Sec. III-E) */

#define FUSION_MAX_TOKENS 1024
#define FUSION_MAX_DIM 1024
/* batches of at most this many samples run their plan (validation, output offsets)
   inside the per-sample kernel; larger ones launch a plan kernel first */
#define FUSION_FUSED_PLAN_MAX_BATCH 1024

/* Size-aware attention (fusion_attention): head width and the longest sample. */
#define FUSION_ATTN_HEAD_DIM 64
#define FUSION_ATTN_MAX_TOKENS 1024

/* Pooling of an MLP exit head (fusion_mlp_head.pool). */
#define FUSION_POOL_CLS 0     /* the CLS row (the paper's CLS-only head, block 10) */
#define FUSION_POOL_SPATIAL 1 /* size-weighted mean of the patch rows (SpatialPool head, block 8) */

/* A ragged batch as seen by the device.  All pointers are device memory. */
typedef struct fusion_ragged {
    int32_t max_batch;      /* host upper bound on the number of samples (>= 0) */
    int32_t max_tokens;     /* host upper bound on N_i, CLS included (1..FUSION_MAX_TOKENS) */
    int64_t max_rows;       /* rows allocated in the token arrays; offsets[B] must not exceed it */
    const int32_t *offsets; /* [max_batch + 1]; entries beyond the actual count are ignored */
    const int32_t *batch;   /* device scalar with the actual count B (<= max_batch); NULL: B = max_batch */
    const int32_t *ids;     /* [max_batch] original sample ids in [0, max_batch); NULL: ids[i] = i */
} fusion_ragged;

/* Exit head of Sec. III-D: LayerNorm(CLS) -> Linear(dim -> classes) -> softmax;
 * a sample exits iff its maximum class probability c satisfies c >= tau (Eq. 7). */
typedef struct fusion_exit_head {
    const void *ln_gamma; /* [dim], dtype */
    const void *ln_beta;  /* [dim], dtype */
    float ln_eps;         /* LayerNorm epsilon (biased variance) */
    const void *weight;   /* [classes, dim] row-major, dtype */
    const float *bias;    /* [classes] float32 */
    int32_t classes;      /* C >= 1 */
    float tau;            /* exit threshold */
} fusion_exit_head;

/* Exit head as a 2-layer MLP (Sec. III-G; Sec. IV-I: the paper's SpatialPool head at
 * block 8 and CLS-only head at block 10): head(z) = W2 GELU(W1 LN(pool(z)) + b1) + b2,
 * then softmax; a sample exits iff its maximum class probability c >= tau (Eq. 7). */
typedef struct fusion_mlp_head {
    int32_t pool;         /* FUSION_POOL_CLS or FUSION_POOL_SPATIAL */
    const void *ln_gamma; /* [dim], dtype */
    const void *ln_beta;  /* [dim], dtype */
    float ln_eps;         /* LayerNorm epsilon (biased variance) */
    const void *w1;       /* [hidden, dim] row-major, dtype */
    const float *b1;      /* [hidden] float32 */
    int32_t hidden;       /* H: a multiple of 16 in [16, FUSION_MAX_DIM] */
    const void *w2;       /* [classes, hidden] row-major, dtype */
    const float *b2;      /* [classes] float32 */
    int32_t classes;      /* C >= 1 */
    float tau;            /* exit threshold */
} fusion_mlp_head;

/* Human-readable name of a return code or of a single FUSION_DEV_* bit. */
const char *fusion_status_string(int code);

/* Library version string (host memory owned by the library). */
const char *fusion_version(void);

/*
 * Profiling aid (no counterpart in the paper): arms the NEXT fusion_* call made
 * from the calling host thread to record up to three CUDA events (cudaEvent_t
 * passed as void*, NULL to skip) on that call's stream: `start` before its first
 * kernel, `mid` between its first kernel (plan or exit check) and its
 * per-sample kernel, `end` after its last kernel.  Inside a stream capture the
 * events are recorded by graph nodes, at every replay.  The events are created
 * and owned by the caller.  Returns FUSION_OK.
 */
int fusion_profile_next(void *start, void *mid, void *end);

/*
 * Launch gate (a failure-detection aid; no counterpart in the paper): while a gate is set,
 * the per-sample kernels of the merge, prune, compact and stage calls made afterwards from
 * the calling host thread wait, before reading any input, until the device int32 *flag is
 * nonzero, polling it at most `polls` more times after the first read (each poll takes
 * about 0.1 to 1 microsecond).  A CTA that gives up raises FUSION_DEV_TIMEOUT and writes no
 * output (nothing asynchronous is in flight at that point).  A caller can launch work ahead
 * of a producer that sets the flag; a test can check that a wait runs out.  flag NULL clears
 * the gate.  Returns FUSION_ERR_INVALID_ARG for polls < 0 with a flag, else FUSION_OK.
 */
int fusion_set_launch_gate(const int32_t *flag, int64_t polls);

/*
 * Bytes of scratch device memory every call needs for a batch bound of
 * max_batch samples and an exit head of `classes` classes (pass the largest
 * head used with this workspace; 1 when no exit check is run).  The workspace
 * must be zero-filled before its first use; every call leaves it zero-filled
 * again when its kernels complete, so it can be reused on the same stream
 * without clearing.  Calls that overlap on the device must not share one.
 */
size_t fusion_workspace_size(int32_t max_batch, int32_t classes);

/*
 * fusion_merge: bipartite soft matching and size-weighted merging of every
 * sample (Sec. III-C, after ToMe; Algorithm 1, merge branch).
 *
 * For sample i with halves A and B: every A token a is paired with the B token
 * j*(a) of largest cosine similarity of the L2-normalised keys
 * (k / max(||k||, 1e-12)); s(a) is that similarity.  The r_eff = min(max(r, 0),
 * |A|) A tokens with the largest s(a) are merged: every B token b becomes
 *     x'_b = sum_{t in S_b} size_t x_t / sum_{t in S_b} size_t,
 *     size'_b = sum size_t,  score'_b = sum score_t,
 * over S_b = {b} and the merged A tokens paired with b.  Other tokens are copied.
 * The sample keeps N_i - r_eff tokens.
 *
 * x [rows, dim] and keys [rows, key_dim]: dtype; keys may be the same pointer
 * as x.  sizes [rows] (> 0), scores [rows] (may be NULL), r [*]: int32.
 * Outputs (capacity in.max_rows rows unless stated):
 *   x_out [rows, dim], sizes_out [rows], scores_out [rows] (NULL iff scores is
 *   NULL), offsets_out [max_batch + 1], keep_idx [rows] (input row of every
 *   output row; may be NULL), dst_map [in.max_rows] (for every input row, the
 *   output row it was copied or merged into; may be NULL), a_match
 *   [in.max_rows] (for A rows the input row of the matched B token, -1 for the
 *   other rows; may be NULL).
 */
int fusion_merge(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *keys,
                 int32_t key_dim, const float *sizes, const float *scores, const int32_t *r,
                 void *x_out, float *sizes_out, float *scores_out, int32_t *offsets_out,
                 int32_t *keep_idx, int32_t *dst_map, int32_t *a_match, void *workspace,
                 size_t workspace_bytes, int32_t *dev_status, void *stream);

/*
 * fusion_exit_check: confidence-based early exit (Sec. III-D, Eq. 6-7).
 *
 * For every sample: u = LayerNorm(CLS row) with gamma, beta, eps and biased
 * variance (rounded to bf16 when dtype is FUSION_BF16); logits l = W u + b;
 * c = max_k softmax(l)_k; exit iff c >= tau.
 * Outputs: exit_mask [max_batch] uint8 (1 = exits), logits [max_batch, classes]
 * float32 (the early prediction: only the rows of samples that exit are written,
 * the other rows are untouched; may be NULL), max_prob [max_batch] float32 (may be
 * NULL).  Entries beyond the actual count are untouched.
 */
int fusion_exit_check(int dtype, fusion_ragged in, const void *x, int32_t dim,
                      fusion_exit_head head, uint8_t *exit_mask, float *logits, float *max_prob,
                      void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream);

/*
 * Scratch bytes of fusion_exit_check_mlp for max_batch samples, token width dim and
 * the head's hidden width and classes; zero-filled before its first use, left
 * zero-filled by every call (as fusion_workspace_size).
 */
size_t fusion_exit_mlp_workspace_size(int32_t max_batch, int32_t dim, int32_t hidden, int32_t classes);

/*
 * fusion_exit_check_mlp: the exit check (Sec. III-D, Eq. 6 and Eq. 7) with an MLP exit
 * head.  For every sample: z = its CLS row (FUSION_POOL_CLS) or sum_t s_t x_t / sum_t s_t
 * over its patch rows (FUSION_POOL_SPATIAL; the CLS row when it has no patch), in
 * float32; u = LayerNorm(z) (gamma, beta, eps, biased variance); h = GELU(W1 u + b1)
 * with GELU(a) = a (1 + erf(a / sqrt 2)) / 2; logits l = W2 h + b2; c = max_k
 * softmax(l)_k; exit iff c >= tau.  For FUSION_BF16, u and h are rounded to bf16 (the
 * operands of the two tensor-core products, float32 accumulation).
 * sizes: [max_rows] float32 token sizes (needed for FUSION_POOL_SPATIAL, else may be
 * NULL).  Outputs as fusion_exit_check: exit_mask [max_batch], logits [max_batch,
 * classes] (may be NULL), max_prob [max_batch] (may be NULL).
 * Errors: FUSION_ERR_INVALID_ARG for NULL or misaligned pointers or a bad pool;
 * FUSION_ERR_SHAPE for a hidden width outside the dim rule or classes < 1;
 * FUSION_ERR_WORKSPACE below fusion_exit_mlp_workspace_size; device bits BAD_BATCH,
 * BAD_OFFSETS (that sample's head input is zero), NONFINITE.
 */
int fusion_exit_check_mlp(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                          fusion_mlp_head head, uint8_t *exit_mask, float *logits, float *max_prob,
                          void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream);

/*
 * fusion_exit_check_noalloc: fusion_exit_check for callers that cannot allocate
 * device memory.  The paper has no counterpart; this is a deployment aid.
 *
 * Some callers have no way to call cudaMalloc (a plugin host that passes only
 * input and output buffers, a C program without a device allocator, a loop where
 * an allocation would stall).  This call takes the same inputs and outputs as
 * fusion_exit_check but no workspace: its scratch lives in a 1 MiB device array
 * inside the library, present on every GPU that loads the library until the
 * process exits.  A batch bound and class count whose scratch exceeds 1 MiB (see
 * fusion_workspace_size) is rejected with FUSION_ERR_WORKSPACE before anything is
 * enqueued.  Every call looks up the array's device address in the current context
 * (a host-side query); the first call on a device may load the library's device code
 * there, so make that first call before any stream capture.  Calls allocate nothing
 * (no cudaMalloc / cudaFree); each one clears the counters it needs with an
 * asynchronous memset on `stream`.  All calls on a device share the one array:
 * calls that may run concurrently on the GPU (unordered streams) race and must
 * not be issued.
 */
int fusion_exit_check_noalloc(int dtype, fusion_ragged in, const void *x, int32_t dim,
                              fusion_exit_head head, uint8_t *exit_mask, float *logits,
                              float *max_prob, int32_t *dev_status, void *stream);

/*
 * fusion_prune: keep CLS and the k_i = ceil(rho * P_i) patch tokens with the
 * largest scores (Sec. III-E, Eq. 8, with the keep count taken per sample), in
 * ascending position.  rho is read as its exact float32 value; k is clamped to
 * [0, P_i] (NaN rho keeps none and raises FUSION_DEV_NONFINITE).
 * Inputs as in fusion_merge (scores required); rho [*] float32 indexed like r.
 * Outputs: x_out, sizes_out, scores_out (may be NULL), offsets_out
 * [max_batch + 1], keep_idx (may be NULL), as in fusion_merge.
 */
int fusion_prune(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                 const float *scores, const float *rho, void *x_out, float *sizes_out,
                 float *scores_out, int32_t *offsets_out, int32_t *keep_idx, void *workspace,
                 size_t workspace_bytes, int32_t *dev_status, void *stream);

/*
 * fusion_compact: stream compaction of the samples that continue (Algorithm 1:
 * a sample that exits returns, so it leaves the batch).  Samples with
 * exit_mask[i] == 0 are copied, in ascending order, into a packed ragged batch.
 * Outputs: x_out, sizes_out, scores_out (NULL iff scores is NULL), offsets_out
 * [max_batch + 1] (the first B'+1 entries are written), ids_out [max_batch]
 * (original id of every surviving sample), batch_out (device scalar, B'),
 * keep_idx [rows] (may be NULL).
 */
int fusion_compact(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                   const float *scores, const uint8_t *exit_mask, void *x_out, float *sizes_out,
                   float *scores_out, int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out,
                   int32_t *keep_idx, void *workspace, size_t workspace_bytes,
                   int32_t *dev_status, void *stream);

/*
 * fusion_merge_router: the per-sample merge counts from the merge router with
 * profile scaling (Sec. III-C, Eq. 4 and Eq. 5), the input r of fusion_merge and
 * fusion_stage:
 *   m_i  = sigmoid(w . z_i + beta), z_i the CLS row of sample i          (Eq. 4)
 *   mt_i = m_i (1 - tau_tgt) / (1 - tau_ref), clamped to [0, 1]          (Eq. 5)
 *   r_i  = floor(mt_i N_i / 2), N_i the sample's token count, CLS included
 * (the merge then clamps r_i to |A|).  tau_tgt is the target keep ratio of the
 * operating profile, tau_ref that of the reference profile the router was
 * trained at.  Evaluated in double, so r_i differs from an exact evaluation only
 * when mt_i N_i / 2 lies within about 1e-15 of an integer.
 * w: [dim] device, the tokens' dtype.  Outputs by original id (in.ids, or the
 * position): r_out [max_batch] int32, m_out [max_batch] float (mt_i; may be
 * NULL).  Samples beyond the device batch count are not written.
 * Errors: FUSION_ERR_INVALID_ARG for NULL pointers or tau_ref >= 1 or a
 * non-finite beta / tau; device bits BAD_BATCH, BAD_OFFSETS, BAD_IDS, NONFINITE
 * (that sample's r is 0).  No workspace.
 */
int fusion_merge_router(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *w,
                        float beta, float tau_tgt, float tau_ref, int32_t *r_out, float *m_out,
                        int32_t *dev_status, void *stream);

/*
 * fusion_attention: the attention of the transformer block that consumes a compacted
 * batch (Algorithm 1, Block_b), with the size-aware (proportional) attention of ToMe, so
 * that a merged token of size s weighs like the s tokens it replaced.  For every sample
 * (rows offsets[i] .. offsets[i+1]-1), head h and query row m of the sample:
 *   out[m, h, :] = sum_j p_j v_j,  p = softmax_j(q_m . k_j / sqrt(64) + log s_j)
 * over the sample's rows j (plain attention when sizes is NULL).  tcgen05 tensor cores:
 * q k^T and p v in bf16 with float32 accumulation, p rounded to bf16 for the second
 * product, the row sum taken in float32 before that rounding.
 * dtype: FUSION_BF16 only.  qkv: [max_rows, 3, heads, 64] bf16 row-major (timm's packed
 * projection output: q, then k, then v, each heads x 64), 16-byte aligned; sizes:
 * [max_rows] float32 token sizes (> 0, within a factor 2^100 of each other inside a sample:
 * the softmax is shifted by max_j q.k / sqrt(64) + max_j log s_j, which exceeds the row's
 * largest logit by at most log(max s / min s)) or NULL; out: [max_rows, heads, 64] bf16,
 * 16-byte aligned; rows outside the samples are not written.
 * Calls with in.max_tokens <= 256 hold each sample in shared memory; longer ones (up to
 * FUSION_ATTN_MAX_TOKENS) stream blocks of 128 keys, two passes per query tile.
 * Errors: FUSION_ERR_DTYPE unless bf16; FUSION_ERR_SHAPE for head_dim != 64, heads < 1 or
 * in.max_tokens > FUSION_ATTN_MAX_TOKENS; FUSION_ERR_INVALID_ARG for NULL or misaligned
 * pointers; device bits BAD_BATCH, BAD_OFFSETS (that sample is not written), TIMEOUT.
 * No workspace.
 */
int fusion_attention(int dtype, fusion_ragged in, const void *qkv, int32_t heads, int32_t head_dim,
                     const float *sizes, void *out, int32_t *dev_status, void *stream);

/*
 * fusion_token_scores: the prune scores from a pruning router with a linear
 * scoring head (Sec. III-E, Eq. 8, s_i = h_b(z_i) with h_b(z) = w . z + b),
 * the input `scores` of fusion_prune and fusion_stage:
 *   scores_out[t] = w . x[t] + b   for every row t in [offsets[0], offsets[B])
 * B the device batch count.  Accumulated in float32 (products of two bf16 values
 * are exact) along a summation tree of depth at most 24, so
 * |error| <= 2^-18 * (sum_j |w_j x[t]_j| + |b|).
 * x: [rows, dim] device, 16-byte aligned; w: [dim] device, the tokens' dtype,
 * 16-byte aligned; b: the head's bias.  scores_out: [max_rows] float32; rows
 * outside [offsets[0], offsets[B]) are not written.  in.ids is ignored (a row's
 * score depends only on the row).
 * Errors: FUSION_ERR_INVALID_ARG for NULL or misaligned pointers or a
 * non-finite b; device bits: BAD_BATCH (nothing written), BAD_OFFSETS (when
 * offsets[0] < 0, offsets[B] < offsets[0] or offsets[B] > max_rows nothing is
 * written; per-sample defects - a decreasing pair, an empty or longer than
 * max_tokens sample - are flagged while every row of the range is still
 * scored), NONFINITE (a non-finite score, written as computed).  No workspace.
 */
int fusion_token_scores(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *w,
                        float b, float *scores_out, int32_t *dev_status, void *stream);

/*
 * fusion_stage: one block's whole adaptation stage, fused (Algorithm 1 body):
 * merge (FUSION_STAGE_MERGE) -> exit check (FUSION_STAGE_EXIT; exited samples
 * leave the batch) -> prune (FUSION_STAGE_PRUNE) -> compacted output.  The
 * result equals fusion_merge, fusion_exit_check, fusion_compact and
 * fusion_prune called in that order.  The exit check reads the input CLS rows:
 * merging never changes CLS, so they equal the merged ones bit for bit.
 *
 * flags: any OR of the FUSION_STAGE_* bits.  head is read only with
 * FUSION_STAGE_EXIT; r only with MERGE; rho only with PRUNE.
 * Outputs: exit_mask, logits, max_prob as in fusion_exit_check (written only
 * with EXIT; logits and max_prob may be NULL); x_out, sizes_out, scores_out,
 * offsets_out, ids_out, batch_out and keep_idx (input row of every output row)
 * as in fusion_compact; a_match [in.max_rows] as in fusion_merge (may be NULL).
 * ids_out and batch_out are written with every flag combination, so the
 * outputs always describe the next block's input batch.
 * With EXIT and the linear head, the per-sample kernel is launched as a
 * programmatic dependent of the exit kernel (its CTAs may become resident while
 * the exit check finishes and read the exit mask only once it has completed);
 * the call's work still runs in stream order with respect to other work on the
 * stream.
 */
int fusion_stage(int dtype, int flags, fusion_ragged in, const void *x, int32_t dim,
                 const void *keys, int32_t key_dim, const float *sizes, const float *scores,
                 const int32_t *r, const float *rho, fusion_exit_head head, uint8_t *exit_mask,
                 float *logits, float *max_prob, void *x_out, float *sizes_out, float *scores_out,
                 int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out, int32_t *keep_idx,
                 int32_t *a_match, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                 void *stream);

/*
 * Bytes of scratch of fusion_stage_mlp with both FUSION_STAGE_MERGE and FUSION_STAGE_EXIT:
 * the MLP head's scratch (fusion_exit_mlp_workspace_size) and room for the merged batch
 * (max_rows token rows of dim elements at 4 bytes each, their sizes, scores and input rows,
 * and max_batch + 1 offsets).  Zero-filled before its first use, left zero-filled by every call.
 */
size_t fusion_stage_mlp_workspace_size(int32_t max_batch, int64_t max_rows, int32_t dim, int32_t hidden,
                                       int32_t classes);

/*
 * fusion_stage_mlp: fusion_stage with one of the paper's MLP exit heads (Sec. III-G: a
 * SpatialPool head at block 8, a CLS-only head at block 10) in place of the linear head.
 * The exit check reads the merged tokens (Sec. III-B): with FUSION_STAGE_MERGE the call merges
 * into its workspace, runs fusion_exit_check_mlp on that batch (pooling the merged rows as
 * stored, rounded to the dtype), then compacts and prunes from it; keep_idx and a_match still
 * refer to the input rows.  Arguments as fusion_stage; head as fusion_exit_check_mlp (read
 * only with FUSION_STAGE_EXIT); workspace: at least fusion_stage_mlp_workspace_size(
 * in.max_batch, in.max_rows, dim, head.hidden, head.classes) bytes with both merging and the
 * exit check, fusion_exit_mlp_workspace_size(in.max_batch, dim, head.hidden, head.classes)
 * with the exit check alone, else fusion_workspace_size(in.max_batch, 1); zero-filled before
 * first use and left so.
 * Errors: those of fusion_stage and fusion_exit_check_mlp.
 */
int fusion_stage_mlp(int dtype, int flags, fusion_ragged in, const void *x, int32_t dim,
                     const void *keys, int32_t key_dim, const float *sizes, const float *scores,
                     const int32_t *r, const float *rho, fusion_mlp_head head, uint8_t *exit_mask,
                     float *logits, float *max_prob, void *x_out, float *sizes_out, float *scores_out,
                     int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out, int32_t *keep_idx,
                     int32_t *a_match, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                     void *stream);

#ifdef __cplusplus
}
#endif

#endif /* FUSION_H */
