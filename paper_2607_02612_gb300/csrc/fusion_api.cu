// C ABI of the Fusion library: argument checks, workspace carving and kernel
// launches.  Every call validates on the host first and enqueues nothing when a
// check fails.
#include <stdint.h>

#include <cmath>

#include "launch.h"

namespace fz {
// The general exit kernel as a programmatic dependent launch (exit.cu), for the MLP head's layers.
cudaError_t launch_exit_pdl(int dtype, const ExitParams &p, cudaStream_t s);
}  // namespace fz

using namespace fz;

namespace {

constexpr const char *kVersion = "fusion-gb300 0.1.0 (sm_103a)";

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_dtype(int dtype) {
    return (dtype == FUSION_F32 || dtype == FUSION_BF16) ? FUSION_OK : FUSION_ERR_DTYPE;
}

int check_dim(int32_t d) {
    return (d >= 16 && d <= FUSION_MAX_DIM && d % 16 == 0) ? FUSION_OK : FUSION_ERR_SHAPE;
}

int check_ragged(const fusion_ragged &in) {
    if (!in.offsets) return FUSION_ERR_INVALID_ARG;
    if (in.max_batch < 0 || in.max_tokens < 1 || in.max_tokens > FUSION_MAX_TOKENS) return FUSION_ERR_SHAPE;
    if (in.max_rows < 0 || in.max_rows > INT32_MAX) return FUSION_ERR_SHAPE;
    return FUSION_OK;
}

int check_workspace(const void *ws, size_t bytes, int32_t max_batch, int32_t classes) {
    if (!ws || !aligned16(ws)) return FUSION_ERR_WORKSPACE;
    return bytes >= ws_layout(max_batch, classes).total ? FUSION_OK : FUSION_ERR_WORKSPACE;
}

int check_head(const fusion_exit_head &h) {
    if (!h.ln_gamma || !h.ln_beta || !h.weight || !h.bias) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(h.ln_gamma) || !aligned16(h.ln_beta) || !aligned16(h.weight)) return FUSION_ERR_INVALID_ARG;
    if (h.classes < 1) return FUSION_ERR_SHAPE;
    return FUSION_OK;
}

Ragged dev(const fusion_ragged &in) {
    return Ragged{in.max_batch, in.max_tokens, (long long)in.max_rows, in.offsets, in.batch, in.ids};
}

Head dev(const fusion_exit_head &h) {
    return Head{h.ln_gamma, h.ln_beta, h.ln_eps, h.weight, h.bias, h.classes, h.tau};
}

struct Ws {
    int *slot;
    int *plan;
    int *counters;
    float2 *partials;
    float *lg;   // logits tiles of the general exit kernel (NULL for heads it does not run)
};

Ws carve(void *ws, int32_t max_batch, int32_t classes) {
    const WsLayout L = ws_layout(max_batch, classes);
    unsigned char *b = static_cast<unsigned char *>(ws);
    return Ws{reinterpret_cast<int *>(b + L.slot), reinterpret_cast<int *>(b + L.plan),
              reinterpret_cast<int *>(b + L.counters), reinterpret_cast<float2 *>(b + L.partials),
              L.total > L.lg ? reinterpret_cast<float *>(b + L.lg) : nullptr};
}

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? FUSION_OK : FUSION_ERR_CUDA; }

// Events armed by fusion_profile_next() for the next call of this host thread.
struct ProfileEvents {
    cudaEvent_t start = nullptr, mid = nullptr, end = nullptr;
};
thread_local ProfileEvents g_profile;

// Launch gate armed by fusion_set_launch_gate() for this host thread's calls.
thread_local const int32_t *g_gate = nullptr;
thread_local unsigned g_gate_spins = 0;

// Takes the armed events (if any) for the call that is starting.
ProfileEvents take_profile() {
    ProfileEvents e = g_profile;
    g_profile = ProfileEvents{};
    return e;
}

// Under stream capture a plain record only orders the graph; an external record becomes a
// node that records the event at every replay.
void record(cudaEvent_t e, cudaStream_t s) {
    if (!e) return;
    cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &st) == cudaSuccess && st == cudaStreamCaptureStatusActive)
        cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
    else
        cudaEventRecord(e, s);
}

#define FZ_TRY(expr)                    \
    do {                                \
        const int rc_ = (expr);         \
        if (rc_ != FUSION_OK) return rc_; \
    } while (0)

ImageParams image_params(const fusion_ragged &in, const void *x, int32_t dim, const void *keys,
                         int32_t key_dim, const float *sizes, const float *scores, const int32_t *r,
                         const float *rho, int do_merge, int do_prune, const Ws &w,
                         const int32_t *offsets_out, void *x_out, float *sizes_out, float *scores_out,
                         int32_t *keep_idx, int32_t *dst_map, int32_t *a_match, int32_t *status,
                         const ImageGeometry &G) {
    ImageParams p{};
    p.in = dev(in);
    p.x = x;
    p.keys = keys ? keys : x;
    p.dim = dim;
    p.kdim = keys ? key_dim : dim;
    p.keys_alias = (keys == nullptr || keys == x) && p.kdim == dim;
    p.sizes = sizes;
    p.scores = scores;
    p.r = r;
    p.rho = rho;
    p.do_merge = do_merge;
    p.do_prune = do_prune;
    p.need_match = a_match != nullptr;
    p.slot = w.slot;
    p.plan = w.plan;
    p.offsets_out = offsets_out;
    p.x_out = x_out;
    p.sizes_out = sizes_out;
    p.scores_out = scores_out;
    p.keep_idx = keep_idx;
    p.gate = g_gate;
    p.gate_spins = g_gate_spins;
    p.dst_map = dst_map;
    p.a_match = a_match;
    p.status = status;
    p.resident = G.resident;
    p.kc = G.kc;
    p.ra = G.ra;
    p.rb = G.rb;
    return p;
}

// Dynamic shared memory per CTA of the tcgen05 kernel: two CTAs share an SM's 228 KB
// (1 KB of it reserved per CTA, plus the kernel's static shared memory), so that one
// CTA's decisions and gather overlap the other's loads.
constexpr int kTcSmemBudgetKb = 111;

// The plan runs inside the per-sample kernel when every CTA can afford to scan the batch.
bool fuse_plan(const fusion_ragged &in) { return in.max_batch >= 1 && in.max_batch <= kFusedPlanMaxBatch; }

// The per-sample kernel: TMA + tcgen05 when the shape allows it, else the general one.
// pdl: the TMA + tcgen05 kernel as a programmatic dependent of the kernel before it (the linear
// exit check of a fused stage, with no event between them).
cudaError_t launch_sample_kernel(int dtype, const ImageParams &p, const ImageGeometry &G, cudaStream_t s,
                                 bool pdl = false) {
    if (p.do_merge) {
        const TcGeometry T = image_tc_geometry(dtype, p.in.max_tokens, p.kdim, p.dim, p.in.max_rows, 1, kTcSmemBudgetKb);
        if (T.ok) return launch_image_tc(p, T, s, pdl);
    }
    return launch_image(dtype, p, G.smem, s);
}

}  // namespace

extern "C" {

const char *fusion_version(void) { return kVersion; }

int fusion_set_launch_gate(const int32_t *flag, int64_t polls) {
    if (flag && polls < 0) return FUSION_ERR_INVALID_ARG;
    g_gate = flag;
    g_gate_spins = flag ? (polls > (int64_t)0xFFFFFFFF ? 0xFFFFFFFFu : (unsigned)polls) : 0u;
    return FUSION_OK;
}

int fusion_profile_next(void *start, void *mid, void *end) {
    g_profile.start = static_cast<cudaEvent_t>(start);
    g_profile.mid = static_cast<cudaEvent_t>(mid);
    g_profile.end = static_cast<cudaEvent_t>(end);
    return FUSION_OK;
}

const char *fusion_status_string(int code) {
    switch (code) {
        case FUSION_OK: return "ok";
        case FUSION_ERR_INVALID_ARG: return "invalid argument (NULL, misaligned pointer or bad flags)";
        case FUSION_ERR_SHAPE: return "shape out of range (dim, key_dim, max_tokens, classes, batch)";
        case FUSION_ERR_DTYPE: return "unsupported dtype";
        case FUSION_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case FUSION_ERR_CUDA: return "CUDA error";
        case FUSION_DEV_BAD_OFFSETS: return "device: malformed offsets";
        case FUSION_DEV_BAD_BATCH: return "device: batch count out of range";
        case FUSION_DEV_NONFINITE: return "device: NaN or Inf in a decision input";
        case FUSION_DEV_INTERNAL: return "device: internal consistency check failed";
        case FUSION_DEV_BAD_IDS: return "device: sample id out of range";
        case FUSION_DEV_TIMEOUT: return "device: a bounded wait timed out";
        default: return "unknown status";
    }
}

size_t fusion_workspace_size(int32_t max_batch, int32_t classes) {
    return ws_layout(max_batch < 0 ? 0 : max_batch, classes < 1 ? 1 : classes).total;
}

int fusion_merge(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *keys,
                 int32_t key_dim, const float *sizes, const float *scores, const int32_t *r,
                 void *x_out, float *sizes_out, float *scores_out, int32_t *offsets_out,
                 int32_t *keep_idx, int32_t *dst_map, int32_t *a_match, void *workspace,
                 size_t workspace_bytes, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!keys) return FUSION_ERR_INVALID_ARG;
    FZ_TRY(check_dim(key_dim));
    if (!x || !sizes || !r || !x_out || !sizes_out || !offsets_out) return FUSION_ERR_INVALID_ARG;
    if ((scores == nullptr) != (scores_out == nullptr)) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(keys) || !aligned16(x_out)) return FUSION_ERR_INVALID_ARG;
    FZ_TRY(check_workspace(workspace, workspace_bytes, in.max_batch, 1));
    const ImageGeometry G = image_geometry(dtype, in.max_tokens, key_dim, 1);
    if (!G.ok) return FUSION_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Ws w = carve(workspace, in.max_batch, 1);
    const ProfileEvents ev = take_profile();

    PlanArgs pa{};
    pa.in = dev(in);
    pa.merge = 1;
    pa.r = r;
    pa.offsets_out = offsets_out;
    pa.slot = w.slot;
    pa.plan = w.plan;
    pa.status = dev_status;
    record(ev.start, s);
    if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pa, s)));
    record(ev.mid, s);
    ImageParams p = image_params(in, x, dim, keys, key_dim, sizes, scores, r, nullptr, 1, 0, w, offsets_out,
                                 x_out, sizes_out, scores_out, keep_idx, dst_map, a_match, dev_status, G);
    p.fused_plan = fuse_plan(in);
    p.plan_args = pa;
    const int rc = cuda_rc(launch_sample_kernel(dtype, p, G, s));
    record(ev.end, s);
    return rc;
}

int fusion_exit_check(int dtype, fusion_ragged in, const void *x, int32_t dim,
                      fusion_exit_head head, uint8_t *exit_mask, float *logits, float *max_prob,
                      void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    FZ_TRY(check_head(head));
    if (!x || !exit_mask || !aligned16(x)) return FUSION_ERR_INVALID_ARG;
    FZ_TRY(check_workspace(workspace, workspace_bytes, in.max_batch, head.classes));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Ws w = carve(workspace, in.max_batch, head.classes);
    ExitParams e{};
    e.in = dev(in);
    e.x = x;
    e.dim = dim;
    e.head = dev(head);
    e.exit_mask = exit_mask;
    e.logits = logits;
    e.max_prob = max_prob;
    e.counters = w.counters;
    e.partials = w.partials;
    e.lg_tmp = logits ? w.lg : nullptr;
    e.n_ctile = ceil_div(head.classes, kExitCT);
    e.n_btile = ceil_div(in.max_batch > 0 ? in.max_batch : 1, kExitBT);
    e.do_plan = 0;
    e.status = dev_status;
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    const int rc = cuda_rc(launch_exit(dtype, e, s));
    record(ev.mid, s);
    record(ev.end, s);
    return rc;
}

int fusion_prune(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                 const float *scores, const float *rho, void *x_out, float *sizes_out,
                 float *scores_out, int32_t *offsets_out, int32_t *keep_idx, void *workspace,
                 size_t workspace_bytes, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!x || !sizes || !scores || !rho || !x_out || !sizes_out || !offsets_out) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(x_out)) return FUSION_ERR_INVALID_ARG;
    FZ_TRY(check_workspace(workspace, workspace_bytes, in.max_batch, 1));
    const ImageGeometry G = image_geometry(dtype, in.max_tokens, dim, 0);
    if (!G.ok) return FUSION_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Ws w = carve(workspace, in.max_batch, 1);
    PlanArgs pa{};
    pa.in = dev(in);
    pa.prune = 1;
    pa.rho = rho;
    pa.offsets_out = offsets_out;
    pa.slot = w.slot;
    pa.plan = w.plan;
    pa.status = dev_status;
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pa, s)));
    record(ev.mid, s);
    ImageParams p = image_params(in, x, dim, nullptr, dim, sizes, scores, nullptr, rho, 0, 1, w, offsets_out,
                                 x_out, sizes_out, scores_out, keep_idx, nullptr, nullptr, dev_status, G);
    p.fused_plan = fuse_plan(in);
    p.plan_args = pa;
    const int rc = cuda_rc(launch_sample_kernel(dtype, p, G, s));
    record(ev.end, s);
    return rc;
}

int fusion_compact(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                   const float *scores, const uint8_t *exit_mask, void *x_out, float *sizes_out,
                   float *scores_out, int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out,
                   int32_t *keep_idx, void *workspace, size_t workspace_bytes,
                   int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!x || !sizes || !exit_mask || !x_out || !sizes_out || !offsets_out || !ids_out || !batch_out)
        return FUSION_ERR_INVALID_ARG;
    if ((scores == nullptr) != (scores_out == nullptr)) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(x_out)) return FUSION_ERR_INVALID_ARG;
    FZ_TRY(check_workspace(workspace, workspace_bytes, in.max_batch, 1));
    const ImageGeometry G = image_geometry(dtype, in.max_tokens, dim, 0);
    if (!G.ok) return FUSION_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Ws w = carve(workspace, in.max_batch, 1);
    PlanArgs pa{};
    pa.in = dev(in);
    pa.exit_mask = exit_mask;
    pa.offsets_out = offsets_out;
    pa.ids_out = ids_out;
    pa.batch_out = batch_out;
    pa.slot = w.slot;
    pa.plan = w.plan;
    pa.status = dev_status;
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pa, s)));
    record(ev.mid, s);
    ImageParams p = image_params(in, x, dim, nullptr, dim, sizes, scores, nullptr, nullptr, 0, 0, w, offsets_out,
                                 x_out, sizes_out, scores_out, keep_idx, nullptr, nullptr, dev_status, G);
    p.fused_plan = fuse_plan(in);
    p.plan_args = pa;
    const int rc = cuda_rc(launch_sample_kernel(dtype, p, G, s));
    record(ev.end, s);
    return rc;
}

int fusion_merge_router(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *w,
                        float beta, float tau_tgt, float tau_ref, int32_t *r_out, float *m_out,
                        int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!x || !w || !r_out) return FUSION_ERR_INVALID_ARG;
    if (!std::isfinite(beta) || !std::isfinite(tau_tgt) || !std::isfinite(tau_ref) || !(tau_ref < 1.0f))
        return FUSION_ERR_INVALID_ARG;
    RouterParams p{};
    p.in = dev(in);
    p.x = x;
    p.dim = dim;
    p.w = w;
    p.beta = beta;
    p.tau_tgt = tau_tgt;
    p.tau_ref = tau_ref;
    p.r_out = r_out;
    p.m_out = m_out;
    p.status = dev_status;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    record(ev.mid, s);
    const int rc = cuda_rc(launch_router(dtype, p, s));
    record(ev.end, s);
    return rc;
}

namespace {
// fusion_exit_check_mlp scratch: the linear exit workspace for `classes`, then the pooled
// rows [max_batch, dim] float32 and the hidden rows [max_batch, hidden] (float32 size).
struct MlpWs {
    size_t u, ulo, hid, lg, total;
};
// The stage's own scratch, the pooled rows (float-float: high then low parts), the hidden rows
// (at most float32) and the second layer's logits tiles (the general exit kernel writes exited
// rows from there).
MlpWs mlp_ws_layout(int32_t max_batch, int32_t dim, int32_t hidden, int32_t classes) {
    const size_t mb = (size_t)(max_batch > 0 ? max_batch : 1);
    const size_t tiles = (size_t)ceil_div(max_batch > 0 ? max_batch : 1, kExitBT) * kExitBT;
    MlpWs L;
    L.u = (ws_layout(max_batch, classes).total + 255) / 256 * 256;
    L.ulo = (L.u + mb * (size_t)dim * sizeof(float) + 255) / 256 * 256;
    L.hid = (L.ulo + mb * (size_t)dim * sizeof(float) + 255) / 256 * 256;
    L.lg = (L.hid + mb * (size_t)hidden * sizeof(float) + 255) / 256 * 256;
    L.total = (L.lg + tiles * (size_t)classes * sizeof(float) + 255) / 256 * 256;
    return L;
}
// fusion_stage_mlp with merging and the exit check: the MLP head's scratch, then the merged
// batch (tokens at 4 bytes per element whatever the dtype, sizes, scores, input row of every
// merged row, offsets) that the head reads and the compaction and pruning start from.
struct StageMlpWs {
    size_t x, sizes, scores, keep, offsets, total;
};
StageMlpWs stage_mlp_ws_layout(int32_t max_batch, int64_t max_rows, int32_t dim, int32_t hidden, int32_t classes) {
    const size_t mr = (size_t)(max_rows > 0 ? max_rows : 1);
    StageMlpWs L;
    L.x = mlp_ws_layout(max_batch, dim, hidden, classes).total;
    L.sizes = align256(L.x + mr * (size_t)dim * 4);
    L.scores = align256(L.sizes + mr * 4);
    L.keep = align256(L.scores + mr * 4);
    L.offsets = align256(L.keep + mr * 4);
    L.total = align256(L.offsets + (size_t)(max_batch > 0 ? max_batch + 1 : 1) * 4);
    return L;
}
}  // namespace

namespace {
int check_mlp_head(const fusion_mlp_head &head, const float *sizes) {
    FZ_TRY(check_dim(head.hidden));
    if (head.classes < 1) return FUSION_ERR_SHAPE;
    if (head.pool != FUSION_POOL_CLS && head.pool != FUSION_POOL_SPATIAL) return FUSION_ERR_INVALID_ARG;
    if (head.pool == FUSION_POOL_SPATIAL && !sizes) return FUSION_ERR_INVALID_ARG;
    if (!head.ln_gamma || !head.ln_beta || !head.w1 || !head.b1 || !head.w2 || !head.b2) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(head.ln_gamma) || !aligned16(head.ln_beta) || !aligned16(head.w1) || !aligned16(head.w2))
        return FUSION_ERR_INVALID_ARG;
    return FUSION_OK;
}

// The MLP exit head's three launches (pool; LayerNorm, first layer and GELU; second layer,
// softmax maximum and exit rule) on the rows of `in`, scratch from a checked workspace.
// `mid` (may be NULL) is recorded between the first layer and the second.
int launch_exit_mlp(int dtype, const fusion_ragged &in, const void *x, int32_t dim, const float *sizes,
                    const fusion_mlp_head &head, uint8_t *exit_mask, float *logits, float *max_prob, void *workspace,
                    int32_t *dev_status, cudaStream_t s, cudaEvent_t mid) {
    const MlpWs L = mlp_ws_layout(in.max_batch, dim, head.hidden, head.classes);
    unsigned char *wb = static_cast<unsigned char *>(workspace);
    float *u = reinterpret_cast<float *>(wb + L.u);
    void *hid = wb + L.hid;
    const Ws w = carve(workspace, in.max_batch, head.classes);
    const int n_btile = ceil_div(in.max_batch > 0 ? in.max_batch : 1, kExitBT);

    PoolParams pp{};
    pp.in = dev(in);
    pp.x = x;
    pp.dim = dim;
    pp.sizes = sizes;
    pp.pool = head.pool;
    pp.u_out = u;
    pp.u_lo = reinterpret_cast<float *>(wb + L.ulo);
    pp.status = dev_status;

    ExitParams l1{};   // LayerNorm, first layer and GELU
    l1.in = dev(in);
    l1.dim = dim;
    l1.head = Head{head.ln_gamma, head.ln_beta, head.ln_eps, head.w1, head.b1, head.hidden, 0.0f};
    l1.counters = w.counters;
    l1.partials = w.partials;
    l1.n_ctile = ceil_div(head.hidden, kExitCT);
    l1.n_btile = n_btile;
    l1.status = dev_status;
    l1.in_mode = 2;
    l1.u_in = u;
    l1.u_in_lo = reinterpret_cast<const float *>(wb + L.ulo);
    l1.out_mode = 1;
    l1.hidden_out = hid;

    ExitParams l2{};   // second layer, softmax maximum and exit rule
    l2.in = dev(in);
    l2.x = hid;
    l2.dim = head.hidden;
    l2.head = Head{nullptr, nullptr, 0.0f, head.w2, head.b2, head.classes, head.tau};
    l2.exit_mask = exit_mask;
    l2.logits = logits;
    l2.max_prob = max_prob;
    l2.counters = w.counters;
    l2.partials = w.partials;
    l2.lg_tmp = logits ? reinterpret_cast<float *>(wb + L.lg) : nullptr;
    l2.n_ctile = ceil_div(head.classes, kExitCT);
    l2.n_btile = n_btile;
    l2.status = dev_status;
    l2.in_mode = 1;
    l2.skip_ln = 1;

    // each layer a programmatic dependent of the kernel before it (exit.cu)
    int rc = cuda_rc(launch_head_pool(dtype, pp, s));
    if (rc == FUSION_OK) rc = cuda_rc(launch_exit_pdl(dtype, l1, s));
    record(mid, s);
    if (rc == FUSION_OK) rc = cuda_rc(launch_exit_pdl(dtype, l2, s));
    return rc;
}
}  // namespace

size_t fusion_stage_mlp_workspace_size(int32_t max_batch, int64_t max_rows, int32_t dim, int32_t hidden,
                                       int32_t classes) {
    return stage_mlp_ws_layout(max_batch < 0 ? 0 : max_batch, max_rows, dim < 16 ? 16 : dim, hidden < 16 ? 16 : hidden,
                               classes < 1 ? 1 : classes)
        .total;
}

size_t fusion_exit_mlp_workspace_size(int32_t max_batch, int32_t dim, int32_t hidden, int32_t classes) {
    if (max_batch < 0) max_batch = 0;
    return mlp_ws_layout(max_batch, dim < 16 ? 16 : dim, hidden < 16 ? 16 : hidden, classes < 1 ? 1 : classes).total;
}

int fusion_exit_check_mlp(int dtype, fusion_ragged in, const void *x, int32_t dim, const float *sizes,
                          fusion_mlp_head head, uint8_t *exit_mask, float *logits, float *max_prob,
                          void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    FZ_TRY(check_mlp_head(head, sizes));
    if (!x || !exit_mask || !aligned16(x)) return FUSION_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace)) return FUSION_ERR_WORKSPACE;
    if (workspace_bytes < mlp_ws_layout(in.max_batch, dim, head.hidden, head.classes).total) return FUSION_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    const int rc = launch_exit_mlp(dtype, in, x, dim, sizes, head, exit_mask, logits, max_prob, workspace, dev_status,
                                   s, ev.mid);
    record(ev.end, s);
    return rc;
}

int fusion_attention(int dtype, fusion_ragged in, const void *qkv, int32_t heads, int32_t head_dim,
                     const float *sizes, void *out, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    if (dtype != FUSION_BF16) return FUSION_ERR_DTYPE;
    FZ_TRY(check_ragged(in));
    if (head_dim != FUSION_ATTN_HEAD_DIM || heads < 1 || heads > 64 || in.max_tokens > FUSION_ATTN_MAX_TOKENS)
        return FUSION_ERR_SHAPE;
    if (!qkv || !out || !aligned16(qkv) || !aligned16(out)) return FUSION_ERR_INVALID_ARG;
    AttnParams p{};
    p.in = dev(in);
    p.qkv = qkv;
    p.heads = heads;
    p.sizes = sizes;
    p.out = out;
    p.status = dev_status;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    record(ev.mid, s);
    const int rc = cuda_rc(launch_attention(p, s));
    record(ev.end, s);
    return rc;
}

int fusion_token_scores(int dtype, fusion_ragged in, const void *x, int32_t dim, const void *w, float b,
                        float *scores_out, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!x || !w || !scores_out || !aligned16(x) || !aligned16(w)) return FUSION_ERR_INVALID_ARG;
    if (!std::isfinite(b)) return FUSION_ERR_INVALID_ARG;
    ScoreParams p{};
    p.in = dev(in);
    p.x = x;
    p.dim = dim;
    p.w = w;
    p.b = b;
    p.scores_out = scores_out;
    p.status = dev_status;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    record(ev.mid, s);
    const int rc = cuda_rc(launch_token_scores(dtype, p, s));
    record(ev.end, s);
    return rc;
}

}  // extern "C"

namespace {
// The fused stage with either exit head: `lin` (the linear head, one exit kernel that may run
// the plan) or `mlp` (the MLP head's three launches on the stage's input rows, then the plan
// kernel when the per-sample kernel does not fuse it).
int stage_impl(int dtype, int flags, const fusion_ragged &in, const void *x, int32_t dim, const void *keys,
               int32_t key_dim, const float *sizes, const float *scores, const int32_t *r, const float *rho,
               const fusion_exit_head *lin, const fusion_mlp_head *mlp, uint8_t *exit_mask, float *logits,
               float *max_prob, void *x_out, float *sizes_out, float *scores_out, int32_t *offsets_out,
               int32_t *ids_out, int32_t *batch_out, int32_t *keep_idx, int32_t *a_match, void *workspace,
               size_t workspace_bytes, int32_t *dev_status, void *stream) {
    FZ_TRY(check_dtype(dtype));
    if (flags < 0 || flags > (FUSION_STAGE_MERGE | FUSION_STAGE_EXIT | FUSION_STAGE_PRUNE))
        return FUSION_ERR_INVALID_ARG;
    const int do_merge = (flags & FUSION_STAGE_MERGE) != 0;
    const int do_exit = (flags & FUSION_STAGE_EXIT) != 0;
    const int do_prune = (flags & FUSION_STAGE_PRUNE) != 0;
    FZ_TRY(check_ragged(in));
    FZ_TRY(check_dim(dim));
    if (!x || !sizes || !x_out || !sizes_out || !offsets_out || !ids_out || !batch_out)
        return FUSION_ERR_INVALID_ARG;
    if ((scores == nullptr) != (scores_out == nullptr)) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(x_out)) return FUSION_ERR_INVALID_ARG;
    if (do_merge) {
        if (!keys || !r || !aligned16(keys)) return FUSION_ERR_INVALID_ARG;
        FZ_TRY(check_dim(key_dim));
    }
    if (do_prune && (!rho || !scores)) return FUSION_ERR_INVALID_ARG;
    if (!do_merge && a_match) return FUSION_ERR_INVALID_ARG;
    const int classes = do_exit ? (mlp ? mlp->classes : lin->classes) : 1;
    if (do_exit) {
        FZ_TRY(mlp ? check_mlp_head(*mlp, sizes) : check_head(*lin));
        if (!exit_mask) return FUSION_ERR_INVALID_ARG;
    }
    if (do_exit && mlp) {   // the MLP head's scratch, whose first part is the stage's own
        if (!workspace || !aligned16(workspace)) return FUSION_ERR_WORKSPACE;
        const size_t need = do_merge ? stage_mlp_ws_layout(in.max_batch, in.max_rows, dim, mlp->hidden, mlp->classes).total
                                     : mlp_ws_layout(in.max_batch, dim, mlp->hidden, mlp->classes).total;
        if (workspace_bytes < need) return FUSION_ERR_WORKSPACE;
    } else {
        FZ_TRY(check_workspace(workspace, workspace_bytes, in.max_batch, classes));
    }
    const ImageGeometry G = image_geometry(dtype, in.max_tokens, do_merge ? key_dim : dim, do_merge);
    if (!G.ok) return FUSION_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Ws w = carve(workspace, in.max_batch, classes);

    const ProfileEvents ev = take_profile();
    record(ev.start, s);
    PlanArgs pa{};
    pa.in = dev(in);
    pa.merge = do_merge;
    pa.prune = do_prune;
    pa.r = r;
    pa.rho = rho;
    pa.exit_mask = do_exit ? exit_mask : nullptr;
    pa.offsets_out = offsets_out;
    pa.ids_out = ids_out;
    pa.batch_out = batch_out;
    pa.slot = w.slot;
    pa.plan = w.plan;
    pa.status = dev_status;
    if (do_exit && mlp && do_merge) {
        // The MLP head reads the merged tokens (Sec. III-B): merge into the workspace, the exit
        // check on that batch, then compaction and pruning from it (keep_idx mapped back to the
        // input rows through the merge's row ids).
        const StageMlpWs M = stage_mlp_ws_layout(in.max_batch, in.max_rows, dim, mlp->hidden, mlp->classes);
        unsigned char *wb = static_cast<unsigned char *>(workspace);
        void *x_m = wb + M.x;
        float *sizes_m = reinterpret_cast<float *>(wb + M.sizes);
        float *scores_m = scores ? reinterpret_cast<float *>(wb + M.scores) : nullptr;
        int32_t *keep_m = reinterpret_cast<int32_t *>(wb + M.keep);
        int32_t *offs_m = reinterpret_cast<int32_t *>(wb + M.offsets);
        PlanArgs pm = pa;
        pm.prune = 0;
        pm.exit_mask = nullptr;
        pm.offsets_out = offs_m;
        pm.ids_out = nullptr;
        pm.batch_out = nullptr;
        if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pm, s)));
        ImageParams q = image_params(in, x, dim, keys, key_dim, sizes, scores, r, nullptr, 1, 0, w, offs_m, x_m, sizes_m,
                                     scores_m, keep_m, nullptr, a_match, dev_status, G);
        q.fused_plan = fuse_plan(in);
        q.plan_args = pm;
        FZ_TRY(cuda_rc(launch_sample_kernel(dtype, q, G, s)));
        fusion_ragged in_m = in;
        in_m.offsets = offs_m;
        FZ_TRY(launch_exit_mlp(dtype, in_m, x_m, dim, sizes_m, *mlp, exit_mask, logits, max_prob, workspace, dev_status,
                               s, nullptr));
        record(ev.mid, s);
        PlanArgs pc = pa;
        pc.in = dev(in_m);
        pc.merge = 0;
        if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pc, s)));
        const ImageGeometry G2 = image_geometry(dtype, in.max_tokens, dim, 0);
        if (!G2.ok) return FUSION_ERR_SHAPE;
        ImageParams c = image_params(in_m, x_m, dim, nullptr, dim, sizes_m, scores_m, nullptr, rho, 0, do_prune, w,
                                     offsets_out, x_out, sizes_out, scores_out, keep_idx, nullptr, nullptr, dev_status, G2);
        c.keep_map = keep_m;
        c.fused_plan = fuse_plan(in);
        c.plan_args = pc;
        const int rc = cuda_rc(launch_sample_kernel(dtype, c, G2, s));
        record(ev.end, s);
        return rc;
    }
    if (do_exit && mlp) {
        FZ_TRY(launch_exit_mlp(dtype, in, x, dim, sizes, *mlp, exit_mask, logits, max_prob, workspace, dev_status, s,
                               nullptr));
        if (!fuse_plan(in)) FZ_TRY(cuda_rc(launch_plan(pa, s)));
    } else if (do_exit) {
        const fusion_exit_head &head = *lin;
        ExitParams e{};
        e.in = dev(in);
        e.x = x;
        e.dim = dim;
        e.head = dev(head);
        e.exit_mask = exit_mask;
        e.logits = logits;
        e.max_prob = max_prob;
        e.counters = w.counters;
        e.partials = w.partials;
        e.lg_tmp = logits ? w.lg : nullptr;
        e.n_ctile = ceil_div(head.classes, kExitCT);
        e.n_btile = ceil_div(in.max_batch > 0 ? in.max_batch : 1, kExitBT);
        e.do_plan = !fuse_plan(in);
        e.plan = pa;
        e.status = dev_status;
        FZ_TRY(cuda_rc(launch_exit(dtype, e, s)));
    } else if (!fuse_plan(in)) {
        FZ_TRY(cuda_rc(launch_plan(pa, s)));
    }
    record(ev.mid, s);
    ImageParams p = image_params(in, x, dim, do_merge ? keys : nullptr, key_dim, sizes, scores, r, rho, do_merge,
                                 do_prune, w, offsets_out, x_out, sizes_out, scores_out, keep_idx, nullptr, a_match,
                                 dev_status, G);
    p.fused_plan = fuse_plan(in);
    p.plan_args = pa;
    const bool pdl = do_exit && !mlp && ev.mid == nullptr;   // right after the cluster or general exit kernel
    const int rc = cuda_rc(launch_sample_kernel(dtype, p, G, s, pdl));
    record(ev.end, s);
    return rc;
}
}  // namespace

extern "C" {

int fusion_stage(int dtype, int flags, fusion_ragged in, const void *x, int32_t dim,
                 const void *keys, int32_t key_dim, const float *sizes, const float *scores,
                 const int32_t *r, const float *rho, fusion_exit_head head, uint8_t *exit_mask,
                 float *logits, float *max_prob, void *x_out, float *sizes_out, float *scores_out,
                 int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out, int32_t *keep_idx,
                 int32_t *a_match, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                 void *stream) {
    return stage_impl(dtype, flags, in, x, dim, keys, key_dim, sizes, scores, r, rho, &head, nullptr, exit_mask, logits,
                      max_prob, x_out, sizes_out, scores_out, offsets_out, ids_out, batch_out, keep_idx, a_match,
                      workspace, workspace_bytes, dev_status, stream);
}

int fusion_stage_mlp(int dtype, int flags, fusion_ragged in, const void *x, int32_t dim,
                     const void *keys, int32_t key_dim, const float *sizes, const float *scores,
                     const int32_t *r, const float *rho, fusion_mlp_head head, uint8_t *exit_mask,
                     float *logits, float *max_prob, void *x_out, float *sizes_out, float *scores_out,
                     int32_t *offsets_out, int32_t *ids_out, int32_t *batch_out, int32_t *keep_idx,
                     int32_t *a_match, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                     void *stream) {
    return stage_impl(dtype, flags, in, x, dim, keys, key_dim, sizes, scores, r, rho, nullptr, &head, exit_mask, logits,
                      max_prob, x_out, sizes_out, scores_out, offsets_out, ids_out, batch_out, keep_idx, a_match,
                      workspace, workspace_bytes, dev_status, stream);
}

}  // extern "C"
