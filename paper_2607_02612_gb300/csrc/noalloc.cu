// fusion_exit_check_noalloc: the exit check with its scratch space built into the
// library, for callers that have no way to allocate device memory.
//
// Some callers cannot call cudaMalloc: a plugin host that hands the library only
// its input and output buffers, a C program without a device allocator of its
// own, or a latency-critical loop where an allocation would stall or is not
// allowed.  This entry point needs nothing from them beyond inputs and outputs:
// the scratch the exit kernel uses (partial softmax sums, completion counters, the
// per-sample plan) lives in one file-scope device array.
//
// Limits and sharing: the array holds kNoAllocScratchBytes bytes on every GPU that
// loads the library, for the life of the process.  The first call on a device may load
// the library's device code there (lazy module loading), so make it before any stream
// capture.  A call whose batch bound and
// class count need more returns FUSION_ERR_WORKSPACE and enqueues nothing.  All
// calls on a device share the same array and it keeps the previous call's
// contents, so each call first clears the counters that must start at zero;
// calls that overlap on the GPU (different streams, no ordering between them)
// race on the array and must not be issued.
#include "launch.h"

namespace {

constexpr size_t kNoAllocScratchBytes = 1u << 20;   // 1 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array in the current device's context.  The host-side
// symbol is only a stand-in, not a device address.  The address is looked up on every
// call (a host-side query), so a context that was torn down and created again (after
// cudaDeviceReset, for instance) never receives a stale address.
int scratch_on_current_device(unsigned char **out) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return FUSION_ERR_CUDA;
    *out = static_cast<unsigned char *>(p);
    return FUSION_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int fusion_exit_check_noalloc(int dtype, fusion_ragged in, const void *x, int32_t dim,
                                         fusion_exit_head head, uint8_t *exit_mask, float *logits,
                                         float *max_prob, int32_t *dev_status, void *stream) {
    using namespace fz;
    if (dtype != FUSION_F32 && dtype != FUSION_BF16) return FUSION_ERR_DTYPE;
    if (!in.offsets || !x || !exit_mask || !aligned16(x)) return FUSION_ERR_INVALID_ARG;
    if (in.max_batch < 0 || in.max_tokens < 1 || in.max_tokens > FUSION_MAX_TOKENS) return FUSION_ERR_SHAPE;
    if (in.max_rows < 0 || in.max_rows > INT32_MAX) return FUSION_ERR_SHAPE;
    if (dim < 16 || dim > FUSION_MAX_DIM || dim % 16 != 0) return FUSION_ERR_SHAPE;
    if (!head.ln_gamma || !head.ln_beta || !head.weight || !head.bias) return FUSION_ERR_INVALID_ARG;
    if (!aligned16(head.ln_gamma) || !aligned16(head.ln_beta) || !aligned16(head.weight))
        return FUSION_ERR_INVALID_ARG;
    if (head.classes < 1) return FUSION_ERR_SHAPE;
    const WsLayout L = ws_layout(in.max_batch, head.classes);
    if (L.total > kNoAllocScratchBytes) return FUSION_ERR_WORKSPACE;

    unsigned char *base = nullptr;
    const int rc = scratch_on_current_device(&base);
    if (rc != FUSION_OK) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    ExitParams e{};
    e.in = Ragged{in.max_batch, in.max_tokens, (long long)in.max_rows, in.offsets, in.batch, in.ids};
    e.x = x;
    e.dim = dim;
    e.head = Head{head.ln_gamma, head.ln_beta, head.ln_eps, head.weight, head.bias, head.classes, head.tau};
    e.exit_mask = exit_mask;
    e.logits = logits;
    e.max_prob = max_prob;
    e.counters = reinterpret_cast<int *>(base + L.counters);
    e.partials = reinterpret_cast<float2 *>(base + L.partials);
    e.lg_tmp = (logits && L.total > L.lg) ? reinterpret_cast<float *>(base + L.lg) : nullptr;
    e.n_ctile = ceil_div(head.classes, kExitCT);
    e.n_btile = ceil_div(in.max_batch > 0 ? in.max_batch : 1, kExitBT);
    e.do_plan = 0;
    e.status = dev_status;
    // the completion counters must start at zero; everything else is written before it is read
    if (cudaMemsetAsync(e.counters, 0, sizeof(int) * (size_t)(e.n_btile + 1), s) != cudaSuccess)
        return FUSION_ERR_CUDA;
    return launch_exit(dtype, e, s) == cudaSuccess ? FUSION_OK : FUSION_ERR_CUDA;
}
