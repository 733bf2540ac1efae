// Merge router with profile scaling (Sec. III-C, Eq. 4 and Eq. 5), the source of the
// per-sample merge counts: m = sigmoid(w . z_CLS + beta), mt = m (1 - tau_tgt) /
// (1 - tau_ref) clamped to [0, 1], r = floor(mt N / 2) with N the sample's token count.
//
// One warp per sample.  The dot product, the exponential and the floor run in double:
// the integer r is decided from a real number, and a few dozen double operations per
// sample decide it in the precision of a double evaluation of the definition (only a
// value within about 1e-15 of an integer can round differently).
#include "launch.h"

namespace fz {
namespace {

constexpr int kRouterWarps = 8;

__device__ __forceinline__ double elem_d(const float *p, long long i) { return (double)p[i]; }
__device__ __forceinline__ double elem_d(const __nv_bfloat16 *p, long long i) {
    return (double)__bfloat162float(p[i]);
}

template <typename T>
__global__ void __launch_bounds__(kRouterWarps * 32) k_router(RouterParams p) {
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * kRouterWarps + (int)(threadIdx.x >> 5);
    const int B = device_batch(p.in);
    if (B < 0) {
        if (i == 0 && lane == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    if (i >= B) return;
    const int o0 = p.in.offsets[i], o1 = p.in.offsets[i + 1];
    const int id = p.in.ids ? p.in.ids[i] : i;
    const int N = o1 - o0;
    if (o0 < 0 || N < 1 || N > p.in.max_tokens || (long long)o1 > p.in.max_rows) {
        if (lane == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        return;
    }
    if (id < 0 || id >= p.in.max_batch) {
        if (lane == 0) raise_status(p.status, FUSION_DEV_BAD_IDS);
        return;
    }
    const T *z = reinterpret_cast<const T *>(p.x) + (long long)o0 * p.dim;   // the CLS row
    const T *w = reinterpret_cast<const T *>(p.w);
    double dot = 0.0;
    for (int j = lane; j < p.dim; j += 32) dot = fma(elem_d(w, j), elem_d(z, j), dot);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
    if (lane != 0) return;
    int r = 0;
    float mt_out = 0.0f;
    if (!isfinite(dot)) {
        raise_status(p.status, FUSION_DEV_NONFINITE);
    } else {
        const double m = 1.0 / (1.0 + exp(-(dot + (double)p.beta)));                 // Eq. 4
        const double scale = (1.0 - (double)p.tau_tgt) / (1.0 - (double)p.tau_ref);   // Eq. 5
        double mt = m * scale;
        mt = mt < 0.0 ? 0.0 : (mt > 1.0 ? 1.0 : mt);
        r = (int)floor(mt * (0.5 * (double)N));
        mt_out = (float)mt;
    }
    p.r_out[id] = r;
    if (p.m_out) p.m_out[id] = mt_out;
}

}  // namespace

cudaError_t launch_router(int dtype, const RouterParams &p, cudaStream_t s) {
    if (p.in.max_batch == 0) return cudaSuccess;
    const dim3 grid((unsigned)((p.in.max_batch + kRouterWarps - 1) / kRouterWarps));
    if (dtype == FUSION_BF16)
        k_router<__nv_bfloat16><<<grid, kRouterWarps * 32, 0, s>>>(p);
    else
        k_router<float><<<grid, kRouterWarps * 32, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace fz
