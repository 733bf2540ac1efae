// Pruning router with a linear scoring head (Sec. III-E, Eq. 8): s_t = w . z_t + b for
// every token row t of a ragged batch, the scores the prune ranks.
//
// A pure stream over the tokens (dim * elem bytes read and 4 bytes written per row).  A
// consumer warp splits into 32 / g lane groups of g lanes, one row per group; lane j of a
// group owns the 16-byte chunks j, j + g, ... of its row.  g is 8, 16 or 32 where that
// splits the C chunks of a row evenly into at most 8 per lane (a group then covers whole
// 128-byte lines), else gcd(C, 32), else 32 with the tail masked.  A warp's task is U
// consecutive groups of rows; tasks go round the warps of a grid of two CTAs per SM.
//
// Each lane streams its own chunks through a private ring of S task-sized stages in shared
// memory with cp.async (16 bytes, L2 only), S - 1 tasks ahead of the one it computes, and
// reads back only what it copied itself, so no barrier or cross-lane wait is needed: 24
// chunks (384 bytes) per lane, 192 KB in flight per SM, none of it in registers.  The
// weights stay in registers for the whole kernel.  Each lane accumulates its elements into
// four partial sums with fma, the group adds its lanes in a butterfly, and the bias comes
// last.
#include "launch.h"

namespace fz {
namespace {

constexpr int kScoreThreads = 256;
constexpr int kScoreMaxK = 8;
constexpr int kScoreLaneChunks = 24;   // ring chunks of 16 bytes per lane

__device__ __forceinline__ void unpack(const uint4 &v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
}
__device__ __forceinline__ void unpack(const uint4 &v, float (&f)[8]) {
    const unsigned u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {   // a bf16 is the high half of the float with the same value
        f[2 * i] = __uint_as_float(u[i] << 16);
        f[2 * i + 1] = __uint_as_float(u[i] & 0xFFFF0000u);
    }
}

// 16-byte asynchronous copy global -> shared; src_bytes = 0 reads nothing and writes zeros.
__device__ __forceinline__ void cp_async_zfill(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Ring geometry for K chunks per lane and row: U groups per task (at least 64 bytes per
// lane), S stages within the lane's chunk budget.
template <int K>
struct ScoreRing {
    static constexpr int U = K >= 4 ? 1 : (4 + K - 1) / K;
    static constexpr int S_fit = kScoreLaneChunks / (U * K);
    static constexpr int S = S_fit > 8 ? 8 : (S_fit < 2 ? 2 : S_fit);
    static constexpr size_t smem = (size_t)S * U * K * kScoreThreads * 16;
};

template <typename T, int K>
__global__ void __launch_bounds__(kScoreThreads, 2) k_token_scores(ScoreParams p) {
    constexpr int E = Elem<T>::kPerChunk;
    constexpr int U = ScoreRing<K>::U, S = ScoreRing<K>::S;
    extern __shared__ __align__(16) uint4 ring[];   // [S][U][K][kScoreThreads]: lane-consecutive chunks
    const int tid = threadIdx.x, lane = tid & 31;
    const int g = p.group;   // lanes per row, a power of two
    const int R = 32 / g;    // rows per group
    const int j = lane & (g - 1);
    const int rsub = lane / g;
    const int C = p.dim / E;

    uint4 wraw[K];   // the weights do not depend on the offsets: request them first
    const uint4 *w4 = reinterpret_cast<const uint4 *>(p.w);
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const int c = j + g * k;
        wraw[k] = c < C ? __ldg(w4 + c) : make_uint4(0u, 0u, 0u, 0u);
    }

    const int B = device_batch(p.in);
    if (B < 0) {
        if (blockIdx.x == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    const int o0 = p.in.offsets[0], o1 = p.in.offsets[B];
    if (o0 < 0 || o1 < o0 || (long long)o1 > p.in.max_rows) {
        if (blockIdx.x == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        return;
    }
    if (blockIdx.x == 0) {   // per-sample defects do not change which rows are scored
        for (int i = tid; i < B; i += kScoreThreads) {
            const int n = p.in.offsets[i + 1] - p.in.offsets[i];
            if (n < 1 || n > p.in.max_tokens) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        }
    }

    const uint4 *x4 = reinterpret_cast<const uint4 *>(p.x);
    const long long groups = ((long long)(o1 - o0) + R - 1) / R;
    const long long tasks = (groups + U - 1) / U;
    const long long W = ((long long)blockIdx.x * kScoreThreads + tid) >> 5;   // this warp
    const long long NW = ((long long)gridDim.x * kScoreThreads) >> 5;
    const long long nt = W < tasks ? (tasks - W + NW - 1) / NW : 0;           // its tasks: W, W + NW, ...
    const uint32_t ring0 = smem_addr(ring) + (uint32_t)tid * 16u;

    // task it -> stage st of the ring (one commit group per task, empty past the last)
    auto issue = [&](long long it, int st) {
        if (it < nt) {
            const long long t = W + it * NW;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const long long row = o0 + (t * U + u) * R + rsub;
#pragma unroll
                for (int k = 0; k < K; ++k) {
                    const int c = j + g * k;
                    const bool v = row < o1 && c < C;
                    cp_async_zfill(ring0 + (uint32_t)(((st * U + u) * K + k) * kScoreThreads) * 16u,
                                   v ? static_cast<const void *>(x4 + row * C + c) : p.x, v ? 16u : 0u);
                }
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    float wf[K][E];
#pragma unroll
    for (int k = 0; k < K; ++k) unpack(wraw[k], wf[k]);
#pragma unroll
    for (int s = 0; s < S - 1; ++s) issue(s, s);
    bool nonfinite = false;
    for (long long it = 0; it < nt; ++it) {   // warp-uniform trip count
        const int st = (int)(it % S);
        issue(it + S - 1, (int)((it + S - 1) % S));
        cp_async_wait<S - 1>();   // this lane's copies of task it have landed
        const long long t = W + it * NW;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const long long row = o0 + (t * U + u) * R + rsub;
            float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int k = 0; k < K; ++k) {
                float f[E];
                unpack(ring[((st * U + u) * K + k) * kScoreThreads + tid], f);
#pragma unroll
                for (int e = 0; e < E; ++e) acc[e & 3] = fmaf(wf[k][e], f[e], acc[e & 3]);
            }
            float a = (acc[0] + acc[1]) + (acc[2] + acc[3]);
            for (int o = g >> 1; o >= 1; o >>= 1) a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
            if (j == 0 && row < o1) {
                const float sc = a + p.b;
                p.scores_out[row] = sc;
                nonfinite |= !isfinite(sc);
            }
        }
    }
    cp_async_wait<0>();
    if (nonfinite) raise_status(p.status, FUSION_DEV_NONFINITE);
}

template <typename T, int K>
cudaError_t launch_k(const ScoreParams &p, int sms, cudaStream_t s) {
    auto kern = k_token_scores<T, K>;
    constexpr size_t smem = ScoreRing<K>::smem;
    // set on every launch: the attribute belongs to the current device
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long R = 32 / p.group;
    const long long tasks = ((p.in.max_rows + R - 1) / R + ScoreRing<K>::U - 1) / ScoreRing<K>::U;
    long long blocks = (tasks + kScoreThreads / 32 - 1) / (kScoreThreads / 32);
    if (blocks > 2LL * sms) blocks = 2LL * sms;   // two CTAs per SM
    if (blocks < 1) blocks = 1;
    kern<<<(unsigned)blocks, kScoreThreads, smem, s>>>(p);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const ScoreParams &p, int K, int sms, cudaStream_t s) {
    switch (K) {
    case 1: return launch_k<T, 1>(p, sms, s);
    case 2: return launch_k<T, 2>(p, sms, s);
    case 3: return launch_k<T, 3>(p, sms, s);
    case 4: return launch_k<T, 4>(p, sms, s);
    case 5: return launch_k<T, 5>(p, sms, s);
    case 6: return launch_k<T, 6>(p, sms, s);
    case 7: return launch_k<T, 7>(p, sms, s);
    case 8: return launch_k<T, 8>(p, sms, s);
    default: return cudaErrorInvalidValue;
    }
}

int gcd_int(int a, int b) {
    while (b) {
        const int t = a % b;
        a = b;
        b = t;
    }
    return a;
}

}  // namespace

ScoreLayout score_layout(int dtype, int dim) {
    const int C = dim / (dtype == FUSION_BF16 ? 8 : 4);
    ScoreLayout L;
    for (int g = 8; g <= 32; g *= 2) {
        if (C % g == 0 && C / g <= kScoreMaxK) {
            L.group = g;
            L.chunks = C / g;
            return L;
        }
    }
    L.group = gcd_int(C, 32);
    L.chunks = C / L.group;
    if (L.chunks > kScoreMaxK) {
        L.group = 32;
        L.chunks = (C + 31) / 32;
    }
    return L;
}

cudaError_t launch_token_scores(int dtype, const ScoreParams &p, cudaStream_t s) {
    if (p.in.max_batch == 0) return cudaSuccess;   // no sample, no row
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const ScoreLayout L = score_layout(dtype, p.dim);
    ScoreParams q = p;
    q.group = L.group;
    return dtype == FUSION_BF16 ? launch_t<__nv_bfloat16>(q, L.chunks, sms, s) : launch_t<float>(q, L.chunks, sms, s);
}

}  // namespace fz
