// Input of an MLP exit head (Sec. III-G: a SpatialPool head at block 8, a CLS-only head
// at block 10): the CLS row, or the size-weighted mean of the patch rows,
// u = sum_t s_t x_t / sum_t s_t over positions 1..N-1 (the CLS row when N = 1), as a
// float-float value per element (u_out + u_lo), so that the LayerNorm of the head rounds its
// bf16 output like an exact evaluation.
//
// One CTA of 512 threads per sample (two per SM, one wave for a few hundred samples).
// Thread (r, c) owns the 16-byte column chunk c and the rows r, r + RL, ... of the sample
// (RL = 512 / chunks per row, at least 1), accumulating s_t x_t as exact products summed
// with compensation; the RL partial sums of a column are added in ascending r through shared
// memory in float-float and divided by the total size.  A stream over the tokens (dim * elem
// bytes read per row): eight rows of loads in flight per thread, about 16 MB over the GPU for
// 256 DeiT-S images.
#include "launch.h"

namespace fz {
namespace {

constexpr int kPoolThreads = 512;
constexpr int kPoolUnroll = 8;

template <typename T>
__global__ void __launch_bounds__(kPoolThreads, 2) k_head_pool(PoolParams p) {
    constexpr int E = Elem<T>::kPerChunk;
    __shared__ float2 red[kPoolThreads * E];  // [RL][dim] partial sums, float-float (RL * dim <= threads * E)
    __shared__ float2 wred[kPoolThreads];     // [RL] partial size sums, float-float
    const int s = blockIdx.x, tid = threadIdx.x;
    const int B = device_batch(p.in);
    if (B < 0) {
        if (s == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    if (s >= B) return;
    const int dim = p.dim;
    float *u = p.u_out + (size_t)s * dim;
    float *ul = p.u_lo + (size_t)s * dim;
    const int o0 = p.in.offsets[s], o1 = p.in.offsets[s + 1], n = o1 - o0;
    if (o0 < 0 || n < 1 || n > p.in.max_tokens || (long long)o1 > p.in.max_rows) {
        if (tid == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        for (int j = tid; j < dim; j += kPoolThreads) {
            u[j] = 0.0f;
            ul[j] = 0.0f;
        }
        return;
    }
    const int nch = dim / E;
    const uint4 *x4 = reinterpret_cast<const uint4 *>(p.x);
    if (p.pool == FUSION_POOL_CLS || n < 2) {
        for (int c = tid; c < nch; c += kPoolThreads) {
            float f[E];
            chunk_to_f(__ldg(x4 + (size_t)o0 * nch + c), f);
#pragma unroll
            for (int e = 0; e < E; ++e) {
                u[c * E + e] = f[e];
                ul[c * E + e] = 0.0f;
            }
        }
        return;
    }
    const int RL = nch < kPoolThreads ? kPoolThreads / nch : 1;
    const int c = tid % nch, r = tid / nch;
    float acc[E], acl[E];   // compensated sums: acc + acl
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = acl[e] = 0.0f;
    float ws = 0.0f, wl = 0.0f;
    if (r < RL) {
        for (int t = o0 + 1 + r; t < o1; t += kPoolUnroll * RL) {   // all loads before their products
            uint4 v[kPoolUnroll];
            float w[kPoolUnroll];
#pragma unroll
            for (int q = 0; q < kPoolUnroll; ++q) {   // rows past the sample add an exact 0
                const int tq = t + q * RL;
                v[q] = tq < o1 ? __ldcs(x4 + (size_t)tq * nch + c) : make_uint4(0u, 0u, 0u, 0u);
                w[q] = tq < o1 ? p.sizes[tq] : 0.0f;
            }
#pragma unroll
            for (int q = 0; q < kPoolUnroll; ++q) {
                float f[E];
                chunk_to_f(v[q], f);
#pragma unroll
                for (int e = 0; e < E; ++e) {   // the product exactly (two_prod), then a two_sum
                    const F2 pr = two_prod(w[q], f[e]);
                    const F2 t = two_sum(acc[e], pr.hi);
                    acc[e] = t.hi;
                    acl[e] = __fadd_rn(acl[e], __fadd_rn(t.lo, pr.lo));
                }
                const F2 tw = two_sum(ws, w[q]);
                ws = tw.hi;
                wl = __fadd_rn(wl, tw.lo);
            }
        }
#pragma unroll
        for (int e = 0; e < E; ++e) red[r * dim + c * E + e] = make_float2(acc[e], acl[e]);
        if (c == 0) wred[r] = make_float2(ws, wl);
    }
    __syncthreads();
    F2 W = {0.0f, 0.0f};
    for (int q = 0; q < RL; ++q) W = f2_add(W, {wred[q].x, wred[q].y});
    if (tid == 0 && !(W.hi > 0.0f && isfinite(W.hi))) raise_status(p.status, FUSION_DEV_NONFINITE);
    for (int j = tid; j < dim; j += kPoolThreads) {
        F2 a = {0.0f, 0.0f};
        for (int q = 0; q < RL; ++q) a = f2_add(a, {red[q * dim + j].x, red[q * dim + j].y});
        const F2 m = f2_div(a, W);
        u[j] = m.hi;
        ul[j] = m.lo;
    }
}

}  // namespace

cudaError_t launch_head_pool(int dtype, const PoolParams &p, cudaStream_t s) {
    if (p.in.max_batch == 0) return cudaSuccess;
    const dim3 grid((unsigned)p.in.max_batch);
    if (dtype == FUSION_BF16)
        k_head_pool<__nv_bfloat16><<<grid, kPoolThreads, 0, s>>>(p);
    else
        k_head_pool<float><<<grid, kPoolThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace fz
