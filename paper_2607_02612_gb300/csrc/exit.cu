// Exit check (Sec. III-D, Eq. 6-7): u = LayerNorm(CLS), logits = W u + b,
// c = max_k softmax(logits)_k, exit iff c >= tau.
//
// Grid: (class tiles of kExitCT) x (sample tiles of kExitBT).  Every CTA computes
// the LayerNorm of its samples' CLS rows, one logits tile (bf16: mma.sync tensor
// cores with float32 accumulation; f32: FFMA) and a partial softmax (tile max and
// sum of exponentials) per sample.  The last CTA of a sample tile to finish
// (atomic counter, no waiting) merges the partials into c and the exit mask; the
// last sample tile to finish runs the compaction plan for the fused stage.
#include "launch.h"

namespace fz {
namespace {

template <typename T>
__device__ __forceinline__ void store_u_chunk(T *dst, const F2 (&t)[Elem<T>::kPerChunk]);

template <>
__device__ __forceinline__ void store_u_chunk<float>(float *dst, const F2 (&t)[4]) {
    // the float nearest to hi + lo is hi (normalised pair)
    *reinterpret_cast<float4 *>(dst) = make_float4(t[0].hi, t[1].hi, t[2].hi, t[3].hi);
}
template <>
__device__ __forceinline__ void store_u_chunk<__nv_bfloat16>(__nv_bfloat16 *dst, const F2 (&t)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q)
        w[q] = (uint32_t)f2_to_bf16_bits(t[2 * q]) | ((uint32_t)f2_to_bf16_bits(t[2 * q + 1]) << 16);
    *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename T>
__global__ void __launch_bounds__(kExitThreads) k_exit(ExitParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int EB = Elem<T>::kBytes;
    const int dim = p.dim;
    const int nchunk = dim / CH;
    const int u_stride = dim + 16 / EB;            // row bytes = 16 (mod 32): conflict-free ldmatrix
    constexpr int w_stride = kExitKC + 16 / EB;
    T *u_s = reinterpret_cast<T *>(sm);
    unsigned char *w_region = sm + ((size_t)kExitBT * u_stride * EB + 15) / 16 * 16;
    float *lg_s = reinterpret_cast<float *>(w_region);   // reused after the GEMM

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ct = blockIdx.x, bt = blockIdx.y;
    const int s0 = bt * kExitBT, c0 = ct * kExitCT;
    const int C = p.head.classes;
    const int Bdev = device_batch(p.in);
    const int B = Bdev < 0 ? 0 : Bdev;
    const bool active = s0 < B;

    if (active) {
        // ---- LayerNorm of the CLS rows, in float-float arithmetic -------------------
        for (int sl = warp; sl < kExitBT; sl += kExitThreads / 32) {
            const int s = s0 + sl;
            T *urow = u_s + (size_t)sl * u_stride;
            long long row = -1;
            if (s < B) {
                row = p.in.offsets[s];
                if (row < 0 || row >= p.in.max_rows) {
                    if (lane == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
                    row = -1;
                }
            }
            if (row < 0) {
                for (int c = lane; c < nchunk; c += 32)
                    *reinterpret_cast<uint4 *>(urow + c * CH) = make_uint4(0, 0, 0, 0);
                continue;
            }
            const T *xr = reinterpret_cast<const T *>(p.x) + row * dim;
            F2 acc = {0.0f, 0.0f};
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH];
                chunk_to_f(ldg16(xr + c * CH), f);
#pragma unroll
                for (int e = 0; e < CH; ++e) acc = f2_add_f(acc, f[e]);
            }
            const F2 fdim = {(float)dim, 0.0f};
            const F2 mean = f2_div(warp_sum_f2(acc), fdim);
            const F2 nmean = {-mean.hi, -mean.lo};
            F2 acc2 = {0.0f, 0.0f};
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH];
                chunk_to_f(ldg16(xr + c * CH), f);
#pragma unroll
                for (int e = 0; e < CH; ++e) {
                    const F2 dl = f2_add_f(nmean, f[e]);
                    acc2 = f2_add(acc2, f2_mul(dl, dl));
                }
            }
            const F2 var = f2_div(warp_sum_f2(acc2), fdim);
            const double rs = 1.0 / sqrt((double)var.hi + (double)var.lo + (double)p.head.eps);
            const F2 rstd = {(float)rs, (float)(rs - (double)(float)rs)};
            if (lane == 0 && !(isfinite(mean.hi) && isfinite(var.hi)))
                raise_status(p.status, FUSION_DEV_NONFINITE);
            const T *g = reinterpret_cast<const T *>(p.head.gamma);
            const T *b = reinterpret_cast<const T *>(p.head.beta);
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH], gf[CH], bf[CH];
                chunk_to_f(ldg16(xr + c * CH), f);
                chunk_to_f(ldg16(g + c * CH), gf);
                chunk_to_f(ldg16(b + c * CH), bf);
                F2 t[CH];
#pragma unroll
                for (int e = 0; e < CH; ++e) {
                    F2 v = f2_mul(f2_add_f(nmean, f[e]), rstd);
                    v = f2_mul(v, {gf[e], 0.0f});
                    t[e] = f2_add_f(v, bf[e]);
                }
                store_u_chunk<T>(urow + c * CH, t);
            }
        }
    }
    __syncthreads();

    // ---- logits tile: [kExitBT samples] x [kExitCT classes] ------------------------
    constexpr bool kBf16 = (EB == 2);
    float acc[kBf16 ? 4 : 4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[a][q] = 0.0f;

    if (active) {
        const T *W = reinterpret_cast<const T *>(p.head.weight);
        constexpr int wchunks = kExitKC / CH;
        for (int k0 = 0; k0 < dim; k0 += kExitKC) {
            const int kw = min(kExitKC, dim - k0);
            for (int it = tid; it < kExitCT * wchunks; it += kExitThreads) {
                const int row = it / wchunks, c = it - row * wchunks;
                T *dst = reinterpret_cast<T *>(w_region) + row * w_stride + c * CH;
                if (c0 + row < C && c * CH < kw)
                    cp_async16(dst, W + (size_t)(c0 + row) * dim + k0 + c * CH);
                else
                    *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
            }
            cp_async_commit();
            cp_async_wait_all();
            __syncthreads();
            float tmp[4][4];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int q = 0; q < 4; ++q) tmp[a][q] = 0.0f;
            if constexpr (kBf16) {
                // warp -> 16 samples (mt) x 32 classes (ng): four m16n8 tiles
                const int mt = warp & 1, ng = warp >> 1;
                const uint32_t ubase = smem_addr(u_s);
                const uint32_t wbase = smem_addr(w_region);
                for (int kk = 0; kk < kw; kk += 16) {
                    uint32_t af[4];
                    const int arow = mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                    const int acol = k0 + kk + (lane >> 4) * 8;
                    ldsm_x4(ubase + (uint32_t)((arow * u_stride + acol) * 2), af[0], af[1], af[2], af[3]);
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr) {
                        const int brow = ng * 32 + (2 * pr + (lane >> 4)) * 8 + (lane & 7);
                        const int bcol = kk + ((lane >> 3) & 1) * 8;
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(wbase + (uint32_t)((brow * w_stride + bcol) * 2), b0, b1, b2, b3);
                        mma_bf16_16816(tmp[2 * pr], af, b0, b1);
                        mma_bf16_16816(tmp[2 * pr + 1], af, b2, b3);
                    }
                }
            } else {
                // warp -> 4 samples; lane -> classes lane + 32 q
                const float *us = reinterpret_cast<const float *>(u_s);
                const float *ws = reinterpret_cast<const float *>(w_region);
                for (int kk = 0; kk < kw; kk += 4) {
                    float4 uv[4], wv[4];
#pragma unroll
                    for (int a = 0; a < 4; ++a)
                        uv[a] = *reinterpret_cast<const float4 *>(us + (warp * 4 + a) * u_stride + k0 + kk);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        wv[q] = *reinterpret_cast<const float4 *>(ws + (lane + 32 * q) * w_stride + kk);
#pragma unroll
                    for (int a = 0; a < 4; ++a)
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            tmp[a][q] = fmaf(uv[a].x, wv[q].x, tmp[a][q]);
                            tmp[a][q] = fmaf(uv[a].y, wv[q].y, tmp[a][q]);
                            tmp[a][q] = fmaf(uv[a].z, wv[q].z, tmp[a][q]);
                            tmp[a][q] = fmaf(uv[a].w, wv[q].w, tmp[a][q]);
                        }
                }
            }
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int q = 0; q < 4; ++q) acc[a][q] += tmp[a][q];
            __syncthreads();
        }
        // ---- logits (+ bias) into shared memory; padded classes get -inf ----------
        if constexpr (kBf16) {
            const int mt = warp & 1, ng = warp >> 1, g = lane >> 2, t4 = lane & 3;
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int row = mt * 16 + g + (e >> 1) * 8;
                    const int col = ng * 32 + q * 8 + 2 * t4 + (e & 1);
                    const int c = c0 + col;
                    lg_s[row * kExitCT + col] = (c < C) ? acc[q][e] + p.head.bias[c] : -INFINITY;
                }
        } else {
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int col = lane + 32 * q;
                    const int c = c0 + col;
                    lg_s[(warp * 4 + a) * kExitCT + col] = (c < C) ? acc[a][q] + p.head.bias[c] : -INFINITY;
                }
        }
        __syncthreads();
        if (p.logits) {
            for (int it = tid; it < kExitBT * kExitCT; it += kExitThreads) {
                const int sl = it / kExitCT, col = it - sl * kExitCT;
                if (s0 + sl < B && c0 + col < C)
                    p.logits[(size_t)(s0 + sl) * C + c0 + col] = lg_s[it];
            }
        }
        // ---- partial softmax of this class tile ------------------------------------
        for (int sl = warp * 4; sl < warp * 4 + 4; ++sl) {
            const int s = s0 + sl;
            float m = -INFINITY;
            for (int col = lane; col < kExitCT; col += 32) m = fmaxf(m, lg_s[sl * kExitCT + col]);
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
            float z = 0.0f;
            for (int col = lane; col < kExitCT; col += 32) {
                const float l = lg_s[sl * kExitCT + col];
                if (l != -INFINITY) z += expf(l - m);
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
            if (lane == 0 && s < B) p.partials[(size_t)s * p.n_ctile + ct] = make_float2(m, z);
        }
    }

    // ---- the last class tile of this sample tile merges the partials ---------------
    __shared__ int s_last;
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = (atomicAdd(&p.counters[bt], 1) == p.n_ctile - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (active) {
        for (int sl = warp * 4; sl < warp * 4 + 4; ++sl) {
            const int s = s0 + sl;
            if (s >= B) continue;
            float m = -INFINITY;
            for (int q = lane; q < p.n_ctile; q += 32) m = fmaxf(m, __ldcg(&p.partials[(size_t)s * p.n_ctile + q]).x);
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
            float z = 0.0f;
            for (int q = lane; q < p.n_ctile; q += 32) {
                const float2 pz = __ldcg(&p.partials[(size_t)s * p.n_ctile + q]);
                z += pz.y * expf(pz.x - m);
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
            if (lane == 0) {
                const float c = 1.0f / z;   // max_k softmax = exp(l_max - l_max) / sum
                p.exit_mask[s] = (c >= p.head.tau) ? 1 : 0;
                if (p.max_prob) p.max_prob[s] = c;
                if (!isfinite(m)) raise_status(p.status, FUSION_DEV_NONFINITE);
            }
        }
    }
    if (tid == 0) p.counters[bt] = 0;

    // ---- the last sample tile runs the plan ------------------------------------------
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = (atomicAdd(&p.counters[p.n_btile], 1) == p.n_btile - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) {
        p.counters[p.n_btile] = 0;
        if (Bdev < 0 && !p.do_plan) raise_status(p.status, FUSION_DEV_BAD_BATCH);
    }
    if (p.do_plan) run_plan(p.plan, reinterpret_cast<int *>(sm));
}

}  // namespace

size_t exit_smem_bytes(int dtype, int dim) {
    const int EB = dtype == FUSION_BF16 ? 2 : 4;
    const size_t u = ((size_t)kExitBT * (dim + 16 / EB) * EB + 15) / 16 * 16;
    size_t w = (size_t)kExitCT * (kExitKC + 16 / EB) * EB;
    const size_t lg = (size_t)kExitBT * kExitCT * sizeof(float);
    if (lg > w) w = lg;
    size_t total = u + w;
    const size_t plan = (4 * kExitThreads + 40) * sizeof(int);
    if (plan > total) total = plan;
    return total;
}

cudaError_t launch_exit(int dtype, const ExitParams &p, cudaStream_t s) {
    const size_t smem = exit_smem_bytes(dtype, p.dim);
    const dim3 grid(p.n_ctile, p.n_btile);
    if (dtype == FUSION_BF16) {
        cudaError_t e = cudaFuncSetAttribute(k_exit<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_exit<__nv_bfloat16><<<grid, kExitThreads, smem, s>>>(p);
    } else {
        cudaError_t e = cudaFuncSetAttribute(k_exit<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_exit<float><<<grid, kExitThreads, smem, s>>>(p);
    }
    return cudaGetLastError();
}

namespace {
__global__ void __launch_bounds__(kPlanThreads) k_plan(PlanArgs a) {
    extern __shared__ int plan_sm[];
    run_plan(a, plan_sm);
}
}  // namespace

cudaError_t launch_plan(const PlanArgs &a, cudaStream_t s) {
    const size_t smem = (4 * kPlanThreads + 40) * sizeof(int);
    k_plan<<<1, kPlanThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace fz
