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

// Head K chunk staged in shared memory (two stages): 128 dims for bf16, 64 for f32.
template <typename T> struct ExitKC;
template <> struct ExitKC<__nv_bfloat16> { static constexpr int v = 128; };
template <> struct ExitKC<float> { static constexpr int v = 64; };

// Neumaier-compensated accumulation: (s, c) carries the sum of every term added
// with an error of a few units in the last place of the result.
__device__ __forceinline__ void neu_add(float &s, float &c, float x) {
    const float t = __fadd_rn(s, x);
    c = __fadd_rn(c, fabsf(s) >= fabsf(x) ? __fadd_rn(__fsub_rn(s, t), x) : __fadd_rn(__fsub_rn(x, t), s));
    s = t;
}

// u = (x - mean) * rstd * gamma + beta for one element, rounded once to the head's
// input type.  A float32 evaluation is exact enough unless it lands within a few
// float32 ulps of a bf16 rounding midpoint (or beta cancels most of it); then the
// float-float evaluation decides.
__device__ __forceinline__ uint16_t ln_out_bf16(float x, F2 mean, F2 rstd, float g, float b) {
    const float d = __fsub_rn(__fsub_rn(x, mean.hi), mean.lo);
    const float v = __fmul_rn(__fmul_rn(d, rstd.hi), g);
    const float u = __fadd_rn(v, b);
    const uint32_t low = __float_as_uint(u) & 0xFFFFu;
    const uint32_t dist = low > 0x8000u ? low - 0x8000u : 0x8000u - low;
    if (dist > 24u && fabsf(u) >= 0.5f * fabsf(v)) {
        const uint32_t bits = __float_as_uint(u);
        if ((bits & 0x7F800000u) == 0x7F800000u) return (uint16_t)((bits >> 16) | ((bits & 0x7FFFFFu) ? 0x40u : 0u));
        return (uint16_t)((bits + (low > 0x8000u ? 0x8000u : 0u)) >> 16);   // not near a tie: plain rounding
    }
    F2 dd = two_sum(x, -mean.hi);
    dd.lo = __fsub_rn(dd.lo, mean.lo);
    F2 t = f2_mul(quick_two_sum(dd.hi, dd.lo), rstd);
    t = f2_mul(t, {g, 0.0f});
    return f2_to_bf16_bits(f2_add_f(t, b));
}
__device__ __forceinline__ float ln_out_f32(float x, F2 mean, F2 rstd, float g, float b) {
    const float d = __fsub_rn(__fsub_rn(x, mean.hi), mean.lo);
    return __fmaf_rn(__fmul_rn(d, rstd.hi), g, b);
}

template <typename T>
__device__ __forceinline__ void issue_w_chunk(const ExitParams &p, unsigned char *stage_buf, int c0, int k0,
                                              int dim, int C, int tid) {
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int EB = Elem<T>::kBytes;
    constexpr int KC = ExitKC<T>::v;
    constexpr int w_stride = KC + 16 / EB;
    constexpr int wchunks = KC / CH;
    const int kw = min(KC, dim - k0);
    const T *W = reinterpret_cast<const T *>(p.head.weight);
    for (int it = tid; it < kExitCT * wchunks; it += kExitThreads) {
        const int row = it / wchunks, c = it - row * wchunks;
        T *dst = reinterpret_cast<T *>(stage_buf) + row * w_stride + c * CH;
        if (c0 + row < C && c * CH < kw)
            cp_async16(dst, W + (size_t)(c0 + row) * dim + k0 + c * CH);
        else
            *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
    }
    cp_async_commit();
}

template <typename T>
struct ExitSmem {
    static constexpr int EB = Elem<T>::kBytes;
    static constexpr int KC = ExitKC<T>::v;
    static constexpr int w_stride = KC + 16 / EB;
    static constexpr size_t w_stage = (size_t)kExitCT * w_stride * EB;
    static __host__ __device__ int u_stride(int dim) { return dim + 16 / EB; }   // row bytes = 16 (mod 32)
    static __host__ __device__ size_t u_bytes(int dim) { return ((size_t)16 * u_stride(dim) * EB + 15) / 16 * 16; }
    static __host__ __device__ size_t total(int dim) {
        size_t t = u_bytes(dim) + 2 * w_stage + kExitCT * sizeof(float);
        const size_t plan = (4 * kExitThreads + 40) * sizeof(int);
        return t > plan ? t : plan;
    }
};

template <typename T>
__global__ void __launch_bounds__(kExitThreads) k_exit(ExitParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    using S = ExitSmem<T>;
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int EB = Elem<T>::kBytes;
    constexpr int KC = S::KC;
    constexpr bool kBf16 = (EB == 2);
    const int dim = p.dim;
    const int nchunk = dim / CH;
    const int u_stride = S::u_stride(dim);
    T *u_s = reinterpret_cast<T *>(sm);                   // 16 rows: CLS rows, then LayerNorm outputs
    unsigned char *w_region = sm + S::u_bytes(dim);
    float *lg_s = reinterpret_cast<float *>(w_region);    // [kExitBT][kExitCT], reused after the GEMM
    float *bias_s = reinterpret_cast<float *>(w_region + 2 * S::w_stage);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ct = blockIdx.x, bt = blockIdx.y;
    const int s0 = bt * kExitBT, c0 = ct * kExitCT;
    const int C = p.head.classes;
    const int Bdev = device_batch(p.in);
    const int B = Bdev < 0 ? 0 : Bdev;
    const bool active = s0 < B;
    const int n_k = (dim + KC - 1) / KC;

    // weight chunks 0 and 1, the CLS rows and the bias tile load together
    if (active) {
        issue_w_chunk<T>(p, w_region, c0, 0, dim, C, tid);
        if (n_k > 1) issue_w_chunk<T>(p, w_region + S::w_stage, c0, KC, dim, C, tid);
        for (int it = tid; it < 16 * nchunk; it += kExitThreads) {
            const int sl = it / nchunk, c = it - sl * nchunk;
            const int s = s0 + sl;
            T *dst = u_s + (size_t)sl * u_stride + c * CH;
            long long row = -1;
            if (sl < kExitBT && s < B) {
                row = p.in.offsets[s];
                if (row < 0 || row >= p.in.max_rows) row = -1;
            }
            if (row >= 0)
                cp_async16(dst, reinterpret_cast<const T *>(p.x) + row * dim + c * CH);
            else
                *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
        }
        cp_async_commit();
        for (int c = tid; c < kExitCT; c += kExitThreads) bias_s[c] = (c0 + c < C) ? p.head.bias[c0 + c] : 0.0f;
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        __syncthreads();

        // ---- LayerNorm of one CLS row per warp (float-float statistics) ---------------
        const int s = s0 + warp;
        bool ok = s < B;
        if (ok) {
            const long long row = p.in.offsets[s];
            if (row < 0 || row >= p.in.max_rows) {
                if (lane == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
                ok = false;
            }
        }
        T *xr = u_s + (size_t)warp * u_stride;
        if (ok) {
            float ss = 0.0f, sc = 0.0f;
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH];
                chunk_to_f(*reinterpret_cast<const uint4 *>(xr + c * CH), f);
#pragma unroll
                for (int e = 0; e < CH; ++e) neu_add(ss, sc, f[e]);
            }
            const F2 fdim = {(float)dim, 0.0f};
            const F2 mean = f2_div(warp_sum_f2(two_sum(ss, sc)), fdim);
            ss = sc = 0.0f;
            float lo = 0.0f;
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH];
                chunk_to_f(*reinterpret_cast<const uint4 *>(xr + c * CH), f);
#pragma unroll
                for (int e = 0; e < CH; ++e) {
                    F2 d = two_sum(f[e], -mean.hi);
                    d.lo = __fsub_rn(d.lo, mean.lo);
                    const F2 sq = two_prod(d.hi, d.hi);
                    neu_add(ss, sc, sq.hi);
                    lo = __fmaf_rn(2.0f * d.hi, d.lo, __fadd_rn(lo, sq.lo));
                }
            }
            const F2 var = f2_div(warp_sum_f2(f2_add_f(two_sum(ss, sc), lo)), fdim);
            const F2 rstd = f2_rsqrt(f2_add_f(var, p.head.eps));
            if (lane == 0 && !(isfinite(mean.hi) && isfinite(var.hi))) raise_status(p.status, FUSION_DEV_NONFINITE);
            const T *g = reinterpret_cast<const T *>(p.head.gamma);
            const T *bb = reinterpret_cast<const T *>(p.head.beta);
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH], gf[CH], bf[CH];
                chunk_to_f(*reinterpret_cast<const uint4 *>(xr + c * CH), f);
                chunk_to_f(ldg16(g + c * CH), gf);
                chunk_to_f(ldg16(bb + c * CH), bf);
                if constexpr (kBf16) {
                    uint32_t w4[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        w4[q] = (uint32_t)ln_out_bf16(f[2 * q], mean, rstd, gf[2 * q], bf[2 * q]) |
                                ((uint32_t)ln_out_bf16(f[2 * q + 1], mean, rstd, gf[2 * q + 1], bf[2 * q + 1]) << 16);
                    *reinterpret_cast<uint4 *>(xr + c * CH) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
                } else {
                    float4 o;
                    o.x = ln_out_f32(f[0], mean, rstd, gf[0], bf[0]);
                    o.y = ln_out_f32(f[1], mean, rstd, gf[1], bf[1]);
                    o.z = ln_out_f32(f[2], mean, rstd, gf[2], bf[2]);
                    o.w = ln_out_f32(f[3], mean, rstd, gf[3], bf[3]);
                    *reinterpret_cast<float4 *>(xr + c * CH) = o;
                }
            }
        } else {
            for (int c = lane; c < nchunk; c += 32) *reinterpret_cast<uint4 *>(xr + c * CH) = make_uint4(0, 0, 0, 0);
        }
    }
    __syncthreads();

    // ---- logits tile [kExitBT samples] x [kExitCT classes], K chunks double-buffered ----
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};   // bf16: two m16n8 fragments' valid rows; f32: 4 classes
    float acc2[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (active) {
        for (int kc = 0; kc < n_k; ++kc) {
            const int k0 = kc * KC;
            const int kw = min(KC, dim - k0);
            unsigned char *wbuf = w_region + (kc & 1) * S::w_stage;
            if (kc + 1 < n_k)
                asm volatile("cp.async.wait_group 1;\n" ::: "memory");
            else
                cp_async_wait_all();
            __syncthreads();
            if constexpr (kBf16) {
                // warp -> the 16-row sample tile (rows 8..15 are zero) x 16 classes
                float t0[4] = {0.0f, 0.0f, 0.0f, 0.0f}, t1[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                const uint32_t ubase = smem_addr(u_s);
                const uint32_t wbase = smem_addr(wbuf);
                const int arow = (lane & 7) + ((lane >> 3) & 1) * 8;
                const int brow = warp * 16 + (lane >> 4) * 8 + (lane & 7);
                for (int kk = 0; kk < kw; kk += 16) {
                    uint32_t af[4], b0, b1, b2, b3;
                    ldsm_x4(ubase + (uint32_t)((arow * u_stride + k0 + kk + (lane >> 4) * 8) * 2), af[0], af[1],
                            af[2], af[3]);
                    ldsm_x4(wbase + (uint32_t)((brow * S::w_stride + kk + ((lane >> 3) & 1) * 8) * 2), b0, b1, b2, b3);
                    mma_bf16_16816(t0, af, b0, b1);
                    mma_bf16_16816(t1, af, b2, b3);
                    if ((kk & 63) == 48) {   // flush the partial sums every 64 dims
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            acc[e] += t0[e];
                            acc2[e] += t1[e];
                            t0[e] = t1[e] = 0.0f;
                        }
                    }
                }
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc[e] += t0[e];
                    acc2[e] += t1[e];
                }
            } else {
                // warp -> sample `warp`; lane -> classes lane + 32 q
                const float *ur = reinterpret_cast<const float *>(u_s) + (size_t)warp * u_stride + k0;
                const float *ws = reinterpret_cast<const float *>(wbuf);
                float t[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                for (int kk = 0; kk < kw; kk += 4) {
                    const float4 uv = *reinterpret_cast<const float4 *>(ur + kk);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float4 wv = *reinterpret_cast<const float4 *>(ws + (lane + 32 * q) * S::w_stride + kk);
                        t[q] = fmaf(uv.x, wv.x, t[q]);
                        t[q] = fmaf(uv.y, wv.y, t[q]);
                        t[q] = fmaf(uv.z, wv.z, t[q]);
                        t[q] = fmaf(uv.w, wv.w, t[q]);
                    }
                    if ((kk & 15) == 12) {   // flush every 16 dims
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            acc[q] += t[q];
                            t[q] = 0.0f;
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < 4; ++q) acc[q] += t[q];
            }
            __syncthreads();   // everyone is done with this stage buffer
            if (kc + 2 < n_k) issue_w_chunk<T>(p, wbuf, c0, k0 + 2 * KC, dim, C, tid);
        }

        // ---- logits (+ bias) into shared memory; padded classes get -inf ---------------
        if constexpr (kBf16) {
            const int g = lane >> 2, t4 = lane & 3;   // fragment rows g (valid) and g + 8 (padding)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int col0 = warp * 16 + 2 * t4 + e, col1 = col0 + 8;
                lg_s[g * kExitCT + col0] = (c0 + col0 < C) ? acc[e] + bias_s[col0] : -INFINITY;
                lg_s[g * kExitCT + col1] = (c0 + col1 < C) ? acc2[e] + bias_s[col1] : -INFINITY;
            }
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int col = lane + 32 * q;
                lg_s[warp * kExitCT + col] = (c0 + col < C) ? acc[q] + bias_s[col] : -INFINITY;
            }
        }
        __syncthreads();
        if (p.logits) {
            for (int it = tid; it < kExitBT * kExitCT; it += kExitThreads) {
                const int sl = it / kExitCT, col = it - sl * kExitCT;
                if (s0 + sl < B && c0 + col < C) p.logits[(size_t)(s0 + sl) * C + c0 + col] = lg_s[it];
            }
        }
        // ---- partial softmax of this class tile: warp -> sample ------------------------
        {
            const int sl = warp, s = s0 + sl;
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
        const int s = s0 + warp;
        if (s < B) {
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
    return dtype == FUSION_BF16 ? ExitSmem<__nv_bfloat16>::total(dim) : ExitSmem<float>::total(dim);
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
