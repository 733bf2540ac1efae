// Exit check (Sec. III-D, Eq. 6-7): u = LayerNorm(CLS), logits = W u + b,
// c = max_k softmax(logits)_k, exit iff c >= tau.  The general kernel also runs the two
// layers of the MLP exit heads (Sec. III-G): the first reads the pooled float32 rows, the
// LayerNorm and GELU(W1 u + b1) rounded to the dtype; the second reads those rows densely,
// without LayerNorm, and ends in the softmax maximum and the exit rule.
//
// Two kernels.  The cluster kernel (heads of at most 8 class tiles) is described below.
// The general one: grid (class tiles of kExitCT) x (sample tiles of kExitBT).  Every CTA computes
// the LayerNorm of its samples' CLS rows, one logits tile (bf16: the weight tile by TMA and one
// tcgen05 product D[128 classes][16 samples] in tensor memory; f32: FFMA) and a partial softmax
// (tile max and sum of exponentials) per sample.  The last CTA of a sample tile to finish
// (atomic counter, no waiting) merges the partials into c and the exit mask; the
// last sample tile to finish runs the compaction plan for the fused stage.
#include <cooperative_groups.h>

#include "launch.h"
#include "ln.cuh"
#include "tc.cuh"

namespace cg = cooperative_groups;

namespace fz {
namespace {

// Head K chunk of the float32 kernels' two cp.async weight stages: 64 dims (bf16 heads arrive by
// TMA in 64-dim stages, kExitWStage; their entry here only sizes the unused float32 layout).
template <typename T> struct ExitKC;
template <> struct ExitKC<__nv_bfloat16> { static constexpr int v = 128; };
template <> struct ExitKC<float> { static constexpr int v = 64; };

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

// ---- the bf16 product of both kernels on tcgen05 ---------------------------------------
constexpr uint32_t kExitWStage = kExitCT * 128u;     // one weight stage: kExitCT rows x 64 bf16 dims

// Byte offset of 16-byte chunk c (8 bf16 dims) of row r in a bf16 u tile: K-blocks of 64 dims,
// each [16 rows][128 bytes] with chunk j of row r at j ^ (r % 8), the K-major,
// 128-byte-swizzled layout of a tcgen05 operand (8-row groups 1024 bytes apart).
__device__ __forceinline__ uint32_t u_tc_off(int r, int c) {
    return (uint32_t)(c >> 3) * 2048u + (uint32_t)r * 128u + ((uint32_t)((c & 7) ^ (r & 7)) << 4);
}
constexpr uint32_t kExitTmemCols = 32;   // D: 128 classes (lanes) x 16 samples (columns)
constexpr int kExitClMaxW = 16;          // most weight stages of a bf16 kernel
constexpr size_t kExitClBudget = 112 * 1024;   // the cluster kernel's dynamic shared memory bound (two CTAs per SM)
// the general kernel's bound: two CTAs per SM with its larger static shared memory
constexpr size_t kExitTcBudget = 110 * 1024;

// Instruction descriptor of D[128][16] (float32) += A[128][16] B[16][16]^T, A and B bf16, K-major.
constexpr uint32_t kExitIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(16 >> 3) << 17) | (8u << 24);

// The general kernel's bf16 shared memory, offsets from a 1024-byte aligned base: the u tile
// (u_tc_off; 16 rows, rows 8..15 zero) | the weight ring (w_stages TMA stages, the whole tile when
// it fits) | the bias tile.  The logits tile [kExitBT][kExitCT] reuses the ring after the product.
struct ExitTcSmem {
    static __host__ __device__ size_t u_bytes(int dim) { return (size_t)((dim + 63) / 64) * 2048; }
    static __host__ __device__ int w_stages(int dim) {
        const int nk = (dim + 63) / 64;
        const size_t rest = u_bytes(dim) + kExitCT * sizeof(float) + 1024;
        int st = rest + 2 * kExitWStage <= kExitTcBudget ? (int)((kExitTcBudget - rest) / kExitWStage) : 2;
        st = st < kExitClMaxW ? st : kExitClMaxW;
        return nk < st ? nk : st;
    }
    static __host__ __device__ size_t w_off(int dim) { return u_bytes(dim); }
    static __host__ __device__ size_t bias_off(int dim) { return w_off(dim) + (size_t)w_stages(dim) * kExitWStage; }
    static __host__ __device__ size_t total(int dim) {
        const size_t t = bias_off(dim) + kExitCT * sizeof(float);
        const size_t plan = plan_smem_bytes(kExitThreads);   // run_plan reuses the buffer from its start
        return (t > plan ? t : plan) + 1024;
    }
};

// D[128 classes][16 samples] = W_tile u^T on tcgen05, by one thread: per 64-dim K-block, wait
// for its weight stage (stages 0..nws-1 already issued), four MMAs (K = 16; fewer in a short
// last block), commit; when the tile is not resident, the stage of the block before is
// refilled by TMA once its MMAs completed (one block late, so that the wait overlaps the
// products just issued).  Every wait is bounded; after a failure the copies and products in
// flight are waited for (bounded) and FUSION_DEV_TIMEOUT is raised.  Returns whether D is
// complete.
__device__ __forceinline__ bool exit_tc_product(const CUtensorMap *wmap, uint32_t tmem, uint32_t ub, uint32_t wr,
                                                int dim, int nws, int c0, unsigned long long *wbar,
                                                unsigned long long *wempty, unsigned long long *wdone, int *status) {
    const int nk = (dim + 63) / 64;
    bool okw = true;
    int waited = 0, issued = 0, loaded = nws;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    for (int kc = 0; kc < nk; ++kc) {
        const int st = kc % nws;
        const uint32_t ph = (uint32_t)(kc / nws) & 1u;
        if (!mbar_wait(smem_addr(&wbar[st]), ph)) {
            okw = false;
            break;
        }
        waited = kc + 1;
        const uint32_t a0 = wr + (uint32_t)st * kExitWStage, b0 = ub + (uint32_t)kc * 2048u;
        const int kw = min(64, dim - kc * 64);
        for (int k = 0; k * 16 < kw; ++k)
            umma_bf16(tmem, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), kExitIdesc, (kc | k) ? 1u : 0u);
        umma_commit(smem_addr(&wempty[st]));
        issued = kc + 1;
        const int kp = kc - 1;   // the block before; its stage next holds block kp + nws
        if (kp >= 0 && kp + nws < nk) {
            const int sp = kp % nws;
            if (!mbar_wait(smem_addr(&wempty[sp]), (uint32_t)(kp / nws) & 1u)) {
                okw = false;
                break;
            }
            mbar_expect_tx(smem_addr(&wbar[sp]), kExitWStage);
            tma_load_2d(wr + (uint32_t)sp * kExitWStage, wmap, (kp + nws) * 64, c0, smem_addr(&wbar[sp]));
            loaded = kp + nws + 1;
        }
    }
    if (okw) {
        umma_commit(smem_addr(wdone));
        okw = mbar_wait(smem_addr(wdone), 0u);
    }
    if (!okw) {
        for (int q = waited; q < loaded; ++q) (void)mbar_wait(smem_addr(&wbar[q % nws]), (uint32_t)(q / nws) & 1u);
        if (issued > 0) (void)mbar_wait(smem_addr(&wempty[(issued - 1) % nws]), (uint32_t)((issued - 1) / nws) & 1u);
        raise_status(status, FUSION_DEV_TIMEOUT);
    }
    return okw;
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
        const size_t plan = plan_smem_bytes(kExitThreads);
        return t > plan ? t : plan;
    }
};

// The float32 logits tile [kExitBT samples] x [kExitCT classes] of one CTA by FFMA, K chunks of
// the head double-buffered (chunks 0 and 1 already in flight); u_s holds the LayerNorm rows.
template <typename T>
__device__ __forceinline__ void exit_gemm(const ExitParams &p, const T *u_s, unsigned char *w_region, int c0, int dim,
                                          int C, int n_k, float (&acc)[4]) {
    static_assert(sizeof(T) == 4, "bf16 heads take the tcgen05 product");
    using S = ExitSmem<T>;
    constexpr int KC = S::KC;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int u_stride = S::u_stride(dim);
    for (int kc = 0; kc < n_k; ++kc) {
        const int k0 = kc * KC;
        const int kw = min(KC, dim - k0);
        unsigned char *wbuf = w_region + (kc & 1) * S::w_stage;
        if (kc + 1 < n_k)
            asm volatile("cp.async.wait_group 1;\n" ::: "memory");
        else
            cp_async_wait_all();
        __syncthreads();
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
        __syncthreads();   // everyone is done with this stage buffer
        if (kc + 2 < n_k) issue_w_chunk<T>(p, wbuf, c0, k0 + 2 * KC, dim, C, tid);
    }
}

// The float32 logits (+ bias) into shared memory; padded classes get -inf.
__device__ __forceinline__ void exit_logits_f32(float *lg_s, const float *bias_s, const float (&acc)[4], int c0, int C) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int col = lane + 32 * q;
        lg_s[warp * kExitCT + col] = (c0 + col < C) ? acc[q] + bias_s[col] : -INFINITY;
    }
}

// The logits tile in shared memory (complete: after a barrier) to the staging rows lg_tmp, from
// which the last CTA of the sample tile writes the rows of the samples that exit.
__device__ __forceinline__ void exit_stage_logits(const ExitParams &p, const float *lg_s, int s0, int c0, int B, int C) {
    if (!p.lg_tmp) return;
    for (int it = threadIdx.x; it < kExitBT * kExitCT; it += kExitThreads) {
        const int sl = it / kExitCT, col = it - sl * kExitCT;
        if (s0 + sl < B && c0 + col < C) p.lg_tmp[(size_t)(s0 + sl) * C + c0 + col] = lg_s[it];
    }
}

// Error scale of a hidden unit's pre-activation a from the tcgen05 product: the bf16 products are
// exact and every K = 16 step adds them into the float32 accumulator, n = dim / 16 steps, each
// with an error below one float32 ulp (2^-23) of its partial sum, truncation included.  For
// partial sums of mixed signs the k-th is typically about sqrt(16 k / dim) ||w|| ||u|| / sqrt(dim),
// and even n errors of one sign at that size sum to about (sqrt(n) / 6) 2^-23 ||w|| ||u||, below
// 2^-22 ||w|| ||u|| up to dim = 1024.  Where the products share a sign, the partial sums grow
// monotonically up to |a|: the second term, n 2^-23 |a|, covers that case.  A typical-case scale,
// not a worst-case bound: rows whose partial sums rise to about sum |w u| / 2 and then cancel can
// exceed it if the accumulator truncates (about 2x at dim = 1024 in a model of the accumulation).
constexpr float kHidErr = 0x1p-22f;

// The exact pre-activation a = w . u + b1 of one hidden unit, by a whole warp: exact bf16 x bf16
// products summed in float-float (each lane a slice of the dims, then a butterfly).  The row u is
// row `row` of a u tile in shared memory (u_tc_off layout); the weight row is row wr of the
// resident weight ring wt (K-block q in stage q, TMA's 128-byte swizzle: chunk j of row r at
// j ^ (r % 8)) or, with wt NULL, the global row wg.  Every lane returns the result.
__device__ __forceinline__ F2 hidden_dot_exact_warp(const unsigned char *wt, int wr, const __nv_bfloat16 *wg,
                                                    const unsigned char *ut, int row, int dim, float b1) {
    const int lane = threadIdx.x & 31;
    F2 acc = {0.0f, 0.0f};
    for (int c = lane * 8; c < dim; c += 256) {
        float wf[8], uf[8];
        const int ch = c >> 3;
        chunk_to_f(wt ? *reinterpret_cast<const uint4 *>(wt + (size_t)(ch >> 3) * kExitWStage + (size_t)wr * 128 +
                                                         (((ch & 7) ^ (wr & 7)) << 4))
                      : ldg16(wg + c),
                   wf);
        chunk_to_f(*reinterpret_cast<const uint4 *>(ut + u_tc_off(row, ch)), uf);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = f2_add_f(acc, __fmul_rn(wf[e], uf[e]));
    }
    return f2_add_f(warp_sum_f2(acc), b1);
}

// GELU of an exact pre-activation (float-float) rounded once to bf16, by one thread: with the
// argument exact, the float GELU of its high part is within about a hundred float ulps of the
// exact value (erfc's error, amplified by its argument for large |a|); only a unit closer than
// that to a bf16 midpoint is evaluated in double, in the erf form.
__device__ __forceinline__ uint16_t gelu_exact_bf16(F2 acc) {
    const float g2 = 0.5f * acc.hi * erfcf(-acc.hi * 0.70710678118654752f);
    const float mid = __uint_as_float((__float_as_uint(g2) & 0xFFFF0000u) | 0x8000u);
    if (isfinite(g2) && fabsf(g2 - mid) > fabsf(g2) * 0x1p-17f) return __bfloat16_as_ushort(__float2bfloat16_rn(g2));
    const double a = (double)acc.hi + (double)acc.lo;
    const double g = 0.5 * a * (1.0 + erf(a / sqrt(2.0)));
    return __bfloat16_as_ushort(__double2bfloat16(g));
}

template <typename T>
__global__ void __launch_bounds__(kExitThreads) k_exit(const __grid_constant__ CUtensorMap wmap, ExitParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ __align__(8) unsigned long long wbar[kExitClMaxW], wempty[kExitClMaxW], wdone;
    __shared__ int s_wfail;
    __shared__ uint32_t tmem_base;
    using S = ExitSmem<T>;
    using TS = ExitTcSmem;
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int EB = Elem<T>::kBytes;
    constexpr int KC = S::KC;
    constexpr bool kBf16 = (EB == 2);
    const int dim = p.dim;
    const int nchunk = dim / CH;
    const int u_stride = S::u_stride(dim);
    // bf16: offsets from a 1024-byte aligned base (ExitTcSmem); float32: the u tile [16][u_stride]
    // | two cp.async weight stages | bias
    unsigned char *base = kBf16 ? reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm) + 1023) &
                                                                    ~uintptr_t(1023))
                                : sm;
    T *u_s = reinterpret_cast<T *>(base);   // 16 rows: CLS rows, then LayerNorm outputs
    // chunk c (CH dims) of row r of the u tile (bf16: the tcgen05 operand layout u_tc_off)
    auto uchunk = [&](int r, int c) -> T * {
        return kBf16 ? reinterpret_cast<T *>(base + u_tc_off(r, c)) : u_s + (size_t)r * u_stride + c * CH;
    };
    unsigned char *w_region = base + (kBf16 ? TS::w_off(dim) : S::u_bytes(dim));
    float *lg_s = reinterpret_cast<float *>(w_region);    // [kExitBT][kExitCT], reused after the product
    float *bias_s = reinterpret_cast<float *>(kBf16 ? base + TS::bias_off(dim) : w_region + 2 * S::w_stage);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ct = blockIdx.x, bt = blockIdx.y;
    const int s0 = bt * kExitBT, c0 = ct * kExitCT;
    const int C = p.head.classes;
    const int Bdev = device_batch(p.in);
    const int B = Bdev < 0 ? 0 : Bdev;
    const bool active = s0 < B;
    const int n_k = (dim + KC - 1) / KC;

    // the weight tile (bf16: TMA stages, the whole tile when it fits; float32: chunks 0 and 1), the
    // CLS rows and the bias tile load together
    if (active) {
        if constexpr (kBf16) {
            if (tid == 0) s_wfail = 0;
            if (warp == 0) {   // the logits tile's accumulator
                asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                                 smem_addr(&tmem_base)),
                             "r"(kExitTmemCols)
                             : "memory");
                asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
            }
            if (tid == 0) {
                const int nws = TS::w_stages(dim);
                for (int q = 0; q < nws; ++q) {
                    mbar_init(smem_addr(&wbar[q]), 1);
                    mbar_init(smem_addr(&wempty[q]), 1);
                }
                mbar_init(smem_addr(&wdone), 1);
                asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
                for (int q = 0; q < nws; ++q) {
                    mbar_expect_tx(smem_addr(&wbar[q]), kExitWStage);
                    tma_load_2d(smem_addr(w_region + (size_t)q * kExitWStage), &wmap, q * 64, c0, smem_addr(&wbar[q]));
                }
            }
        } else {
            issue_w_chunk<T>(p, w_region, c0, 0, dim, C, tid);
            if (n_k > 1) issue_w_chunk<T>(p, w_region + S::w_stage, c0, KC, dim, C, tid);
        }
        // launched as a programmatic dependent of the kernel before it (the MLP head's layers):
        // the weights above are this call's own input; the rows below may be that kernel's output
        asm volatile("griddepcontrol.wait;" ::: "memory");
        for (int it = tid; it < 16 * nchunk; it += kExitThreads) {
            const int sl = it / nchunk, c = it - sl * nchunk;
            const int s = s0 + sl;
            T *dst = uchunk(sl, c);
            long long row = -1;   // in_mode 2: the LayerNorm reads u_in and fills the tile
            if (sl < kExitBT && s < B && p.in_mode != 2) {
                row = p.in_mode == 0 ? (long long)p.in.offsets[s] : (long long)s;
                if (p.in_mode == 0 && (row < 0 || row >= p.in.max_rows)) row = -1;
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
        if (ok && p.in_mode == 0) {
            const long long row = p.in.offsets[s];
            if (row < 0 || row >= p.in.max_rows) {
                if (lane == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
                ok = false;
            }
        }
        // the row's chunk c as floats: from the tile, or from the float32 input rows
        const float *ur = p.in_mode == 2 && ok ? p.u_in + (size_t)s * dim : nullptr;
        const float *url = ur && p.u_in_lo ? p.u_in_lo + (size_t)s * dim : nullptr;   // float-float low parts
        auto in_lo = [&](int c, float (&f)[CH]) {
#pragma unroll
            for (int e = 0; e < CH; e += 4) {
                const float4 v = url ? *reinterpret_cast<const float4 *>(url + c * CH + e) : make_float4(0.f, 0.f, 0.f, 0.f);
                f[e] = v.x;
                f[e + 1] = v.y;
                f[e + 2] = v.z;
                f[e + 3] = v.w;
            }
        };
        auto in_chunk = [&](int c, float (&f)[CH]) {
            if (ur) {
#pragma unroll
                for (int e = 0; e < CH; e += 4) {
                    const float4 v = *reinterpret_cast<const float4 *>(ur + c * CH + e);
                    f[e] = v.x;
                    f[e + 1] = v.y;
                    f[e + 2] = v.z;
                    f[e + 3] = v.w;
                }
            } else {
                chunk_to_f(*reinterpret_cast<const uint4 *>(uchunk(warp, c)), f);
            }
        };
        if (ok && !p.skip_ln) {
            float ss = 0.0f, sc = 0.0f, sl_lo = 0.0f;
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH], fl[CH];
                in_chunk(c, f);
#pragma unroll
                for (int e = 0; e < CH; ++e) neu_add(ss, sc, f[e]);
                if (url) {
                    in_lo(c, fl);
#pragma unroll
                    for (int e = 0; e < CH; ++e) sl_lo = __fadd_rn(sl_lo, fl[e]);
                }
            }
            const F2 rdim = f2_recip((float)dim);
            const F2 mean = f2_mul(warp_sum_f2(url ? f2_add_f(two_sum(ss, sc), sl_lo) : two_sum(ss, sc)), rdim);
            ss = sc = 0.0f;
            float lo = 0.0f;
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH], fl[CH];
                in_chunk(c, f);
                in_lo(c, fl);
#pragma unroll
                for (int e = 0; e < CH; ++e) {
                    F2 d = two_sum(f[e], -mean.hi);
                    d.lo = url ? __fadd_rn(__fsub_rn(d.lo, mean.lo), fl[e]) : __fsub_rn(d.lo, mean.lo);
                    const F2 sq = two_prod(d.hi, d.hi);
                    neu_add(ss, sc, sq.hi);
                    lo = __fmaf_rn(2.0f * d.hi, d.lo, __fadd_rn(lo, sq.lo));
                }
            }
            const F2 var = f2_mul(warp_sum_f2(f2_add_f(two_sum(ss, sc), lo)), rdim);
            const F2 rstd = f2_rsqrt(f2_add_f(var, p.head.eps));
            if (lane == 0 && !(isfinite(mean.hi) && isfinite(var.hi))) raise_status(p.status, FUSION_DEV_NONFINITE);
            const T *g = reinterpret_cast<const T *>(p.head.gamma);
            const T *bb = reinterpret_cast<const T *>(p.head.beta);
            for (int c = lane; c < nchunk; c += 32) {
                float f[CH], fl[CH], gf[CH], bf[CH];
                in_chunk(c, f);
                in_lo(c, fl);
                chunk_to_f(ldg16(g + c * CH), gf);
                chunk_to_f(ldg16(bb + c * CH), bf);
                if constexpr (kBf16) {
                    uint32_t w4[4];
                    if (url) {
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            w4[q] = (uint32_t)ln_out_bf16_lo(f[2 * q], fl[2 * q], mean, rstd, gf[2 * q], bf[2 * q]) |
                                    ((uint32_t)ln_out_bf16_lo(f[2 * q + 1], fl[2 * q + 1], mean, rstd, gf[2 * q + 1],
                                                              bf[2 * q + 1])
                                     << 16);
                    } else {
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            w4[q] = (uint32_t)ln_out_bf16(f[2 * q], mean, rstd, gf[2 * q], bf[2 * q]) |
                                    ((uint32_t)ln_out_bf16(f[2 * q + 1], mean, rstd, gf[2 * q + 1], bf[2 * q + 1]) << 16);
                    }
                    *reinterpret_cast<uint4 *>(uchunk(warp, c)) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
                } else {
                    float4 o;
                    o.x = url ? ln_out_f32_lo(f[0], fl[0], mean, rstd, gf[0], bf[0]) : ln_out_f32(f[0], mean, rstd, gf[0], bf[0]);
                    o.y = url ? ln_out_f32_lo(f[1], fl[1], mean, rstd, gf[1], bf[1]) : ln_out_f32(f[1], mean, rstd, gf[1], bf[1]);
                    o.z = url ? ln_out_f32_lo(f[2], fl[2], mean, rstd, gf[2], bf[2]) : ln_out_f32(f[2], mean, rstd, gf[2], bf[2]);
                    o.w = url ? ln_out_f32_lo(f[3], fl[3], mean, rstd, gf[3], bf[3]) : ln_out_f32(f[3], mean, rstd, gf[3], bf[3]);
                    *reinterpret_cast<float4 *>(uchunk(warp, c)) = o;
                }
            }
        } else if (!ok) {   // (skip_ln: the loaded rows stay as they are)
            for (int c = lane; c < nchunk; c += 32) *reinterpret_cast<uint4 *>(uchunk(warp, c)) = make_uint4(0, 0, 0, 0);
        }
    }
    // bf16: the u tile, written by the generic proxy (stores and cp.async), is read by the tensor
    // core (async proxy) after the barrier
    if constexpr (kBf16) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();

    // ---- logits tile [kExitBT samples] x [kExitCT classes] -----------------------------
    // GELU(a) = a (1 + erf(a / sqrt 2)) / 2 = a erfc(-a / sqrt 2) / 2 for the hidden layer of an MLP
    // head; the erfc form is accurate in float for both signs.  bf16: a unit whose GELU lies within
    // the error scale of the product (kHidErr ||w_j|| ||u|| + n 2^-23 |a|, and the bias addition)
    // plus that of the float evaluation of a bf16 rounding midpoint is evaluated again exactly: the
    // dot product in float-float from exact bf16 x bf16 products, GELU in double.
    bool failed = false;   // bf16: a bounded wait of the product ran out (status raised; no output)
    if (active) {
        if constexpr (kBf16) {
            const uint32_t tmem = tmem_base;
            const int nws = TS::w_stages(dim);
            if (tid == 0)
                s_wfail = exit_tc_product(&wmap, tmem, smem_addr(base), smem_addr(w_region), dim, nws, c0, wbar,
                                          wempty, &wdone, p.status)
                              ? 0
                              : 1;
            __syncthreads();
            // the product is done: a programmatic dependent (the MLP head's next layer) may start its
            // prologue now; it reads nothing of ours before this grid completes
            asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            failed = s_wfail != 0;
            if (p.out_mode == 1) {
                // ---- hidden layer: a = D + b1 straight from tensor memory, the weight ring intact ----
                __shared__ float wn2[2][kExitCT], un[kExitBT];   // ||w_j||^2 in two halves; ||u||
                const bool resident = nws * 64 >= dim;           // every K-block in its own stage
                {   // ||w_j||^2, two threads per row: from the ring (a row's 8 chunks in any order; rows
                    // past C and dims past dim are zero), else from global memory, 8 loads at a time
                    const int r = tid & (kExitCT - 1), h = tid / kExitCT;
                    float acc = 0.0f;
                    if (resident) {
                        for (int q = h; q < nws; q += 2) {
                            const unsigned char *row = w_region + (size_t)q * kExitWStage + (size_t)r * 128;
#pragma unroll
                            for (int j2 = 0; j2 < 8; ++j2) {
                                float f[8];
                                chunk_to_f(*reinterpret_cast<const uint4 *>(row + 16 * j2), f);
#pragma unroll
                                for (int e = 0; e < 8; ++e) acc = fmaf(f[e], f[e], acc);
                            }
                        }
                    } else if (c0 + r < C) {
                        const T *wr = reinterpret_cast<const T *>(p.head.weight) + (size_t)(c0 + r) * dim;
                        for (int cb = h; cb < nchunk; cb += 16) {
                            uint4 v[8];
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                v[q] = cb + 2 * q < nchunk ? ldg16(wr + (cb + 2 * q) * CH) : make_uint4(0, 0, 0, 0);
#pragma unroll
                            for (int q = 0; q < 8; ++q) {
                                float f[CH];
                                chunk_to_f(v[q], f);
#pragma unroll
                                for (int e = 0; e < CH; ++e) acc = fmaf(f[e], f[e], acc);
                            }
                        }
                    }
                    wn2[h][r] = acc;
                }
                {   // ||u||^2 of each sample's row (warp -> sample slot)
                    float acc = 0.0f;
                    for (int c = lane; c < nchunk; c += 32) {
                        float f[CH];
                        chunk_to_f(*reinterpret_cast<const uint4 *>(uchunk(warp, c)), f);
#pragma unroll
                        for (int e = 0; e < CH; ++e) acc = fmaf(f[e], f[e], acc);
                    }
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
                    if (lane == 0) un[warp] = sqrtf(acc);
                }
                __syncthreads();
                // thread -> unit (class col = 32 (warp % 4) + lane: its tensor-memory lane; samples
                // 4 (warp / 4) .. + 3: columns of D)
                const int col = 32 * (warp & 3) + lane, sb = 4 * (warp >> 2);
                uint32_t v[16] = {};
                if (!failed) tmem_ld16(tmem + ((uint32_t)(32 * (warp & 3)) << 16), v);   // (failed: uniform)
                const float wn = sqrtf(1.0001f * (wn2[0][col] + wn2[1][col]));
                // the second term of the error scale: n = dim / 16 accumulation steps (kHidErr), plus
                // the bias addition and the float32 evaluation of a
                const float a_rel = 0x1p-20f + (float)((dim + 15) / 16) * 0x1p-23f;
                uint16_t *ho = reinterpret_cast<uint16_t *>(p.hidden_out);
                uint16_t hb[4];
                F2 ax[4];            // exact pre-activations of this thread's flagged units
                unsigned fl = 0;     // its units near a rounding midpoint (bit i: sample sb + i)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int sl = sb + i;
                    const bool valid = s0 + sl < B && c0 + col < C && !failed;
                    const float a = __uint_as_float(warp >= 4 ? v[4 + i] : v[i]) + bias_s[col];
                    const float g = 0.5f * a * erfcf(-a * 0.70710678118654752f);
                    const float ea = kHidErr * wn * un[sl] + fabsf(a) * a_rel;
                    const float eg = 1.13f * ea + fabsf(g) * 0x1p-16f;
                    const float mid = __uint_as_float((__float_as_uint(g) & 0xFFFF0000u) | 0x8000u);
                    const bool exact = valid && !(isfinite(g) && fabsf(g - mid) > eg);
                    hb[i] = __bfloat16_as_ushort(__float2bfloat16_rn(g));
                    ax[i] = {0.0f, 0.0f};
                    if (exact) fl |= 1u << i;
                    // their exact dot products, one at a time by the whole warp
                    for (unsigned mask = __ballot_sync(0xFFFFFFFFu, exact); mask; mask &= mask - 1) {
                        const int src = __ffs(mask) - 1;
                        const int scol = __shfl_sync(0xFFFFFFFFu, col, src);
                        const F2 e = hidden_dot_exact_warp(
                            resident ? w_region : nullptr, scol,
                            reinterpret_cast<const __nv_bfloat16 *>(p.head.weight) + (size_t)(c0 + scol) * dim, base,
                            sl, dim, bias_s[scol]);
                        if (lane == src) ax[i] = e;
                    }
                }
                // their GELU, every thread its own (the double-precision fallback then runs once per
                // unit, not once per lane of a warp)
                for (unsigned m = fl; m; m &= m - 1) {
                    const int i = __ffs(m) - 1;
                    const F2 x = i == 0 ? ax[0] : i == 1 ? ax[1] : i == 2 ? ax[2] : ax[3];
                    const uint16_t e = gelu_exact_bf16(x);
                    hb[0] = i == 0 ? e : hb[0];
                    hb[1] = i == 1 ? e : hb[1];
                    hb[2] = i == 2 ? e : hb[2];
                    hb[3] = i == 3 ? e : hb[3];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (s0 + sb + i < B && c0 + col < C && !failed) ho[(size_t)(s0 + sb + i) * C + c0 + col] = hb[i];
            } else if (warp < 4 && !failed) {
                // logits (+ bias) into shared memory over the ring: warp w < 4 reads the lanes
                // (classes) 32w.. of D
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16), v);
                const int cls = warp * 32 + lane;
#pragma unroll
                for (int n = 0; n < kExitBT; ++n)
                    lg_s[n * kExitCT + cls] = (c0 + cls < C) ? __uint_as_float(v[n]) + bias_s[cls] : -INFINITY;
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncthreads();
            if (warp == 0)
                asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kExitTmemCols)
                             : "memory");
        } else {
            float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};   // 4 classes of sample `warp`
            exit_gemm<T>(p, u_s, w_region, c0, dim, C, n_k, acc);
            exit_logits_f32(lg_s, bias_s, acc, c0, C);
            __syncthreads();
            if (p.out_mode == 1) {   // hidden layer: GELU in float32
                for (int it = tid; it < kExitBT * kExitCT; it += kExitThreads) {
                    const int sl = it / kExitCT, col = it - sl * kExitCT;
                    const float a = lg_s[it];
                    if (s0 + sl < B && c0 + col < C)
                        reinterpret_cast<float *>(p.hidden_out)[(size_t)(s0 + sl) * C + c0 + col] =
                            0.5f * a * erfcf(-a * 0.70710678118654752f);
                }
            }
        }
        if (p.out_mode == 0) {
            if (!failed) exit_stage_logits(p, lg_s, s0, c0, B, C);
            // ---- partial softmax of this class tile: warp -> sample ------------------------
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
            // a tile whose product timed out sends z = -1: no decision for its samples
            if (lane == 0 && s < B)
                p.partials[(size_t)s * p.n_ctile + ct] = failed ? make_float2(0.0f, -1.0f) : make_float2(m, z);
        }
    }
    if (p.out_mode == 1) return;   // no softmax across the tiles of a hidden layer

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
            bool bad = false;
            for (int q = lane; q < p.n_ctile; q += 32) {
                const float2 pz = __ldcg(&p.partials[(size_t)s * p.n_ctile + q]);
                m = fmaxf(m, pz.x);
                bad = bad || pz.y < 0.0f;
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
            if (!__any_sync(0xFFFFFFFFu, bad)) {   // else a product timed out: no decision (status raised)
                float z = 0.0f;
                for (int q = lane; q < p.n_ctile; q += 32) {
                    const float2 pz = __ldcg(&p.partials[(size_t)s * p.n_ctile + q]);
                    z += pz.y * expf(pz.x - m);
                }
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
                const float c = 1.0f / z;   // max_k softmax = exp(l_max - l_max) / sum
                const bool ex = c >= p.head.tau;
                if (lane == 0) {
                    p.exit_mask[s] = ex ? 1 : 0;
                    if (p.max_prob) p.max_prob[s] = c;
                    if (!isfinite(m)) raise_status(p.status, FUSION_DEV_NONFINITE);
                }
                if (ex && p.logits && p.lg_tmp)   // logits only for the samples that exit
                    for (int col = lane; col < p.head.classes; col += 32)
                        p.logits[(size_t)s * p.head.classes + col] =
                            __ldcg(&p.lg_tmp[(size_t)s * p.head.classes + col]);
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

__device__ __forceinline__ float to_float(float v) { return v; }
__device__ __forceinline__ float to_float(__nv_bfloat16 v) { return __bfloat162float(v); }

// ---------------------------------------------------------------------------
// The exit check as thread-block clusters: the n_ctile (<= 8) class tiles of one sample
// tile (8 samples) form a cluster.  Cluster rank r computes the
// LayerNorm of the tile's samples r, r + n_ctile, ... with several warps per row (one pass:
// sum and sum of squares in float-float, var = E[x^2] - mean^2) and stores the normalised
// row into the shared memory of every CTA of the cluster; each CTA then computes its logits
// tile and partial softmax, sends (max, sum of exponentials) to the sample's owner, and the
// owner merges them.  bf16: the head's weight tile arrives by TMA from the kernel's start
// (all of it when it fits, else a ring), and the logits tile is one tcgen05 product
// D[128 classes][16 samples] in tensor memory; float32: cp.async stages and FFMA.  No global
// atomics unless the plan kernel's work runs here (batches above the fused-plan bound).
// ---------------------------------------------------------------------------

template <typename T>
struct ExitClSmem {
    static constexpr int EB = Elem<T>::kBytes;
    static constexpr bool kTc = EB == 2;
    // samples per cluster (the tensor-memory product's N = 16 carries 8 of them: with 16,
    // a CTA needs the SM for itself and the clusters no longer fit in one wave)
    static constexpr int BT = kExitBT;
    using B = ExitSmem<T>;
    // u tile (16 GEMM rows; bf16: swizzled K-blocks) | W stages (bf16: w_stages(dim) TMA stages,
    // the whole tile when it fits; float32: two cp.async stages) | own raw CLS rows (BT; bf16:
    // none here, they use rows 8..15 of the u tile, which feed only unused columns) | gamma |
    // beta | bias | partials [BT][8] | reduction scratch | row flags.  bf16 offsets count from a
    // 1024-byte aligned base (the total includes the slack).
    static __host__ __device__ size_t u_bytes(int dim) { return kTc ? (size_t)((dim + 63) / 64) * 2048 : B::u_bytes(dim); }
    static __host__ __device__ size_t rest_bytes(int dim) {   // everything but the W stages
        return u_bytes(dim) + x_bytes(dim) + 2 * (((size_t)dim * EB + 15) / 16 * 16) +
               kExitCT * sizeof(float) + (size_t)BT * 8 * sizeof(float2) + (kExitThreads / 32) * 8 * sizeof(float) +
               (size_t)BT * sizeof(int);
    }
    static __host__ __device__ int w_stages(int dim) {
        if (!kTc) return 2;
        const int nk = (dim + 63) / 64;
        const size_t rest = rest_bytes(dim) + 1024;
        int st = rest + 2 * kExitWStage <= kExitClBudget ? (int)((kExitClBudget - rest) / kExitWStage) : 2;
        st = st < kExitClMaxW ? st : kExitClMaxW;
        return nk < st ? nk : st;
    }
    static __host__ __device__ size_t w_bytes(int dim) { return kTc ? (size_t)w_stages(dim) * kExitWStage : 2 * B::w_stage; }
    static __host__ __device__ size_t x_bytes(int dim) { return kTc ? 0 : (size_t)BT * B::u_stride(dim) * EB; }
    static __host__ __device__ size_t w_off(int dim) { return u_bytes(dim); }
    static __host__ __device__ size_t x_off(int dim) { return w_off(dim) + w_bytes(dim); }
    static __host__ __device__ size_t g_off(int dim) { return x_off(dim) + x_bytes(dim); }
    static __host__ __device__ size_t be_off(int dim) { return g_off(dim) + ((size_t)dim * EB + 15) / 16 * 16; }
    static __host__ __device__ size_t bias_off(int dim) { return be_off(dim) + ((size_t)dim * EB + 15) / 16 * 16; }
    static __host__ __device__ size_t part_off(int dim) { return bias_off(dim) + kExitCT * sizeof(float); }
    static __host__ __device__ size_t red_off(int dim) { return part_off(dim) + (size_t)BT * 8 * sizeof(float2); }
    static __host__ __device__ size_t flag_off(int dim) { return red_off(dim) + (size_t)(kExitThreads / 32) * 8 * sizeof(float); }
    static __host__ __device__ size_t total(int dim) {
        const size_t t = flag_off(dim) + (size_t)BT * sizeof(int);
        const size_t plan = w_off(dim) + plan_smem_bytes(kExitThreads);   // run_plan reuses the W stages
        return (t > plan ? t : plan) + (kTc ? 1024 : 0);
    }
};

template <typename T>
__global__ void __launch_bounds__(kExitThreads) k_exit_cl(const __grid_constant__ CUtensorMap wmap, ExitParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ __align__(8) unsigned long long wbar[kExitClMaxW], wempty[kExitClMaxW], wdone;
    __shared__ int s_wfail;
    __shared__ uint32_t tmem_base;
    using S = ExitSmem<T>;
    using L = ExitClSmem<T>;
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int EB = Elem<T>::kBytes;
    constexpr int KC = S::KC;
    constexpr bool kBf16 = (EB == 2);
    constexpr int kWarps = kExitThreads / 32;
    constexpr int BT = L::BT;
    cg::cluster_group cl = cg::this_cluster();
    const int ncl = (int)cl.num_blocks(), rank = (int)cl.block_rank();
    const int dim = p.dim, nchunk = dim / CH, u_stride = S::u_stride(dim);
    unsigned char *base = kBf16 ? reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm) + 1023) &
                                                                    ~uintptr_t(1023))
                                : sm;
    T *u_s = reinterpret_cast<T *>(base);   // float32: [16][u_stride]; bf16: see u_tc_off
    T *x_s = reinterpret_cast<T *>(base + L::x_off(dim));
    // chunk c of own raw CLS row j: float32 [BT][u_stride]; bf16 rows 8 + j of the u tile
    auto raw_chunk = [&](int j, int c) -> T * {
        return kBf16 ? reinterpret_cast<T *>(base + u_tc_off(8 + j, c)) : x_s + (size_t)j * u_stride + c * CH;
    };
    T *g_s = reinterpret_cast<T *>(base + L::g_off(dim));
    T *be_s = reinterpret_cast<T *>(base + L::be_off(dim));
    unsigned char *w_region = base + L::w_off(dim);   // bf16: 1024-byte aligned TMA stages
    float *lg_s = reinterpret_cast<float *>(w_region);   // [BT][kExitCT], reused after the GEMM
    float *bias_s = reinterpret_cast<float *>(base + L::bias_off(dim));
    float2 *part_s = reinterpret_cast<float2 *>(base + L::part_off(dim));
    float *red = reinterpret_cast<float *>(base + L::red_off(dim));
    int *rowflag_s = reinterpret_cast<int *>(base + L::flag_off(dim));   // [BT]: 1 row, 0 none, -1 bad

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ct = blockIdx.x, bt = blockIdx.y;
    const int s0 = bt * BT, c0 = ct * kExitCT;
    const int C = p.head.classes;
    const int Bdev = device_batch(p.in);
    const int B = Bdev < 0 ? 0 : Bdev;
    const bool active = s0 < B;   // uniform over the cluster (same sample tile)
    const int n_k = (dim + KC - 1) / KC;
    // rows of this CTA: slot j -> sample slot sl = rank + j * ncl (nrp slots, a power of two);
    // G >= 1 warps per row, ngr = kWarps / G rows at a time
    int nrp = 1;
    while (nrp * ncl < BT) nrp <<= 1;
    const int G = nrp >= kWarps ? 1 : kWarps / nrp;
    const int ngr = kWarps / G;
    const int jw = warp / G, gt = tid - jw * G * 32;   // row of this warp in a round, thread index in its group

    if (tid == 0) s_wfail = 0;
    if (active && kBf16 && warp == 0) {   // the logits tile's accumulator
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(kExitTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (active && kBf16 && tid == 0) {
        // the head's first weight chunks first: they depend on nothing and take longest to land
        const int nws = L::w_stages(dim);
        for (int q = 0; q < nws; ++q) {
            mbar_init(smem_addr(&wbar[q]), 1);
            mbar_init(smem_addr(&wempty[q]), 1);
        }
        mbar_init(smem_addr(&wdone), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        for (int q = 0; q < nws; ++q) {
            mbar_expect_tx(smem_addr(&wbar[q]), kExitWStage);
            tma_load_2d(smem_addr(w_region + (size_t)q * kExitWStage), &wmap, q * 64, c0, smem_addr(&wbar[q]));
        }
    }
    if (active) {
        // own CLS rows, gamma and beta (group 0), then the bias
        for (int it = tid; it < BT * nchunk; it += kExitThreads) {
            const int jj = it / nchunk, c = it - jj * nchunk;
            const int sli = rank + jj * ncl, si = s0 + sli;
            T *dst = raw_chunk(jj, c);
            long long row = -1;
            const bool want = sli < BT && si < B;
            if (want) {
                row = p.in.offsets[si];
                if (row < 0 || row >= p.in.max_rows) row = -1;
            }
            if (c == 0) rowflag_s[jj] = want ? (row >= 0 ? 1 : -1) : 0;
            if (row >= 0)
                cp_async16(dst, reinterpret_cast<const T *>(p.x) + row * dim + c * CH);
            else
                *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
        }
        for (int c = tid; c < 2 * nchunk; c += kExitThreads) {
            const bool isg = c < nchunk;
            const int cc = isg ? c : c - nchunk;
            cp_async16((isg ? g_s : be_s) + cc * CH,
                       reinterpret_cast<const T *>(isg ? p.head.gamma : p.head.beta) + cc * CH);
        }
        for (int c = tid; c < kExitCT; c += kExitThreads) {
            if (c0 + c < C)
                cp_async4(bias_s + c, p.head.bias + c0 + c);
            else
                bias_s[c] = 0.0f;
        }
        cp_async_commit();
        // padding rows 8..15 of the GEMM's A tile (float32; for bf16 they feed only the unused
        // columns 8..15 of the tensor-memory product)
        for (int it = tid; !kBf16 && it < 8 * nchunk; it += kExitThreads) {
            const int r = 8 + it / nchunk, c = it % nchunk;
            *reinterpret_cast<uint4 *>(u_s + (size_t)r * u_stride + c * CH) = make_uint4(0, 0, 0, 0);
        }
    }
    // every CTA of the cluster runs before any remote shared-memory store; nothing written before
    // it is read remotely, so the arrive need not release anything
    asm volatile("barrier.cluster.arrive.relaxed.aligned;\n\tbarrier.cluster.wait.aligned;" ::: "memory");
    if (active) {
        cp_async_wait_all();
        __syncthreads();
        // float32: the head's first two weight chunks load while the LayerNorm runs (issued
        // only now: every CTA's 64 KB of cp.async at once would hold up the CLS rows above)
        if constexpr (!kBf16) {
            issue_w_chunk<T>(p, w_region, c0, 0, dim, C, tid);
            if (n_k > 1) issue_w_chunk<T>(p, w_region + S::w_stage, c0, KC, dim, C, tid);
        }

        // ---- LayerNorm, G warps per row: one pass of sum and sum of squares -----------
        for (int jb = 0; jb < nrp; jb += ngr) {   // rounds of ngr rows (uniform trip count)
            const int j = jb + jw, sl = rank + j * ncl;
            const bool has_row = j < nrp && sl < BT;
            const int rflag = has_row ? rowflag_s[j] : 0;   // checked by the load loop above
            if (rflag < 0 && gt == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
            const bool ok = rflag > 0;
            const F2 rdim = f2_recip((float)dim);
            float s1 = 0.0f, c1 = 0.0f, s2 = 0.0f, c2 = 0.0f, l2 = 0.0f;
            if (ok) {
                for (int e = gt; e < dim; e += G * 32) {
                    const float v = to_float(raw_chunk(j, e / CH)[e % CH]);
                    neu_add(s1, c1, v);
                    const F2 sq = two_prod(v, v);
                    neu_add(s2, c2, sq.hi);
                    l2 = __fadd_rn(l2, sq.lo);
                }
            }
            F2 a1 = warp_sum_f2(two_sum(s1, c1));
            F2 a2 = warp_sum_f2(f2_add_f(two_sum(s2, c2), l2));
            if (lane == 0) {
                red[warp * 8 + 0] = a1.hi;
                red[warp * 8 + 1] = a1.lo;
                red[warp * 8 + 2] = a2.hi;
                red[warp * 8 + 3] = a2.lo;
            }
            __syncthreads();
            if (ok) {
                // the group's G (a power of two) warp sums: every aligned run of G lanes adds them
                // as a butterfly, so all lanes hold the same bits (f2_add is symmetric)
                const int wq = jw * G + (lane & (G - 1));
                F2 t1 = {red[wq * 8 + 0], red[wq * 8 + 1]}, t2 = {red[wq * 8 + 2], red[wq * 8 + 3]};
                for (int m = G >> 1; m >= 1; m >>= 1) {
                    t1 = f2_add(t1, f2_shfl_xor(t1, m));
                    t2 = f2_add(t2, f2_shfl_xor(t2, m));
                }
                const F2 mean = f2_mul(t1, rdim);
                const F2 ex2 = f2_mul(t2, rdim);
                const F2 m2 = f2_mul(mean, mean);
                F2 var = f2_add(ex2, {-m2.hi, -m2.lo});
                if (var.hi < 0.0f) var = {0.0f, 0.0f};
                const F2 rstd = f2_rsqrt(f2_add_f(var, p.head.eps));
                if (gt == 0 && !(isfinite(mean.hi) && isfinite(var.hi))) raise_status(p.status, FUSION_DEV_NONFINITE);
                for (int c = gt; c < nchunk; c += G * 32) {
                    float f[CH], gf[CH], bf[CH];
                    chunk_to_f(*reinterpret_cast<const uint4 *>(raw_chunk(j, c)), f);
                    chunk_to_f(*reinterpret_cast<const uint4 *>(g_s + c * CH), gf);
                    chunk_to_f(*reinterpret_cast<const uint4 *>(be_s + c * CH), bf);
                    uint4 outv;
                    if constexpr (kBf16) {
                        uint32_t w4[4];
    #pragma unroll
                        for (int q = 0; q < 4; ++q)
                            w4[q] = (uint32_t)ln_out_bf16(f[2 * q], mean, rstd, gf[2 * q], bf[2 * q]) |
                                    ((uint32_t)ln_out_bf16(f[2 * q + 1], mean, rstd, gf[2 * q + 1], bf[2 * q + 1]) << 16);
                        outv = make_uint4(w4[0], w4[1], w4[2], w4[3]);
                    } else {
                        outv = make_uint4(__float_as_uint(ln_out_f32(f[0], mean, rstd, gf[0], bf[0])),
                                          __float_as_uint(ln_out_f32(f[1], mean, rstd, gf[1], bf[1])),
                                          __float_as_uint(ln_out_f32(f[2], mean, rstd, gf[2], bf[2])),
                                          __float_as_uint(ln_out_f32(f[3], mean, rstd, gf[3], bf[3])));
                    }
                    T *dst = kBf16 ? reinterpret_cast<T *>(base + u_tc_off(sl, c)) : u_s + (size_t)sl * u_stride + c * CH;
                    for (int r = 0; r < ncl; ++r) *reinterpret_cast<uint4 *>(cl.map_shared_rank(dst, r)) = outv;
                }
            } else if (has_row) {
                for (int c = gt; c < nchunk; c += G * 32) {
                    T *dst = kBf16 ? reinterpret_cast<T *>(base + u_tc_off(sl, c)) : u_s + (size_t)sl * u_stride + c * CH;
                    for (int r = 0; r < ncl; ++r)
                        *reinterpret_cast<uint4 *>(cl.map_shared_rank(dst, r)) = make_uint4(0, 0, 0, 0);
                }
            }
            __syncthreads();   // the reduction scratch is reused by the next round
        }
    }
    // bf16: the u tile, written by the generic proxy here and in the other CTAs, is read by the
    // tensor core (async proxy) after the barrier
    if constexpr (kBf16) asm volatile("fence.proxy.async.shared::cluster;" ::: "memory");
    cl.sync();   // all LayerNorm rows are in every CTA's shared memory

    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};   // float32: 4 classes of sample `warp`
    if (active) {
        if constexpr (kBf16) {
            // ---- D[128 classes][16 samples] = W_tile u^T on tcgen05 (exit_tc_product) ----------
            const uint32_t tmem = tmem_base;
            if (tid == 0)
                s_wfail = exit_tc_product(&wmap, tmem, smem_addr(base), smem_addr(w_region), dim, L::w_stages(dim), c0,
                                          wbar, wempty, &wdone, p.status)
                              ? 0
                              : 1;
            __syncthreads();
            // the product is done: a programmatic dependent (the fused stage's per-sample kernel)
            // may start its prologue now; it reads nothing of ours before this grid completes
            asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            // logits (+ bias) into shared memory: warp w < 4 reads the lanes (classes) 32w.. of D
            // (not after a timed-out wait: the product may be incomplete)
            if (warp < 4 && s_wfail == 0) {
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16), v);
                const int cls = warp * 32 + lane;
#pragma unroll
                for (int n = 0; n < BT; ++n)
                    lg_s[n * kExitCT + cls] = (c0 + cls < C) ? __uint_as_float(v[n]) + bias_s[cls] : -INFINITY;
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncthreads();
            if (warp == 0)
                asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kExitTmemCols)
                             : "memory");
        } else {
            exit_gemm<T>(p, u_s, w_region, c0, dim, C, n_k, acc);
            exit_logits_f32(lg_s, bias_s, acc, c0, C);
            __syncthreads();
        }
        // partial softmax of this class tile, warp -> sample slots warp, warp + 8, ...; to every
        // CTA of the cluster (a tile whose product timed out sends z = -1: no decision)
        const bool failed = s_wfail != 0;
        for (int slw = warp; slw < BT; slw += kWarps) {
            const int sw = s0 + slw;
            float m = -INFINITY;
            for (int col = lane; col < kExitCT; col += 32) m = fmaxf(m, lg_s[slw * kExitCT + col]);
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
            float z = 0.0f;
            for (int col = lane; col < kExitCT; col += 32) {
                const float l = lg_s[slw * kExitCT + col];
                if (l != -INFINITY) z += expf(l - m);
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
            if (lane < ncl && sw < B)
                *cl.map_shared_rank(part_s + slw * 8 + rank, lane) = failed ? make_float2(0.0f, -1.0f) : make_float2(m, z);
        }
    }
    cl.sync();   // every CTA holds every partial of the tile's samples
    // Every CTA merges the partials in the same order (so all agree on every decision); the
    // owner writes the exit mask and c, every CTA its logits tile of the samples that exit.
    for (int slw = warp; active && slw < BT; slw += kWarps) {
        const int sw = s0 + slw;
        if (sw >= B) continue;
        float m = -INFINITY;
        bool bad = false;
        for (int q = lane; q < ncl; q += 32) {
            const float2 pz = part_s[slw * 8 + q];
            m = fmaxf(m, pz.x);
            bad = bad || pz.y < 0.0f;
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        if (__any_sync(0xFFFFFFFFu, bad)) continue;   // a product timed out: no decision (status raised)
        float z = 0.0f;
        for (int q = lane; q < ncl; q += 32) {
            const float2 pz = part_s[slw * 8 + q];
            z += pz.y * expf(pz.x - m);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
        const float c = 1.0f / z;   // max_k softmax = exp(l_max - l_max) / sum
        const bool ex = c >= p.head.tau;
        if (slw % ncl == rank && lane == 0) {
            p.exit_mask[sw] = ex ? 1 : 0;
            if (p.max_prob) p.max_prob[sw] = c;
            if (!isfinite(m)) raise_status(p.status, FUSION_DEV_NONFINITE);
        }
        if (ex && p.logits)   // logits only for the samples that exit
            for (int col = lane; col < kExitCT; col += 32)
                if (c0 + col < C) p.logits[(size_t)sw * C + c0 + col] = lg_s[slw * kExitCT + col];
    }
    if (!p.do_plan) {
        if (Bdev < 0 && bt == 0 && rank == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    // ---- the last cluster to finish runs the plan (batches above the fused-plan bound) ----
    __threadfence();
    cl.sync();   // this cluster's exit masks are written
    __shared__ int s_last;
    if (tid == 0) {
        s_last = 0;
        if (rank == 0) {
            __threadfence();
            s_last = (atomicAdd(&p.counters[p.n_btile], 1) == p.n_btile - 1);
        }
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) p.counters[p.n_btile] = 0;
    run_plan(p.plan, reinterpret_cast<int *>(w_region));
}

}  // namespace

size_t exit_smem_bytes(int dtype, int dim) {
    return dtype == FUSION_BF16 ? ExitTcSmem::total(dim) : ExitSmem<float>::total(dim);
}

namespace {
// bf16: the head weights [C][dim] as TMA boxes of 64 dims x 128 classes, 128-byte swizzle (the
// tcgen05 A operand); rows past C read as zero.  float32: no map (the kernels use cp.async).
cudaError_t head_weight_map(int dtype, const ExitParams &p, CUtensorMap *wmap) {
    *wmap = CUtensorMap{};
    if (dtype != FUSION_BF16) return cudaSuccess;
    EncodeTiledFn enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    cuuint64_t dims[2] = {(cuuint64_t)p.dim, (cuuint64_t)p.head.classes};
    cuuint64_t strides[1] = {(cuuint64_t)p.dim * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)kExitCT};
    cuuint32_t estr[2] = {1, 1};
    if (enc(wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p.head.weight), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    return cudaSuccess;
}

// The general kernel; pdl: as a programmatic dependent of the kernel before it on the stream.
template <typename T>
cudaError_t launch_exit_general(const ExitParams &p, cudaStream_t s, bool pdl) {
    CUtensorMap wmap;
    cudaError_t e = head_weight_map(sizeof(T) == 2 ? FUSION_BF16 : FUSION_F32, p, &wmap);
    if (e != cudaSuccess) return e;
    const size_t smem = exit_smem_bytes(sizeof(T) == 2 ? FUSION_BF16 : FUSION_F32, p.dim);
    e = cudaFuncSetAttribute(k_exit<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.n_ctile, p.n_btile);
    cfg.blockDim = dim3(kExitThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_exit<T>, wmap, p);
}
}  // namespace

template <typename T>
cudaError_t launch_exit_cluster(const ExitParams &p, cudaStream_t s) {
    CUtensorMap wmap;
    cudaError_t he = head_weight_map(sizeof(T) == 2 ? FUSION_BF16 : FUSION_F32, p, &wmap);
    if (he != cudaSuccess) return he;
    const size_t smem = ExitClSmem<T>::total(p.dim);
    cudaError_t e = cudaFuncSetAttribute(k_exit_cl<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ExitParams q = p;   // sample tiles of this kernel's size (the plan's cluster count), at least
                        // one: with max_batch == 0 the kernel still runs the plan
    q.n_btile = ceil_div(p.in.max_batch > 0 ? p.in.max_batch : 1, ExitClSmem<T>::BT);
    q.lg_tmp = nullptr;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(q.n_ctile, q.n_btile);
    cfg.blockDim = dim3(kExitThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = p.n_ctile;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_exit_cl<T>, wmap, q);
}

cudaError_t launch_exit(int dtype, const ExitParams &p, cudaStream_t s) {
    // the class tiles of a sample tile as one cluster (portable size: at most 8 tiles,
    // 1024 classes); larger heads take the kernel with a global last-CTA merge
    if (p.n_ctile <= kExitClMaxTiles && p.in_mode == 0 && !p.skip_ln && p.out_mode == 0)
        return dtype == FUSION_BF16 ? launch_exit_cluster<__nv_bfloat16>(p, s) : launch_exit_cluster<float>(p, s);
    return dtype == FUSION_BF16 ? launch_exit_general<__nv_bfloat16>(p, s, false) : launch_exit_general<float>(p, s, false);
}

// The general kernel as a programmatic dependent launch: its CTAs may start as the previous
// kernel on the stream triggers or finishes and wait for its results after issuing their
// weight loads.
cudaError_t launch_exit_pdl(int dtype, const ExitParams &p, cudaStream_t s) {
    return dtype == FUSION_BF16 ? launch_exit_general<__nv_bfloat16>(p, s, true) : launch_exit_general<float>(p, s, true);
}

namespace {
__global__ void __launch_bounds__(kPlanThreads) k_plan(PlanArgs a) {
    extern __shared__ int plan_sm[];
    run_plan(a, plan_sm);
}
}  // namespace

cudaError_t launch_plan(const PlanArgs &a, cudaStream_t s) {
    const size_t smem = plan_smem_bytes(kPlanThreads);
    k_plan<<<1, kPlanThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace fz
