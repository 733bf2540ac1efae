// Device helpers shared by the Fusion kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "fusion.h"

namespace fz {

// ---------------------------------------------------------------------------
// launch-side views of the C structs
// ---------------------------------------------------------------------------
struct Ragged {
    int max_batch;
    int max_tokens;
    long long max_rows;
    const int *offsets;
    const int *batch;
    const int *ids;
};

struct Head {
    const void *gamma;
    const void *beta;
    float eps;
    const void *weight;
    const float *bias;
    int classes;
    float tau;
};

// Geometry shared by the exit kernel, its workspace and the host.
constexpr int kExitBT = 8;      // samples per exit CTA (one LayerNorm per warp)
constexpr int kExitCT = 128;    // classes per exit CTA
constexpr int kExitThreads = 256;

constexpr int kPlanThreads = 1024;
constexpr int kImageThreads = 512;
constexpr int kImageWarps = kImageThreads / 32;

// Workspace layout (bytes from the workspace base; every block 256-aligned).
// The slot map and the plan come first, so their offsets depend on max_batch
// only; the exit counters and partial softmax sums follow, then the logits tiles of
// the general exit kernel (heads of more than kExitClMaxTiles class tiles only: its
// CTAs cannot wait for one another, so the last CTA of a sample tile copies the rows
// of the samples that exit from there).
constexpr int kExitClMaxTiles = 8;   // class tiles of the cluster exit kernel (portable cluster size)
struct WsLayout {
    size_t slot;       // int[max_batch]: output sample of every input sample
    size_t plan;       // int[4]: batch valid, survivor count
    size_t counters;   // int[n_btile + 1], zero between calls
    size_t partials;   // float2[n_btile * kExitBT * n_ctile]
    size_t lg;         // float[n_btile * kExitBT][classes] (empty for heads of <= kExitClMaxTiles tiles)
    size_t total;
};

__host__ __device__ inline size_t align256(size_t v) { return (v + 255) & ~size_t(255); }
__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }

__host__ __device__ inline WsLayout ws_layout(int max_batch, int classes) {
    WsLayout L;
    const int nbt = ceil_div(max_batch > 0 ? max_batch : 1, kExitBT);
    const int nct = ceil_div(classes > 0 ? classes : 1, kExitCT);
    size_t off = 0;
    L.slot = off;
    off += align256(sizeof(int) * (size_t)(max_batch > 0 ? max_batch : 1));
    L.plan = off;
    off += align256(sizeof(int) * 4);
    L.counters = off;
    off += align256(sizeof(int) * (size_t)(nbt + 1));
    L.partials = off;
    off += align256(sizeof(float) * 2 * (size_t)nbt * kExitBT * (size_t)nct);
    L.lg = off;
    if (nct > kExitClMaxTiles) off += align256(sizeof(float) * (size_t)nbt * kExitBT * (size_t)(classes > 0 ? classes : 1));
    L.total = off;
    return L;
}

// ---------------------------------------------------------------------------
// status and sample access
// ---------------------------------------------------------------------------
__device__ __forceinline__ void raise_status(int *st, int bits) {
    if (st) atomicOr(st, bits);
}

// Actual sample count (device scalar or the host bound); -1 when out of range.
__device__ __forceinline__ int device_batch(const Ragged &in) {
    if (!in.batch) return in.max_batch;
    const int b = *in.batch;
    return (b < 0 || b > in.max_batch) ? -1 : b;
}

// ---------------------------------------------------------------------------
// element types
// ---------------------------------------------------------------------------
template <typename T> struct Elem;
template <> struct Elem<float> {
    static constexpr int kBytes = 4;
    static constexpr int kPerChunk = 4;   // elements per 16-byte chunk
    __device__ __forceinline__ static float to_f(float v) { return v; }
};
template <> struct Elem<__nv_bfloat16> {
    static constexpr int kBytes = 2;
    static constexpr int kPerChunk = 8;
    __device__ __forceinline__ static float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
};

// Decode the elements of one 16-byte chunk.
__device__ __forceinline__ void chunk_to_f(const uint4 &c, float (&v)[4]) {
    v[0] = __uint_as_float(c.x);
    v[1] = __uint_as_float(c.y);
    v[2] = __uint_as_float(c.z);
    v[3] = __uint_as_float(c.w);
}
__device__ __forceinline__ void chunk_to_f(const uint4 &c, float (&v)[8]) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        v[2 * q] = __uint_as_float(w[q] << 16);
        v[2 * q + 1] = __uint_as_float(w[q] & 0xFFFF0000u);
    }
}

// ---------------------------------------------------------------------------
// data movement and tensor-core helpers (inline PTX)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gsrc) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(smem_addr(smem_dst)), "l"(gsrc)
                 : "memory");
}
__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gsrc) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(smem_addr(smem_dst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

__device__ __forceinline__ uint4 ldg16(const void *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

// Four 8x8 b16 matrices from shared memory; lane l supplies the row address of
// matrix l/8, row l%8.
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D += A(16x16, row) * B(16x8, col), bf16 inputs, f32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// ---------------------------------------------------------------------------
// ordering keys: larger key = larger value, then lower index
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t ordered_bits(float f) {
    f = (f == 0.0f) ? 0.0f : f;   // -0 and +0 compare equal
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float from_ordered_bits(uint32_t o) {
    const uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
    return __uint_as_float(u);
}
__device__ __forceinline__ unsigned long long rank_key(float v, int idx) {
    return ((unsigned long long)ordered_bits(v) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)idx);
}

// ---------------------------------------------------------------------------
// float-float ("double-float") arithmetic: value = hi + lo, |lo| <= ulp(hi)/2.
// The error-free transformations use the _rn intrinsics so that the compiler
// cannot contract or reassociate them.
// ---------------------------------------------------------------------------
struct F2 {
    float hi, lo;
};
__device__ __forceinline__ F2 two_sum(float a, float b) {
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return {s, e};
}
__device__ __forceinline__ F2 quick_two_sum(float a, float b) {   // |a| >= |b|
    const float s = __fadd_rn(a, b);
    return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ F2 two_prod(float a, float b) {
    const float p = __fmul_rn(a, b);
    return {p, __fmaf_rn(a, b, -p)};
}
__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
    F2 s = two_sum(a.hi, b.hi);
    const F2 t = two_sum(a.lo, b.lo);
    s.lo = __fadd_rn(s.lo, t.hi);
    s = quick_two_sum(s.hi, s.lo);
    s.lo = __fadd_rn(s.lo, t.lo);
    return quick_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ F2 f2_add_f(F2 a, float b) {
    F2 s = two_sum(a.hi, b);
    s.lo = __fadd_rn(s.lo, a.lo);
    return quick_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ F2 f2_mul(F2 a, F2 b) {
    F2 p = two_prod(a.hi, b.hi);
    p.lo = __fmaf_rn(a.hi, b.lo, p.lo);
    p.lo = __fmaf_rn(a.lo, b.hi, p.lo);
    return quick_two_sum(p.hi, p.lo);
}
// a / b for float-float operands, about 44 correct bits.
__device__ __forceinline__ F2 f2_div(F2 a, F2 b) {
    const float q1 = __fdiv_rn(a.hi, b.hi);
    const F2 r = f2_add(a, f2_mul({-q1, 0.0f}, b));
    const float q2 = __fdiv_rn(r.hi, b.hi);
    return quick_two_sum(q1, q2);
}
// 1 / n in float-float for a positive float n: the correctly rounded reciprocal r plus the
// remainder 1 - r n (exact in one fma for a correctly rounded r) times r, about 46 correct
// bits.  It needs no data, so a caller computes it before a reduction rather than after.
__device__ __forceinline__ F2 f2_recip(float n) {
    const float r = __frcp_rn(n);
    return quick_two_sum(r, __fmul_rn(__fmaf_rn(-r, n, 1.0f), r));
}
// 1 / sqrt(v) for a positive float-float v: one Newton step in float-float on the
// float32 estimate, about 44 correct bits.
__device__ __forceinline__ F2 f2_rsqrt(F2 v) {
    const float y = rsqrtf(v.hi);
    const F2 vy2 = f2_mul(v, two_prod(y, y));                    // v * y^2 ~ 1
    const F2 e = f2_add({1.0f, 0.0f}, {-vy2.hi, -vy2.lo});       // 1 - v y^2, tiny
    const float corr = __fmul_rn(__fmul_rn(0.5f, y), e.hi);      // y e / 2
    return quick_two_sum(y, corr);
}
__device__ __forceinline__ F2 f2_shfl_xor(F2 v, int m) {
    return {__shfl_xor_sync(0xFFFFFFFFu, v.hi, m), __shfl_xor_sync(0xFFFFFFFFu, v.lo, m)};
}
__device__ __forceinline__ F2 warp_sum_f2(F2 v) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) v = f2_add(v, f2_shfl_xor(v, m));
    return v;
}

// Round hi + lo (a float-float value) to the nearest bfloat16, ties to even.
// The only case where lo matters is hi lying exactly on a bf16 rounding midpoint.
__device__ __forceinline__ uint16_t f2_to_bf16_bits(F2 v) {
    const uint32_t u = __float_as_uint(v.hi);
    if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0x007FFFFFu) ? 0x40u : 0u));
    const uint32_t low = u & 0xFFFFu;
    uint32_t up = u >> 16;
    if (low > 0x8000u) {
        up += 1;
    } else if (low == 0x8000u) {
        // exactly on a midpoint of |hi|: lo decides, ties to even
        const bool away = (v.lo != 0.0f) && ((v.lo > 0.0f) == (v.hi > 0.0f));
        const bool toward = (v.lo != 0.0f) && !away;
        if (away || (!toward && (up & 1u))) up += 1;
    }
    return (uint16_t)up;
}

// ---------------------------------------------------------------------------
// block-wide exclusive scan of v[0..n) in shared memory, in chunks of 2 * blockDim.x
// elements (one chunk for n <= 2 * blockDim.x).  All threads must call; tmp needs 33 ints.
// Returns the total.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int block_scan_excl(int *v, int n, int *tmp) {
    const int t = threadIdx.x;
    const int lane = t & 31, w = t >> 5, nw = (blockDim.x + 31) >> 5;
    int base = 0;
    for (int c0 = 0; c0 < n; c0 += 2 * (int)blockDim.x) {
        const int i0 = c0 + 2 * t, i1 = i0 + 1;
        const int a = (i0 < n) ? v[i0] : 0;
        const int b = (i1 < n) ? v[i1] : 0;
        const int s = a + b;
        int incl = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) tmp[w] = incl;
        __syncthreads();
        if (w == 0) {
            const int x = (lane < nw) ? tmp[lane] : 0;
            int ix = x;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, ix, o);
                if (lane >= o) ix += y;
            }
            if (lane < nw) tmp[lane] = ix - x;
            if (lane == 31) tmp[32] = ix;
        }
        __syncthreads();
        const int excl = base + tmp[w] + incl - s;
        if (i0 < n) v[i0] = excl;
        if (i1 < n) v[i1] = excl + a;
        base += tmp[32];
        __syncthreads();
    }
    return base;
}

// ceil(rho * P) with rho taken exactly, clamped to [0, P]; NaN keeps nothing; NaN and
// +-inf set `nonfinite`.  P < 2^24 and rho has 24 significant bits, so the product is
// exactly p + e with p = fl(rho * P) and e = fma(rho, P, -p).  No integer lies strictly
// between p and the exact product (integers up to 2^24 are floats and p is the nearest
// float), so the ceiling is ceil(p), except when p is itself an integer: then it is
// p + 1 if e > 0.
__device__ __forceinline__ int keep_count(float rho, int P, bool &nonfinite) {
    if (isnan(rho) || isinf(rho)) nonfinite = true;
    if (P <= 0 || isnan(rho)) return 0;
    const float fP = (float)P;
    const float prod = __fmul_rn(rho, fP);
    const float err = __fmaf_rn(rho, fP, -prod);
    if (!(prod > 0.0f || (prod == 0.0f && err > 0.0f))) return 0;
    if (prod >= fP) return P;
    float c = ceilf(prod);
    if (c == prod && err > 0.0f) c += 1.0f;
    const int k = (int)c;
    return k > P ? P : k;
}

__device__ __forceinline__ int merge_count(int r, int P) {
    const int nA = P / 2;
    return r < 0 ? 0 : (r > nA ? nA : r);
}

}  // namespace fz
