// LayerNorm pieces of the exit kernels (Sec. III-D, Eq. 6: the exit head's LayerNorm of the
// CLS row): compensated sums and the output element rounded once to the head's input type.
#pragma once

#include "common.cuh"

namespace fz {

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

// ln_out_bf16 / ln_out_f32 for a float-float input element x + xlo (|xlo| <= ulp(x) / 2).
__device__ __forceinline__ uint16_t ln_out_bf16_lo(float x, float xlo, F2 mean, F2 rstd, float g, float b) {
    const float d = __fadd_rn(__fsub_rn(__fsub_rn(x, mean.hi), mean.lo), xlo);
    const float v = __fmul_rn(__fmul_rn(d, rstd.hi), g);
    const float u = __fadd_rn(v, b);
    const uint32_t low = __float_as_uint(u) & 0xFFFFu;
    const uint32_t dist = low > 0x8000u ? low - 0x8000u : 0x8000u - low;
    if (dist > 24u && fabsf(u) >= 0.5f * fabsf(v)) {
        const uint32_t bits = __float_as_uint(u);
        if ((bits & 0x7F800000u) == 0x7F800000u) return (uint16_t)((bits >> 16) | ((bits & 0x7FFFFFu) ? 0x40u : 0u));
        return (uint16_t)((bits + (low > 0x8000u ? 0x8000u : 0u)) >> 16);
    }
    F2 dd = two_sum(x, -mean.hi);
    dd.lo = __fadd_rn(__fsub_rn(dd.lo, mean.lo), xlo);
    F2 t = f2_mul(quick_two_sum(dd.hi, dd.lo), rstd);
    t = f2_mul(t, {g, 0.0f});
    return f2_to_bf16_bits(f2_add_f(t, b));
}
__device__ __forceinline__ float ln_out_f32_lo(float x, float xlo, F2 mean, F2 rstd, float g, float b) {
    const float d = __fadd_rn(__fsub_rn(__fsub_rn(x, mean.hi), mean.lo), xlo);
    return __fmaf_rn(__fmul_rn(d, rstd.hi), g, b);
}

}  // namespace fz
