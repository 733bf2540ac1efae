// Size-aware attention over a ragged batch: the transformer block that consumes a compacted
// batch (Algorithm 1, Block_b), with the proportional attention of ToMe so that a merged
// token of size s weighs like the s tokens it replaced.  For every sample, head h and query
// row m of the sample:
//   out[m, h] = sum_j softmax_j(q_m . k_j / sqrt(dh) + log s_j) v_j.
//
// One CTA of 256 threads per (head, sample), dh = 64, bf16.  Samples of at most 256 tokens
// (calls whose max_tokens is at most 256) keep the whole sample in shared memory (k_attn_tc);
// longer samples, up to 1024 tokens, stream key blocks (k_attn_tc_long, below).
// TMA brings the sample's query tiles of 128 rows, its K rows and its V rows (one 128-byte
// row of 64 dims each, 128-byte swizzle) from the packed qkv matrix.  Q and K are K-major
// operands; V, rows of keys with the dims contiguous, is the MN-major B operand of the second
// product as it lies (8-key swizzle atoms 1024 bytes apart); its rows past the sample are
// zeroed once it has landed.  Per query tile t: S_t = Q_t K^T (M = 128, N = tokens
// rounded up to 16, K = 64) accumulates in tensor-memory columns [0, N);
// warp w and warp w + 4 share the rows of lane quadrant w, each taking half of the columns
// (maxima and sums meet in shared memory): logits scaled by log2(e) / sqrt(dh) plus
// log2(s_j), masked past the sample, shifted by max_j S scale + max_j log2 s_j (an upper bound of
// the row maximum within log2(max s / min s), so sizes within a factor 2^100 of each other keep
// every probability a normal float), exp2 (ex2.approx), the row sum, and the
// unnormalised probabilities P_t as bf16 pairs written back over S's first columns; O_t = P_t V
// (M = 128, N = 64, K = tokens rounded up to 16, A = P from tensor memory) accumulates in
// columns [128, 192); the epilogue divides each row by its sum and stores bf16.  P is rounded to
// bf16 (the operand type of the second product); the sum is taken before that.  Without a P
// buffer a CTA needs Q, K and V only (84 KB for 197 tokens) and 256 tensor-memory columns, so
// two CTAs share an SM; the query tiles of a sample run one after the other.
//
// Every wait on an mbarrier is bounded; on a timeout the CTA raises FUSION_DEV_TIMEOUT, skips
// its outputs, waits (bounded) for the operations it started and frees its tensor memory.
#include "launch.h"
#include "tc.cuh"

namespace fz {
namespace {

constexpr int kAttnThreads = 256;
constexpr int kAttnDh = 64;
constexpr int kAttnMaxN = 256;
constexpr uint32_t kQTileBytes = 128 * 128;   // 128 rows x one K-block of 64 bf16
constexpr uint32_t kAttnTmemCols = 256;       // S (<= 256 columns); P over its first half; O at 128

__device__ __forceinline__ float ex2(float x) {   // 2^x, one MUFU instruction (2^-inf = 0)
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// max(a, b, c) in one instruction (three-source max.f32 of sm_100 and later); exact
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
// max of m and the 16 values of a tensor-memory chunk: a tree of three-source maxima (8
// instructions, 3 deep, against 16 in a chain)
__device__ __forceinline__ float max16(float m, const uint32_t (&v)[16]) {
    const float a = max3(__uint_as_float(v[0]), __uint_as_float(v[1]), __uint_as_float(v[2]));
    const float b = max3(__uint_as_float(v[3]), __uint_as_float(v[4]), __uint_as_float(v[5]));
    const float c = max3(__uint_as_float(v[6]), __uint_as_float(v[7]), __uint_as_float(v[8]));
    const float d = max3(__uint_as_float(v[9]), __uint_as_float(v[10]), __uint_as_float(v[11]));
    const float e = max3(__uint_as_float(v[12]), __uint_as_float(v[13]), __uint_as_float(v[14]));
    return max3(m, max3(a, b, c), max3(d, e, __uint_as_float(v[15])));
}

struct AttnMaps {
    CUtensorMap b32, b8;   // qkv rows, boxes of 64 dims x 32 / 8 rows, 128-byte swizzle
};

// The two warps that share lane quadrant w (warps w and w + 4) meet at named barrier 1 + w.
__device__ __forceinline__ void pair_sync(int warp) {
    switch (warp & 3) {   // literal ids: the kernel reserves barriers 0..4 only
    case 0: asm volatile("bar.sync 1, 64;" ::: "memory"); break;
    case 1: asm volatile("bar.sync 2, 64;" ::: "memory"); break;
    case 2: asm volatile("bar.sync 3, 64;" ::: "memory"); break;
    default: asm volatile("bar.sync 4, 64;" ::: "memory"); break;
    }
}
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}
// D (tensor memory) += A (tensor memory, 128 lanes x 16 bf16 packed in 8 columns) x B (shared memory).
__device__ __forceinline__ void umma_bf16_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc, uint32_t idesc,
                                             uint32_t accumulate) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(tmem_d),
        "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__global__ void __launch_bounds__(kAttnThreads, 2)
    k_attn_tc(const __grid_constant__ AttnMaps maps, AttnParams p) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
    // bar_ld: query tile 0 and K (the first product's operands); bar_ld2: V and the other query tiles
    __shared__ __align__(8) unsigned long long bar_ld, bar_ld2, bar_s, bar_o;
    __shared__ uint32_t tmem_base;
    __shared__ int s_fail, s_issued;   // s_issued: operations started (for the drain on a timeout)
    __shared__ __align__(16) float lsz[kAttnMaxN];   // log2 of the key sizes
    __shared__ float red[2][128];      // the two column halves' row maxima, then row sums
    __shared__ float s_lszmax;         // max_j log2 s_j

    const int tid = threadIdx.x, warp = tid >> 5;
    const int h = blockIdx.x, i = blockIdx.y;
    const int B = device_batch(p.in);
    if (B < 0) {
        if (h == 0 && i == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    if (i >= B) return;
    const int o0 = p.in.offsets[i], n = p.in.offsets[i + 1] - o0;
    if (o0 < 0 || n < 1 || n > p.in.max_tokens || n > kAttnMaxN || (long long)o0 + n > p.in.max_rows) {
        if (h == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        return;
    }
    const int H = p.heads;
    const int npad = (n + 15) & ~15;              // keys rounded up to the MMA granularity
    const int T = (n + 127) >> 7;                 // query tiles
    unsigned char *Q = sm;                        // T tiles of 128 rows
    unsigned char *Kr = sm + (size_t)T * kQTileBytes;
    unsigned char *Vr = Kr + (size_t)npad * 128;  // V rows (MN-major B operand)

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(kAttnTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid == 0) {
        s_fail = 0;
        s_issued = 0;
        mbar_init(smem_addr(&bar_ld), 1);
        mbar_init(smem_addr(&bar_ld2), 1);
        mbar_init(smem_addr(&bar_s), 1);
        mbar_init(smem_addr(&bar_o), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();

    // ---- loads: the query tiles, K and V by TMA (rows rounded up to 8); query tile 0 and K on
    // ---- bar_ld (the first product starts once they landed), V and the other tiles on bar_ld2 --
    if (tid == 0) {
        const int rk = (n + 7) & ~7;
        auto qrows = [&](int t) { return (min(128, n - 128 * t) + 7) & ~7; };
        uint32_t bytes2 = (uint32_t)rk * 128u;
        for (int t = 1; t < T; ++t) bytes2 += (uint32_t)qrows(t) * 128u;
        mbar_expect_tx(smem_addr(&bar_ld), (uint32_t)(rk + qrows(0)) * 128u);
        mbar_expect_tx(smem_addr(&bar_ld2), bytes2);
        auto rows = [&](unsigned char *dst, int x, int y0, int cnt, unsigned long long *bar) {   // cnt: multiple of 8
            int r = 0;
            for (; r + 32 <= cnt; r += 32) tma_load_2d(smem_addr(dst + r * 128), &maps.b32, x, y0 + r, smem_addr(bar));
            for (; r < cnt; r += 8) tma_load_2d(smem_addr(dst + r * 128), &maps.b8, x, y0 + r, smem_addr(bar));
        };
        rows(Q, h * kAttnDh, o0, qrows(0), &bar_ld);
        rows(Kr, (H + h) * kAttnDh, o0, rk, &bar_ld);
        rows(Vr, (2 * H + h) * kAttnDh, o0, rk, &bar_ld2);
        for (int t = 1; t < T; ++t) rows(Q + (size_t)t * kQTileBytes, h * kAttnDh, o0 + 128 * t, qrows(t), &bar_ld2);
        s_issued = 1;
    }
    for (int j = tid; j < npad; j += kAttnThreads)
        lsz[j] = j < n ? (p.sizes ? log2f(p.sizes[o0 + j]) : 0.0f) : 0.0f;
    if (tid == 0 && !mbar_wait(smem_addr(&bar_ld), 0)) s_fail = 1;
    __syncthreads();
    if (warp == 0) {   // max_j log2 s_j over the sample
        float lm = -INFINITY;
        for (int j = threadIdx.x; j < n; j += 32) lm = fmaxf(lm, lsz[j]);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) lm = fmaxf(lm, __shfl_xor_sync(0xFFFFFFFFu, lm, o));
        if (threadIdx.x == 0) s_lszmax = lm;
    }
    __syncthreads();

    const uint32_t tmem = tmem_base;
    const int half = warp >> 2;                 // column half of the row
    const int r = tid & 127;                    // row of the tile = tensor-memory lane
    const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const int nch = npad >> 4;                  // 16-column chunks of S
    const int cA = (nch + 1) >> 1;              // chunks [0, cA) to half 0, [cA, nch) to half 1
    const int c_lo = half ? cA : 0, c_hi = half ? nch : cA;
    constexpr float kScale2 = 0.18033688011112042f;   // log2(e) / sqrt(64)
    const uint32_t idesc_s = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(npad >> 3) << 17) | (8u << 24);
    // B = V as it lies: MN-major (bit 16), 8-key swizzle atoms 1024 bytes apart
    const uint32_t idesc_o =
        (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(kAttnDh >> 3) << 17) | (8u << 24);

    bool stop = s_fail != 0;   // read between two barriers: the same in every thread
    for (int t = 0; t < T && !stop; ++t) {
        // ---- S = Q_t K^T into columns [0, npad) ---------------------------------------------
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
            for (int k = 0; k < 4; ++k)
                umma_bf16(tmem, sw128_desc(smem_addr(Q + (size_t)t * kQTileBytes) + k * 32), sw128_desc(smem_addr(Kr) + k * 32),
                          idesc_s, k ? 1u : 0u);
            umma_commit(smem_addr(&bar_s));
            s_issued = 2 + 2 * t;
        }
        if (!mbar_wait(smem_addr(&bar_s), (uint32_t)t & 1u)) atomicOr(&s_fail, 2);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const bool rows_here = 128 * t + 32 * (warp & 3) < n;   // warp-uniform: a warp of rows past the sample idles
        // ---- the softmax shift: max_j S * scale + max_j log2 s_j, an upper bound of the row's largest
        // ---- logit by at most log2(max s / min s) (the result does not depend on the shift) -------
        float mx = -INFINITY;
        if (rows_here) {
            for (int c = c_lo; c < c_hi; ++c) {
                uint32_t v[16];
                tmem_ld16(lane_addr + (uint32_t)(16 * c), v);
                if (16 * c + 16 <= n) {
                    mx = max16(mx, v);
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (16 * c + e < n) mx = fmaxf(mx, __uint_as_float(v[e]));
                }
            }
        }
        red[half][r] = mx;
        pair_sync(warp);
        mx = fmaf(fmaxf(red[0][r], red[1][r]), kScale2, s_lszmax);
        // ---- P = 2^(logit - max) as bf16 pairs, and the row sum; P goes over S's first columns once
        // ---- every S column of the row has been read (the other half reads some of them) ----------
        float2 lsum2 = make_float2(0.0f, 0.0f);   // even and odd columns (packed float32 pairs)
        uint32_t pk[8][8];   // this half's chunks, at most 8
        if (rows_here) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int c = c_lo + q;
                if (c < c_hi) {
                    uint32_t v[16];
                    tmem_ld16(lane_addr + (uint32_t)(16 * c), v);
                    float pr[16];
#pragma unroll
                    for (int e = 0; e < 16; e += 2) {   // fma then subtract, two columns per instruction
                        const float2 x = __fadd2_rn(
                            __ffma2_rn(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])),
                                       make_float2(kScale2, kScale2), *reinterpret_cast<const float2 *>(&lsz[16 * c + e])),
                            make_float2(-mx, -mx));
                        pr[e] = ex2(x.x);
                        pr[e + 1] = ex2(x.y);
                    }
                    if (16 * c + 16 > n) {
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            if (16 * c + e >= n) pr[e] = 0.0f;
                    }
#pragma unroll
                    for (int e = 0; e < 16; e += 2) {
                        lsum2 = __fadd2_rn(lsum2, make_float2(pr[e], pr[e + 1]));
                        const __nv_bfloat162 b2 = __floats2bfloat162_rn(pr[e], pr[e + 1]);
                        pk[q][e >> 1] = *reinterpret_cast<const uint32_t *>(&b2);
                    }
                }
            }
        }
        pair_sync(warp);   // every S column of these rows read; both halves' maxima read
        if (rows_here) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (c_lo + q < c_hi) tmem_st8(lane_addr + (uint32_t)(8 * (c_lo + q)), pk[q]);
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        }
        red[half][r] = lsum2.x + lsum2.y;
        if (t == 0) {
            // V and the other query tiles: landed while this tile's softmax ran; V rows n .. npad-1
            // (another sample's rows or stale memory) read as zero in P V
            if (tid == 0 && !mbar_wait(smem_addr(&bar_ld2), 0)) atomicOr(&s_fail, 8);
            __syncthreads();
            if (s_fail == 0)
                for (int c = tid; c < (npad - n) * 8; c += kAttnThreads)
                    reinterpret_cast<uint4 *>(Vr + (size_t)n * 128)[c] = make_uint4(0u, 0u, 0u, 0u);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // visible to the tensor core
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();   // all of P stored before the second product
        const float lsum = red[0][r] + red[1][r];
        // ---- O = P V into columns [128, 192) ---------------------------------------------------
        const bool ok_s = s_fail == 0;   // the S waits' outcome, after the barrier above
        if (tid == 0 && ok_s) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            for (int kk = 0; kk < npad / 16; ++kk)
                umma_bf16_ts(tmem + 128u, tmem + 8u * kk, sw128_desc(smem_addr(Vr) + kk * 2048u), idesc_o, kk ? 1u : 0u);
            umma_commit(smem_addr(&bar_o));
            s_issued = 3 + 2 * t;
        }
        if (ok_s && !mbar_wait(smem_addr(&bar_o), (uint32_t)t & 1u)) atomicOr(&s_fail, 4);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // ---- epilogue: this half's 32 dims of O / row sum -> bf16 -------------------------------
        if (rows_here) {
            uint32_t o[32];
            tmem_ld16(lane_addr + 128u + 32u * half, *reinterpret_cast<uint32_t(*)[16]>(o));
            tmem_ld16(lane_addr + 144u + 32u * half, *reinterpret_cast<uint32_t(*)[16]>(o + 16));
            const int m = 128 * t + r;
            if (m < n && s_fail == 0) {
                const float inv = 1.0f / lsum;
                uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                                       (size_t)(o0 + m) * H * kAttnDh + (size_t)h * kAttnDh + 32 * half);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 y = __fmul2_rn(
                            make_float2(__uint_as_float(o[8 * c + 2 * e]), __uint_as_float(o[8 * c + 2 * e + 1])),
                            make_float2(inv, inv));
                        const __nv_bfloat162 b2 = __floats2bfloat162_rn(y.x, y.y);
                        w[e] = *reinterpret_cast<const uint32_t *>(&b2);
                    }
                    dst[c] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();   // O read and the sums consumed before the next tile's S overwrites them
        stop = s_fail != 0;
        __syncthreads();   // nobody writes s_fail again before every thread has read it
    }
    if (tid == 0 && s_fail != 0) {   // let everything this CTA started finish before it leaves
        raise_status(p.status, FUSION_DEV_TIMEOUT);
        mbar_wait(smem_addr(&bar_ld), 0);
        mbar_wait(smem_addr(&bar_ld2), 0);
        const int k = s_issued;   // 2 + 2t: S of tile t issued; 3 + 2t: also its O
        if (k >= 2) mbar_wait(smem_addr(&bar_s), (uint32_t)((k - 2) >> 1) & 1u);
        if (k >= 3 && (k & 1)) mbar_wait(smem_addr(&bar_o), (uint32_t)((k - 3) >> 1) & 1u);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kAttnTmemCols) : "memory");
}

// ---------------------------------------------------------------------------
// Samples of 257 .. 1024 tokens.  The keys come in blocks of 128 (K, and V for the second
// pass), double-buffered by TMA one step ahead; per query tile a first pass over the key blocks
// takes the softmax shift (max_j S scale + max_j log2 s_j, as above) and a second pass forms P
// over S's first columns and accumulates O = P V over the key blocks in columns [128, 192).
// Q tiles are double-buffered too; every step waits for the previous step's products, so a
// buffer is refilled only once nothing reads it.
// ---------------------------------------------------------------------------
constexpr int kLongMaxN = 1024;
constexpr uint32_t kKvBytes = 128 * 128;   // a block of 128 key rows (K or V)

__global__ void __launch_bounds__(kAttnThreads, 2)
    k_attn_tc_long(const __grid_constant__ AttnMaps maps, AttnParams p) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) unsigned long long bar_ld[2], bar_s, bar_o;
    __shared__ uint32_t tmem_base;
    __shared__ int s_fail, s_ld, s_ns, s_no;   // steps whose loads were issued; products S and O issued
    __shared__ __align__(16) float lsz[kLongMaxN];
    __shared__ float red[2][128];
    __shared__ float s_lszmax;

    const int tid = threadIdx.x, warp = tid >> 5;
    const int h = blockIdx.x, i = blockIdx.y;
    const int B = device_batch(p.in);
    if (B < 0) {
        if (h == 0 && i == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_BATCH);
        return;
    }
    if (i >= B) return;
    const int o0 = p.in.offsets[i], n = p.in.offsets[i + 1] - o0;
    if (o0 < 0 || n < 1 || n > p.in.max_tokens || n > kLongMaxN || (long long)o0 + n > p.in.max_rows) {
        if (h == 0 && tid == 0) raise_status(p.status, FUSION_DEV_BAD_OFFSETS);
        return;
    }
    const int H = p.heads;
    const int T = (n + 127) >> 7;          // query tiles
    const int nkv = (n + 127) >> 7;        // key blocks
    const int steps = T * 2 * nkv;         // (tile, pass, block) in that order
    unsigned char *Qb = sm;                                 // [2] query tiles
    unsigned char *Kb = sm + 2 * kQTileBytes;               // [2] key blocks
    unsigned char *Vb = Kb + 2 * kKvBytes;                  // [2] value blocks

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(kAttnTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // the loads of step k into buffer k & 1: the key block, the value block in the second pass,
    // the query tile at a tile's first step
    auto issue = [&](int k) {
        const int t = k / (2 * nkv), pass = (k / nkv) & 1, kb = k % nkv;
        const int buf = k & 1;
        const int rows_k = min(128, n - 128 * kb), rk = (rows_k + 7) & ~7;
        const bool q = pass == 0 && kb == 0;
        const int rq = (min(128, n - 128 * t) + 7) & ~7;
        uint32_t bytes = (uint32_t)rk * 128u * (pass ? 2u : 1u) + (q ? (uint32_t)rq * 128u : 0u);
        const uint32_t bar = smem_addr(&bar_ld[buf]);
        mbar_expect_tx(bar, bytes);
        auto rows = [&](unsigned char *dst, int x, int y0, int cnt) {
            int r = 0;
            for (; r + 32 <= cnt; r += 32) tma_load_2d(smem_addr(dst + r * 128), &maps.b32, x, y0 + r, bar);
            for (; r < cnt; r += 8) tma_load_2d(smem_addr(dst + r * 128), &maps.b8, x, y0 + r, bar);
        };
        rows(Kb + buf * kKvBytes, (H + h) * kAttnDh, o0 + 128 * kb, rk);
        if (pass) rows(Vb + buf * kKvBytes, (2 * H + h) * kAttnDh, o0 + 128 * kb, rk);
        if (q) rows(Qb + (t & 1) * kQTileBytes, h * kAttnDh, o0 + 128 * t, rq);
    };
    if (tid == 0) {
        s_fail = 0;
        s_ns = s_no = 0;
        mbar_init(smem_addr(&bar_ld[0]), 1);
        mbar_init(smem_addr(&bar_ld[1]), 1);
        mbar_init(smem_addr(&bar_s), 1);
        mbar_init(smem_addr(&bar_o), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        issue(0);
        s_ld = 1;
    }
    for (int j = tid; j < n; j += kAttnThreads) lsz[j] = p.sizes ? log2f(p.sizes[o0 + j]) : 0.0f;
    __syncthreads();
    if (warp == 0) {
        float lm = -INFINITY;
        for (int j = threadIdx.x; j < n; j += 32) lm = fmaxf(lm, lsz[j]);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) lm = fmaxf(lm, __shfl_xor_sync(0xFFFFFFFFu, lm, o));
        if (threadIdx.x == 0) s_lszmax = lm;
    }
    __syncthreads();

    const uint32_t tmem = tmem_base;
    const int half = warp >> 2;
    const int r = tid & 127;
    const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    constexpr float kScale2 = 0.18033688011112042f;   // log2(e) / sqrt(64)
    const uint32_t idesc_o =
        (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(kAttnDh >> 3) << 17) | (8u << 24);
    float mraw = -INFINITY, mx = 0.0f;
    float2 lsum2 = make_float2(0.0f, 0.0f);   // even and odd columns (packed float32 pairs)
    bool stop = false;
    for (int k = 0; k < steps && !stop; ++k) {
        const int t = k / (2 * nkv), pass = (k / nkv) & 1, kb = k % nkv;
        const int buf = k & 1;
        const int rows_k = min(128, n - 128 * kb), npadb = (rows_k + 15) & ~15;
        const bool rows_here = 128 * t + 32 * (warp & 3) < n;   // warp-uniform
        const int nch = npadb >> 4, cA = (nch + 1) >> 1;
        const int c_lo = half ? cA : 0, c_hi = half ? nch : cA;
        // ---- this step's blocks landed; the next step's loads go out -------------------------
        if (tid == 0) {
            if (!mbar_wait(smem_addr(&bar_ld[buf]), (uint32_t)(k >> 1) & 1u)) {
                s_fail = 1;
            } else if (k + 1 < steps) {
                issue(k + 1);
                s_ld = k + 2;
            }
        }
        __syncthreads();
        if (s_fail & 1) break;   // uniform: bit 1 is written only before the barrier above
        if (pass == 1 && rows_k < npadb)   // value rows past the sample read as zero in P V
            for (int c = tid; c < (npadb - rows_k) * 8; c += kAttnThreads)
                reinterpret_cast<uint4 *>(Vb + buf * kKvBytes + (size_t)rows_k * 128)[c] = make_uint4(0u, 0u, 0u, 0u);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        // ---- S = Q_t K_kb^T --------------------------------------------------------------------
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t idesc_s = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(npadb >> 3) << 17) | (8u << 24);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                umma_bf16(tmem, sw128_desc(smem_addr(Qb + (t & 1) * kQTileBytes) + kk * 32),
                          sw128_desc(smem_addr(Kb + buf * kKvBytes) + kk * 32), idesc_s, kk ? 1u : 0u);
            umma_commit(smem_addr(&bar_s));
            s_ns = s_ns + 1;
        }
        if (!mbar_wait(smem_addr(&bar_s), (uint32_t)k & 1u)) atomicOr(&s_fail, 2);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if (pass == 0) {
            // ---- first pass: running maximum of S over this half's columns ---------------------
            if (rows_here) {
                for (int c = c_lo; c < c_hi; ++c) {
                    uint32_t v[16];
                    tmem_ld16(lane_addr + (uint32_t)(16 * c), v);
                    if (16 * c + 16 <= rows_k) {
                        mraw = max16(mraw, v);
                    } else {
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            if (16 * c + e < rows_k) mraw = fmaxf(mraw, __uint_as_float(v[e]));
                    }
                }
            }
            if (kb == nkv - 1) {   // the tile's shift from both halves
                red[half][r] = mraw;
                pair_sync(warp);
                mx = fmaf(fmaxf(red[0][r], red[1][r]), kScale2, s_lszmax);
                pair_sync(warp);
            }
        } else {
            // ---- second pass: P over S's first columns, then O += P V_kb ----------------------
            uint32_t pk[4][8];   // this half's chunks, at most 4
            if (rows_here) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int c = c_lo + q;
                    if (c < c_hi) {
                        uint32_t v[16];
                        tmem_ld16(lane_addr + (uint32_t)(16 * c), v);
                        float pr[16];
#pragma unroll
                        for (int e = 0; e < 16; e += 2) {   // fma then subtract, two columns per instruction
                            const float2 x = __fadd2_rn(
                                __ffma2_rn(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])),
                                           make_float2(kScale2, kScale2),
                                           *reinterpret_cast<const float2 *>(&lsz[128 * kb + 16 * c + e])),
                                make_float2(-mx, -mx));
                            pr[e] = 16 * c + e < rows_k ? ex2(x.x) : 0.0f;
                            pr[e + 1] = 16 * c + e + 1 < rows_k ? ex2(x.y) : 0.0f;
                        }
#pragma unroll
                        for (int e = 0; e < 16; e += 2) {
                            lsum2 = __fadd2_rn(lsum2, make_float2(pr[e], pr[e + 1]));
                            const __nv_bfloat162 b2 = __floats2bfloat162_rn(pr[e], pr[e + 1]);
                            pk[q][e >> 1] = *reinterpret_cast<const uint32_t *>(&b2);
                        }
                    }
                }
            }
            pair_sync(warp);   // every S column of these rows read
            if (rows_here) {
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (c_lo + q < c_hi) tmem_st8(lane_addr + (uint32_t)(8 * (c_lo + q)), pk[q]);
                asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncthreads();
            const bool ok_s = s_fail == 0;
            if (tid == 0 && ok_s) {
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                for (int kk = 0; kk < npadb / 16; ++kk)
                    umma_bf16_ts(tmem + 128u, tmem + 8u * kk, sw128_desc(smem_addr(Vb + buf * kKvBytes) + kk * 2048u),
                                 idesc_o, (kb | kk) ? 1u : 0u);
                umma_commit(smem_addr(&bar_o));
                s_no = s_no + 1;
            }
            if (ok_s && !mbar_wait(smem_addr(&bar_o), (uint32_t)(t * nkv + kb) & 1u)) atomicOr(&s_fail, 4);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            if (kb == nkv - 1) {
                // ---- the tile's epilogue: O / row sum -> bf16 --------------------------------------
                red[half][r] = lsum2.x + lsum2.y;
                __syncthreads();
                const float l = red[0][r] + red[1][r];
                if (rows_here && s_fail == 0) {
                    uint32_t o[32];
                    tmem_ld16(lane_addr + 128u + 32u * half, *reinterpret_cast<uint32_t(*)[16]>(o));
                    tmem_ld16(lane_addr + 144u + 32u * half, *reinterpret_cast<uint32_t(*)[16]>(o + 16));
                    const int m = 128 * t + r;
                    if (m < n) {
                        const float inv = 1.0f / l;
                        uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                                               (size_t)(o0 + m) * H * kAttnDh + (size_t)h * kAttnDh +
                                                               32 * half);
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            uint32_t w[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const float2 y = __fmul2_rn(
                                    make_float2(__uint_as_float(o[8 * c + 2 * e]), __uint_as_float(o[8 * c + 2 * e + 1])),
                                    make_float2(inv, inv));
                                const __nv_bfloat162 b2 = __floats2bfloat162_rn(y.x, y.y);
                                w[e] = *reinterpret_cast<const uint32_t *>(&b2);
                            }
                            dst[c] = make_uint4(w[0], w[1], w[2], w[3]);
                        }
                    }
                }
                mraw = -INFINITY;
                lsum2 = make_float2(0.0f, 0.0f);
            }
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();   // S, P and O read before the next step's products overwrite them
        stop = s_fail != 0;
        __syncthreads();
    }
    if (tid == 0 && s_fail != 0) {   // let everything this CTA started finish before it leaves
        raise_status(p.status, FUSION_DEV_TIMEOUT);
        for (int b = 0; b < 2; ++b) {
            const int last = s_ld - 1 - ((s_ld - 1 - b) & 1);   // the last step issued into buffer b
            if (last >= 0) mbar_wait(smem_addr(&bar_ld[b]), (uint32_t)(last >> 1) & 1u);
        }
        if (s_ns > 0) mbar_wait(smem_addr(&bar_s), (uint32_t)(s_ns - 1) & 1u);
        if (s_no > 0) mbar_wait(smem_addr(&bar_o), (uint32_t)(s_no - 1) & 1u);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kAttnTmemCols) : "memory");
}

}  // namespace

size_t attn_smem_bytes(int max_tokens) {
    if (max_tokens > kAttnMaxN) return 1024u + 2u * kQTileBytes + 4u * kKvBytes;   // two Q tiles, two K and V blocks
    const int npad = (max_tokens + 15) & ~15, T = (max_tokens + 127) >> 7;
    return 1024u + (size_t)T * kQTileBytes + 2u * (size_t)npad * 128u;   // alignment, Q tiles, K, V
}

cudaError_t launch_attention(const AttnParams &p, cudaStream_t s) {
    if (p.in.max_batch == 0 || p.heads == 0) return cudaSuccess;
    EncodeTiledFn enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const size_t smem = attn_smem_bytes(p.in.max_tokens);
    AttnMaps maps;
    for (int b = 0; b < 2; ++b) {
        cuuint64_t dims[2] = {(cuuint64_t)3 * p.heads * kAttnDh, (cuuint64_t)p.in.max_rows};
        cuuint64_t strides[1] = {(cuuint64_t)3 * p.heads * kAttnDh * 2};
        cuuint32_t box[2] = {64, b == 0 ? 32u : 8u};
        cuuint32_t estr[2] = {1, 1};
        if (enc(b == 0 ? &maps.b32 : &maps.b8, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p.qkv), dims,
                strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    auto kern = p.in.max_tokens > kAttnMaxN ? k_attn_tc_long : k_attn_tc;   // whole samples resident, or key blocks
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<dim3((unsigned)p.heads, (unsigned)p.in.max_batch), kAttnThreads, smem, s>>>(maps, p);
    return cudaGetLastError();
}

}  // namespace fz
