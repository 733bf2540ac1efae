// Size-aware attention over a ragged batch: the transformer block that consumes a compacted
// batch (Algorithm 1, Block_b), with the proportional attention of ToMe so that a merged
// token of size s weighs like the s tokens it replaced.  For every sample, head h and query
// row m of the sample:
//   out[m, h] = sum_j softmax_j(q_m . k_j / sqrt(dh) + log s_j) v_j.
//
// One CTA of 256 threads per (head, sample); samples of at most 256 tokens, dh = 64, bf16.
// TMA brings the sample's query tiles of 128 rows, its K rows and its V rows (one 128-byte
// row of 64 dims each, 128-byte swizzle) from the packed qkv matrix.  Q and K are K-major
// operands; V, rows of keys with the dims contiguous, is the MN-major B operand of the second
// product as it lies (8-key swizzle atoms 1024 bytes apart); its rows past the sample are
// zeroed once it has landed.  Per query tile t: S_t = Q_t K^T (M = 128, N = tokens
// rounded up to 16, K = 64) accumulates in tensor-memory columns [256 t, 256 t + N); warps
// 4t..4t+3 then take one row each per thread: logits scaled by log2(e) / sqrt(dh) plus
// log2(s_j), masked past the sample, the row maximum, exp2 (ex2.approx), the row sum, and the unnormalised
// probabilities P_t as bf16 into shared memory (swizzled K-major again, over the dead Q and K
// tiles).  O_t = P_t V (M = 128, N = 64, K = tokens rounded up to 16) accumulates over the first
// 64 columns of S_t's region; the epilogue divides each row by its sum and stores bf16.  P is
// rounded to bf16 (the operand type of the second product); the sum is taken before that.
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

__device__ __forceinline__ float ex2(float x) {   // 2^x, one MUFU instruction (2^-inf = 0)
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

struct AttnMaps {
    CUtensorMap b32, b8;   // qkv rows, boxes of 64 dims x 32 / 8 rows, 128-byte swizzle
};

__global__ void __launch_bounds__(kAttnThreads, 1)
    k_attn_tc(const __grid_constant__ AttnMaps maps, AttnParams p) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) unsigned long long bar_ld, bar_s, bar_o;
    __shared__ uint32_t tmem_base;
    __shared__ int s_fail, s_issued;   // s_issued: 1 = the products S were issued, 2 = also O
    __shared__ float lsz[kAttnMaxN];   // log2 of the key sizes

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
    const int nkb = (npad + 63) >> 6;             // K-blocks of 64 keys in P and V^T
    unsigned char *U = sm;                        // Q tiles and K, later the P tiles
    unsigned char *Kr = U + (size_t)T * kQTileBytes;
    unsigned char *Vr = sm + p.u_bytes;           // V rows (MN-major B operand)

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(p.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid == 0) {
        s_fail = 0;
        s_issued = 0;
        mbar_init(smem_addr(&bar_ld), 1);
        mbar_init(smem_addr(&bar_s), 1);
        mbar_init(smem_addr(&bar_o), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();

    // ---- loads: K rows and the query tiles by TMA (rows rounded up to 8) --------------------
    if (tid == 0) {
        const int rk = (n + 7) & ~7;
        uint32_t bytes = 2u * (uint32_t)rk * 128u;
        for (int t = 0; t < T; ++t) bytes += (uint32_t)((min(128, n - 128 * t) + 7) & ~7) * 128u;
        mbar_expect_tx(smem_addr(&bar_ld), bytes);
        auto rows = [&](unsigned char *dst, int x, int y0, int cnt) {   // cnt is a multiple of 8
            int r = 0;
            for (; r + 32 <= cnt; r += 32) tma_load_2d(smem_addr(dst + r * 128), &maps.b32, x, y0 + r, smem_addr(&bar_ld));
            for (; r < cnt; r += 8) tma_load_2d(smem_addr(dst + r * 128), &maps.b8, x, y0 + r, smem_addr(&bar_ld));
        };
        rows(Kr, (H + h) * kAttnDh, o0, rk);
        rows(Vr, (2 * H + h) * kAttnDh, o0, rk);
        for (int t = 0; t < T; ++t) rows(U + (size_t)t * kQTileBytes, h * kAttnDh, o0 + 128 * t, (min(128, n - 128 * t) + 7) & ~7);
    }
    // ---- key log-sizes; once V has landed, its rows past the sample are zeroed ----------------
    for (int j = tid; j < npad; j += kAttnThreads)
        lsz[j] = j < n ? (p.sizes ? log2f(p.sizes[o0 + j]) : 0.0f) : 0.0f;
    __syncthreads();
    const uint32_t tmem = tmem_base;

    // ---- S_t = Q_t K^T ----------------------------------------------------------------------
    if (tid == 0) {
        if (mbar_wait(smem_addr(&bar_ld), 0)) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(npad >> 3) << 17) | (8u << 24);
            for (int t = 0; t < T; ++t)
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem + 256u * t, sw128_desc(smem_addr(U + (size_t)t * kQTileBytes) + k * 32),
                              sw128_desc(smem_addr(Kr) + k * 32), idesc, k ? 1u : 0u);
            umma_commit(smem_addr(&bar_s));
            s_issued = 1;
        } else {
            s_fail = 1;
        }
    }
    __syncthreads();
    // V rows n .. npad-1 (another sample's rows or stale memory) read as zero in P V
    if (s_fail == 0 && npad > n) {
        for (int c = tid; c < (npad - n) * 8; c += kAttnThreads)
            reinterpret_cast<uint4 *>(Vr + (size_t)n * 128)[c] = make_uint4(0u, 0u, 0u, 0u);
    }
    if (s_fail == 0 && !mbar_wait(smem_addr(&bar_s), 0)) atomicOr(&s_fail, 2);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    __syncthreads();

    // ---- softmax rows: warps 4t .. 4t + 3 take tile t, one row per thread --------------------
    const int t = warp >> 2;
    const int r = tid & 127;   // row of the tile = tensor-memory lane
    const int m = 128 * t + r; // query row of the sample
    const uint32_t lane_addr = tmem + 256u * t + ((uint32_t)((warp & 3) * 32) << 16);
    constexpr float kScale2 = 0.18033688011112042f;   // log2(e) / sqrt(64)
    float lsum = 0.0f;
    if (s_fail == 0 && t < T) {   // warp-uniform: every lane takes part in the tensor-memory loads
        float mx = -INFINITY;
        for (int c0 = 0; c0 < npad; c0 += 16) {
            uint32_t v[16];
            tmem_ld16(lane_addr + (uint32_t)c0, v);
            if (c0 + 16 <= n) {
#pragma unroll
                for (int e = 0; e < 16; ++e) mx = fmaxf(mx, fmaf(__uint_as_float(v[e]), kScale2, lsz[c0 + e]));
            } else {
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (c0 + e < n) mx = fmaxf(mx, fmaf(__uint_as_float(v[e]), kScale2, lsz[c0 + e]));
            }
        }
        unsigned char *P = U + (size_t)t * nkb * kQTileBytes;
        for (int c0 = 0; c0 < npad; c0 += 16) {
            uint32_t v[16];
            tmem_ld16(lane_addr + (uint32_t)c0, v);
            float pr[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) pr[e] = ex2(fmaf(__uint_as_float(v[e]), kScale2, lsz[c0 + e]) - mx);
            if (c0 + 16 > n) {
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (c0 + e >= n) pr[e] = 0.0f;
            }
            uint32_t pk[8];
#pragma unroll
            for (int e = 0; e < 16; e += 2) {
                lsum += pr[e] + pr[e + 1];
                const __nv_bfloat162 b2 = __floats2bfloat162_rn(pr[e], pr[e + 1]);
                pk[e >> 1] = *reinterpret_cast<const uint32_t *>(&b2);
            }
            unsigned char *blk = P + (size_t)(c0 >> 6) * kQTileBytes + r * 128;
            const int cc = (c0 & 63) >> 3;
            *reinterpret_cast<uint4 *>(blk + ((cc ^ (r & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            *reinterpret_cast<uint4 *>(blk + (((cc + 1) ^ (r & 7)) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // P visible to the tensor core
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();

    // ---- O_t = P_t V over the first 64 columns of S_t ------------------------------------------
    if (tid == 0 && s_fail == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // B = V as it lies: MN-major (bit 16), 8-key swizzle atoms 1024 bytes apart
        const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(kAttnDh >> 3) << 17) |
                               (8u << 24);
        for (int tt = 0; tt < T; ++tt) {
            const uint32_t pa = smem_addr(U + (size_t)tt * nkb * kQTileBytes);
            for (int kk = 0; kk < npad / 16; ++kk)
                umma_bf16(tmem + 256u * tt, sw128_desc(pa + (kk >> 2) * kQTileBytes + (kk & 3) * 32),
                          sw128_desc(smem_addr(Vr) + kk * 2048u), idesc, kk ? 1u : 0u);
        }
        umma_commit(smem_addr(&bar_o));
        s_issued = 2;
    }
    __syncthreads();
    if (s_fail == 0 && !mbar_wait(smem_addr(&bar_o), 0)) atomicOr(&s_fail, 4);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    __syncthreads();

    // ---- epilogue: O / row sum -> bf16 --------------------------------------------------------
    if (s_fail == 0 && t < T) {
        uint32_t o[64];
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 16) tmem_ld16(lane_addr + (uint32_t)c0, *reinterpret_cast<uint32_t(*)[16]>(o + c0));
        if (m < n) {
            const float inv = 1.0f / lsum;
            uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                                   (size_t)(o0 + m) * H * kAttnDh + (size_t)h * kAttnDh);
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(o[8 * c + 2 * e]) * inv,
                                                                    __uint_as_float(o[8 * c + 2 * e + 1]) * inv);
                    w[e] = *reinterpret_cast<const uint32_t *>(&b2);
                }
                dst[c] = make_uint4(w[0], w[1], w[2], w[3]);
            }
        }
    }
    if (tid == 0 && s_fail != 0) {   // let everything this CTA started finish before it leaves
        raise_status(p.status, FUSION_DEV_TIMEOUT);
        mbar_wait(smem_addr(&bar_ld), 0);
        if (s_issued >= 1) mbar_wait(smem_addr(&bar_s), 0);
        if (s_issued >= 2) mbar_wait(smem_addr(&bar_o), 0);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
}

}  // namespace

AttnGeometry attn_geometry(int max_tokens) {
    AttnGeometry g{};
    const int npad = (max_tokens + 15) & ~15, T = (max_tokens + 127) >> 7, nkb = (npad + 63) >> 6;
    const uint32_t qk = (uint32_t)T * kQTileBytes + (uint32_t)npad * 128u;
    const uint32_t pt = (uint32_t)T * (uint32_t)nkb * kQTileBytes;
    g.u_bytes = ((qk > pt ? qk : pt) + 1023u) & ~1023u;
    g.smem = 1024u + g.u_bytes + (uint32_t)npad * 128u;
    g.tmem_cols = 256u * (uint32_t)T;
    return g;
}

cudaError_t launch_attention(const AttnParams &p, cudaStream_t s) {
    if (p.in.max_batch == 0 || p.heads == 0) return cudaSuccess;
    EncodeTiledFn enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const AttnGeometry g = attn_geometry(p.in.max_tokens);
    AttnParams q = p;
    q.u_bytes = g.u_bytes;
    q.tmem_cols = g.tmem_cols;
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
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem);
    if (e != cudaSuccess) return e;
    k_attn_tc<<<dim3((unsigned)p.heads, (unsigned)p.in.max_batch), kAttnThreads, g.smem, s>>>(maps, q);
    return cudaGetLastError();
}

}  // namespace fz
