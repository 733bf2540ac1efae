// Per-sample merge (Sec. III-C) -> prune (Sec. III-E) -> gather into the
// compacted output batch.  One CTA per input sample; a sample that exited (or is
// beyond the device batch count) returns at once.
//
// Merge decisions.  The keys of half A (even positions) and half B (odd
// positions) are staged in shared memory in a chunk-major layout: the 16-byte
// chunk c of the token with half-index t lives at region + (c * R + t) * 16,
// with R = 1 (mod 8) rows per chunk column, so that ldmatrix row groups and
// row-wise 16-byte reads are bank-conflict free.  When every key dim fits
// (resident), the keys are staged once and, when they are the token rows
// themselves, the gather reads them back from shared memory instead of HBM.
// Otherwise the key dims stream through in chunks, once per pass over the
// output strips.
//
// S = A_hat * B_hat^T is computed strip by strip (16 A rows x 32 B columns per
// warp): bf16 keys on the tensor cores (mma.sync m16n8k16, f32 accumulate),
// f32 keys with FFMA.  Partial sums are flushed into the running sum every 64
// key dims, which keeps the rounding error of long dot products small.  The
// cosine is dot * invnorm_a * invnorm_b; every A row keeps the packed maximum
// (value, lowest B index) through a shared-memory 64-bit atomicMax.
//
// Output.  Each output row is either a copy of its input row or, for a B token
// that received merged A tokens, the size-weighted mean of its sources computed
// in float-float arithmetic and rounded once (bf16: ties to even, from a value
// with about 44 correct bits, so the rounding matches the exact mean).
#include "sample.cuh"

namespace fz {
namespace {

constexpr int kSPW = 2;   // output strips per warp per pass (accumulators live in registers)

__host__ __device__ inline int rows_odd8(int n) {   // smallest R >= n with R % 8 == 1
    if (n < 1) n = 1;
    return n + ((9 - n % 8) % 8);
}

// Staging area: A region (stage_chunks x ra rows) then B region (stage_chunks x rb rows)
// of 16-byte chunks, plus a tail for padded strip rows read past the end.
__host__ __device__ inline size_t stage_a_bytes(int stage_chunks, int ra) { return (size_t)stage_chunks * ra * 16; }
__host__ __device__ inline size_t stage_total(int stage_chunks, int ra, int rb) {
    return (size_t)stage_chunks * (ra + rb) * 16 + 512;
}

// ---------------------------------------------------------------------------
// similarity + row argmax over one sample
// ---------------------------------------------------------------------------
template <typename T>
__device__ void sim_argmax(const ImageParams &p, unsigned char *sm, size_t stage_b, MetaPtrs &m, int start,
                           int nA, int nB) {
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr bool kBf16 = (Elem<T>::kBytes == 2);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, t4 = lane & 3;
    const T *keys = reinterpret_cast<const T *>(p.keys);
    const int kdim = p.kdim;
    unsigned char *regA = sm;
    unsigned char *regB = sm + stage_b;
    float *ssA = m.inv_a;   // squared norms, then inverse norms
    float *ssB = m.inv_b;
    unsigned long long *best = m.best;
    const int ra = p.ra, rb = p.rb;

    const int MT = (nA + 15) / 16, NG = (nB + 31) / 32;
    const int S = MT * NG;
    constexpr int per_pass = kImageWarps * kSPW;
    const int n_pass = (S + per_pass - 1) / per_pass;
    const int kc = p.kc;
    const int n_kchunk = (kdim + kc - 1) / kc;
    bool staged = false;

    for (int pass = 0; pass < n_pass; ++pass) {
        float acc[kSPW][4][4];
#pragma unroll
        for (int a = 0; a < kSPW; ++a)
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][q][e] = 0.0f;

        for (int kci = 0; kci < n_kchunk; ++kci) {
            const int k0 = kci * kc;
            const int kw = min(kc, kdim - k0);
            const int nch = kw / CH;   // 16-byte chunks per staged row
            if (!(p.resident && staged)) {
                __syncthreads();   // previous readers of the staging area are done
                const int total = (nA + nB) * nch;
                for (int it = tid; it < total; it += kImageThreads) {
                    const int tok = it / nch, c = it - tok * nch;
                    long long row;
                    unsigned char *dst;
                    if (tok < nA) {
                        row = start + 2 + 2 * tok;
                        dst = regA + ((size_t)c * ra + tok) * 16;
                    } else {
                        const int n = tok - nA;
                        row = start + 1 + 2 * n;
                        dst = regB + ((size_t)c * rb + n) * 16;
                    }
                    cp_async16(dst, keys + row * kdim + k0 + c * CH);
                }
                cp_async_commit();
                cp_async_wait_all();
                __syncthreads();
                staged = true;
                if (pass == 0) {
                    // squared key norms, accumulated chunk by chunk (one warp per token)
                    for (int tok = warp; tok < nA + nB; tok += kImageWarps) {
                        const bool isA = tok < nA;
                        const int tix = isA ? tok : tok - nA;
                        const unsigned char *base = isA ? regA : regB;
                        const int R = isA ? ra : rb;
                        float sq = 0.0f;
                        for (int c = lane; c < nch; c += 32) {
                            float f[CH];
                            chunk_to_f(*reinterpret_cast<const uint4 *>(base + ((size_t)c * R + tix) * 16), f);
#pragma unroll
                            for (int e = 0; e < CH; ++e) sq = fmaf(f[e], f[e], sq);
                        }
#pragma unroll
                        for (int o = 16; o >= 1; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
                        if (lane == 0) {
                            if (isA) ssA[tix] += sq;
                            else ssB[tix] += sq;
                        }
                    }
                }
            }

            // ---- tile products for this chunk of key dims ---------------------------
#pragma unroll
            for (int sl = 0; sl < kSPW; ++sl) {
                const int s = pass * per_pass + sl * kImageWarps + warp;
                if (s >= S) continue;
                const int mt = s / NG, ng = s - mt * NG;
                float tmp[4][4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int e = 0; e < 4; ++e) tmp[q][e] = 0.0f;
                if constexpr (kBf16) {
                    const uint32_t baseA = smem_addr(regA), baseB = smem_addr(regB);
                    const int arow = mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                    for (int kk = 0; kk < nch / 2; ++kk) {
                        uint32_t af[4];
                        const int achunk = 2 * kk + (lane >> 4);
                        ldsm_x4(baseA + (uint32_t)(((size_t)achunk * ra + arow) * 16), af[0], af[1], af[2], af[3]);
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            const int brow = ng * 32 + (2 * pr + (lane >> 4)) * 8 + (lane & 7);
                            const int bchunk = 2 * kk + ((lane >> 3) & 1);
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4(baseB + (uint32_t)(((size_t)bchunk * rb + brow) * 16), b0, b1, b2, b3);
                            mma_bf16_16816(tmp[2 * pr], af, b0, b1);
                            mma_bf16_16816(tmp[2 * pr + 1], af, b2, b3);
                        }
                        if ((kk & 3) == 3) {
#pragma unroll
                            for (int q = 0; q < 4; ++q)
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    acc[sl][q][e] += tmp[q][e];
                                    tmp[q][e] = 0.0f;
                                }
                        }
                    }
                } else {
                    const int r0 = mt * 16 + g;
                    for (int c = 0; c < nch; ++c) {
                        const float4 a0 = *reinterpret_cast<const float4 *>(regA + ((size_t)c * ra + r0) * 16);
                        const float4 a1 = *reinterpret_cast<const float4 *>(regA + ((size_t)c * ra + r0 + 8) * 16);
#pragma unroll
                        for (int q = 0; q < 4; ++q)
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                const int col = ng * 32 + q * 8 + 2 * t4 + e;
                                const float4 b = *reinterpret_cast<const float4 *>(regB + ((size_t)c * rb + col) * 16);
                                float v0 = tmp[q][e], v1 = tmp[q][2 + e];
                                v0 = fmaf(a0.x, b.x, v0); v0 = fmaf(a0.y, b.y, v0);
                                v0 = fmaf(a0.z, b.z, v0); v0 = fmaf(a0.w, b.w, v0);
                                v1 = fmaf(a1.x, b.x, v1); v1 = fmaf(a1.y, b.y, v1);
                                v1 = fmaf(a1.z, b.z, v1); v1 = fmaf(a1.w, b.w, v1);
                                tmp[q][e] = v0;
                                tmp[q][2 + e] = v1;
                            }
                        if ((c & 3) == 3) {
#pragma unroll
                            for (int q = 0; q < 4; ++q)
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    acc[sl][q][e] += tmp[q][e];
                                    tmp[q][e] = 0.0f;
                                }
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[sl][q][e] += tmp[q][e];
            }
        }

        if (pass == 0) {
            __syncthreads();
            for (int tok = tid; tok < nA + nB; tok += kImageThreads) {
                float *ss = tok < nA ? ssA + tok : ssB + (tok - nA);
                const float v = *ss;
                if (!isfinite(v)) raise_status(p.status, FUSION_DEV_NONFINITE);
                *ss = 1.0f / fmaxf(sqrtf(v), 1e-12f);   // now the inverse norm
            }
            __syncthreads();
        }

        // ---- epilogue: cosine, row maximum with lowest column on ties ---------------
#pragma unroll
        for (int sl = 0; sl < kSPW; ++sl) {
            const int s = pass * per_pass + sl * kImageWarps + warp;
            if (s >= S) continue;
            const int mt = s / NG, ng = s - mt * NG;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const int row = mt * 16 + g + half * 8;
                unsigned long long bk = 0ull;
                if (row < nA) {
                    const float ia = ssA[row];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int col = ng * 32 + q * 8 + 2 * t4 + e;
                            if (col < nB) {
                                const float v = (acc[sl][q][half * 2 + e] * ia) * ssB[col];
                                const unsigned long long k = rank_key(v, col);
                                bk = k > bk ? k : bk;
                            }
                        }
                }
                unsigned long long o1 = __shfl_xor_sync(0xFFFFFFFFu, bk, 1);
                bk = o1 > bk ? o1 : bk;
                unsigned long long o2 = __shfl_xor_sync(0xFFFFFFFFu, bk, 2);
                bk = o2 > bk ? o2 : bk;
                if (t4 == 0 && row < nA) atomicMax(best + row, bk);
            }
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// the per-sample kernel
// ---------------------------------------------------------------------------
// Chunk c of input token pos from the chunk-major staging area (CLS from global).
template <typename T>
struct ChunkMajorLoader {
    const unsigned char *regA, *regB;
    int ra, rb;
    GlobalLoader<T> g;
    __device__ __forceinline__ uint4 operator()(int pos, int c) const {
        if (pos == 0) return g(0, c);
        if (pos & 1) return *reinterpret_cast<const uint4 *>(regB + ((size_t)c * rb + (pos - 1) / 2) * 16);
        return *reinterpret_cast<const uint4 *>(regA + ((size_t)c * ra + (pos - 2) / 2) * 16);
    }
};

template <typename T>
__global__ void __launch_bounds__(kImageThreads, 1) k_image(ImageParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    constexpr int CH = Elem<T>::kPerChunk;
    SampleInfo s;
    if (!sample_begin<kImageThreads>(p, blockIdx.x, s)) return;
    const int tid = threadIdx.x;
    const int stage_chunks = p.resident ? p.kdim / CH : p.kc / CH;
    const size_t stage_b = p.do_merge ? stage_a_bytes(stage_chunks, p.ra) : 0;
    const size_t stage = p.do_merge ? stage_total(stage_chunks, p.ra, p.rb) : 0;
    MetaPtrs m(sm, meta_layout(p.in.max_tokens, stage));
    meta_init<kImageThreads>(p, s, m);
    for (int a = tid; a < s.nA; a += kImageThreads) m.inv_a[a] = 0.0f;
    for (int n = tid; n < s.nB; n += kImageThreads) m.inv_b[n] = 0.0f;
    __syncthreads();

    // merge decisions: pair every A token with its best B token, keep the r best
    if (s.decide) {
        sim_argmax<T>(p, sm, stage_b, m, s.start, s.nA, s.nB);
        select_top_r<kImageThreads>(s, m);
    }
    const GlobalLoader<T> gl{reinterpret_cast<const T *>(p.x), (long long)s.start, p.dim};
    if (s.decide && p.resident && p.keys_alias) {
        const ChunkMajorLoader<T> ld{sm, sm + stage_b, p.ra, p.rb, gl};
        finish_sample<T, kImageThreads>(p, s, m, ld);
    } else {
        finish_sample<T, kImageThreads>(p, s, m, gl);
    }
}

}  // namespace

ImageGeometry image_geometry(int dtype, int max_tokens, int kdim, int do_merge) {
    ImageGeometry G{};
    const int eb = dtype == FUSION_BF16 ? 2 : 4;
    const int CH = 16 / eb;
    const int nA = (max_tokens - 1) / 2, nB = max_tokens / 2;
    G.ra = rows_odd8(nA);
    G.rb = rows_odd8(nB);
    constexpr size_t kBudget = 227 * 1024 - 2048;   // leave room for static shared memory
    const size_t meta = meta_layout(max_tokens, 0).total;
    if (!do_merge) {
        G.ok = meta <= kBudget;
        G.smem = meta;
        return G;
    }
    const size_t full = meta_layout(max_tokens, stage_total(kdim / CH, G.ra, G.rb)).total;
    if (full <= kBudget) {
        G.ok = 1;
        G.resident = 1;
        G.kc = kdim;
        G.smem = full;
        return G;
    }
    const size_t per_dim = (size_t)(G.ra + G.rb) * eb;   // staged bytes per key dim
    if (meta + 1024 >= kBudget) return G;
    int kc = (int)((kBudget - meta - 1024) / per_dim) / 16 * 16;
    if (kc > kdim) kc = kdim;
    if (kc < 16) return G;
    G.ok = 1;
    G.resident = 0;
    G.kc = kc;
    G.smem = meta_layout(max_tokens, stage_total(kc / CH, G.ra, G.rb)).total;
    return G;
}

cudaError_t launch_image(int dtype, const ImageParams &p, size_t smem, cudaStream_t s) {
    if (p.in.max_batch == 0) return cudaSuccess;
    const dim3 grid(p.in.max_batch);
    if (dtype == FUSION_BF16) {
        cudaError_t e = cudaFuncSetAttribute(k_image<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_image<__nv_bfloat16><<<grid, kImageThreads, smem, s>>>(p);
    } else {
        cudaError_t e = cudaFuncSetAttribute(k_image<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_image<float><<<grid, kImageThreads, smem, s>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace fz
