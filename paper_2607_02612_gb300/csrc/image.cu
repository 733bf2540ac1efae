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
#include "launch.h"

namespace fz {
namespace {

constexpr int kSPW = 2;   // output strips per warp per pass (accumulators live in registers)

struct ImgLayout {
    size_t stage_a, stage_b;
    size_t best, ss_a, ss_b, match, sel, mflag, kflag, opos, srcpos, scnt, slist, msize, mscore, tmp;
    size_t total;
};

__host__ __device__ inline ImgLayout img_layout(int nmax, int ra, int rb, int stage_chunks, int stage) {
    const int nA = (nmax - 1) / 2 > 0 ? (nmax - 1) / 2 : 1;
    const int nB = nmax / 2 > 0 ? nmax / 2 : 1;
    ImgLayout L;
    size_t off = 0;
    L.stage_a = off;
    if (stage) off += (size_t)stage_chunks * ra * 16;
    L.stage_b = off;
    if (stage) off += (size_t)stage_chunks * rb * 16 + 512;   // tail: padded strip rows read past the end
    off = (off + 15) / 16 * 16;
    L.best = off;   off += sizeof(unsigned long long) * nA;
    L.ss_a = off;   off += sizeof(float) * nA;
    L.ss_b = off;   off += sizeof(float) * nB;
    L.match = off;  off += sizeof(int) * nA;
    L.sel = off;    off += sizeof(int) * nA;
    L.mflag = off;  off += sizeof(int) * nmax;
    L.kflag = off;  off += sizeof(int) * nmax;
    L.opos = off;   off += sizeof(int) * (nmax + 1);
    L.srcpos = off; off += sizeof(int) * nmax;
    L.scnt = off;   off += sizeof(int) * (nB + 1);
    L.slist = off;  off += sizeof(int) * nA;
    L.msize = off;  off += sizeof(float) * nmax;
    L.mscore = off; off += sizeof(float) * nmax;
    L.tmp = off;    off += sizeof(int) * 40;
    L.total = (off + 15) / 16 * 16;
    return L;
}

__host__ __device__ inline int rows_odd8(int n) {   // smallest R >= n with R % 8 == 1
    if (n < 1) n = 1;
    return n + ((9 - n % 8) % 8);
}

// ---------------------------------------------------------------------------
// similarity + row argmax over one sample
// ---------------------------------------------------------------------------
template <typename T>
__device__ void sim_argmax(const ImageParams &p, unsigned char *sm, const ImgLayout &L, int start,
                           int nA, int nB) {
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr bool kBf16 = (Elem<T>::kBytes == 2);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, t4 = lane & 3;
    const T *keys = reinterpret_cast<const T *>(p.keys);
    const int kdim = p.kdim;
    unsigned char *regA = sm + L.stage_a;
    unsigned char *regB = sm + L.stage_b;
    float *ssA = reinterpret_cast<float *>(sm + L.ss_a);
    float *ssB = reinterpret_cast<float *>(sm + L.ss_b);
    unsigned long long *best = reinterpret_cast<unsigned long long *>(sm + L.best);
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
template <typename T>
__device__ __forceinline__ uint4 load_src_chunk(const ImageParams &p, const unsigned char *sm,
                                                const ImgLayout &L, bool from_smem, int start, int pos,
                                                int c) {
    constexpr int CH = Elem<T>::kPerChunk;
    if (from_smem && pos > 0) {
        if (pos & 1) return *reinterpret_cast<const uint4 *>(sm + L.stage_b + ((size_t)c * p.rb + (pos - 1) / 2) * 16);
        return *reinterpret_cast<const uint4 *>(sm + L.stage_a + ((size_t)c * p.ra + (pos - 2) / 2) * 16);
    }
    return ldg16(reinterpret_cast<const T *>(p.x) + ((long long)start + pos) * p.dim + c * CH);
}

__device__ __forceinline__ uint4 pack_chunk(const F2 (&q)[4]) {
    return make_uint4(__float_as_uint(q[0].hi), __float_as_uint(q[1].hi), __float_as_uint(q[2].hi),
                      __float_as_uint(q[3].hi));
}
__device__ __forceinline__ uint4 pack_chunk(const F2 (&q)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
        w[k] = (uint32_t)f2_to_bf16_bits(q[2 * k]) | ((uint32_t)f2_to_bf16_bits(q[2 * k + 1]) << 16);
    return make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename T>
__global__ void __launch_bounds__(kImageThreads, 1) k_image(ImageParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    constexpr int CH = Elem<T>::kPerChunk;
    const int tid = threadIdx.x;
    const int i = blockIdx.x;
    const int B = device_batch(p.in);
    if (B < 0 || i >= B) return;
    if (p.plan[0] == 0) return;
    const int j = p.slot[i];
    if (j < 0) return;

    const int start = p.in.offsets[i];
    const int N = p.in.offsets[i + 1] - start;
    const int out_start = p.offsets_out[j];
    const int out_n = p.offsets_out[j + 1] - out_start;
    const int id = p.in.ids ? p.in.ids[i] : i;
    const int P = N - 1, nA = P / 2, nB = (P + 1) / 2;
    const int r_eff = p.do_merge ? merge_count(p.r[id], P) : 0;
    const bool decide = p.do_merge && nA > 0 && (r_eff > 0 || p.need_match);

    const int stage_chunks = p.resident ? p.kdim / CH : p.kc / CH;
    const ImgLayout L = img_layout(p.in.max_tokens, p.ra, p.rb, stage_chunks, p.do_merge);
    unsigned long long *best = reinterpret_cast<unsigned long long *>(sm + L.best);
    float *ssA = reinterpret_cast<float *>(sm + L.ss_a);
    float *ssB = reinterpret_cast<float *>(sm + L.ss_b);
    int *match = reinterpret_cast<int *>(sm + L.match);
    int *sel = reinterpret_cast<int *>(sm + L.sel);
    int *mflag = reinterpret_cast<int *>(sm + L.mflag);
    int *kflag = reinterpret_cast<int *>(sm + L.kflag);
    int *opos = reinterpret_cast<int *>(sm + L.opos);
    int *srcpos = reinterpret_cast<int *>(sm + L.srcpos);
    int *scnt = reinterpret_cast<int *>(sm + L.scnt);
    int *slist = reinterpret_cast<int *>(sm + L.slist);
    float *msize = reinterpret_cast<float *>(sm + L.msize);
    float *mscore = reinterpret_cast<float *>(sm + L.mscore);
    int *tmp = reinterpret_cast<int *>(sm + L.tmp);

    for (int m = tid; m < nA; m += kImageThreads) {
        best[m] = 0ull;
        ssA[m] = 0.0f;
        sel[m] = 0;
        match[m] = 0;
    }
    for (int n = tid; n <= nB; n += kImageThreads) {
        if (n < nB) ssB[n] = 0.0f;
        scnt[n] = 0;
    }
    __syncthreads();

    // ---- merge decisions: pair every A token with its best B token, keep the r best
    if (decide) {
        sim_argmax<T>(p, sm, L, start, nA, nB);
        for (int m = tid; m < nA; m += kImageThreads)
            match[m] = (int)(0xFFFFFFFFu - (uint32_t)(best[m] & 0xFFFFFFFFull));
        if (r_eff > 0) {
            for (int m = tid; m < nA; m += kImageThreads) {
                const unsigned long long km = (best[m] & 0xFFFFFFFF00000000ull) | (0xFFFFFFFFull - (unsigned)m);
                int rank = 0;
                for (int q = 0; q < nA; ++q) {
                    const unsigned long long kq = (best[q] & 0xFFFFFFFF00000000ull) | (0xFFFFFFFFull - (unsigned)q);
                    rank += (kq > km) ? 1 : 0;
                }
                sel[m] = rank < r_eff ? 1 : 0;
            }
        }
        __syncthreads();
    }

    // ---- merged token set: survivors keep ascending position ------------------------
    for (int pos = tid; pos < N; pos += kImageThreads)
        mflag[pos] = (pos >= 2 && !(pos & 1) && sel[(pos - 2) / 2]) ? 0 : 1;
    if (r_eff > 0)
        for (int m = tid; m < nA; m += kImageThreads)
            if (sel[m]) atomicAdd(&scnt[match[m]], 1);
    __syncthreads();
    block_scan_excl(scnt, nB + 1, tmp);   // scnt[n] = first slot of B token n's sources
    if (r_eff > 0) {
        for (int m = tid; m < nA; m += kImageThreads) {
            if (!sel[m]) continue;
            const int n = match[m];
            int before = 0;
            for (int q = 0; q < m; ++q) before += (sel[q] && match[q] == n) ? 1 : 0;
            slist[scnt[n] + before] = m;   // sources of every B token in ascending A order
        }
    }
    __syncthreads();

    // merged sizes and scores (sums over the sources, exact in double)
    for (int pos = tid; pos < N; pos += kImageThreads) {
        if (!mflag[pos]) continue;
        double sz = p.sizes[start + pos];
        double sc = p.scores ? (double)p.scores[start + pos] : 0.0;
        if (pos & 1) {
            const int n = (pos - 1) / 2;
            for (int q = scnt[n]; q < scnt[n + 1]; ++q) {
                const int a = start + 2 + 2 * slist[q];
                sz += p.sizes[a];
                if (p.scores) sc += (double)p.scores[a];
            }
        }
        msize[pos] = (float)sz;
        mscore[pos] = (float)sc;
        if (p.scores && !isfinite(mscore[pos]) && pos > 0) raise_status(p.status, FUSION_DEV_NONFINITE);
    }
    __syncthreads();

    // ---- prune: CLS + the k highest merged scores, lowest position on ties -----------
    if (p.do_prune) {
        bool nf = false;
        const int k = keep_count(p.rho[id], N - r_eff - 1, nf);
        for (int pos = tid; pos < N; pos += kImageThreads) {
            int keep = 0;
            if (pos == 0) {
                keep = 1;
            } else if (mflag[pos]) {
                const unsigned long long kp = rank_key(mscore[pos], pos);
                int rank = 0;
                for (int q = 1; q < N; ++q)
                    rank += (mflag[q] && rank_key(mscore[q], q) > kp) ? 1 : 0;
                keep = rank < k ? 1 : 0;
            }
            kflag[pos] = keep;
            opos[pos] = keep;
        }
    } else {
        for (int pos = tid; pos < N; pos += kImageThreads) {
            kflag[pos] = mflag[pos];
            opos[pos] = mflag[pos];
        }
    }
    __syncthreads();
    const int total = block_scan_excl(opos, N, tmp);
    if (total != out_n) {   // the plan and the decisions disagree: a library bug
        if (tid == 0) raise_status(p.status, FUSION_DEV_INTERNAL);
        return;
    }
    for (int pos = tid; pos < N; pos += kImageThreads)
        if (kflag[pos]) srcpos[opos[pos]] = pos;
    __syncthreads();

    // ---- index outputs ----------------------------------------------------------------
    for (int o = tid; o < out_n; o += kImageThreads) {
        const int pos = srcpos[o];
        const long long orow = (long long)out_start + o;
        p.sizes_out[orow] = msize[pos];
        if (p.scores_out) p.scores_out[orow] = mscore[pos];
        if (p.keep_idx) p.keep_idx[orow] = start + pos;
    }
    if (p.a_match)
        for (int pos = tid; pos < N; pos += kImageThreads)
            p.a_match[start + pos] = (pos >= 2 && !(pos & 1)) ? start + 1 + 2 * match[(pos - 2) / 2] : -1;
    if (p.dst_map && !p.do_prune)
        for (int pos = tid; pos < N; pos += kImageThreads) {
            const bool gone = pos >= 2 && !(pos & 1) && sel[(pos - 2) / 2];
            const int dest = gone ? 1 + 2 * match[(pos - 2) / 2] : pos;
            p.dst_map[start + pos] = out_start + opos[dest];
        }

    // ---- token rows: copies and size-weighted means, 16 bytes per thread --------------
    const int ncx = p.dim / CH;
    const bool from_smem = decide && p.resident && p.keys_alias;
    T *xo = reinterpret_cast<T *>(p.x_out);
    for (int it = tid; it < out_n * ncx; it += kImageThreads) {
        const int o = it / ncx, c = it - o * ncx;
        const int pos = srcpos[o];
        const uint4 self = load_src_chunk<T>(p, sm, L, from_smem, start, pos, c);
        uint4 outv = self;
        if (pos & 1) {
            const int n = (pos - 1) / 2;
            const int q0 = scnt[n], q1 = scnt[n + 1];
            if (q1 > q0) {
                float f[CH];
                chunk_to_f(self, f);
                const float sb = p.sizes[start + pos];
                F2 den = {sb, 0.0f};
                F2 num[CH];
#pragma unroll
                for (int e = 0; e < CH; ++e) num[e] = two_prod(sb, f[e]);
                for (int q = q0; q < q1; ++q) {
                    const int apos = 2 + 2 * slist[q];
                    const float sa = p.sizes[start + apos];
                    den = f2_add_f(den, sa);
                    chunk_to_f(load_src_chunk<T>(p, sm, L, from_smem, start, apos, c), f);
#pragma unroll
                    for (int e = 0; e < CH; ++e) num[e] = f2_add(num[e], two_prod(sa, f[e]));
                }
                F2 qv[CH];
#pragma unroll
                for (int e = 0; e < CH; ++e) qv[e] = f2_div(num[e], den);
                outv = pack_chunk(qv);
            }
        }
        *reinterpret_cast<uint4 *>(xo + ((long long)out_start + o) * p.dim + c * CH) = outv;
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
    const size_t meta = img_layout(max_tokens, G.ra, G.rb, 0, 0).total;
    if (!do_merge) {
        G.ok = meta <= kBudget;
        G.smem = meta;
        return G;
    }
    const size_t per_dim = (size_t)(G.ra + G.rb) * eb;   // staged bytes per key dim
    const size_t full = img_layout(max_tokens, G.ra, G.rb, kdim / CH, 1).total;
    if (full <= kBudget) {
        G.ok = 1;
        G.resident = 1;
        G.kc = kdim;
        G.smem = full;
        return G;
    }
    if (meta + 1024 >= kBudget) return G;
    int kc = (int)((kBudget - meta - 1024) / per_dim) / 16 * 16;
    if (kc > kdim) kc = kdim;
    if (kc < 16) return G;
    G.ok = 1;
    G.resident = 0;
    G.kc = kc;
    G.smem = img_layout(max_tokens, G.ra, G.rb, kc / CH, 1).total;
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
