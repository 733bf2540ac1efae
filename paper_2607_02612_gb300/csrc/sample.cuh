// Per-sample work shared by the two per-sample kernels (image.cu: mma.sync / FFMA
// decisions; image_tc.cu: TMA + tcgen05 decisions): the sample's bookkeeping, the
// top-r selection from the row maxima (Sec. III-C), the merged token set with its
// size-weighted means, pruning (Sec. III-E) and the gather into the compacted output.
#pragma once

#include "launch.h"

namespace fz {

// ---------------------------------------------------------------------------
// metadata in shared memory, after the kernel's staging area
// ---------------------------------------------------------------------------
struct Meta {
    size_t best, rk, pk, inv_a, inv_b, match, sel, mflag, kflag, opos, srcpos, scnt, slist, msize, mscore, invd,
        tsize, tscore, tmp, total;
};

__host__ __device__ inline Meta meta_layout(int nmax, size_t base) {
    const int nA = (nmax - 1) / 2 > 0 ? (nmax - 1) / 2 : 1;
    const int nB = nmax / 2 > 0 ? nmax / 2 : 1;
    Meta L;
    size_t off = (base + 15) / 16 * 16;
    L.best = off;   off += sizeof(unsigned long long) * nA;
    L.rk = off;     off += sizeof(unsigned long long) * nA;
    L.pk = off;     off += sizeof(unsigned long long) * nmax;
    L.inv_a = off;  off += sizeof(float) * nA;
    L.inv_b = off;  off += sizeof(float) * nB;
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
    off = (off + 7) / 8 * 8;
    L.invd = off;   off += sizeof(float2) * nmax;
    L.tsize = off;  off += sizeof(float) * nmax;
    L.tscore = off; off += sizeof(float) * nmax;
    L.tmp = off;    off += sizeof(int) * 40;
    L.total = (off + 15) / 16 * 16;
    return L;
}

struct MetaPtrs {
    unsigned long long *best, *rk, *pk;
    float *inv_a, *inv_b;
    int *match, *sel, *mflag, *kflag, *opos, *srcpos, *scnt, *slist;
    float *msize, *mscore;
    float2 *invd;
    float *tsize, *tscore;
    int *tmp;
    __device__ MetaPtrs(unsigned char *sm, const Meta &L)
        : best(reinterpret_cast<unsigned long long *>(sm + L.best)),
          rk(reinterpret_cast<unsigned long long *>(sm + L.rk)),
          pk(reinterpret_cast<unsigned long long *>(sm + L.pk)),
          inv_a(reinterpret_cast<float *>(sm + L.inv_a)),
          inv_b(reinterpret_cast<float *>(sm + L.inv_b)),
          match(reinterpret_cast<int *>(sm + L.match)),
          sel(reinterpret_cast<int *>(sm + L.sel)),
          mflag(reinterpret_cast<int *>(sm + L.mflag)),
          kflag(reinterpret_cast<int *>(sm + L.kflag)),
          opos(reinterpret_cast<int *>(sm + L.opos)),
          srcpos(reinterpret_cast<int *>(sm + L.srcpos)),
          scnt(reinterpret_cast<int *>(sm + L.scnt)),
          slist(reinterpret_cast<int *>(sm + L.slist)),
          msize(reinterpret_cast<float *>(sm + L.msize)),
          mscore(reinterpret_cast<float *>(sm + L.mscore)),
          invd(reinterpret_cast<float2 *>(sm + L.invd)),
          tsize(reinterpret_cast<float *>(sm + L.tsize)),
          tscore(reinterpret_cast<float *>(sm + L.tscore)),
          tmp(reinterpret_cast<int *>(sm + L.tmp)) {}
};

struct SampleInfo {
    int start, N, out_start, out_n, id, P, nA, nB, r_eff;
    bool decide;   // the merge decisions are needed (something merges, or matches are requested)
};

// The input sample this CTA handles; false when there is nothing to do (beyond the
// device batch count, an invalid call, or a sample that exited).
__device__ __forceinline__ bool sample_info(const ImageParams &p, int i, SampleInfo &s) {
    const int B = device_batch(p.in);
    if (B < 0 || i >= B) return false;
    if (p.plan[0] == 0) return false;
    const int j = p.slot[i];
    if (j < 0) return false;
    s.start = p.in.offsets[i];
    s.N = p.in.offsets[i + 1] - s.start;
    s.out_start = p.offsets_out[j];
    s.out_n = p.offsets_out[j + 1] - s.out_start;
    s.id = p.in.ids ? p.in.ids[i] : i;
    s.P = s.N - 1;
    s.nA = s.P / 2;
    s.nB = (s.P + 1) / 2;
    s.r_eff = p.do_merge ? merge_count(p.r[s.id], s.P) : 0;
    s.decide = p.do_merge && s.nA > 0 && (s.r_eff > 0 || p.need_match);
    return true;
}

template <int NT>
__device__ __forceinline__ void meta_init(const ImageParams &p, const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    for (int a = tid; a < s.nA; a += NT) {
        m.best[a] = 0ull;
        m.sel[a] = 0;
        m.match[a] = 0;
    }
    for (int n = tid; n <= s.nB; n += NT) m.scnt[n] = 0;
    for (int pos = tid; pos < s.N; pos += NT) {
        m.tsize[pos] = p.sizes[s.start + pos];
        m.tscore[pos] = p.scores ? p.scores[s.start + pos] : 0.0f;
    }
}

// best[a] holds the packed (similarity, lowest B index) maximum of every A row.  Writes
// match[a] and, when tokens merge, sel[a] for the r_eff A tokens of largest similarity
// (lowest position on ties).  Ends with a barrier.
template <int NT>
__device__ __forceinline__ void select_top_r(const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    for (int a = tid; a < s.nA; a += NT) m.match[a] = (int)(0xFFFFFFFFu - (uint32_t)(m.best[a] & 0xFFFFFFFFull));
    if (s.r_eff > 0) {
        for (int a = tid; a < s.nA; a += NT)
            m.rk[a] = (m.best[a] & 0xFFFFFFFF00000000ull) | (0xFFFFFFFFull - (unsigned)a);
        __syncthreads();
        for (int a = tid; a < s.nA; a += NT) {
            const unsigned long long ka = m.rk[a];
            int rank = 0;
#pragma unroll 8
            for (int q = 0; q < s.nA; ++q) rank += m.rk[q] > ka ? 1 : 0;
            m.sel[a] = rank < s.r_eff ? 1 : 0;
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// exact rounding of the size-weighted mean
// ---------------------------------------------------------------------------
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

// num / den for the merged mean, as a float-float value whose rounding to the
// output type is the rounding of the exact quotient.
//   bf16: num * (1/den) in float-float (exact when den is a power of two).  Otherwise,
//   when the product lies within a few float32 ulps of a bf16 rounding midpoint m, the
//   side of m is decided exactly from the sign of num - m * den (an exact tie stays a
//   tie, so it rounds to even).
//   f32: the float-float division.
__device__ __forceinline__ F2 mean_of(F2 num, F2 den, F2 inv, __nv_bfloat16) {
    const F2 q = f2_mul(num, inv);
    const uint32_t bits = __float_as_uint(q.hi);
    const uint32_t low = bits & 0xFFFFu;
    const uint32_t dist = low > 0x8000u ? low - 0x8000u : 0x8000u - low;
    const bool pow2 = den.lo == 0.0f && (__float_as_uint(den.hi) & 0x007FFFFFu) == 0u;
    if (pow2 || dist > 8u) return q;
    const float mid = __uint_as_float((bits & 0xFFFF0000u) | 0x8000u);
    const F2 md = f2_mul({mid, 0.0f}, den);
    const F2 r = f2_add(num, {-md.hi, -md.lo});
    const float side = r.hi != 0.0f ? r.hi : r.lo;   // sign of (q - mid) * den
    const float tiny = copysignf(1e-30f, side);
    return side == 0.0f ? F2{mid, 0.0f} : F2{mid, tiny};
}
__device__ __forceinline__ F2 mean_of(F2 num, F2 den, F2, float) { return f2_div(num, den); }

// Accumulator of exact products: hi parts summed with two_sum, the rounding errors and
// product remainders summed plainly (about 44 correct bits for a few terms).
struct Acc2 {
    float hi = 0.0f, lo = 0.0f;
    __device__ __forceinline__ void add_prod(float a, float b) {
        const F2 pr = two_prod(a, b);
        const F2 sm = two_sum(hi, pr.hi);
        hi = sm.hi;
        lo = __fadd_rn(lo, __fadd_rn(sm.lo, pr.lo));
    }
    __device__ __forceinline__ F2 value() const { return quick_two_sum(hi, lo); }
};

// Loads the 16-byte chunk c of the input token at `pos` straight from global memory.
template <typename T>
struct GlobalLoader {
    const T *x;
    long long row0;
    int dim;
    __device__ __forceinline__ uint4 operator()(int pos, int c) const {
        return ldg16(x + (row0 + pos) * dim + c * Elem<T>::kPerChunk);
    }
};

// ---------------------------------------------------------------------------
// merged token set -> merged sizes / scores -> prune -> outputs
// ---------------------------------------------------------------------------
// Requires sel / match / scnt / tsize / tscore ready (after a barrier).  `load(pos, c)`
// returns the 16-byte chunk c of input token pos.  Returns false (after raising
// FUSION_DEV_INTERNAL) if the token count disagrees with the plan; uniform per CTA.
template <typename T, int NT, typename Loader>
__device__ bool finish_sample(const ImageParams &p, const SampleInfo &s, MetaPtrs &m, const Loader &load) {
    constexpr int CH = Elem<T>::kPerChunk;
    const int tid = threadIdx.x;
    const int N = s.N;

    // merged token set: survivors keep ascending position
    for (int pos = tid; pos < N; pos += NT)
        m.mflag[pos] = (pos >= 2 && !(pos & 1) && m.sel[(pos - 2) / 2]) ? 0 : 1;
    if (s.r_eff > 0)
        for (int a = tid; a < s.nA; a += NT)
            if (m.sel[a]) atomicAdd(&m.scnt[m.match[a]], 1);
    __syncthreads();
    block_scan_excl(m.scnt, s.nB + 1, m.tmp);   // scnt[n] = first slot of B token n's sources
    if (s.r_eff > 0) {
        for (int a = tid; a < s.nA; a += NT) {
            if (!m.sel[a]) continue;
            const int n = m.match[a];
            int before = 0;
            for (int q = 0; q < a; ++q) before += (m.sel[q] && m.match[q] == n) ? 1 : 0;
            m.slist[m.scnt[n] + before] = a;   // sources of every B token in ascending A order
        }
    }
    __syncthreads();

    // merged sizes and scores: float-float sums over the sources (exact for a few terms),
    // rounded once; merged B tokens also keep 1 / (sum of sizes) for the weighted mean
    for (int pos = tid; pos < N; pos += NT) {
        if (!m.mflag[pos]) continue;
        F2 sz = {m.tsize[pos], 0.0f};
        F2 sc = {m.tscore[pos], 0.0f};
        bool merged = false;
        if (pos & 1) {
            const int n = (pos - 1) / 2;
            for (int q = m.scnt[n]; q < m.scnt[n + 1]; ++q) {
                const int a = 2 + 2 * m.slist[q];
                sz = f2_add_f(sz, m.tsize[a]);
                sc = f2_add_f(sc, m.tscore[a]);
                merged = true;
            }
        }
        m.msize[pos] = sz.hi;
        m.mscore[pos] = sc.hi;
        if (merged) {
            const F2 inv = f2_div({1.0f, 0.0f}, sz);
            m.invd[pos] = make_float2(inv.hi, inv.lo);
        }
        if (p.scores && !isfinite(m.mscore[pos]) && pos > 0) raise_status(p.status, FUSION_DEV_NONFINITE);
    }
    __syncthreads();

    // prune: CLS + the k highest merged scores, lowest position on ties
    if (p.do_prune) {
        bool nf = false;
        const int k = keep_count(p.rho[s.id], N - s.r_eff - 1, nf);
        // key 0 marks a non-candidate (CLS or merged away); every candidate key is > 0
        for (int pos = tid; pos < N; pos += NT)
            m.pk[pos] = (pos > 0 && m.mflag[pos]) ? rank_key(m.mscore[pos], pos) : 0ull;
        __syncthreads();
        for (int pos = tid; pos < N; pos += NT) {
            int keep = 0;
            if (pos == 0) {
                keep = 1;
            } else if (m.mflag[pos]) {
                const unsigned long long kp = m.pk[pos];
                int rank = 0;
#pragma unroll 8
                for (int q = 1; q < N; ++q) rank += m.pk[q] > kp ? 1 : 0;
                keep = rank < k ? 1 : 0;
            }
            m.kflag[pos] = keep;
            m.opos[pos] = keep;
        }
    } else {
        for (int pos = tid; pos < N; pos += NT) {
            m.kflag[pos] = m.mflag[pos];
            m.opos[pos] = m.mflag[pos];
        }
    }
    __syncthreads();
    const int total = block_scan_excl(m.opos, N, m.tmp);
    if (total != s.out_n) {   // the plan and the decisions disagree: a library bug
        if (tid == 0) raise_status(p.status, FUSION_DEV_INTERNAL);
        return false;
    }
    for (int pos = tid; pos < N; pos += NT)
        if (m.kflag[pos]) m.srcpos[m.opos[pos]] = pos;
    __syncthreads();

    // index outputs
    const int start = s.start, out_start = s.out_start, out_n = s.out_n;
    for (int o = tid; o < out_n; o += NT) {
        const int pos = m.srcpos[o];
        const long long orow = (long long)out_start + o;
        p.sizes_out[orow] = m.msize[pos];
        if (p.scores_out) p.scores_out[orow] = m.mscore[pos];
        if (p.keep_idx) p.keep_idx[orow] = start + pos;
    }
    if (p.a_match)
        for (int pos = tid; pos < N; pos += NT)
            p.a_match[start + pos] = (pos >= 2 && !(pos & 1)) ? start + 1 + 2 * m.match[(pos - 2) / 2] : -1;
    if (p.dst_map && !p.do_prune)
        for (int pos = tid; pos < N; pos += NT) {
            const bool gone = pos >= 2 && !(pos & 1) && m.sel[(pos - 2) / 2];
            const int dest = gone ? 1 + 2 * m.match[(pos - 2) / 2] : pos;
            p.dst_map[start + pos] = out_start + m.opos[dest];
        }

    // token rows: copies and size-weighted means, 16 bytes per thread.  (o, c) walks the
    // output rows chunk by chunk without a division per step.
    const int ncx = p.dim / CH;
    const int ostep = NT / ncx, cstep = NT - ostep * ncx;
    T *xo = reinterpret_cast<T *>(p.x_out);
    int o = tid / ncx, c = tid - (tid / ncx) * ncx;
    for (; o < out_n;) {
        const int pos = m.srcpos[o];
        const uint4 self = load(pos, c);
        uint4 outv = self;
        if (pos & 1) {
            const int n = (pos - 1) / 2;
            const int q0 = m.scnt[n], q1 = m.scnt[n + 1];
            if (q1 > q0) {
                float f[CH];
                chunk_to_f(self, f);
                const float sb = m.tsize[pos];
                Acc2 num[CH];
#pragma unroll
                for (int e = 0; e < CH; ++e) num[e].add_prod(sb, f[e]);
                F2 den = {sb, 0.0f};
                for (int q = q0; q < q1; ++q) {
                    const int apos = 2 + 2 * m.slist[q];
                    const float sa = m.tsize[apos];
                    den = f2_add_f(den, sa);
                    chunk_to_f(load(apos, c), f);
#pragma unroll
                    for (int e = 0; e < CH; ++e) num[e].add_prod(sa, f[e]);
                }
                const float2 iv = m.invd[pos];
                F2 qv[CH];
#pragma unroll
                for (int e = 0; e < CH; ++e) qv[e] = mean_of(num[e].value(), den, {iv.x, iv.y}, T{});
                outv = pack_chunk(qv);
            }
        }
        *reinterpret_cast<uint4 *>(xo + ((long long)out_start + o) * p.dim + c * CH) = outv;
        o += ostep;
        c += cstep;
        if (c >= ncx) {
            c -= ncx;
            ++o;
        }
    }
    return true;
}

}  // namespace fz
