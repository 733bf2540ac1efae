// Per-sample work shared by the two per-sample kernels (image.cu: mma.sync / FFMA
// decisions; image_tc.cu: TMA + tcgen05 decisions): the sample's bookkeeping, the
// top-r selection from the row maxima (Sec. III-C), the merged token set with its
// size-weighted means, pruning (Sec. III-E) and the gather into the compacted output.
#pragma once

#include "launch.h"

namespace fz {

// A and B indices are below FUSION_MAX_TOKENS / 2 <= 2^kKeyShift, so (B index, A index)
// packs into one int that orders by B token first.
constexpr int kKeyShift = 10;
static_assert(FUSION_MAX_TOKENS / 2 <= (1 << kKeyShift), "token index does not fit the merge key");
constexpr int kMergedCount = 36;   // tmp[] slot of the number of B tokens that receive sources
constexpr int kGatherChunks = 2048;   // copy chunks in flight per CTA
constexpr int kSrcU = 2;           // merge sources fetched ahead

// ---------------------------------------------------------------------------
// metadata in shared memory, after the kernel's staging area
// ---------------------------------------------------------------------------
struct Meta {
    size_t best, rk, pk, inv_a, inv_b, match, sel, mkey, mflag, kflag, opos, srcpos, scnt, slist, mlist, msize,
        mscore, invd, tsize, tscore, tmp, total;
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
    L.mkey = off;   off += sizeof(int) * nA;
    L.mflag = off;  off += sizeof(int) * nmax;
    L.kflag = off;  off += sizeof(int) * nmax;
    L.opos = off;   off += sizeof(int) * (nmax + 1);
    L.srcpos = off; off += sizeof(int) * nmax;
    L.scnt = off;   off += sizeof(int) * (nB + 1);
    L.slist = off;  off += sizeof(int) * nA;
    L.mlist = off;  off += sizeof(int) * nB;
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
    MetaPtrs() = default;
    // only the arrays a merged mean reads (sizes, source lists, inverse size sums)
    __device__ static MetaPtrs views(const float *tsize, const int *slist, const float2 *invd) {
        MetaPtrs m{};
        m.tsize = const_cast<float *>(tsize);
        m.slist = const_cast<int *>(slist);
        m.invd = const_cast<float2 *>(invd);
        return m;
    }
    unsigned long long *best, *rk, *pk;
    float *inv_a, *inv_b;
    int *match, *sel, *mkey, *mflag, *kflag, *opos, *srcpos, *scnt, *slist, *mlist;
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
          mkey(reinterpret_cast<int *>(sm + L.mkey)),
          mflag(reinterpret_cast<int *>(sm + L.mflag)),
          kflag(reinterpret_cast<int *>(sm + L.kflag)),
          opos(reinterpret_cast<int *>(sm + L.opos)),
          srcpos(reinterpret_cast<int *>(sm + L.srcpos)),
          scnt(reinterpret_cast<int *>(sm + L.scnt)),
          slist(reinterpret_cast<int *>(sm + L.slist)),
          mlist(reinterpret_cast<int *>(sm + L.mlist)),
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
// The grid has one CTA per possible sample (i < max_batch), so every load of the first
// group is in bounds whatever the device batch count says; they issue together, and the
// second group (which needs the output slot and the original id) follows.
__device__ __forceinline__ bool sample_info(const ImageParams &p, int i, SampleInfo &s) {
    const int bval = p.in.batch ? *p.in.batch : p.in.max_batch;
    const int valid = p.plan[0];
    const int j = p.slot[i];
    const int o0 = p.in.offsets[i], o1 = p.in.offsets[i + 1];
    const int id = p.in.ids ? p.in.ids[i] : i;
    if (bval < 0 || bval > p.in.max_batch || i >= bval || valid == 0 || j < 0) return false;
    s.start = o0;
    s.N = o1 - o0;
    s.out_start = p.offsets_out[j];
    s.out_n = p.offsets_out[j + 1] - s.out_start;
    s.id = id;
    s.P = s.N - 1;
    s.nA = s.P / 2;
    s.nB = (s.P + 1) / 2;
    s.r_eff = p.do_merge ? merge_count(p.r[s.id], s.P) : 0;
    s.decide = p.do_merge && s.nA > 0 && (s.r_eff > 0 || p.need_match);
    return true;
}

// The plan of one call computed inside the per-sample kernel, for batches of at most
// kFusedPlanMaxBatch samples: every CTA runs through the whole batch (validation, which
// samples continue, their output token counts) and keeps the exclusive prefix before its
// own sample, so all CTAs agree on validity and no plan kernel runs first.  The loads of
// the first group are in bounds for any j < max_batch, so they issue before the device
// batch count is known.  CTA 0 writes the batch-level outputs and raises the status.
// Must be called by every thread of the CTA.

// dep_wait: the kernel may run as a programmatic dependent of the exit check, whose exit mask
// is read only after `griddepcontrol.wait`; everything else the plan reads (offsets, ids, merge
// counts, keep ratios) is this call's input and loads before it.
template <int NT>
__device__ bool sample_plan(const ImageParams &p, int i, SampleInfo &s, bool dep_wait = false) {
    const PlanArgs &a = p.plan_args;
    constexpr int kW = NT / 32;
    __shared__ int red[6][kW];
    __shared__ int own[6];   // start, N, id, continues, count, merge count of sample i
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int bval = a.in.batch ? *a.in.batch : a.in.max_batch;
    int bad = 0, nf = 0, pre_s = 0, pre_r = 0, tot_s = 0, tot_r = 0;
    bool waited = !dep_wait;   // uniform
    for (int j0 = 0; j0 < a.in.max_batch; j0 += NT) {
        const int j = j0 + t;
        const bool inb = j < a.in.max_batch;
        const int o0 = inb ? a.in.offsets[j] : 0, o1 = inb ? a.in.offsets[j + 1] : 0;
        const int idr = inb ? (a.in.ids ? a.in.ids[j] : j) : 0;
        const bool id_ok = idr >= 0 && idr < a.in.max_batch;
        // merge count and keep ratio by id, for every in-bounds id (used for continuing samples only)
        const int rr = (inb && id_ok && a.merge) ? a.r[idr] : 0;
        const float rh = (inb && id_ok && a.prune) ? a.rho[idr] : 0.0f;
        if (!waited) {
            asm volatile("griddepcontrol.wait;" ::: "memory");
            waited = true;
        }
        const int ex = (inb && a.exit_mask) ? a.exit_mask[j] : 0;
        if (!inb || j >= bval) continue;
        const int N = o1 - o0;
        const bool ok = o0 >= 0 && N >= 1 && N <= a.in.max_tokens && (long long)o1 <= a.in.max_rows;
        if (!ok) bad |= FUSION_DEV_BAD_OFFSETS;
        if (!id_ok) bad |= FUSION_DEV_BAD_IDS;
        const int surv = ex == 0 ? 1 : 0;
        int cnt = 0, rm = 0;
        if (ok && id_ok && surv) {
            int n = N;
            if (a.merge) {
                rm = merge_count(rr, N - 1);
                n -= rm;
            }
            if (a.prune) {
                bool f = false;
                n = 1 + keep_count(rh, n - 1, f);
                if (f) nf = 1;
            }
            cnt = n;
        }
        tot_s += surv;
        tot_r += cnt;
        if (j < i) {
            pre_s += surv;
            pre_r += cnt;
        }
        if (j == i) {
            own[0] = o0;
            own[1] = N;
            own[2] = idr;
            own[3] = surv;
            own[4] = cnt;
            own[5] = rm;
        }
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        bad |= __shfl_xor_sync(0xFFFFFFFFu, bad, m);
        nf |= __shfl_xor_sync(0xFFFFFFFFu, nf, m);
        pre_s += __shfl_xor_sync(0xFFFFFFFFu, pre_s, m);
        pre_r += __shfl_xor_sync(0xFFFFFFFFu, pre_r, m);
        tot_s += __shfl_xor_sync(0xFFFFFFFFu, tot_s, m);
        tot_r += __shfl_xor_sync(0xFFFFFFFFu, tot_r, m);
    }
    if (lane == 0) {
        red[0][w] = bad;
        red[1][w] = nf;
        red[2][w] = pre_s;
        red[3][w] = pre_r;
        red[4][w] = tot_s;
        red[5][w] = tot_r;
    }
    __syncthreads();
    bad = nf = pre_s = pre_r = tot_s = tot_r = 0;
#pragma unroll
    for (int k = 0; k < kW; ++k) {
        bad |= red[0][k];
        nf |= red[1][k];
        pre_s += red[2][k];
        pre_r += red[3][k];
        tot_s += red[4][k];
        tot_r += red[5][k];
    }
    const bool batch_ok = bval >= 0 && bval <= a.in.max_batch;
    if (!batch_ok) bad |= FUSION_DEV_BAD_BATCH;
    if (i == 0 && t == 0) {
        if (bad) raise_status(a.status, bad);
        if (nf) raise_status(a.status, FUSION_DEV_NONFINITE);
        a.offsets_out[bad ? 0 : tot_s] = bad ? 0 : tot_r;
        if (a.batch_out) *a.batch_out = bad ? 0 : tot_s;
    }
    if (bad || i >= bval || !own[3]) return false;
    if (t == 0) {
        a.offsets_out[pre_s] = pre_r;
        if (a.ids_out) a.ids_out[pre_s] = own[2];
    }
    s.start = own[0];
    s.N = own[1];
    s.out_start = pre_r;
    s.out_n = own[4];
    s.id = own[2];
    s.P = s.N - 1;
    s.nA = s.P / 2;
    s.nB = (s.P + 1) / 2;
    s.r_eff = p.do_merge ? own[5] : 0;   // the plan's merge flag is the call's
    s.decide = p.do_merge && s.nA > 0 && (s.r_eff > 0 || p.need_match);
    return true;
}

// The launch gate (fusion_set_launch_gate): thread 0 polls the flag, at most `spins` more
// times after the first read, and the CTA learns the result through shared memory.  Called
// before any load of the call's inputs and before any asynchronous copy, so a CTA that gives up
// has nothing in flight.
__device__ __forceinline__ bool gate_open(const int *gate, unsigned spins) {
    __shared__ int s_open;
    if (threadIdx.x == 0) {
        int ok = 0;
        for (unsigned it = 0;; ++it) {
            int v;
            asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(gate) : "memory");
            if (v != 0) {
                ok = 1;
                break;
            }
            if (it >= spins) break;
            __nanosleep(128);
        }
        s_open = ok;
    }
    __syncthreads();
    return s_open != 0;
}

// Either the fused plan or the plan kernel's results, once the launch gate (if any) is open;
// a CTA whose gate wait gives up raises FUSION_DEV_TIMEOUT and writes nothing.
template <int NT>
// dep_wait: see sample_plan; without the fused plan the wait comes first (the plan's results may be
// the predecessor's output).
__device__ __forceinline__ bool sample_begin(const ImageParams &p, int i, SampleInfo &s, bool dep_wait = false) {
    if (p.gate && !gate_open(p.gate, p.gate_spins)) {
        if (threadIdx.x == 0) raise_status(p.status, FUSION_DEV_TIMEOUT);
        return false;
    }
    if (dep_wait && !p.fused_plan) asm volatile("griddepcontrol.wait;" ::: "memory");
    return p.fused_plan ? sample_plan<NT>(p, i, s, dep_wait) : sample_info(p, i, s);
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
    if (tid == 0) m.tmp[kMergedCount] = 0;
    for (int pos = tid; pos < s.N; pos += NT) {
        m.tsize[pos] = p.sizes[s.start + pos];
        m.tscore[pos] = p.scores ? p.scores[s.start + pos] : 0.0f;
    }
}

// meta_init in two parts, for a kernel whose own bulk loads would otherwise sit ahead of the
// token sizes and scores in the memory queues: the copies of the sizes and scores go out first
// (cp.async, no registers held), the rest of the metadata after, and the copies are waited for
// at its end (before the caller's barrier).
template <int NT>
__device__ __forceinline__ void meta_prefetch(const ImageParams &p, const SampleInfo &s, MetaPtrs &m) {
    for (int pos = threadIdx.x; pos < s.N; pos += NT) {
        cp_async4(&m.tsize[pos], p.sizes + s.start + pos);
        if (p.scores) cp_async4(&m.tscore[pos], p.scores + s.start + pos);
    }
    cp_async_commit();
}
template <int NT>
__device__ __forceinline__ void meta_init_rest(const ImageParams &p, const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    for (int a = tid; a < s.nA; a += NT) {
        m.best[a] = 0ull;
        m.sel[a] = 0;
        m.match[a] = 0;
    }
    for (int n = tid; n <= s.nB; n += NT) m.scnt[n] = 0;
    if (tid == 0) m.tmp[kMergedCount] = 0;
    if (!p.scores)
        for (int pos = tid; pos < s.N; pos += NT) m.tscore[pos] = 0.0f;
    cp_async_wait_all();
}

// best[a] holds the packed (similarity, lowest B index) maximum of every A row.  Writes
// match[a] and, when tokens merge, sel[a] for the r_eff A tokens of largest similarity
// (lowest position on ties) and mkey[rank] = (match[a] << kKeyShift) | a for each of them.
// Ends with a barrier.
template <int NT>
__device__ __forceinline__ void select_top_r(const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    for (int a = tid; a < s.nA; a += NT) m.match[a] = (int)(0xFFFFFFFFu - (uint32_t)(m.best[a] & 0xFFFFFFFFull));
    if (s.r_eff > 0) {
        // the ordered similarity of every A row (the high half of its key)
        uint32_t *rv = reinterpret_cast<uint32_t *>(m.rk);
        for (int a = tid; a < s.nA; a += NT) rv[a] = (uint32_t)(m.best[a] >> 32);
        __syncthreads();
        for (int a = tid; a < s.nA; a += NT) {
            // rank of a: the rows of larger similarity, and the rows of equal similarity at a
            // lower position (32-bit comparisons in two ranges instead of 64-bit keys)
            const uint32_t va = rv[a];
            int rank = 0;
#pragma unroll 8
            for (int q = 0; q < a; ++q) rank += rv[q] >= va ? 1 : 0;
#pragma unroll 8
            for (int q = a + 1; q < s.nA; ++q) rank += rv[q] > va ? 1 : 0;
            m.sel[a] = rank < s.r_eff ? 1 : 0;
            if (rank < s.r_eff) m.mkey[rank] = (m.match[a] << kKeyShift) | a;
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

// bf16 bits of num / den rounded to nearest even.  A power-of-two den (uniform over a
// merged row; every merge of two unit-size tokens) scales num exactly, so the float-float
// product rounds directly, as in mean_of.  Otherwise q1 = num.hi * inv.hi carries three
// relative errors of at most 2^-24 each (num.lo dropped, inv.lo dropped, the product's
// rounding), so it lies within 4 float32 ulps of the exact quotient: when it is more than
// 8 ulps from every bf16 rounding midpoint it rounds like the exact quotient; otherwise
// the float-float path above decides.
// The rare case near a midpoint, out of line so that the common path stays short.
static __device__ __noinline__ uint16_t mean_bits_slow(F2 num, F2 den, F2 inv) {
    return f2_to_bf16_bits(mean_of(num, den, inv, __nv_bfloat16{}));
}
__device__ __forceinline__ uint16_t mean_bits(F2 num, F2 den, F2 inv, bool pow2, __nv_bfloat16) {
    if (pow2) return f2_to_bf16_bits(f2_mul(num, inv));
    const uint32_t u = __float_as_uint(__fmul_rn(num.hi, inv.hi));
    const uint32_t low = u & 0xFFFFu;
    const uint32_t dist = low > 0x8000u ? low - 0x8000u : 0x8000u - low;
    if (dist > 8u && (u & 0x7F800000u) != 0x7F800000u) return (uint16_t)((u + 0x8000u) >> 16);
    return mean_bits_slow(num, den, inv);
}

// Accumulator of exact products: hi parts summed with two_sum, the rounding errors and
// product remainders summed plainly (about 44 correct bits for a few terms).
struct Acc2 {
    float hi = 0.0f, lo = 0.0f;
    __device__ __forceinline__ void first_prod(float a, float b) {   // add_prod from zero
        const F2 pr = two_prod(a, b);
        hi = pr.hi;
        lo = pr.lo;
    }
    __device__ __forceinline__ void add_prod(float a, float b) {
        const F2 pr = two_prod(a, b);
        const F2 sm = two_sum(hi, pr.hi);
        hi = sm.hi;
        lo = __fadd_rn(lo, __fadd_rn(sm.lo, pr.lo));
    }
    __device__ __forceinline__ F2 value() const { return quick_two_sum(hi, lo); }
};

__device__ __forceinline__ uint4 merged_pack(const Acc2 (&num)[8], F2 den, F2 inv, __nv_bfloat16) {
    const bool pow2 = den.lo == 0.0f && (__float_as_uint(den.hi) & 0x007FFFFFu) == 0u;
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
        w[k] = (uint32_t)mean_bits(num[2 * k].value(), den, inv, pow2, __nv_bfloat16{}) |
               ((uint32_t)mean_bits(num[2 * k + 1].value(), den, inv, pow2, __nv_bfloat16{}) << 16);
    return make_uint4(w[0], w[1], w[2], w[3]);
}
__device__ __forceinline__ uint4 merged_pack(const Acc2 (&num)[4], F2 den, F2 inv, float) {
    F2 q[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) q[e] = mean_of(num[e].value(), den, inv, 0.0f);
    return pack_chunk(q);
}

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
// One chunk of a merged output row (Sec. III-C): chunk c of B token `pos` and of its
// first kSrcU sources, fetched ahead of the arithmetic so the loads overlap other work.
struct MergedItem {
    int pos, c, q0, q1;   // pos < 0: nothing to do
    uint4 self, av[kSrcU];
};

// Item t of the merged chunks [c_lo, c_lo + w) of every merged row.
template <typename Loader>
__device__ __forceinline__ void merged_fetch(const MetaPtrs &m, int t, int n_items, int w, int c_lo, const Loader &load,
                                             MergedItem &it) {
    it.pos = -1;
    if (t >= n_items) return;
    const int k = t / w;
    const int pos = 1 + 2 * m.mlist[k];
    if (!m.kflag[pos]) return;   // pruned after merging
    it.pos = pos;
    it.c = c_lo + t - k * w;
    const int n = (pos - 1) >> 1;
    it.q0 = m.scnt[n];
    it.q1 = m.scnt[n + 1];
    it.self = load(pos, it.c);
#pragma unroll
    for (int u = 0; u < kSrcU; ++u)
        if (it.q0 + u < it.q1) it.av[u] = load(2 + 2 * m.slist[it.q0 + u], it.c);
}

// The size-weighted mean of a fetched item: the B token first, then its sources in
// ascending A order, products summed exactly enough that the result rounds once.
template <typename T, typename Loader>
__device__ __forceinline__ uint4 merged_compute(const MetaPtrs &m, const MergedItem &it, const Loader &load) {
    constexpr int CH = Elem<T>::kPerChunk;
    float f[CH];
    chunk_to_f(it.self, f);
    const float sb = m.tsize[it.pos];
    Acc2 num[CH];
#pragma unroll
    for (int e = 0; e < CH; ++e) num[e].first_prod(sb, f[e]);
    F2 den = {sb, 0.0f};
#pragma unroll
    for (int u = 0; u < kSrcU; ++u) {
        if (it.q0 + u >= it.q1) break;
        const float sa = m.tsize[2 + 2 * m.slist[it.q0 + u]];
        den = f2_add_f(den, sa);
        chunk_to_f(it.av[u], f);
#pragma unroll
        for (int e = 0; e < CH; ++e) num[e].add_prod(sa, f[e]);
    }
    for (int q = it.q0 + kSrcU; q < it.q1; ++q) {
        const int ap = 2 + 2 * m.slist[q];
        const float sa = m.tsize[ap];
        den = f2_add_f(den, sa);
        chunk_to_f(load(ap, it.c), f);
#pragma unroll
        for (int e = 0; e < CH; ++e) num[e].add_prod(sa, f[e]);
    }
    const float2 iv = m.invd[it.pos];
    return merged_pack(num, den, {iv.x, iv.y}, T{});
}

// A size whose product with any bf16 value (8 significant bits) is exact in float: at most
// 16 significant bits, at least 1 (so products with subnormal values stay on the float
// grid) and below 2^64.
__device__ __forceinline__ bool short_size(float s) {
    return s >= 1.0f && s < 0x1p64f && (__float_as_uint(s) & 0xFFu) == 0u;
}

// The exact float-float mean of a chunk, out of line; everything passed by value so the
// caller keeps its state in registers.
template <typename Loader>
__device__ __noinline__ uint4 merged_exact_bf16(const float *tsize, const int *slist, const float2 *invd, int pos, int c,
                                                int q0, int q1, uint4 self, uint4 av0, uint4 av1, Loader load) {
    MergedItem it;
    it.pos = pos;
    it.c = c;
    it.q0 = q0;
    it.q1 = q1;
    it.self = self;
    it.av[0] = av0;
    it.av[1] = av1;
    MetaPtrs m = MetaPtrs::views(tsize, slist, invd);
    return merged_compute<__nv_bfloat16>(m, it, load);
}

// A bf16 merged chunk, exactly rounded, in float.  When every size is short, every
// product s x is exact; a two_sum chain over the products then shows whether their float
// sum num is the exact numerator (it is unless the terms lie more than 2^24 apart).  With
// num exact and den (the float sum of the sizes) exact:
//  * q0 = num * inv.hi lies within a few float ulps of the exact mean t = num / den, so t
//    lies in the bf16 interval [b, b+1] that holds q0 or within a few float ulps of its
//    ends, where the rounding is that of the nearest end anyway;
//  * m, the midpoint of that interval, decides the rounding: R = fma(m, -den, num) is
//    num - m den rounded once, so its sign (and whether it is zero) is that of t - m:
//    t beyond m rounds away from b, short of m to b, exactly on m to the even end.
// When the products are exact but their float sum is not, the chain's rounding errors,
// summed beside it, make the float-float numerator that the out-of-line computation would
// form from the same products in the same order (its product remainders are zero), and
// mean_bits rounds it here.  Otherwise (long sizes, an inexact sum of sizes, non-finite
// values) the float-float computation runs, out of line.
template <typename Loader>
__device__ __forceinline__ uint4 merged_fast_bf16(const MetaPtrs &m, const MergedItem &it, const Loader &load) {
    const float sb = m.tsize[it.pos];
    const float2 iv = m.invd[it.pos];   // 1 / den as float-float
    float num[8], lo[8], x[8];
    chunk_to_f(it.self, x);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        num[e] = __fmul_rn(sb, x[e]);
        lo[e] = 0.0f;
    }
    float den = sb;
    bool ok = short_size(sb);   // every product exact, the sum of sizes exact
    bool exact = true;          // and the sum of products too
    for (int q = it.q0; q < it.q1; ++q) {
        const int u = q - it.q0;
        const int ap = 2 + 2 * m.slist[q];
        const float sa = m.tsize[ap];
        const F2 dd = two_sum(den, sa);
        den = dd.hi;
        ok = ok && short_size(sa) && dd.lo == 0.0f;
        chunk_to_f(u == 0 ? it.av[0] : u == 1 ? it.av[1] : load(ap, it.c), x);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const F2 t = two_sum(num[e], __fmul_rn(sa, x[e]));
            num[e] = t.hi;
            lo[e] = __fadd_rn(lo[e], t.lo);
            exact = exact && t.lo == 0.0f;
        }
    }
    if (!ok)
        return merged_exact_bf16(m.tsize, m.slist, m.invd, it.pos, it.c, it.q0, it.q1, it.self, it.av[0], it.av[1], load);
    if (!exact) {
        const F2 dn = {den, 0.0f};
        const F2 inv = {iv.x, iv.y};
        const bool pow2 = (__float_as_uint(den) & 0x007FFFFFu) == 0u;
        uint32_t w[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
            w[k] = (uint32_t)mean_bits(quick_two_sum(num[2 * k], lo[2 * k]), dn, inv, pow2, __nv_bfloat16{}) |
                   ((uint32_t)mean_bits(quick_two_sum(num[2 * k + 1], lo[2 * k + 1]), dn, inv, pow2, __nv_bfloat16{})
                    << 16);
        return make_uint4(w[0], w[1], w[2], w[3]);
    }
    uint32_t bits[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const uint32_t uq = __float_as_uint(__fmul_rn(num[e], iv.x));
        ok = ok && ((uq >> 23) & 0xFFu) != 0xFFu;
        const float mid = __uint_as_float((uq & 0xFFFF0000u) | 0x8000u);
        const float R = __fmaf_rn(mid, -den, num[e]);
        const uint32_t b = uq >> 16;
        const bool neg = (uq >> 31) != 0u;
        const bool up = R == 0.0f ? (b & 1u) != 0u : ((R > 0.0f) != neg);
        bits[e] = b + (up ? 1u : 0u);
    }
    if (!ok)
        return merged_exact_bf16(m.tsize, m.slist, m.invd, it.pos, it.c, it.q0, it.q1, it.self, it.av[0], it.av[1], load);
    return make_uint4(bits[0] | (bits[1] << 16), bits[2] | (bits[3] << 16), bits[4] | (bits[5] << 16),
                      bits[6] | (bits[7] << 16));
}

template <typename T, typename Loader>
__device__ __forceinline__ uint4 merged_value(const MetaPtrs &m, const MergedItem &it, const Loader &load) {
    if constexpr (Elem<T>::kBytes == 2)
        return merged_fast_bf16(m, it, load);
    else
        return merged_compute<T>(m, it, load);
}

// The decisions after the matching, up to the output position of every kept token:
// merged set, merged sizes and scores, pruning, the scan of kept tokens and the source of
// every output row.  Requires sel / match / mkey / tsize / tscore ready (after a barrier);
// needs s.out_n but not s.out_start.  Returns false (after raising FUSION_DEV_INTERNAL) if
// the token count disagrees with the plan; uniform per CTA.
template <int NT>
__device__ bool finish_decide(const ImageParams &p, const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    const int N = s.N, nB = s.nB, R = s.r_eff;

    // merged token set: survivors keep ascending position (mflag 1; 0 = merged away).
    // The selected A tokens, keyed (B index, A index), give every B token the slice
    // scnt[n] .. scnt[n+1] of slist holding its sources in ascending A order.
    for (int pos = tid; pos < N; pos += NT)
        m.mflag[pos] = (pos >= 2 && !(pos & 1) && m.sel[(pos - 2) / 2]) ? 0 : 1;
    if (R > 0) {
        for (int t = tid; t < R; t += NT) {
            const int key = m.mkey[t];
            int slot = 0;
            for (int u = 0; u < R; ++u) slot += m.mkey[u] < key ? 1 : 0;
            m.slist[slot] = key & ((1 << kKeyShift) - 1);
        }
        for (int n = tid; n < nB; n += NT) {
            int lt = 0, eq = 0;
            for (int u = 0; u < R; ++u) {
                const int b = m.mkey[u] >> kKeyShift;
                lt += b < n ? 1 : 0;
                eq += b == n ? 1 : 0;
            }
            m.scnt[n] = lt;
            if (eq > 0) m.mlist[atomicAdd(&m.tmp[kMergedCount], 1)] = n;
        }
        if (tid == 0) m.scnt[nB] = R;
    }
    __syncthreads();

    // merged sizes and scores: float-float sums over the sources (exact for a few terms),
    // rounded once; merged B tokens (mflag 2) also keep 1 / (sum of sizes) for the mean
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
            m.mflag[pos] = 2;
        }
        if (p.scores && !isfinite(m.mscore[pos]) && pos > 0) raise_status(p.status, FUSION_DEV_NONFINITE);
    }
    __syncthreads();

    // prune: CLS + the k highest merged scores, lowest position on ties
    if (p.do_prune) {
        bool nf = false;
        const int k = keep_count(p.rho[s.id], N - R - 1, nf);
        // the ordered merged score of every candidate; 0 marks a non-candidate (CLS or merged
        // away), below every candidate's value (ordered values of floats are >= 1)
        uint32_t *pv = reinterpret_cast<uint32_t *>(m.pk);
        for (int pos = tid; pos < N; pos += NT) pv[pos] = (pos > 0 && m.mflag[pos]) ? ordered_bits(m.mscore[pos]) : 0u;
        __syncthreads();
        for (int pos = tid; pos < N; pos += NT) {
            int keep = 0;
            if (pos == 0) {
                keep = 1;
            } else if (m.mflag[pos]) {
                // rank: candidates of larger score, and of equal score at a lower position
                const uint32_t vp = pv[pos];
                int rank = 0;
#pragma unroll 8
                for (int q = 1; q < pos; ++q) rank += pv[q] >= vp ? 1 : 0;
#pragma unroll 8
                for (int q = pos + 1; q < N; ++q) rank += pv[q] > vp ? 1 : 0;
                keep = rank < k ? 1 : 0;
            }
            m.kflag[pos] = keep;
            m.opos[pos] = keep;
        }
    } else {
        for (int pos = tid; pos < N; pos += NT) {
            const int keep = m.mflag[pos] ? 1 : 0;
            m.kflag[pos] = keep;
            m.opos[pos] = keep;
        }
    }
    __syncthreads();
    const int total = block_scan_excl(m.opos, N, m.tmp);
    if (total != s.out_n) {   // the plan and the decisions disagree: a library bug
        if (tid == 0) raise_status(p.status, FUSION_DEV_INTERNAL);
        return false;
    }
    // source of every output row; merged rows are stored complemented (negative)
    for (int pos = tid; pos < N; pos += NT)
        if (m.kflag[pos]) m.srcpos[m.opos[pos]] = m.mflag[pos] == 2 ? ~pos : pos;
    __syncthreads();
    return true;
}

// Index outputs of a decided sample (after finish_decide): sizes, scores and input row of every
// output row at s.out_start, and the match / destination maps when requested.
template <int NT>
__device__ void write_index_outputs(const ImageParams &p, const SampleInfo &s, MetaPtrs &m) {
    const int tid = threadIdx.x;
    const int N = s.N;
    const int start = s.start, out_start = s.out_start, out_n = s.out_n;
    for (int o = tid; o < out_n; o += NT) {
        const int sp = m.srcpos[o];
        const int pos = sp < 0 ? ~sp : sp;
        const long long orow = (long long)out_start + o;
        p.sizes_out[orow] = m.msize[pos];
        if (p.scores_out) p.scores_out[orow] = m.mscore[pos];
        if (p.keep_idx) p.keep_idx[orow] = p.keep_map ? p.keep_map[start + pos] : start + pos;
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
}

// The token rows of a decided sample, 16-byte chunks [c_lo, c_hi) of every output row: copied
// rows with kGatherU chunks in flight per thread ((o, c) walks the rows chunk by chunk without
// a division per step), then the merged rows' size-weighted means with the next item's loads
// in flight.  `load(pos, c)` returns chunk c of input token pos.
template <typename T, int NT, typename Loader>
__device__ void write_rows(const ImageParams &p, const SampleInfo &s, MetaPtrs &m, const Loader &load, int c_lo,
                           int c_hi) {
    constexpr int CH = Elem<T>::kPerChunk;
    constexpr int kGatherU = kGatherChunks / NT;
    const int tid = threadIdx.x;
    const int out_n = s.out_n;
    const int dim = p.dim, w = c_hi - c_lo;
    if (w <= 0) return;
    const int ostep = NT / w, cstep = NT - ostep * w;
    T *xo = reinterpret_cast<T *>(p.x_out) + (long long)s.out_start * dim;
    const int n_items = m.tmp[kMergedCount] * w;   // merged chunks of the range
    MergedItem cur;
    merged_fetch(m, tid, n_items, w, c_lo, load, cur);   // lands while the copies run
    int o = tid / w, c = tid - (tid / w) * w;
    while (o < out_n) {
        int src[kGatherU], cc[kGatherU], dst[kGatherU];
#pragma unroll
        for (int u = 0; u < kGatherU; ++u) {
            src[u] = o < out_n ? m.srcpos[o] : -1;   // < 0: merged row or past the end
            cc[u] = c_lo + c;
            dst[u] = o * dim + (c_lo + c) * CH;
            o += ostep;
            c += cstep;
            if (c >= w) {
                c -= w;
                ++o;
            }
        }
        uint4 v[kGatherU];
#pragma unroll
        for (int u = 0; u < kGatherU; ++u)
            if (src[u] >= 0) v[u] = load(src[u], cc[u]);
#pragma unroll
        for (int u = 0; u < kGatherU; ++u)
            if (src[u] >= 0) *reinterpret_cast<uint4 *>(xo + dst[u]) = v[u];
    }
    for (int t = tid; t < n_items; t += NT) {
        MergedItem nxt;
        merged_fetch(m, t + NT, n_items, w, c_lo, load, nxt);
        if (cur.pos >= 0)
            *reinterpret_cast<uint4 *>(xo + m.opos[cur.pos] * dim + cur.c * CH) = merged_value<T>(m, cur, load);
        cur = nxt;
    }
}

// The outputs of a decided sample (after finish_decide) at s.out_start.
template <typename T, int NT, typename Loader>
__device__ void finish_write(const ImageParams &p, const SampleInfo &s, MetaPtrs &m, const Loader &load) {
    write_index_outputs<NT>(p, s, m);
    write_rows<T, NT>(p, s, m, load, 0, p.dim / Elem<T>::kPerChunk);
}

// finish_decide then finish_write (the plan's output offsets already known).
template <typename T, int NT, typename Loader>
__device__ bool finish_sample(const ImageParams &p, const SampleInfo &s, MetaPtrs &m, const Loader &load) {
    if (!finish_decide<NT>(p, s, m)) return false;
    finish_write<T, NT>(p, s, m, load);
    return true;
}

}  // namespace fz
