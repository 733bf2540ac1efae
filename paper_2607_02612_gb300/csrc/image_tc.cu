// Per-sample merge -> prune -> gather for bf16 tokens on the 5th-generation tensor
// cores (tcgen05) with TMA, for samples of at most 257 tokens (|A|, |B| <= 128).
//
// One CTA of 256 threads per input sample.  The keys of half A (even positions) and
// half B (odd positions) arrive by TMA tensor loads in K-blocks of 64 dims, 128-byte
// swizzled: K-block kb of a half is a [rows][128 B] tile, 16-byte chunk j of row t
// stored at chunk position j ^ (t % 8).  Two tensor maps per parity of the global row
// index (every other row of the token matrix) cover boxes of 32 and 8 rows, so any
// half of any sample loads in whole 8-row groups.  The K-blocks stream through a ring
// of stages (the whole sample stays resident when it fits).
//
// Thread 0 produces (TMA), thread 32 issues tcgen05.mma (M = 128 A rows, N = |B|
// rounded up to 16, K = 16 per instruction, f32 accumulation in tensor memory), and
// every thread accumulates the squared norm of one A or B row from the same stages.
// A stage is released when the MMAs that read it completed (tcgen05.commit) and all
// warps are done with it.  The epilogue reads S from tensor memory, one A row per
// thread (two warpgroups split the columns), forms cos = dot * inv|a| * inv|b| and
// keeps the largest value with the lowest B index.  Everything after the decisions
// (top-r, merged set, sums, pruning, gather) is the shared finish phase.
//
// Every wait on an mbarrier is bounded; on a timeout the CTA raises
// FUSION_DEV_TIMEOUT, skips its outputs and frees its tensor memory.
#include <cuda.h>

#include <algorithm>

#include "sample.cuh"
#include "tc.cuh"

namespace fz {
namespace {

constexpr int kTcThreads = 256;
constexpr int kMaxStages = 16;

struct TcMaps {
    CUtensorMap e32, o32, e8, o8;   // even / odd rows, boxes of 32 / 8 rows x 64 dims
    // even / odd rows seen as (64 dims, row, K-block) with the K-block stride 128 B: a box of
    // 8 rows x all K-blocks lands as [K-block][8 rows][128 B], one 1 KB swizzle atom per K-block
    CUtensorMap ge, go;
};

// ss + sc += part, Neumaier-compensated.
__device__ __forceinline__ void neumaier_add(float &ss, float &sc, float part) {
    const float t = __fadd_rn(ss, part);
    sc = __fadd_rn(sc, fabsf(ss) >= fabsf(part) ? __fadd_rn(__fsub_rn(ss, t), part) : __fadd_rn(__fsub_rn(part, t), ss));
    ss = t;
}
// Sum of squares of the 8 bf16 values of a 16-byte chunk.
__device__ __forceinline__ float chunk_sq(uint4 v) {
    float f[8];
    chunk_to_f(v, f);
    float part = 0.0f;
#pragma unroll
    for (int e = 0; e < 8; ++e) part = fmaf(f[e], f[e], part);
    return part;
}

// Chunk c of input token pos for the finish phase, wherever the sample's rows are: one type
// for every layout, so the finish phase is compiled once (its code is fetched cold after every
// flush of L2, and a second copy for another layout made stages slower).
//   rows in global memory (g != null): chunk c of token pos at g + pos * rb + 16 c;
//   rows in shared memory: CLS from its staged copy; row r of a half (positions 2, 4, ... or
//   1, 3, ...) at h + (r / 8) G + (r % 8) 128, its 16-byte chunk c (c / 8) K + 16 ((c % 8) ^
//   (r % 8)) further (ring: h = the half's base in stage 0, G = 1024, K = kbs; grouped layout:
//   h = the half's first group, G = n_kb KB, K = 1024).
// The branch is uniform over the CTA.
struct RowLoader {
    const unsigned char *g;   // the sample's first row in global memory, or null
    uint32_t rb;               // bytes of a token row
    const unsigned char *cls, *hA, *hB;
    uint32_t G, K;
    __device__ __forceinline__ uint4 operator()(int pos, int c) const {
        if (g) return ldg16(g + (size_t)pos * rb + (size_t)c * 16);
        if (pos == 0) return *reinterpret_cast<const uint4 *>(cls + (size_t)c * 16);
        const bool isB = pos & 1;
        const unsigned r = (unsigned)(isB ? (pos - 1) >> 1 : (pos - 2) >> 1);
        const unsigned x = r & 7u, cc = (unsigned)c;
        const unsigned char *base = (isB ? hB : hA) + (size_t)(r >> 3) * G + (size_t)(cc >> 3) * K;
        return *reinterpret_cast<const uint4 *>(base + x * 128u + (((cc & 7u) ^ x) << 4));
    }
};

// The ring of K-block stages of one sample, sized for it: S stages of kbs bytes, K-block kb
// in stage kb % S with half A at the stage's start and half B after rowsA rows.  The boxes of
// one K-block: half A then half B, in 32-row boxes while 32 rows remain, then 8-row boxes.
struct Ring {
    int S, rowsA, rowsB, npad, nbA, per_kb;
    uint32_t kbs;
};
__device__ __forceinline__ Ring ring_for(int nA, int nB, int nkb, const TcGeometry &g) {
    Ring R;
    R.rowsA = (nA + 7) & ~7;
    R.rowsB = (nB + 7) & ~7;
    R.npad = (nB + 15) & ~15;   // MMA N: |B| rounded up to 16
    R.kbs = (uint32_t)(R.rowsA + R.rowsB) * 128u;
    // An MMA reads 128 A rows and npad B rows from a stage, past its end when the sample is
    // small, which stays inside the buffer.
    const uint32_t reach = (uint32_t)max(16384, (R.rowsA + R.npad) * 128);
    int S = min(min(nkb, kMaxStages), (int)(g.stage_region / R.kbs));
    while (S > 1 && (uint32_t)(S - 1) * R.kbs + reach > g.usable) --S;
    R.S = S;
    R.nbA = (nA >> 5) + (((nA & 31) + 7) >> 3);
    R.per_kb = R.nbA + (nB >> 5) + (((nB & 31) + 7) >> 3);
    return R;
}
// Box b of K-block kb of the sample whose rows start at `start` (half A: positions 2, 4, ...,
// half B: 1, 3, ..., each contiguous in the even or odd row view).
__device__ __forceinline__ void issue_box(const TcMaps &maps, const Ring &R, int start, int nA, int nB,
                                          unsigned char *sm, unsigned long long *bar_full, int kb, int b) {
    const int st = kb % R.S;
    const int half = b >= R.nbA ? 1 : 0;
    const int q = half ? b - R.nbA : b;
    const int n32 = (half ? nB : nA) >> 5;
    const bool big = q < n32;
    const int row0 = big ? q * 32 : n32 * 32 + (q - n32) * 8;
    const bool odd = half ? ((start + 1) & 1) : ((start + 2) & 1);
    const CUtensorMap *map = big ? (odd ? &maps.o32 : &maps.e32) : (odd ? &maps.o8 : &maps.e8);
    const int y = half ? (start + 1) >> 1 : (start + 2) >> 1;
    const uint32_t dst = smem_addr(sm + (half ? (size_t)R.rowsA * 128 : (size_t)0) + (size_t)st * R.kbs + (size_t)row0 * 128);
    tma_load_2d(dst, map, kb * 64, y + row0, smem_addr(&bar_full[st]));
}
// Every barrier a ring can use, from one thread at kernel entry: the fence that publishes the
// initialisation waits for the thread's outstanding memory operations, so it runs before the
// thread has issued any.
__device__ __forceinline__ void ring_barriers_init(unsigned long long *bar_full, unsigned long long *bar_empty,
                                                   unsigned long long *bar_done) {
    for (int st = 0; st < kMaxStages; ++st) {
        mbar_init(smem_addr(&bar_full[st]), 1);
        mbar_init(smem_addr(&bar_empty[st]), 1 + kTcThreads / 32);
    }
    mbar_init(smem_addr(bar_done), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// From the 32 lanes of one warp, once the barriers are initialised and that is visible to the
// warp: the first min(S, nkb) K-blocks.
__device__ __forceinline__ void ring_start(const TcMaps &maps, const Ring &R, int start, int nA, int nB, int nkb,
                                           unsigned char *sm, unsigned long long *bar_full) {
    const int lane = threadIdx.x & 31;
    __syncwarp();
    const int S0 = min(R.S, nkb);
    if (lane < S0) mbar_expect_tx(smem_addr(&bar_full[lane]), R.kbs);
    for (int t = lane; t < S0 * R.per_kb; t += 32)
        issue_box(maps, R, start, nA, nB, sm, bar_full, t / R.per_kb, t % R.per_kb);
}
// A sample that fits in shared memory, grouped: half A in 8-row groups g at g * nkb KB, each
// group [K-block][8 rows][128 B], half B after it the same way, all behind bar_full[0]; one box
// per group (the K-block ring needs per_kb boxes per K-block).  The rows of the last group past
// the half belong to the next sample or lie past the tensor (zero fill) and are never used.
// From the 32 lanes of one warp, once the barriers are initialised and that is visible to it.
__device__ __forceinline__ void group_start(const TcMaps &maps, const Ring &R, int start, int nkb, unsigned char *sm,
                                            unsigned long long *bar_full) {
    const int lane = threadIdx.x & 31;
    const int GA = R.rowsA >> 3, GB = R.rowsB >> 3;
    const uint32_t gstride = (uint32_t)nkb * 1024u;
    __syncwarp();
    if (lane == 0) mbar_expect_tx(smem_addr(&bar_full[0]), (uint32_t)(GA + GB) * gstride);
    const bool oddA = (start + 2) & 1, oddB = (start + 1) & 1;
    const int yA = (start + 2) >> 1, yB = (start + 1) >> 1;
    for (int b = lane; b < GA + GB; b += 32) {
        const bool isB = b >= GA;
        const int q = isB ? b - GA : b;
        const CUtensorMap *map = (isB ? oddB : oddA) ? &maps.go : &maps.ge;
        const uint32_t dst = smem_addr(sm + (size_t)(isB ? GA + q : q) * gstride);
        tma_load_3d(dst, map, 0, (isB ? yB : yA) + 8 * q, 0, smem_addr(&bar_full[0]));
    }
}
// The sample's token sizes and scores and its CLS row into shared memory (cp.async, one
// group; waited for in meta_init_rest).
__device__ __forceinline__ void prefetch_own(const ImageParams &p, int start, int N, const MetaPtrs &m, uint4 *cls) {
    for (int pos = threadIdx.x; pos < N; pos += kTcThreads) {
        cp_async4(&m.tsize[pos], p.sizes + start + pos);
        if (p.scores) cp_async4(&m.tscore[pos], p.scores + start + pos);
    }
    const uint4 *row = reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(p.x) + (long long)start * p.dim);
    for (int c = threadIdx.x; c < p.dim / 8; c += kTcThreads) cp_async16(&cls[c], row + c);
    cp_async_commit();
}

__global__ void __launch_bounds__(kTcThreads, 2)
    k_image_tc(const __grid_constant__ TcMaps maps, ImageParams p, TcGeometry g) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) unsigned long long bar_full[kMaxStages], bar_empty[kMaxStages], bar_done;
    __shared__ uint32_t tmem_base;
    __shared__ int s_fail;
    __shared__ unsigned long long half_best[kTcThreads / 2];

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // Tensor memory first: an SM admits another CTA of a kernel that allocates tensor
    // memory only once the resident one has given up its allocation permit.
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(g.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // the tensor maps' descriptors travel while the sample's metadata loads
    if (tid >= 32 && tid < 36) {
        const CUtensorMap *mp = tid == 32 ? &maps.e32 : tid == 33 ? &maps.o32 : tid == 34 ? &maps.e8 : &maps.o8;
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(mp)) : "memory");
    }
    // the ring's barriers, before this thread issues any memory operation (warp 0 issues the
    // tokens' loads after a CTA barrier: the fused plan's, or the one below)
    if (tid == 36) ring_barriers_init(bar_full, bar_empty, &bar_done);
    if (g.grouped && (tid == 38 || tid == 39))
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tid == 38 ? &maps.ge : &maps.go)) : "memory");
    if (tid == 0) s_fail = 0;   // visible after the barriers below, before any other write
    const int nkb = g.n_kb;
    MetaPtrs m(sm, meta_layout(p.in.max_tokens, g.meta_base));
    uint4 *cls = reinterpret_cast<uint4 *>(sm + g.cls_base);
    // launched as a programmatic dependent of the exit check: everything above (tensor memory,
    // barriers, descriptor prefetch) and the plan's loads of this call's own inputs overlap that
    // kernel's end; the exit mask is read after `griddepcontrol.wait` (without a programmatic
    // predecessor the wait returns at once)
    SampleInfo s;
    if (!sample_begin<kTcThreads>(p, blockIdx.x, s, true)) {   // uniform over the CTA
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        if (warp == 0)
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(g.tmem_cols)
                         : "memory");
        return;
    }
    if (!p.fused_plan) __syncthreads();   // uniform: the fused plan has barriers of its own
    const bool dec = s.decide;
    const Ring R = ring_for(s.nA, s.nB, nkb, g);
    const int S = R.S, npad = R.npad;
    const uint32_t kbs = R.kbs;
    unsigned char *regA = sm;                         // stage st, half A: regA + st * kbs
    unsigned char *regB = sm + (size_t)R.rowsA * 128;  // stage st, half B: regB + st * kbs (ring layout)
    auto produce = [&](int kb) {   // a whole K-block from one thread
        mbar_expect_tx(smem_addr(&bar_full[kb % S]), kbs);
        for (int b = 0; b < R.per_kb; ++b) issue_box(maps, R, s.start, s.nA, s.nB, sm, bar_full, kb, b);
    };

    // the sample's sizes, scores and CLS row first (a few KB that would otherwise queue behind the
    // bulk loads), then its tokens: the grouped layout or the ring's first stages (warp 0)
    prefetch_own(p, s.start, s.N, m, cls);
    const bool grouped = g.grouped && S >= nkb;   // the layout of this sample (uniform)
    const uint32_t gstride = (uint32_t)nkb * 1024u;
    unsigned char *gB = sm + (size_t)(R.rowsA >> 3) * gstride;   // grouped layout: half B
    if (warp == 0 && dec) {
        if (grouped)
            group_start(maps, R, s.start, nkb, sm, bar_full);
        else
            ring_start(maps, R, s.start, s.nA, s.nB, nkb, sm, bar_full);
    }
    meta_init_rest<kTcThreads>(p, s, m);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

    if (dec) {
        const uint32_t tmem = tmem_base;

        // instruction descriptor: f32 accumulator, bf16 A and B, K-major, N = |B| rounded to 16, M = 128
        const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(npad >> 3) << 17) | (8u << 24);
        // Squared row norms: for a sample that stays resident, after all stages landed with
        // kT threads per row; otherwise one thread per row, K-block by K-block as the ring turns.
        const bool resident = S >= nkb;
        const bool isA = tid < 128;
        const int row = isA ? tid : tid - 128;
        const bool has_row = !resident && row < (isA ? s.nA : s.nB);
        float ss = 0.0f, sc = 0.0f;
        bool ok = true;
        if (grouped) {   // everything behind one barrier; all products at once
            if (!mbar_wait(smem_addr(&bar_full[0]), 0u)) {
                ok = false;
            } else if (tid == 32) {
                const uint32_t a0 = smem_addr(sm), b0 = smem_addr(gB);
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        umma_bf16(tmem, sw128_desc_sbo(a0 + kb * 1024 + k * 32, gstride),
                                  sw128_desc_sbo(b0 + kb * 1024 + k * 32, gstride), idesc, (kb | k) ? 1u : 0u);
                umma_commit(smem_addr(&bar_done));
            }
        }
        for (int kb = 0; kb < (grouped ? 0 : nkb); ++kb) {
            const int st = kb % S;
            const uint32_t par = (uint32_t)(kb / S) & 1u;
            if (!mbar_wait(smem_addr(&bar_full[st]), par)) {
                ok = false;
                break;
            }
            if (tid == 32) {
                const uint32_t a0 = smem_addr(regA + (size_t)st * kbs), b0 = smem_addr(regB + (size_t)st * kbs);
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), idesc, (kb | k) ? 1u : 0u);
                umma_commit(smem_addr(&bar_empty[st]));
                if (kb == nkb - 1) umma_commit(smem_addr(&bar_done));
            }
            if (has_row) {   // squared norm of this thread's row, chunk by chunk
                const unsigned char *base = (isA ? regA : regB) + (size_t)st * kbs + row * 128;
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    neumaier_add(ss, sc, chunk_sq(*reinterpret_cast<const uint4 *>(base + ((j ^ (row & 7)) << 4))));
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_addr(&bar_empty[st]));
            if (tid == 0 && kb + S < nkb) {   // refill this stage once everyone is done with it
                if (!mbar_wait(smem_addr(&bar_empty[st]), par)) {
                    ok = false;
                    break;
                }
                produce(kb + S);
            }
        }
        if (!ok) atomicOr(&s_fail, 1);
        int nrow = row;        // row of this thread: A rows, then B rows
        bool owner = has_row;  // writes the row's inverse norm
        if (resident) {   // uniform over the CTA: every lane reaches the shuffles
            // kT threads per row (the largest power of two up to 8 that fits), each taking
            // every kT-th chunk of the row; the partial sums meet by shuffles
            const int R = s.nA + s.nB;
            const int kT = R <= 32 ? 8 : R <= 64 ? 4 : R <= 128 ? 2 : 1;
            const int r = tid / kT, part = tid % kT;
            if (r < R) {
                const bool rA = r < s.nA;
                const int rr = rA ? r : r - s.nA;
                const unsigned char *base = grouped ? (rA ? sm : gB) + (size_t)(rr >> 3) * gstride + (rr & 7) * 128
                                                    : (rA ? regA : regB) + (size_t)rr * 128;
                const uint32_t kstep = grouped ? 1024u : kbs;   // bytes from one K-block of the row to the next
                for (int c = part; c < nkb * 8; c += kT)
                    neumaier_add(ss, sc, chunk_sq(*reinterpret_cast<const uint4 *>(
                                             base + (size_t)(c >> 3) * kstep + (((c & 7) ^ (rr & 7)) << 4))));
            }
            for (int mk = 1; mk < kT; mk <<= 1) {   // kT divides 32: groups stay inside a warp
                const float oss = __shfl_xor_sync(0xFFFFFFFFu, ss, mk), osc = __shfl_xor_sync(0xFFFFFFFFu, sc, mk);
                neumaier_add(ss, sc, oss);
                sc = __fadd_rn(sc, osc);
            }
            owner = r < R && part == 0;
            nrow = r;
        } else if (has_row) {
            nrow = isA ? row : s.nA + row;
        }
        if (owner) {
            const float sq = __fadd_rn(ss, sc);
            if (!isfinite(sq)) raise_status(p.status, FUSION_DEV_NONFINITE);
            const float inv = 1.0f / fmaxf(sqrtf(sq), 1e-12f);
            if (nrow < s.nA)
                m.inv_a[nrow] = inv;
            else
                m.inv_b[nrow - s.nA] = inv;
        }
        __syncthreads();
        bool mma_ok = s_fail == 0 && mbar_wait(smem_addr(&bar_done), 0);
        if (!mma_ok) atomicOr(&s_fail, 2);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        __syncthreads();
        if (s_fail == 0) {
            // epilogue: thread -> A row (tid % 128); the two warpgroups take the low / high columns
            const int wg = tid >> 7;
            const int r = tid & 127;
            const int half_cols = ((npad / 16 + 1) / 2) * 16;
            const int c_lo = wg ? half_cols : 0, c_hi = wg ? npad : half_cols;
            const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
            const float ia = r < s.nA ? m.inv_a[r] : 0.0f;
            // the largest cosine of the thread's columns and its lowest column: the columns go up,
            // so a strict comparison keeps the first of equal values (and -0 equals +0)
            float bv = -INFINITY;
            int bi = -1;
            for (int c0 = c_lo; c0 < c_hi; c0 += 16) {
                uint32_t v[16];
                tmem_ld16(lane_addr + (uint32_t)c0, v);
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int col = c0 + e;
                    if (col < s.nB) {
                        const float cs = (__uint_as_float(v[e]) * ia) * m.inv_b[col];
                        if (cs > bv || bi < 0) {
                            bv = cs;
                            bi = col;
                        }
                    }
                }
            }
            const unsigned long long bk = (r < s.nA && bi >= 0) ? rank_key(bv, bi) : 0ull;
            if (wg == 1) half_best[r] = bk;
            __syncthreads();
            if (wg == 0 && r < s.nA) {
                const unsigned long long o = half_best[r];
                m.best[r] = o > bk ? o : bk;
            }
        } else {
            if (tid == 0) raise_status(p.status, FUSION_DEV_TIMEOUT);
        }
        __syncthreads();
        if (s_fail == 0) select_top_r<kTcThreads>(s, m);
    }

    if (s_fail == 0) {
        const uint32_t rb = (uint32_t)p.dim * 2u;   // bytes of a token row
        RowLoader ld{reinterpret_cast<const unsigned char *>(p.x) + (size_t)s.start * rb, rb,
                     reinterpret_cast<const unsigned char *>(cls), nullptr, nullptr, 0u, 0u};
        if (dec && S >= nkb && p.keys_alias) {   // the whole sample is in shared memory
            ld.g = nullptr;
            ld.hA = sm;
            ld.hB = grouped ? gB : regB;
            ld.G = grouped ? gstride : 1024u;
            ld.K = grouped ? 1024u : kbs;
        }
        finish_sample<__nv_bfloat16, kTcThreads>(p, s, m, ld);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(g.tmem_cols)
                     : "memory");
}

// ---------------------------------------------------------------------------
// Samples whose halves exceed one tile (|A| or |B| above 128; ViT-L/16 at 384: 288 x 288 x
// 1024): one CTA per SM, tensor memory of 256 or 512 columns.  Half A is taken in M-tiles of
// 128 rows; half B in N-blocks of at most 256 columns, all of them held in tensor memory at once.
// For every M-tile the K-blocks of (that tile's A rows, all B rows) stream by TMA through the
// ring (stage q = M-tile q / n_kb, K-block q % n_kb); the B rows are loaded again for every
// M-tile (from L2 after the first).  The tile's products accumulate over its K-blocks, its
// epilogue keeps each A row's best column, and the next tile reuses the accumulators.  Row
// norms: A rows of each tile and, during the first tile, the B rows, one thread per row.
// ---------------------------------------------------------------------------
constexpr int kTiledMaxStages = 8;

__global__ void __launch_bounds__(kTcThreads, 1)
    k_image_tc_tiled(const __grid_constant__ TcMaps maps, ImageParams p, TcGeometry g) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) unsigned long long bar_full[kTiledMaxStages], bar_empty[kTiledMaxStages], bar_done, bar_drain;
    __shared__ uint32_t tmem_base;
    __shared__ int s_fail;
    __shared__ unsigned long long half_best[kTcThreads / 2];

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_base)),
                     "r"(g.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid >= 32 && tid < 36) {
        const CUtensorMap *mp = tid == 32 ? &maps.e32 : tid == 33 ? &maps.o32 : tid == 34 ? &maps.e8 : &maps.o8;
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(mp)) : "memory");
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");   // as in k_image_tc: the exit check's grid first
    SampleInfo s;
    if (!sample_begin<kTcThreads>(p, blockIdx.x, s)) {
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        if (warp == 0)
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(g.tmem_cols)
                         : "memory");
        return;
    }
    const bool dec = s.decide;
    const int nkb = g.n_kb;
    int issued = 0;   // stages issued (thread 0's count; warp 0 issues the first ones)
    const int nM = (s.nA + 127) >> 7;               // M-tiles of half A
    const int rowsB = (s.nB + 7) & ~7;
    const int npad = (s.nB + 15) & ~15;             // columns of the product
    const int nNB = (npad + 255) >> 8;              // N-blocks of at most 256 columns
    // stage: [128 A rows][rowsB B rows] x 128 B; an MMA reads 128 A rows and up to npad B rows
    const uint32_t aBytes = 128u * 128u;
    const uint32_t kbs = aBytes + (uint32_t)rowsB * 128u;
    const uint32_t reach = aBytes + (uint32_t)npad * 128u;
    const int nq = nM * nkb;
    int S = min(min(nq, kTiledMaxStages), (int)(g.stage_region / kbs));
    while (S > 1 && (uint32_t)(S - 1) * kbs + reach > g.usable) --S;
    const int yB = (s.start + 1) >> 1, yA0 = (s.start + 2) >> 1;
    const bool oddA = (s.start + 2) & 1, oddB = (s.start + 1) & 1;
    // boxes of stage q: the A rows of its M-tile (32-row boxes, then 8-row boxes), then all B rows
    auto tile_rows = [&](int mt) { return min(128, s.nA - mt * 128); };
    auto nboxes = [&](int n) { return (n >> 5) + (((n & 31) + 7) >> 3); };
    auto stage_tx = [&](int mt) { return (uint32_t)(((tile_rows(mt) + 7) & ~7) + rowsB) * 128u; };
    auto issue_box = [&](int q, int b) {
        const int st = q % S, mt = q / nkb, kb = q - mt * nkb;
        const int nA_t = tile_rows(mt);
        const int nbA = nboxes(nA_t);
        const bool half = b >= nbA;   // B rows
        const int qq = half ? b - nbA : b;
        const int n = half ? s.nB : nA_t;
        const int n32 = n >> 5;
        const bool big = qq < n32;
        const int row0 = big ? qq * 32 : n32 * 32 + (qq - n32) * 8;
        const bool odd = half ? oddB : oddA;
        const CUtensorMap *map = big ? (odd ? &maps.o32 : &maps.e32) : (odd ? &maps.o8 : &maps.e8);
        unsigned char *base = sm + (size_t)st * kbs + (half ? aBytes : 0u);
        tma_load_2d(smem_addr(base + (size_t)row0 * 128), map, kb * 64, (half ? yB : yA0 + mt * 128) + row0,
                    smem_addr(&bar_full[st]));
    };
    auto boxes_of = [&](int q) { return nboxes(tile_rows(q / nkb)) + nboxes(s.nB); };
    auto produce = [&](int q) {
        mbar_expect_tx(smem_addr(&bar_full[q % S]), stage_tx(q / nkb));
        const int nb = boxes_of(q);
        for (int b = 0; b < nb; ++b) issue_box(q, b);
    };

    MetaPtrs m(sm, meta_layout(p.in.max_tokens, g.meta_base));
    meta_prefetch<kTcThreads>(p, s, m);
    if (warp == 0) {
        if (lane == 0) s_fail = 0;
        if (dec) {
            if (lane < S) {
                mbar_init(smem_addr(&bar_full[lane]), 1);
                mbar_init(smem_addr(&bar_empty[lane]), 1 + kTcThreads / 32);
            }
            if (lane == 31) mbar_init(smem_addr(&bar_done), 1);
            if (lane == 30) mbar_init(smem_addr(&bar_drain), 1);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            issued = min(S, nq);
            for (int q = 0; q < min(S, nq); ++q) {   // each stage's boxes from all lanes
                if (lane == 0) mbar_expect_tx(smem_addr(&bar_full[q]), stage_tx(q / nkb));
                __syncwarp();
                const int nb = boxes_of(q);
                for (int b = lane; b < nb; b += 32) issue_box(q, b);
            }
        }
    }
    meta_init_rest<kTcThreads>(p, s, m);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

    if (dec) {
        const uint32_t tmem = tmem_base;
        bool ok = true;
        for (int mt = 0; mt < nM && ok; ++mt) {
            const int nA_t = tile_rows(mt);
            // norms: thread t < 128 owns A row t of this tile; during tile 0 threads 128.. own the
            // B rows 128 apart
            float ssA = 0.0f, scA = 0.0f;
            float ssB[4] = {0.0f, 0.0f, 0.0f, 0.0f}, scB[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            for (int kb = 0; kb < nkb; ++kb) {
                const int q = mt * nkb + kb;
                const int st = q % S;
                const uint32_t par = (uint32_t)(q / S) & 1u;
                if (!mbar_wait(smem_addr(&bar_full[st]), par)) {
                    ok = false;
                    break;
                }
                const unsigned char *stA = sm + (size_t)st * kbs, *stB = stA + aBytes;
                if (tid == 32) {
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    for (int nb = 0; nb < nNB; ++nb) {
                        const int ncols = min(256, npad - nb * 256);
                        const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(ncols >> 3) << 17) |
                                               (8u << 24);
                        const uint32_t a0 = smem_addr(stA), b0 = smem_addr(stB + (size_t)nb * 256 * 128);
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            umma_bf16(tmem + (uint32_t)(nb * 256), sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32),
                                      idesc, (kb | k) ? 1u : 0u);
                    }
                    umma_commit(smem_addr(&bar_empty[st]));
                    if (kb == nkb - 1) umma_commit(smem_addr(&bar_done));
                }
                if (tid < 128) {
                    if (tid < nA_t) {
                        const unsigned char *rb = stA + tid * 128;
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            neumaier_add(ssA, scA, chunk_sq(*reinterpret_cast<const uint4 *>(rb + ((j ^ (tid & 7)) << 4))));
                    }
                } else if (mt == 0) {
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int br = tid - 128 + u * 128;
                        if (br < s.nB) {
                            const unsigned char *rb = stB + br * 128;
#pragma unroll
                            for (int j = 0; j < 8; ++j)
                                neumaier_add(ssB[u], scB[u],
                                             chunk_sq(*reinterpret_cast<const uint4 *>(rb + ((j ^ (br & 7)) << 4))));
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_empty[st]));
                if (tid == 0 && q + S < nq) {   // refill this stage (possibly with the next tile's K-block)
                    if (!mbar_wait(smem_addr(&bar_empty[st]), par)) {
                        ok = false;
                        break;
                    }
                    produce(q + S);
                    ++issued;
                }
            }
            if (!ok) atomicOr(&s_fail, 1);
            if (tid < nA_t) {
                const float sq = __fadd_rn(ssA, scA);
                if (!isfinite(sq)) raise_status(p.status, FUSION_DEV_NONFINITE);
                m.inv_a[mt * 128 + tid] = 1.0f / fmaxf(sqrtf(sq), 1e-12f);
            }
            if (mt == 0 && tid >= 128) {
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int br = tid - 128 + u * 128;
                    if (br < s.nB) {
                        const float sq = __fadd_rn(ssB[u], scB[u]);
                        if (!isfinite(sq)) raise_status(p.status, FUSION_DEV_NONFINITE);
                        m.inv_b[br] = 1.0f / fmaxf(sqrtf(sq), 1e-12f);
                    }
                }
            }
            __syncthreads();
            const bool mma_ok = s_fail == 0 && mbar_wait(smem_addr(&bar_done), (uint32_t)mt & 1u);
            if (!mma_ok) atomicOr(&s_fail, 2);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            __syncthreads();
            if (s_fail != 0) {
                ok = false;
                break;
            }
            // epilogue of the tile: thread -> A row (tid % 128); the warpgroups split the columns
            const int wg = tid >> 7, r = tid & 127;
            const int half_cols = ((npad / 16 + 1) / 2) * 16;
            const int c_lo = wg ? half_cols : 0, c_hi = wg ? npad : half_cols;
            const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
            const int arow = mt * 128 + r;
            const float ia = r < nA_t ? m.inv_a[arow] : 0.0f;
            float bv = -INFINITY;   // as in k_image_tc: strict comparison over rising columns
            int bi = -1;
            for (int c0 = c_lo; c0 < c_hi; c0 += 16) {
                uint32_t v[16];
                tmem_ld16(lane_addr + (uint32_t)c0, v);
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int col = c0 + e;
                    if (col < s.nB) {
                        const float cs = (__uint_as_float(v[e]) * ia) * m.inv_b[col];
                        if (cs > bv || bi < 0) {
                            bv = cs;
                            bi = col;
                        }
                    }
                }
            }
            const unsigned long long bk = (r < nA_t && bi >= 0) ? rank_key(bv, bi) : 0ull;
            if (wg == 1) half_best[r] = bk;
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncthreads();   // the next tile's products overwrite the accumulators after this
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            if (wg == 0 && r < nA_t) {
                const unsigned long long o = half_best[r];
                m.best[arow] = o > bk ? o : bk;
            }
            __syncthreads();   // half_best is reused by the next tile
        }
        if (s_fail != 0) {
            // a wait gave up: let the copies and products in flight land (bounded) before the
            // shared and tensor memory are released
            if (tid == 0) {
                raise_status(p.status, FUSION_DEV_TIMEOUT);
                for (int q = max(0, issued - S); q < issued; ++q)
                    (void)mbar_wait(smem_addr(&bar_full[q % S]), (uint32_t)(q / S) & 1u);
            }
            if (tid == 32) {
                umma_commit(smem_addr(&bar_drain));
                (void)mbar_wait(smem_addr(&bar_drain), 0u);
            }
        } else {
            select_top_r<kTcThreads>(s, m);
        }
        __syncthreads();
    }
    if (s_fail == 0) {
        const GlobalLoader<__nv_bfloat16> gl{reinterpret_cast<const __nv_bfloat16 *>(p.x), (long long)s.start, p.dim};
        finish_sample<__nv_bfloat16, kTcThreads>(p, s, m, gl);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(g.tmem_cols)
                     : "memory");
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int ceil8(int v) { return (v + 7) & ~7; }

}  // namespace

namespace {
// Geometry of k_image_tc_tiled: one CTA per SM, a ring of [128 A rows | all B rows] stages.
TcGeometry tiled_geometry(int max_tokens, int kdim) {
    TcGeometry g{};
    const int nBmax = max_tokens / 2;
    const int npad_max = (nBmax + 15) & ~15;
    g.tiled = 1;
    g.n_kb = kdim / 64;
    g.tmem_cols = npad_max <= 256 ? 256 : 512;
    g.kb_a = 128u * 128u;
    g.kb_b = (uint32_t)ceil8(nBmax) * 128u;
    const size_t per_stage = g.kb_a + g.kb_b;
    const size_t reach = g.kb_a + (size_t)npad_max * 128;
    const size_t budget = 227 * 1024 - 4096;   // room for static shared memory
    auto need = [&](int S) {
        const size_t meta_base = (size_t)S * per_stage + 2048;
        return std::max(meta_layout(max_tokens, meta_base).total, (size_t)(S - 1) * per_stage + reach);
    };
    int S = kTiledMaxStages;
    while (S > 2 && need(S) + 1024 > budget) --S;
    if (need(S) + 1024 > budget) return TcGeometry{};
    g.stages = S;
    g.stage_region = (uint32_t)(S * per_stage);
    g.meta_base = (uint32_t)(S * per_stage + 2048);
    g.usable = (uint32_t)need(S);
    g.smem = g.usable + 1024;
    g.ok = 1;
    return g;
}
}  // namespace

TcGeometry image_tc_geometry(int dtype, int max_tokens, int kdim, int dim, long long max_rows, int do_merge,
                             int stage_budget_kb) {
    TcGeometry g{};
    if (dtype != FUSION_BF16 || !do_merge || kdim % 64 != 0 || max_rows < 2) return g;
    const int nAmax = (max_tokens - 1) / 2, nBmax = max_tokens / 2;
    if (nAmax > 128 || nBmax > 128) return tiled_geometry(max_tokens, kdim);
    g.n_kb = kdim / 64;
    g.kb_a = (uint32_t)ceil8(nAmax > 0 ? nAmax : 1) * 128u;
    g.kb_b = (uint32_t)ceil8(nBmax > 0 ? nBmax : 1) * 128u;
    int cols = 32;
    while (cols < ((nBmax + 15) & ~15)) cols <<= 1;
    g.tmem_cols = cols;
    const size_t per_stage = g.kb_a + g.kb_b;
    // the largest read from a stage base: 128 A rows, or half A and npad B rows
    const size_t npad_max = (size_t)((nBmax + 15) & ~15);
    const size_t reach = std::max<size_t>(16384, g.kb_a + npad_max * 128);
    size_t budget = (size_t)stage_budget_kb * 1024;
    if (budget > 227 * 1024 - 4096) budget = 227 * 1024 - 4096;   // room for static shared memory
    // usable bytes for S stages at max_tokens: the ring, the metadata, the CLS row (dim bf16)
    auto need = [&](int S) {
        const size_t meta_base = (size_t)S * per_stage + 2048;
        return std::max(meta_layout(max_tokens, meta_base).total + (size_t)dim * 2, (size_t)(S - 1) * per_stage + reach);
    };
    int S = g.n_kb < kMaxStages ? g.n_kb : kMaxStages;
    while (S > 2 && need(S) + 1024 > budget) --S;
    if (need(S) + 1024 > budget) return g;
    g.stages = S;
    g.stage_region = (uint32_t)(S * per_stage);
    g.meta_base = (uint32_t)(S * per_stage + 2048);
    g.cls_base = (uint32_t)meta_layout(max_tokens, g.meta_base).total;
    g.usable = (uint32_t)need(S);
    // The grouped layout for samples that fit: an MMA reads 128 A rows, 16 groups of n_kb KB from
    // the start of the buffer, and up to one group past half B (npad rows), so the buffer must
    // cover both; when the budget allows it, it does.
    const size_t gstride = (size_t)g.n_kb * 1024;
    const size_t g_need = std::max({(size_t)g.usable, 16 * gstride, (size_t)g.stage_region + gstride});
    if (g_need + 1024 <= budget) {
        g.grouped = 1;
        g.usable = (uint32_t)g_need;
    }
    g.smem = g.usable + 1024;
    g.ok = 1;
    return g;
}

cudaError_t launch_image_tc(const ImageParams &p, const TcGeometry &g, cudaStream_t s, bool pdl) {
    if (p.in.max_batch == 0) return cudaSuccess;
    EncodeTiledFn enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    TcMaps maps{};
    const cuuint64_t rows_even = (cuuint64_t)((p.in.max_rows + 1) / 2), rows_odd = (cuuint64_t)(p.in.max_rows / 2);
    const char *keys = reinterpret_cast<const char *>(p.keys);
    for (int i = 0; i < 4; ++i) {
        const int odd = i & 1, box_rows = i < 2 ? 32 : 8;
        cuuint64_t dims[2] = {(cuuint64_t)p.kdim, odd ? rows_odd : rows_even};
        cuuint64_t strides[1] = {(cuuint64_t)p.kdim * 2 * 2};   // every other row
        cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
        cuuint32_t estr[2] = {1, 1};
        CUtensorMap *dst = i == 0 ? &maps.e32 : i == 1 ? &maps.o32 : i == 2 ? &maps.e8 : &maps.o8;
        void *base = const_cast<char *>(keys + (odd ? (size_t)p.kdim * 2 : 0));
        if (enc(dst, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    for (int odd = 0; odd < 2 && g.grouped; ++odd) {   // (64 dims, row, K-block), box 8 rows x all K-blocks
        cuuint64_t dims[3] = {64, odd ? rows_odd : rows_even, (cuuint64_t)(p.kdim / 64)};
        cuuint64_t strides[2] = {(cuuint64_t)p.kdim * 2 * 2, 128};
        cuuint32_t box[3] = {64, 8, (cuuint32_t)(p.kdim / 64)};
        cuuint32_t estr[3] = {1, 1, 1};
        void *base = const_cast<char *>(keys + (odd ? (size_t)p.kdim * 2 : 0));
        if (enc(odd ? &maps.go : &maps.ge, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    auto kernel = g.tiled ? k_image_tc_tiled : k_image_tc;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem);
    if (e != cudaSuccess) return e;
    // the largest shared-memory carveout, so that both CTAs of an SM are resident from the start
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.in.max_batch);
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = g.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, maps, p, g);
}

}  // namespace fz
