// The per-call plan: validates the ragged batch, decides which samples continue,
// computes every sample's output token count and scans them into the output
// offsets.  Output counts follow from the inputs alone: merging removes
// r_eff = clamp(r, 0, floor(P/2)) tokens (Sec. III-C) and pruning then keeps
// 1 + ceil(rho * P') (Sec. III-E), so the scan needs no merge decision.
#pragma once

#include "common.cuh"

namespace fz {

struct PlanArgs {
    Ragged in;
    int merge;                 // counts include merging
    int prune;                 // counts include pruning
    const int *r;              // [*] merge counts (by original id)
    const float *rho;          // [*] keep ratios (by original id)
    const uint8_t *exit_mask;  // [B] 1 = exits (leaves the batch); NULL = all continue
    int *offsets_out;          // [max_batch + 1]
    int *ids_out;              // [max_batch] or NULL
    int *batch_out;            // device scalar or NULL
    int *slot;                 // workspace [max_batch]: output sample of every input sample, -1 if gone
    int *plan;                 // workspace [4]: ok flag, survivor count
    int *status;
};

// Samples staged in shared memory per round of the plan.
constexpr int kPlanChunk = 2048;

// Shared memory run_plan needs for a block of nt threads: per round the chunk's offsets, ids,
// counts and flags, then the block scan's scratch.
__host__ __device__ inline size_t plan_smem_bytes(int nt) {
    return (size_t)(3 * kPlanChunk + 1 + 2 * nt + 40) * sizeof(int) + kPlanChunk;
}

// Run by ONE thread block (any size, multiple of 32) with plan_smem_bytes(blockDim.x) of shared
// memory at `smem`.  The batch is taken in rounds of kPlanChunk samples: the round's offsets,
// ids and exit flags are staged in shared memory with every load in flight at once, then the
// merge counts and keep ratios by id; each thread sums a contiguous segment of the round, the
// segment totals are scanned, and each thread writes its segment's slots, offsets and ids.
__device__ inline void run_plan(const PlanArgs &a, int *smem) {
    const int nt = blockDim.x;
    int *o_s = smem;                          // [kPlanChunk + 1] offsets of the round
    int *id_s = o_s + kPlanChunk + 1;         // [kPlanChunk] ids
    int *cnt_s = id_s + kPlanChunk;           // [kPlanChunk] output counts (0 when the sample is gone)
    int *flags = cnt_s + kPlanChunk;          // [nt] segment survivor counts, then their scan
    int *cnts = flags + nt;                   // [nt] segment row counts, then their scan
    int *tmp = cnts + nt;                     // 40 ints
    unsigned char *sv_s = reinterpret_cast<unsigned char *>(tmp + 40);   // [kPlanChunk] survives
    __shared__ int s_bad, s_nonfinite;
    const int t = threadIdx.x;
    if (t == 0) {
        s_bad = 0;
        s_nonfinite = 0;
    }
    __syncthreads();

    int B = device_batch(a.in);
    if (B < 0) {
        if (t == 0) {
            raise_status(a.status, FUSION_DEV_BAD_BATCH);
            a.plan[0] = 0;
            a.plan[1] = 0;
            a.offsets_out[0] = 0;
            if (a.batch_out) *a.batch_out = 0;
        }
        return;
    }

    int base_s = 0;   // survivors so far
    int base_r = 0;   // output rows so far
    for (int c0 = 0; c0 < B; c0 += kPlanChunk) {
        const int n = min(kPlanChunk, B - c0);
        for (int k = t; k <= n; k += nt) o_s[k] = a.in.offsets[c0 + k];
        for (int k = t; k < n; k += nt) {
            id_s[k] = a.in.ids ? a.in.ids[c0 + k] : c0 + k;
            sv_s[k] = (a.exit_mask == nullptr || __ldcg(a.exit_mask + c0 + k) == 0) ? 1 : 0;
        }
        __syncthreads();
        for (int k = t; k < n; k += nt) {
            const int o0 = o_s[k], o1 = o_s[k + 1];
            const int N = o1 - o0;
            const bool ok = o0 >= 0 && N >= 1 && N <= a.in.max_tokens && (long long)o1 <= a.in.max_rows;
            const int id = id_s[k];
            const bool id_ok = id >= 0 && id < a.in.max_batch;
            if (!ok) atomicOr(&s_bad, FUSION_DEV_BAD_OFFSETS);
            if (!id_ok) atomicOr(&s_bad, FUSION_DEV_BAD_IDS);
            int cnt = 0;
            if (ok && id_ok && sv_s[k]) {
                int nn = N;
                if (a.merge) nn -= merge_count(a.r[id], N - 1);
                if (a.prune) {
                    bool nf = false;
                    nn = 1 + keep_count(a.rho[id], nn - 1, nf);
                    if (nf) s_nonfinite = 1;
                }
                cnt = nn;
            }
            cnt_s[k] = cnt;
        }
        __syncthreads();
        // contiguous segments of the round, one per thread
        const int seg = (n + nt - 1) / nt;
        const int k0 = min(n, t * seg), k1 = min(n, k0 + seg);
        int ss = 0, rr = 0;
        for (int k = k0; k < k1; ++k) {
            ss += sv_s[k];
            rr += cnt_s[k];
        }
        flags[t] = ss;
        cnts[t] = rr;
        __syncthreads();
        const int tot_s = block_scan_excl(flags, nt, tmp);
        const int tot_r = block_scan_excl(cnts, nt, tmp);
        int js = base_s + flags[t], jr = base_r + cnts[t];
        for (int k = k0; k < k1; ++k) {
            const int i = c0 + k;
            if (sv_s[k]) {
                a.slot[i] = js;
                a.offsets_out[js] = jr;
                if (a.ids_out) a.ids_out[js] = id_s[k];
                ++js;
                jr += cnt_s[k];
            } else {
                a.slot[i] = -1;
            }
        }
        base_s += tot_s;
        base_r += tot_r;
        __syncthreads();   // the staging arrays are reused by the next round
    }
    if (t == 0) {
        a.offsets_out[base_s] = base_r;
        if (a.batch_out) *a.batch_out = base_s;
        a.plan[0] = s_bad ? 0 : 1;
        a.plan[1] = base_s;
        if (s_bad) raise_status(a.status, s_bad);
        if (s_nonfinite) raise_status(a.status, FUSION_DEV_NONFINITE);
    }
}

}  // namespace fz
