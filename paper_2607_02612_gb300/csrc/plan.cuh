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

// Run by ONE thread block (any size, multiple of 32).  smem: 4*blockDim.x + 40 ints.
__device__ inline void run_plan(const PlanArgs &a, int *smem) {
    int *flags = smem;                      // [2 * blockDim]
    int *cnts = smem + blockDim.x * 2;      // reuse: counts scanned after flags (second half)
    int *tmp = smem + blockDim.x * 4;       // 33 ints
    __shared__ int s_bad, s_nonfinite;
    const int t = threadIdx.x;
    const int per = 2 * blockDim.x;
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
    for (int t0 = 0; t0 < B; t0 += per) {
        for (int e = 0; e < 2; ++e) {
            const int i = t0 + 2 * t + e;
            int surv = 0, cnt = 0;
            if (i < B) {
                const int o0 = a.in.offsets[i], o1 = a.in.offsets[i + 1];
                const int N = o1 - o0;
                const bool ok = o0 >= 0 && N >= 1 && N <= a.in.max_tokens && (long long)o1 <= a.in.max_rows;
                const int id = a.in.ids ? a.in.ids[i] : i;
                const bool id_ok = id >= 0 && id < a.in.max_batch;
                if (!ok) atomicOr(&s_bad, FUSION_DEV_BAD_OFFSETS);
                if (!id_ok) atomicOr(&s_bad, FUSION_DEV_BAD_IDS);
                surv = (a.exit_mask == nullptr || __ldcg(a.exit_mask + i) == 0) ? 1 : 0;
                if (ok && id_ok && surv) {
                    int n = N;
                    if (a.merge) n -= merge_count(a.r[id], N - 1);
                    if (a.prune) {
                        bool nf = false;
                        n = 1 + keep_count(a.rho[id], n - 1, nf);
                        if (nf) s_nonfinite = 1;
                    }
                    cnt = n;
                }
            }
            flags[2 * t + e] = surv;
            cnts[2 * t + e] = cnt;
        }
        __syncthreads();
        const int tot_s = block_scan_excl(flags, per, tmp);
        const int tot_r = block_scan_excl(cnts, per, tmp);
        for (int e = 0; e < 2; ++e) {
            const int i = t0 + 2 * t + e;
            if (i < B) {
                const bool surv = (a.exit_mask == nullptr || __ldcg(a.exit_mask + i) == 0);
                const int j = base_s + flags[2 * t + e];
                a.slot[i] = surv ? j : -1;
                if (surv) {
                    a.offsets_out[j] = base_r + cnts[2 * t + e];
                    if (a.ids_out) a.ids_out[j] = a.in.ids ? a.in.ids[i] : i;
                }
            }
        }
        base_s += tot_s;
        base_r += tot_r;
        __syncthreads();
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
