"""GPU-vs-oracle comparison helpers for the parity tests.

Rules (one place, used by every parity test):
* index outputs (matches, kept rows, exit mask, offsets, ids) must be bit-exact;
* a decision whose oracle margin is below NEAR_TIE (1e-6: argmax gap, top-r boundary
  gap, prune boundary gap, |c - tau|) may legitimately go either way under a different
  summation order: such decisions are counted and reported, and a sample whose output
  differs only because of one is excluded from the remaining comparisons (and from
  later stages of a chain) instead of failing the test;
* floating-point token rows, logits and max-probs must match within TOL[dtype] relative
  to the oracle row's largest magnitude (f32 1e-5, bf16 2e-2); sizes and scores of kept
  tokens must match exactly.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Set

import numpy as np
import torch

import oracle
from paper_2607_02612_gb300 import runner
from paper_2607_02612_gb300 import _binding as fb
from workloads import Batch, bf16_bits_to_f32

NEAR_TIE = 1e-6
TOL = {"f32": 1e-5, "bf16": 2e-2}
# MLP exit heads (derivation in test_gpu_exit_mlp): logits relative to the row's largest
# magnitude, max_prob relative; exit decisions are held to the NEAR_TIE rule like the linear head
MLP_TOL_LOGITS = {"f32": 1e-4, "bf16": 1e-4}
MLP_TOL_MAXP = {"f32": 1e-4, "bf16": 1e-4}


@dataclass
class Report:
    near_ties: Dict[str, int] = field(default_factory=lambda: {"argmax": 0, "topr": 0, "prune": 0, "exit": 0})
    near_tie_mismatch: Dict[str, int] = field(default_factory=lambda: {"merge": 0, "exit": 0, "rows": 0})
    excluded: Set[int] = field(default_factory=set)
    max_rel_err: Dict[str, float] = field(default_factory=lambda: {"x": 0.0, "logits": 0.0, "max_prob": 0.0})
    non_bitexact_x: int = 0
    compared_samples: int = 0
    failures: List[str] = field(default_factory=list)

    def fail(self, msg: str):
        if len(self.failures) < 20:
            self.failures.append(msg)

    def check(self):
        assert not self.failures, "\n".join(self.failures)

    def summary(self) -> str:
        return (f"samples={self.compared_samples} near_ties={self.near_ties} "
                f"near_tie_mismatch={self.near_tie_mismatch} excluded={len(self.excluded)} "
                f"max_rel_err={self.max_rel_err} non_bitexact_x={self.non_bitexact_x}")


def as_float(a: np.ndarray, dtype: str) -> np.ndarray:
    return bf16_bits_to_f32(a) if dtype == "bf16" else np.asarray(a, np.float32)


def to_host(o: Dict[str, Optional[torch.Tensor]], dtype: str) -> Dict[str, np.ndarray]:
    out = {}
    for k, v in o.items():
        if v is None:
            out[k] = None
        elif k == "x":
            out[k] = runner.tokens_to_numpy(v, dtype)
        else:
            out[k] = v.cpu().numpy()
    return out


def device_batch(b: Batch, device="cuda", max_tokens=None) -> runner.DeviceBatch:
    return runner.device_batch(b.dtype, b.offsets, b.x, b.keys, b.sizes, b.scores, ids=b.ids,
                               max_tokens=max_tokens, device=device)


def rel_err_rows(g: np.ndarray, o: np.ndarray) -> np.ndarray:
    """Per-row max |g - o| / max |o| (rows of a 2-D array)."""
    scale = np.maximum(np.max(np.abs(o), axis=1), 1e-30)
    return np.max(np.abs(g.astype(np.float64) - o.astype(np.float64)), axis=1) / scale


# ---------------------------------------------------------------------------
# exit check
# ---------------------------------------------------------------------------
def compare_exit(rep: Report, dtype: str, ids: np.ndarray, g_mask, g_logits, g_maxp, o: dict,
                 skip: Set[int] = frozenset()):
    gap = o["exit_gap"]
    rep.near_ties["exit"] += int(np.sum(gap < NEAR_TIE))
    for i in range(len(ids)):
        if int(ids[i]) in skip:
            continue
        if g_mask[i] != o["exit_mask"][i]:
            if gap[i] < NEAR_TIE:
                rep.near_tie_mismatch["exit"] += 1
                rep.excluded.add(int(ids[i]))
            else:
                rep.fail(f"exit mask differs for sample id {ids[i]} (c={o['max_prob'][i]}, gap={gap[i]:.3g})")
    keep = np.array([int(t) not in skip for t in ids], bool)
    if g_logits is not None:
        # logits are the early prediction: written for the samples that exit, the other rows
        # are left as they were (zero in every caller here)
        ex = keep & (o["exit_mask"] == 1) & (g_mask == o["exit_mask"])
        if ex.any():
            e = rel_err_rows(g_logits[ex], o["logits"][ex])
            rep.max_rel_err["logits"] = max(rep.max_rel_err["logits"], float(e.max()))
            bad = np.nonzero(e > TOL[dtype])[0]
            for b in bad[:3]:
                rep.fail(f"logits of sample {np.nonzero(ex)[0][b]} off by {e[b]:.3g} (rel)")
        stay = keep & (g_mask == 0)
        if stay.any() and np.any(g_logits[stay] != 0):
            rep.fail(f"logits written for {int(np.sum(np.any(g_logits[stay] != 0, axis=1)))} samples that continue")
    if g_maxp is not None and keep.any():
        e = np.abs(g_maxp[keep].astype(np.float64) - o["max_prob"][keep]) / np.maximum(o["max_prob"][keep], 1e-30)
        rep.max_rel_err["max_prob"] = max(rep.max_rel_err["max_prob"], float(e.max()))
        if e.max() > TOL[dtype]:
            rep.fail(f"max_prob off by {e.max():.3g} (rel)")


# ---------------------------------------------------------------------------
# token outputs of one stage, per sample
# ---------------------------------------------------------------------------
def sample_near_tie(o: dict, in_offsets: np.ndarray, i: int) -> bool:
    a, b = int(in_offsets[i]), int(in_offsets[i + 1])
    ag = o.get("argmax_gap")
    if ag is not None and np.any(ag[a:b] < NEAR_TIE):
        return True
    for k in ("topr_gap", "prune_gap"):
        v = o.get(k)
        if v is not None and v[i] < NEAR_TIE:
            return True
    return False


def count_decision_near_ties(rep: Report, o: dict):
    if o.get("argmax_gap") is not None:
        rep.near_ties["argmax"] += int(np.sum(o["argmax_gap"] < NEAR_TIE))
    if o.get("topr_gap") is not None:
        rep.near_ties["topr"] += int(np.sum(o["topr_gap"] < NEAR_TIE))
    if o.get("prune_gap") is not None:
        rep.near_ties["prune"] += int(np.sum(o["prune_gap"] < NEAR_TIE))


def compare_tokens(rep: Report, dtype: str, o_in_off, o_in_ids, g_in_off, g_in_ids, g: dict, o: dict,
                   g_ids, o_ids, skip: Set[int] = frozenset(), a_match_gpu=None):
    """Compare the output samples of one call sample by sample, matched by original id.
    (o_in_off, o_in_ids) and (g_in_off, g_in_ids) describe the input batch each side
    saw (they differ only after an earlier near-tie exit flip); kept rows and matches
    are compared as positions within their sample.  g / o hold x, sizes, scores,
    offsets, keep_idx of the GPU and of the oracle."""
    o_in_off = np.asarray(o_in_off)
    g_in_off = np.asarray(g_in_off)
    o_pos = {int(t): i for i, t in enumerate(o_in_ids)}
    g_pos = {int(t): i for i, t in enumerate(g_in_ids)}
    g_of_id = {int(t): j for j, t in enumerate(g_ids)}
    o_of_id = {int(t): j for j, t in enumerate(o_ids)}
    gx = as_float(g["x"], dtype)
    ox = as_float(o["x"], dtype)
    for t, jo in o_of_id.items():
        if t in skip or t in rep.excluded:
            continue
        i = o_pos[t]
        near = sample_near_tie(o, o_in_off, i)
        if t not in g_of_id:
            rep.fail(f"sample id {t} missing from the GPU output")
            continue
        jg = g_of_id[t]
        ig = g_pos[t]
        so, sg = int(o_in_off[i]), int(g_in_off[ig])
        n_in = int(o_in_off[i + 1]) - so
        if int(g_in_off[ig + 1]) - sg != n_in:
            rep.fail(f"sample id {t}: GPU input has {int(g_in_off[ig + 1]) - sg} tokens, oracle {n_in}")
            continue
        a0, a1 = int(o["offsets"][jo]), int(o["offsets"][jo + 1])
        b0, b1 = int(g["offsets"][jg]), int(g["offsets"][jg + 1])
        if a_match_gpu is not None and o.get("a_match") is not None:
            om = o["a_match"][so:so + n_in]
            gm = a_match_gpu[sg:sg + n_in]
            om = np.where(om >= 0, om - so, -1)
            gm = np.where(gm >= 0, gm - sg, -1)
            if not np.array_equal(om, gm):
                bad = np.nonzero(om != gm)[0]
                if not np.all(o["argmax_gap"][so + bad] < NEAR_TIE):
                    rep.fail(f"a_match differs for sample id {t} at positions {bad[:5]} "
                             f"(gaps {o['argmax_gap'][so + bad[:5]]})")
                    continue
                rep.near_tie_mismatch["merge"] += 1
        ok = (a1 - a0) == (b1 - b0) and np.array_equal(o["keep_idx"][a0:a1] - so, g["keep_idx"][b0:b1] - sg)
        if ok and not np.array_equal(o["sizes"][a0:a1], g["sizes"][b0:b1]):
            ok = False
        if ok and o.get("scores") is not None and g.get("scores") is not None and \
                not np.array_equal(o["scores"][a0:a1], g["scores"][b0:b1]):
            ok = False
        if not ok:
            if near:
                rep.near_tie_mismatch["rows"] += 1
                rep.excluded.add(t)
            else:
                rep.fail(f"kept rows / sizes / scores differ for sample id {t}: oracle "
                         f"{(o['keep_idx'][a0:a0 + 8] - so)}.. gpu {(g['keep_idx'][b0:b0 + 8] - sg)}..")
            continue
        rep.compared_samples += 1
        if a1 > a0:
            e = rel_err_rows(gx[b0:b1], ox[a0:a1])
            rep.max_rel_err["x"] = max(rep.max_rel_err["x"], float(e.max()))
            if e.max() > TOL[dtype]:
                rep.fail(f"token rows of sample id {t} off by {e.max():.3g} (rel)")
            if dtype == "bf16":
                rep.non_bitexact_x += int(np.sum(g["x"][b0:b1] != o["x"][a0:a1]))
            else:
                rep.non_bitexact_x += int(np.sum(gx[b0:b1] != ox[a0:a1]))


def compare_chain(rep: Report, workload, g_outs, o_outs, fresh_logits: bool = True):
    """fresh_logits: the logits buffers were zero before the run, so rows of samples that
    continue must still be zero (False when the buffers are reused across inputs)."""
    """Stage-by-stage comparison of a chain; samples that diverged at a near tie are
    excluded from the later stages."""
    b = workload.batch
    dtype = b.dtype
    B = b.batch
    o_ids_in = g_ids_in = np.arange(B, dtype=np.int32) if b.ids is None else np.asarray(b.ids)
    o_off_in = g_off_in = b.offsets
    for s, (g, o) in enumerate(zip(g_outs, o_outs)):
        spec = workload.stages[s]
        count_decision_near_ties(rep, o)
        g_nb = int(g["batch"][0])
        g_ids_out = g["ids"][:g_nb]
        if spec.exit:
            mlp = getattr(spec, "mlp_head", None) is not None
            tol_l = MLP_TOL_LOGITS[dtype] if mlp else TOL[dtype]
            tol_p = MLP_TOL_MAXP[dtype] if mlp else TOL[dtype]
            gpos = {int(t): i for i, t in enumerate(g_ids_in)}
            for i, t in enumerate(o_ids_in):
                t = int(t)
                if t in rep.excluded:
                    continue
                if t not in gpos:
                    rep.fail(f"stage {s}: sample id {t} missing from the GPU input")
                    continue
                ig = gpos[t]
                gap = o["exit_gap"][i]
                near = NEAR_TIE
                if gap < near:
                    rep.near_ties["exit"] += 1
                if g["exit_mask"][ig] != o["exit_mask"][i]:
                    if gap < near:
                        rep.near_tie_mismatch["exit"] += 1
                        rep.excluded.add(t)
                        continue
                    rep.fail(f"stage {s}: exit mask differs for sample id {t} "
                             f"(c={o['max_prob'][i]}, gap={gap:.3g})")
                    continue
                if o["exit_mask"][i]:   # logits are written only for the samples that exit
                    e = rel_err_rows(g["logits"][ig:ig + 1], o["logits"][i:i + 1])[0]
                    rep.max_rel_err["logits"] = max(rep.max_rel_err["logits"], float(e))
                    if e > tol_l:
                        rep.fail(f"stage {s}: logits of sample id {t} off by {e:.3g}")
                elif fresh_logits and np.any(g["logits"][ig] != 0):
                    rep.fail(f"stage {s}: logits written for sample id {t}, which continues")
                ep = abs(float(g["max_prob"][ig]) - float(o["max_prob"][i])) / max(float(o["max_prob"][i]), 1e-30)
                rep.max_rel_err["max_prob"] = max(rep.max_rel_err["max_prob"], ep)
                if ep > tol_p:
                    rep.fail(f"stage {s}: max_prob of sample id {t} off by {ep:.3g}")
        compare_tokens(rep, dtype, o_off_in, o_ids_in, g_off_in, g_ids_in, g, o, g_ids_out, o["ids"])
        o_ids_in, o_off_in = o["ids"], o["offsets"]
        g_ids_in, g_off_in = g_ids_out, g["offsets"][:g_nb + 1]


# ---------------------------------------------------------------------------
# running a stage / chain on the GPU
# ---------------------------------------------------------------------------
def flags_of(spec) -> int:
    return ((fb.FUSION_STAGE_MERGE if spec.merge else 0) | (fb.FUSION_STAGE_EXIT if spec.exit else 0) |
            (fb.FUSION_STAGE_PRUNE if spec.prune else 0))


def stage_tensors(spec, dtype: str, device="cuda"):
    r = torch.from_numpy(spec.r).to(device) if spec.r is not None else None
    rho = torch.from_numpy(spec.rho).to(device) if spec.rho is not None else None
    head = runner.head_tensors(spec.head, dtype, device) if spec.head is not None else None
    return r, rho, head


def chain_on_gpu(workload, stages: Optional[int] = None, device="cuda", graph: bool = False):
    """Run the workload's schedule through the fused stage call; return per-stage host outputs."""
    b = workload.batch
    specs = workload.stages[:stages]
    classes = max([s.head.classes for s in specs if s.head is not None] + [1])
    fz = runner.Fusion(b.batch, classes, device)
    db = device_batch(b, device)
    cstages = []
    for s in specs:
        r, rho, head = stage_tensors(s, b.dtype, device)
        mh = getattr(s, "mlp_head", None)
        mlp = runner.mlp_head_tensors(mh, b.dtype, device) if mh is not None else None
        cstages.append(runner.ChainStage(flags_of(s), r, rho, None if mlp is not None else head, mlp))
    ch = runner.Chain(fz, db, cstages)
    if graph:
        ch.run()
        g = ch.capture()
        g.replay()
    else:
        ch.run()
    torch.cuda.synchronize()
    outs = [to_host(o, b.dtype) for o in ch.outs]
    return outs, int(fz.status.item())
