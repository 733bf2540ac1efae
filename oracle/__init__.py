"""CPU oracle for the Fusion staged token-adaptation step.

TEST INFRASTRUCTURE ONLY: imported by the test suite, by the smoke check of
``__graft_entry__`` and by the CPU-baseline leg of ``bench.py``.  The CUDA
library never imports, links or calls anything here, and nothing here imports
the CUDA library.

The arithmetic lives in ``fusion_oracle.c`` (plain C, double precision,
compiled with gcc by :func:`build`).  This module marshals numpy arrays and
composes the four operators in the order of Algorithm 1 / Sec. III-B:
merge, then the exit check on the merged (unpruned) tokens, then, for the
samples that continue, pruning; exited samples leave the batch (compaction).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Dict, List, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fusion_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")

F32, BF16 = 0, 1
_DT = {"f32": F32, "bf16": BF16}

_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into oracle/_build/liboracle.so with gcc (host code only)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def configure(lib):
    """Declare the C signatures on a loaded oracle library (also used on test builds)."""
    P = ctypes.c_void_p
    i32, dbl = ctypes.c_int, ctypes.c_double
    lib.orc_merge.argtypes = [i32, i32, P, i32, P, P, i32, P, P, P, P, P, P, P, P, P, P, P, P]
    lib.orc_exit.argtypes = [i32, i32, P, i32, P, P, P, dbl, P, P, i32, dbl, P, P, P, P, P]
    lib.orc_prune.argtypes = [i32, i32, P, i32, P, P, P, P, P, P, P, P, P, P]
    lib.orc_compact.argtypes = [i32, i32, P, i32, P, P, P, P, P, P, P, P, P, P, P, P]
    lib.orc_merge_router.argtypes = [i32, i32, P, P, i32, P, P, dbl, dbl, dbl, P, P, P]
    lib.orc_merge_router.restype = ctypes.c_int
    lib.orc_token_scores.argtypes = [i32, i32, P, i32, P, P, dbl, P]
    lib.orc_exit_mlp.argtypes = [i32, i32, P, i32, P, P, i32, P, P, dbl, P, P, i32, P, P, i32, dbl,
                                 P, P, P, P, P, P]
    lib.orc_exit_mlp.restype = ctypes.c_int
    lib.orc_attention.argtypes = [i32, i32, P, i32, i32, P, P, P]
    lib.orc_attention.restype = ctypes.c_int
    lib.orc_token_scores.restype = ctypes.c_int
    lib.orc_double_to_bf16.argtypes = [dbl]
    lib.orc_double_to_bf16.restype = ctypes.c_uint16
    lib.orc_bf16_to_double.argtypes = [ctypes.c_uint16]
    lib.orc_bf16_to_double.restype = dbl
    for f in (lib.orc_merge, lib.orc_exit, lib.orc_prune, lib.orc_compact):
        f.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    if _lib is None:
        build()
        _lib = configure(ctypes.CDLL(_LIB))
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def _elem_dtype(dtype: str):
    return np.uint16 if dtype == "bf16" else np.float32


def _check(rc: int, what: str):
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed with code {rc}")


# ---------------------------------------------------------------------------
# scalar conversions (exposed for pinning)
# ---------------------------------------------------------------------------
def double_to_bf16(v: float) -> int:
    return int(_load().orc_double_to_bf16(float(v)))


def bf16_to_double(h: int) -> float:
    return float(_load().orc_bf16_to_double(int(h)))


# ---------------------------------------------------------------------------
# the four operators
# ---------------------------------------------------------------------------
def merge(dtype: str, offsets, x, keys, sizes, scores, r) -> Dict[str, np.ndarray]:
    """Sec. III-C merge of every sample.  Returns x, sizes, scores, offsets, keep_idx,
    dst_map, a_match, argmax_gap, topr_gap."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    keys = _c(keys, et)
    sizes = _c(sizes, np.float32)
    scores = _c(scores, np.float32)
    r = _c(r, np.int32)
    B = len(offsets) - 1
    T, d = x.shape
    dk = keys.shape[1]
    x_out = np.zeros_like(x)
    sizes_out = np.zeros(T, np.float32)
    scores_out = None if scores is None else np.zeros(T, np.float32)
    offsets_out = np.zeros(B + 1, np.int32)
    keep = np.full(T, -1, np.int32)
    dst = np.full(T, -1, np.int32)
    amatch = np.full(T, -1, np.int32)
    agap = np.full(T, np.inf)
    rgap = np.full(B, np.inf)
    rc = lib.orc_merge(_DT[dtype], B, _p(offsets), d, _p(x), _p(keys), dk, _p(sizes), _p(scores),
                       _p(r), _p(x_out), _p(sizes_out), _p(scores_out), _p(offsets_out), _p(keep),
                       _p(dst), _p(amatch), _p(agap), _p(rgap))
    _check(rc, "merge")
    t = int(offsets_out[-1])
    return dict(x=x_out[:t], sizes=sizes_out[:t],
                scores=None if scores_out is None else scores_out[:t], offsets=offsets_out,
                keep_idx=keep[:t], dst_map=dst, a_match=amatch, argmax_gap=agap, topr_gap=rgap)


def exit_check(dtype: str, offsets, x, head) -> Dict[str, np.ndarray]:
    """Sec. III-D exit check on the CLS row of every sample.  Returns exit_mask, logits,
    max_prob, exit_gap, u (the head input)."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    B = len(offsets) - 1
    d = x.shape[1]
    W = _c(head.weight, et)
    C = W.shape[0]
    mask = np.zeros(B, np.uint8)
    logits = np.zeros((B, C), np.float32)
    maxp = np.zeros(B, np.float32)
    gap = np.full(B, np.inf)
    u = np.zeros((B, d), np.float64)
    rc = lib.orc_exit(_DT[dtype], B, _p(offsets), d, _p(x), _p(_c(head.gamma, et)),
                      _p(_c(head.beta, et)), float(head.eps), _p(W),
                      _p(_c(head.bias, np.float32)), C, float(np.float32(head.tau)),
                      _p(mask), _p(logits), _p(maxp), _p(gap), _p(u))
    _check(rc, "exit")
    return dict(exit_mask=mask, logits=logits, max_prob=maxp, exit_gap=gap, u=u)


def exit_mlp(dtype: str, offsets, x, sizes, head) -> Dict[str, np.ndarray]:
    """Sec. III-D exit check with an MLP exit head (``workloads.MlpHead``): pool (CLS row or
    size-weighted patch mean) -> LayerNorm -> W1, GELU -> W2 -> softmax maximum.  Returns
    exit_mask, logits, max_prob, exit_gap, pool (the head input), hidden."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    B = len(offsets) - 1
    d = x.shape[1]
    W1, W2 = _c(head.w1, et), _c(head.w2, et)
    H, C = W1.shape[0], W2.shape[0]
    mask = np.zeros(B, np.uint8)
    logits = np.zeros((B, C), np.float32)
    maxp = np.zeros(B, np.float32)
    gap = np.full(B, np.inf)
    z = np.zeros((B, d), np.float64)
    hid = np.zeros((B, H), np.float64)
    rc = lib.orc_exit_mlp(_DT[dtype], B, _p(offsets), d, _p(x), _p(_c(sizes, np.float32)), int(head.pool),
                          _p(_c(head.gamma, et)), _p(_c(head.beta, et)), float(head.eps), _p(W1),
                          _p(_c(head.b1, np.float32)), H, _p(W2), _p(_c(head.b2, np.float32)), C,
                          float(np.float32(head.tau)), _p(mask), _p(logits), _p(maxp), _p(gap), _p(z), _p(hid))
    _check(rc, "exit_mlp")
    return dict(exit_mask=mask, logits=logits, max_prob=maxp, exit_gap=gap, pool=z, hidden=hid)


def attention(dtype: str, offsets, qkv, heads: int, sizes=None) -> np.ndarray:
    """Size-aware (proportional) attention per sample and head over a ragged batch:
    softmax(q k^T / sqrt(dh) + log s) v.  qkv [rows, 3 * heads * dh] (timm's packed q, k, v);
    sizes [rows] or None (plain attention).  Returns [rows, heads * dh] float64 (rows outside
    the samples are 0)."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    qkv = _c(qkv, et)
    rows = qkv.shape[0]
    dh = qkv.shape[1] // (3 * heads)
    out = np.zeros((rows, heads * dh), np.float64)
    sz = None if sizes is None else _c(sizes, np.float32)
    _check(lib.orc_attention(_DT[dtype], len(offsets) - 1, _p(offsets), heads, dh, _p(qkv),
                             None if sz is None else _p(sz), _p(out)), "attention")
    return out


def merge_router(dtype: str, offsets, x, w, beta: float, tau_tgt: float, tau_ref: float, ids=None,
                 n_ids: Optional[int] = None) -> Dict[str, np.ndarray]:
    """Sec. III-C router with profile scaling (Eq. 4-5) on the CLS row of every sample:
    r = floor(clamp(sigmoid(w . z_CLS + beta) (1 - tau_tgt) / (1 - tau_ref), 0, 1) N / 2).
    The arguments beta, tau_tgt, tau_ref are taken as float32 values (the library's
    argument type).  Returns r (int32), mt (the scaled ratio) and r_gap (margin of the
    floor decision), each indexed by original sample id (ids, or the position)."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    B = len(offsets) - 1
    d = x.shape[1]
    ids_a = None if ids is None else _c(ids, np.int32)
    n = n_ids if n_ids is not None else (int(ids_a.max()) + 1 if ids_a is not None and B > 0 else B)
    r = np.zeros(n, np.int32)
    mt = np.zeros(n, np.float64)
    gap = np.full(n, np.inf)
    rc = lib.orc_merge_router(_DT[dtype], B, _p(offsets), _p(ids_a), d, _p(x), _p(_c(w, et)),
                              float(np.float32(beta)), float(np.float32(tau_tgt)), float(np.float32(tau_ref)),
                              _p(r), _p(mt), _p(gap))
    _check(rc, "merge_router")
    return dict(r=r, mt=mt, r_gap=gap)


def token_scores(dtype: str, offsets, x, w, b: float) -> np.ndarray:
    """Sec. III-E, Eq. 8 pruning router with a linear scoring head: s = w . z + b for every
    token row of the batch (double, rounded once to float32; b taken as a float32 value)."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    B = len(offsets) - 1
    out = np.zeros(x.shape[0], np.float32)
    _check(lib.orc_token_scores(_DT[dtype], B, _p(offsets), x.shape[1], _p(x), _p(_c(w, et)),
                                float(np.float32(b)), _p(out)), "token_scores")
    return out


def prune(dtype: str, offsets, x, sizes, scores, rho) -> Dict[str, np.ndarray]:
    """Sec. III-E pruning of every sample.  Returns x, sizes, scores, offsets, keep_idx,
    prune_gap."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    sizes = _c(sizes, np.float32)
    scores = _c(scores, np.float32)
    rho = _c(rho, np.float32)
    B = len(offsets) - 1
    T, d = x.shape
    x_out = np.zeros_like(x)
    sizes_out = np.zeros(T, np.float32)
    scores_out = np.zeros(T, np.float32)
    offsets_out = np.zeros(B + 1, np.int32)
    keep = np.full(T, -1, np.int32)
    gap = np.full(B, np.inf)
    rc = lib.orc_prune(_DT[dtype], B, _p(offsets), d, _p(x), _p(sizes), _p(scores), _p(rho),
                       _p(x_out), _p(sizes_out), _p(scores_out), _p(offsets_out), _p(keep),
                       _p(gap))
    _check(rc, "prune")
    t = int(offsets_out[-1])
    return dict(x=x_out[:t], sizes=sizes_out[:t], scores=scores_out[:t], offsets=offsets_out,
                keep_idx=keep[:t], prune_gap=gap)


def compact(dtype: str, offsets, x, sizes, scores, exit_mask, ids=None) -> Dict[str, np.ndarray]:
    """Drop exited samples, keep survivors in ascending order.  Returns x, sizes, scores,
    offsets, ids, keep_idx, n_out."""
    lib = _load()
    et = _elem_dtype(dtype)
    offsets = _c(offsets, np.int32)
    x = _c(x, et)
    sizes = _c(sizes, np.float32)
    scores = _c(scores, np.float32)
    mask = _c(exit_mask, np.uint8)
    ids = _c(ids, np.int32)
    B = len(offsets) - 1
    T, d = x.shape
    x_out = np.zeros_like(x)
    sizes_out = np.zeros(T, np.float32)
    scores_out = None if scores is None else np.zeros(T, np.float32)
    offsets_out = np.zeros(B + 1, np.int32)
    ids_out = np.zeros(B, np.int32)
    keep = np.full(T, -1, np.int32)
    n = np.zeros(1, np.int32)
    rc = lib.orc_compact(_DT[dtype], B, _p(offsets), d, _p(x), _p(sizes), _p(scores), _p(mask),
                         _p(ids), _p(x_out), _p(sizes_out), _p(scores_out), _p(offsets_out),
                         _p(ids_out), _p(keep), _p(n))
    _check(rc, "compact")
    nb = int(n[0])
    t = int(offsets_out[nb])
    return dict(x=x_out[:t], sizes=sizes_out[:t],
                scores=None if scores_out is None else scores_out[:t],
                offsets=offsets_out[:nb + 1], ids=ids_out[:nb], keep_idx=keep[:t], n_out=nb)


# ---------------------------------------------------------------------------
# one stage and a chain of stages (Algorithm 1 body, Sec. III-B order)
# ---------------------------------------------------------------------------
def stage(batch, spec) -> Dict[str, object]:
    """One block's adaptation stage on a ``workloads.Batch``.

    Order (Sec. III-B): merge (if enabled) -> exit check on the merged tokens
    (if enabled; exited samples leave the batch) -> prune the survivors (if
    enabled).  Per-sample router outputs spec.r / spec.rho are indexed by the
    samples' original ids.  With spec.mlp_head (an MLP exit head, Sec. III-G) the
    exit check reads the merged tokens as stored (rounded to the dtype), as Sec. III-B
    defines it for every exit head.  Returns the output batch fields plus exit_mask, logits, max_prob
    (indexed by input sample), keep_idx (input row of every output row), a_match
    (input rows) and the decision margins."""
    dtype = batch.dtype
    B = batch.batch
    ids = np.arange(B, dtype=np.int32) if batch.ids is None else np.asarray(batch.ids, np.int32)
    T = int(batch.offsets[-1])
    res: Dict[str, object] = {}
    x, sizes, scores, offsets = batch.x[:T], batch.sizes[:T], batch.scores[:T], batch.offsets
    keep = np.arange(T, dtype=np.int32)
    res["a_match"] = np.full(T, -1, np.int32)
    res["argmax_gap"] = np.full(T, np.inf)
    res["topr_gap"] = np.full(B, np.inf)
    if spec.merge:
        m = merge(dtype, offsets, x, batch.keys[:T], sizes, scores, spec.r[ids])
        x, sizes, scores, offsets = m["x"], m["sizes"], m["scores"], m["offsets"]
        keep = m["keep_idx"]
        res.update(a_match=m["a_match"], argmax_gap=m["argmax_gap"], topr_gap=m["topr_gap"],
                   dst_map=m["dst_map"])
    mask = np.zeros(B, np.uint8)
    res["exit_gap"] = np.full(B, np.inf)
    if spec.exit:
        if getattr(spec, "mlp_head", None) is not None:
            e = exit_mlp(dtype, offsets, x, sizes, spec.mlp_head)
            mask = e["exit_mask"]
            res.update(exit_mask=mask, logits=e["logits"], max_prob=e["max_prob"], exit_gap=e["exit_gap"])
        else:
            e = exit_check(dtype, offsets, x, spec.head)
            mask = e["exit_mask"]
            res.update(exit_mask=mask, logits=e["logits"], max_prob=e["max_prob"],
                       exit_gap=e["exit_gap"], u=e["u"])
        c = compact(dtype, offsets, x, sizes, scores, mask, ids)
        x, sizes, scores, offsets = c["x"], c["sizes"], c["scores"], c["offsets"]
        keep = keep[c["keep_idx"]]
        out_ids = c["ids"]
    else:
        out_ids = ids.copy()
    surv = np.nonzero(mask == 0)[0]
    res["prune_gap"] = np.full(B, np.inf)
    if spec.prune:
        p = prune(dtype, offsets, x, sizes, scores, spec.rho[out_ids])
        x, sizes, scores, offsets = p["x"], p["sizes"], p["scores"], p["offsets"]
        keep = keep[p["keep_idx"]]
        res["prune_gap"][surv] = p["prune_gap"]
    res.update(x=x, sizes=sizes, scores=scores, offsets=offsets, ids=out_ids, keep_idx=keep,
               n_out=len(out_ids), exit_mask=mask)
    return res


def next_batch(batch, res):
    """The batch a stage hands to the next block: its outputs, keys aliasing x."""
    from workloads import Batch
    return Batch(batch.dtype, res["offsets"], res["x"], res["x"], res["sizes"], res["scores"],
                 res["ids"])


def chain(workload, stages: Optional[int] = None) -> List[Dict[str, object]]:
    """Run the workload's schedule of stages; keys of stage s+1 are the tokens stage s wrote."""
    out = []
    b = workload.batch
    for s, spec in enumerate(workload.stages[:stages]):
        res = stage(b, spec)
        out.append(res)
        b = next_batch(b, res)
    return out
