"""The exit check with the paper's MLP exit heads (Sec. III-D, Eq. 6-7; SpatialPool head at
block 8, CLS-only head at block 10, each a 2-layer MLP) on the GPU against the oracle.

Where the kernels' arithmetic differs from the oracle's double evaluation: the pool is summed
in float-float (exact products, compensated sums) and the LayerNorm statistics too, so the bf16
LayerNorm output rounds as the oracle's does (a float evaluation is kept only when it lies more
than 24 float ulps from a bf16 rounding midpoint); the hidden layer's GELU is evaluated in
float in the erfc form and a unit within the product's error scale of a bf16 midpoint is
evaluated again exactly (float-float dot product, GELU in double), so the bf16 hidden units
match; the two products accumulate in float32.  What remains is float32 accumulation and the
softmax: logits within 1e-4 of the row's largest magnitude (both dtypes), max_prob within 1e-4
relative, and exit decisions equal wherever the oracle's margin |c - tau| is at least 1e-6
(closer ones are counted and reported)."""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle  # noqa: E402
import parity as P  # noqa: E402
import paper_2607_02612_gb300 as fz  # noqa: E402
from paper_2607_02612_gb300 import runner  # noqa: E402
from workloads import POOL_CLS, POOL_SPATIAL, make_mlp_head, make_workload  # noqa: E402

pytestmark = pytest.mark.gpu

TOL_LOGITS = {"f32": 1e-4, "bf16": 1e-4}
TOL_MAXP = {"f32": 1e-4, "bf16": 1e-4}


def _run(b, head, batch=None, max_tokens=None):
    f = runner.Fusion(b.batch, 1)
    db = P.device_batch(b, max_tokens=max_tokens)
    if batch is not None:
        db.batch = torch.full((1,), batch, dtype=torch.int32, device="cuda")
    ht = runner.mlp_head_tensors(head, b.dtype)
    o = f.exit_check_mlp(db, ht)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in o.items()}, int(f.status.item()), f, db, ht


def _compare(dtype, g, o, label, n=None):
    n = len(o["max_prob"]) if n is None else n
    ex = (o["exit_mask"][:n] == 1) & (g["exit_mask"][:n] == 1)   # logits: the rows of samples that exit
    e = P.rel_err_rows(g["logits"][:n][ex], o["logits"][:n][ex]) if ex.any() else np.zeros(1)
    assert e.max() <= TOL_LOGITS[dtype], (label, float(e.max()), int(e.argmax()))
    assert not np.any(g["logits"][:n][g["exit_mask"][:n] == 0]), (label, "logits written for samples that continue")
    pe = np.abs(g["max_prob"][:n].astype(np.float64) - o["max_prob"][:n]) / o["max_prob"][:n]
    assert pe.max() <= TOL_MAXP[dtype], (label, float(pe.max()))
    near = o["exit_gap"][:n] < P.NEAR_TIE
    diff = g["exit_mask"][:n] != o["exit_mask"][:n]
    assert not (diff & ~near).any(), (label, np.nonzero(diff & ~near)[0][:5])
    print(f"[{label}] {n} samples, {int(o['exit_mask'][:n].sum())} exit, logits rel err {e.max():.2e}, "
          f"max_prob rel err {pe.max():.2e}, {int(near.sum())} near the threshold, {int(diff.sum())} differ")


def _head_with_median_tau(b, pool, hidden, classes, seed):
    """A random head whose threshold is the oracle's median max_prob (about half exit)."""
    head = make_mlp_head(np.random.default_rng(seed), pool, b.dim, hidden, classes, b.dtype)
    o = oracle.exit_mlp(b.dtype, b.offsets, b.x, b.sizes, head)
    head.tau = float(np.float32(np.median(o["max_prob"])))
    return head, oracle.exit_mlp(b.dtype, b.offsets, b.x, b.sizes, head)


@pytest.mark.parametrize("name,pool", [("deit_s_chain12_bf16_b256", POOL_SPATIAL), ("deit_s_chain12_bf16_b256", POOL_CLS),
                                       ("deit_s_stage_f32_b8", POOL_SPATIAL), ("deit_s_stage_f32_b8", POOL_CLS),
                                       ("ragged_b8192_n65_chain4_f32", POOL_SPATIAL)])
def test_exit_mlp_matches_oracle(name, pool):
    w = make_workload(name, batch=512 if "ragged" in name else None)
    b = w.batch
    head, o = _head_with_median_tau(b, pool, 2 * b.dim, 1000, 3 + pool)
    g, st, *_ = _run(b, head)
    assert st == 0, st
    _compare(b.dtype, g, o, f"{name} pool {pool}")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_exit_mlp_shapes(dtype):
    """Hidden widths and class counts off the tile sizes; samples with one token (SpatialPool
    falls back to the CLS row) and with two; a device batch count below the bound."""
    rng = np.random.default_rng(17)
    Ns = [1, 2, 9, 197, 3, 64, 1, 130, 17, 5, 33]
    offsets = np.concatenate([[0], np.cumsum(Ns)]).astype(np.int32)
    d = 192
    xf = (rng.standard_normal((int(offsets[-1]), d)) * 1.3).astype(np.float32)
    from workloads import Batch, f32_to_bf16_bits
    x = f32_to_bf16_bits(xf) if dtype == "bf16" else xf
    sizes = rng.integers(1, 5, int(offsets[-1])).astype(np.float32)
    b = Batch(dtype, offsets, x, x, sizes, np.zeros(len(sizes), np.float32), None)
    for hidden, classes in ((48, 7), (400, 129), (1024, 300)):
        head, o = _head_with_median_tau(b, POOL_SPATIAL, hidden, classes, hidden)
        g, st, *_ = _run(b, head)
        assert st == 0
        _compare(dtype, g, o, f"{dtype} H {hidden} C {classes}")
    nb = 6
    g, st, *_ = _run(b, head, batch=nb)
    assert st == 0
    o = oracle.exit_mlp(dtype, offsets[:nb + 1], x, sizes, head)
    _compare(dtype, g, o, f"{dtype} device count {nb}", n=nb)
    assert not g["exit_mask"][nb:].any() and not g["max_prob"][nb:].any()


def test_exit_mlp_repeat_and_malformed():
    """A second call on the same scratch gives the same bits (the counters are left zero);
    offsets beyond max_rows raise BAD_OFFSETS."""
    w = make_workload("deit_s_chain12_bf16_b256", batch=32)
    b = w.batch
    head, o = _head_with_median_tau(b, POOL_SPATIAL, 768, 1000, 9)
    g1, st, f, db, ht = _run(b, head)
    g2 = {k: v.cpu().numpy() for k, v in f.exit_check_mlp(db, ht).items()}
    torch.cuda.synchronize()
    assert st == 0 and int(f.status.item()) == 0
    for k in g1:
        np.testing.assert_array_equal(g1[k], g2[k], err_msg=k)
    bad = b.offsets.copy()
    bad[5:] += 10**6
    db.offsets = torch.from_numpy(bad).cuda()
    f.exit_check_mlp(db, ht)
    torch.cuda.synchronize()
    assert int(f.status.item()) & fz.FUSION_DEV_BAD_OFFSETS
