"""The linear pruning router (Sec. III-E, Eq. 8: s = w . z + b per token row) on the GPU
against the oracle: every score within the float32 dot-product error bound the header
states, 2^-18 (sum_j |w_j z_j| + |b|), plus the oracle's own rounding; every lane layout
the kernel picks (one per class of dim); rows outside the batch untouched; the device
batch count; malformed inputs; and a prune ranked by these scores."""
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
from workloads import StageSpec, bf16_bits_to_f32, f32_to_bf16_bits, make_score_head, make_workload  # noqa: E402

pytestmark = pytest.mark.gpu

BOUND = 2.0 ** -18
SENTINEL = -12345.0


def _tensor(a, dtype):
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).cuda()


def _bound(dtype, x, w, b):
    xf = np.abs(P.as_float(x, dtype).astype(np.float64))
    wf = np.abs(P.as_float(w, dtype).astype(np.float64))
    return BOUND * (xf @ wf + abs(b))


def _scores(dtype, offsets, x, w, b, max_batch=None, max_tokens=1024, batch=None, status=None):
    """Run fusion_token_scores on a sentinel-filled output; return (scores, status)."""
    B = len(offsets) - 1
    xt, wt = _tensor(x, dtype), _tensor(w, dtype)
    offs = torch.from_numpy(np.asarray(offsets, np.int32)).cuda()
    bt = None if batch is None else torch.full((1,), batch, dtype=torch.int32, device="cuda")
    rg = fz.ragged(B if max_batch is None else max_batch, max_tokens, x.shape[0], offs, bt)
    out = torch.full((x.shape[0],), SENTINEL, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    code = fz.FUSION_BF16 if dtype == "bf16" else fz.FUSION_F32
    fz.check(fz.fusion_token_scores(code, rg, xt, x.shape[1], wt, b, out, st))
    torch.cuda.synchronize()
    return out.cpu().numpy(), int(st.item())


def _check(dtype, offsets, x, w, b, label, **kw):
    g, st = _scores(dtype, offsets, x, w, b, **kw)
    nb = len(offsets) - 1 if kw.get("batch") is None else kw["batch"]
    o0, o1 = int(offsets[0]), int(offsets[nb])
    ref = oracle.token_scores(dtype, np.asarray(offsets[:nb + 1], np.int32), x, w, b)
    tol = _bound(dtype, x, w, b) + np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    err = np.abs(g[o0:o1].astype(np.float64) - ref[o0:o1])
    bad = err > tol[o0:o1]
    assert not bad.any(), (label, np.nonzero(bad)[0][:5], err[bad][:5], tol[o0:o1][bad][:5])
    assert np.all(g[:o0] == SENTINEL) and np.all(g[o1:] == SENTINEL), label
    exact = int(np.sum(g[o0:o1] == ref[o0:o1]))
    print(f"[{label}] {o1 - o0} rows, {exact} equal to the oracle's bits, max err/bound "
          f"{(err / np.maximum(tol[o0:o1], 1e-300)).max() if o1 > o0 else 0:.3g}")
    return g, st


@pytest.mark.parametrize("name", ["deit_s_chain12_bf16_b256", "deit_s_stage_f32_b8", "ragged_b8192_n65_chain4_f32"])
def test_scores_match_oracle(name):
    w = make_workload(name, batch=512 if "ragged" in name else None)
    b = w.batch
    h = make_score_head(np.random.default_rng(11), b.dim, b.dtype)
    _, st = _check(b.dtype, b.offsets, b.x, h.w, h.b, name)
    assert st == 0


# one dim per lane layout: (g lanes per row, K chunks per lane) from 8, 16 or 32 lanes, gcd(C, 32) or the
# masked whole-warp fallback, C = dim * elem / 16
LAYOUTS = [("bf16", d) for d in (16, 48, 80, 112, 144, 256, 384, 512, 768, 1008, 1024)] + \
          [("f32", d) for d in (16, 48, 112, 128, 144, 240, 384, 1008, 1024)]


@pytest.mark.parametrize("dtype,dim", LAYOUTS)
def test_scores_every_lane_layout(dtype, dim):
    rng = np.random.default_rng(dim)
    Ns = [1, 77, 300, 2, 197]
    lead, tail = 5, 9
    offsets = (lead + np.concatenate([[0], np.cumsum(Ns)])).astype(np.int32)
    xf = rng.standard_normal((int(offsets[-1]) + tail, dim)).astype(np.float32)
    x = f32_to_bf16_bits(xf) if dtype == "bf16" else xf
    h = make_score_head(rng, dim, dtype)
    _, st = _check(dtype, offsets, x, h.w, h.b, f"{dtype} dim {dim}")
    assert st == 0


def test_scores_device_batch_count_and_empty():
    rng = np.random.default_rng(12)
    offsets = np.array([0, 3, 10, 18, 30], np.int32)
    x = f32_to_bf16_bits(rng.standard_normal((30, 384)).astype(np.float32))
    h = make_score_head(rng, 384, "bf16")
    _, st = _check("bf16", offsets, x, h.w, h.b, "device count 2 of 4", batch=2)
    assert st == 0
    g, st = _scores("bf16", offsets, x, h.w, h.b, batch=0)
    assert st == 0 and np.all(g == SENTINEL)


def test_scores_malformed_inputs():
    rng = np.random.default_rng(13)
    offsets = np.array([0, 3, 10, 18], np.int32)
    x = rng.standard_normal((18, 64)).astype(np.float32)
    h = make_score_head(rng, 64, "f32")
    bad = offsets.copy()
    bad[-1] = 19                                          # past max_rows: nothing written
    g, st = _scores("f32", bad, x, h.w, h.b)
    assert st & fz.FUSION_DEV_BAD_OFFSETS and np.all(g == SENTINEL)
    g, st = _scores("f32", offsets, x, h.w, h.b, batch=4)  # device count above max_batch
    assert st & fz.FUSION_DEV_BAD_BATCH and np.all(g == SENTINEL)
    empty = np.array([0, 3, 3, 18], np.int32)             # an empty sample: flagged, rows still scored
    g, st = _check("f32", empty, x, h.w, h.b, "empty sample")
    assert st & fz.FUSION_DEV_BAD_OFFSETS
    long = np.array([0, 3, 10, 18], np.int32)             # a sample longer than max_tokens
    _, st = _scores("f32", long, x, h.w, h.b, max_tokens=7)
    assert st & fz.FUSION_DEV_BAD_OFFSETS
    xi = x.copy()
    xi[5, 7] = np.inf                                     # a non-finite score is flagged
    g, st = _scores("f32", offsets, xi, h.w, h.b)
    assert st & fz.FUSION_DEV_NONFINITE and not np.isfinite(g[5]) and np.all(np.isfinite(np.delete(g, 5)))


def test_prune_ranked_by_router_scores():
    """fusion_stage (merge) -> fusion_token_scores -> fusion_prune equals the oracle's merge ->
    token_scores -> prune; a sample may differ only where its prune boundary is closer than
    the scores' error bound (counted and reported)."""
    w = make_workload("deit_s_chain12_bf16_b256", batch=64)
    b = w.batch
    spec = next(s for s in w.stages if s.merge)
    h = make_score_head(np.random.default_rng(14), b.dim, b.dtype)
    rho = np.random.default_rng(15).uniform(0.3, 0.9, b.batch).astype(np.float32)
    f = runner.Fusion(b.batch, 1)
    db = P.device_batch(b)
    mo = f.stage(db, fz.FUSION_STAGE_MERGE, torch.from_numpy(spec.r).cuda())
    mb = runner.output_batch(db, mo)
    mb.scores = f.token_scores(mb, _tensor(h.w, b.dtype), h.b)
    po = P.to_host(f.prune(mb, torch.from_numpy(rho).cuda()), b.dtype)
    torch.cuda.synchronize()
    assert int(f.status.item()) == 0

    om = oracle.stage(b, StageSpec(True, False, False, r=spec.r))
    os_ = oracle.token_scores(b.dtype, om["offsets"], om["x"], h.w, h.b)
    op = oracle.prune(b.dtype, om["offsets"], om["x"], om["sizes"], os_, rho)
    tol = _bound(b.dtype, om["x"], h.w, h.b) + np.spacing(np.abs(os_)).astype(np.float64)
    g_off, o_off = po["offsets"], op["offsets"]
    near = 0
    for i in range(b.batch):
        gi = po["keep_idx"][g_off[i]:g_off[i + 1]]
        oi = op["keep_idx"][o_off[i]:o_off[i + 1]]
        if g_off[i + 1] - g_off[i] == o_off[i + 1] - o_off[i] and np.array_equal(gi, oi):
            np.testing.assert_array_equal(po["x"][g_off[i]:g_off[i + 1]], op["x"][o_off[i]:o_off[i + 1]])
            continue
        rows = slice(om["offsets"][i], om["offsets"][i + 1])
        assert op["prune_gap"][i] <= 2 * tol[rows].max(), (i, op["prune_gap"][i])
        near += 1
    print(f"[merge -> scores -> prune] {b.batch} samples, {near} decided by a near-tie")
