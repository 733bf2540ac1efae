"""The merge router with profile scaling (Sec. III-C, Eq. 4-5) on the GPU against the
oracle: merge counts bit-exact (a decision closer than 1e-9 to an integer boundary is
counted and reported), scaled ratios within float rounding, outputs at the original
sample id, degenerate profiles, malformed inputs, and a merge driven by the router."""
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
from workloads import StageSpec, make_router, make_workload  # noqa: E402

pytestmark = pytest.mark.gpu

NEAR = 1e-9   # a floor decision this close to an integer may round either way


def _check(b, rs, label, batch=None, ids=None, n_ids=None):
    f = runner.Fusion(b.batch, 1)
    db = P.device_batch(b)
    if batch is not None:
        db.batch = torch.full((1,), batch, dtype=torch.int32, device="cuda")
    if ids is not None:
        db.ids = torch.from_numpy(ids).cuda()
    o = f.merge_router(db, torch.from_numpy(rs.w.copy()).cuda() if b.dtype == "f32" else
                       torch.from_numpy(rs.w.view(np.int16).copy()).cuda(), rs.beta, rs.tau_tgt, rs.tau_ref)
    torch.cuda.synchronize()
    assert int(f.status.item()) == 0, label
    nb = b.batch if batch is None else batch
    ref = oracle.merge_router(b.dtype, b.offsets[:nb + 1], b.x, rs.w, rs.beta, rs.tau_tgt, rs.tau_ref,
                              ids=None if ids is None else ids[:nb], n_ids=n_ids or b.batch)
    where = np.arange(nb) if ids is None else ids[:nb]
    g_r = o["r"].cpu().numpy()[where]
    g_m = o["m"].cpu().numpy()[where]
    near = ref["r_gap"][where] < NEAR
    bad = (g_r != ref["r"][where]) & ~near
    assert not bad.any(), (label, np.nonzero(bad)[0][:5], g_r[bad][:5], ref["r"][where][bad][:5])
    np.testing.assert_allclose(g_m, ref["mt"][where], rtol=1e-6, atol=1e-7, err_msg=label)
    print(f"[{label}] {len(where)} samples, {int(near.sum())} near-integer decisions, r mean {g_r.mean():.2f}")
    return o, ref


@pytest.mark.parametrize("name", ["deit_s_chain12_bf16_b256", "deit_s_stage_f32_b8", "ragged_b8192_n65_chain4_f32"])
def test_router_matches_oracle(name):
    w = make_workload(name, batch=512 if "ragged" in name else None)
    rs = make_router(np.random.default_rng(5), w.batch.dim, w.batch.dtype)
    _check(w.batch, rs, name)


def test_router_outputs_by_id_and_device_count():
    w = make_workload("deit_s_chain12_bf16_b256", batch=64)
    rs = make_router(np.random.default_rng(6), w.batch.dim, "bf16")
    ids = np.random.default_rng(7).permutation(64).astype(np.int32)
    o, _ = _check(w.batch, rs, "ids + device count 40", batch=40, ids=ids, n_ids=64)
    untouched = np.setdiff1d(np.arange(64), ids[:40])
    assert np.all(o["r"].cpu().numpy()[untouched] == 0)


def test_router_degenerate_profiles():
    w = make_workload("deit_s_chain12_bf16_b256", batch=32)
    b = w.batch
    rs = make_router(np.random.default_rng(8), b.dim, "bf16", tau_tgt=1.0)   # keep everything: r = 0
    o, _ = _check(b, rs, "tau_tgt = 1")
    assert np.all(o["r"].cpu().numpy() == 0)
    rs.beta, rs.tau_tgt, rs.tau_ref = 80.0, 0.0, 0.5                           # saturated and clamped
    o, _ = _check(b, rs, "saturated")
    np.testing.assert_array_equal(o["r"].cpu().numpy(), np.diff(b.offsets) // 2)


def test_router_bad_offsets_raise_status():
    w = make_workload("deit_s_stage_f32_b8")
    b = w.batch
    rs = make_router(np.random.default_rng(9), b.dim, "f32")
    f = runner.Fusion(b.batch, 1)
    db = P.device_batch(b)
    bad = b.offsets.copy()
    bad[3] = bad[2] - 1
    rg = fz.ragged(db.max_batch, db.max_tokens, db.max_rows, torch.from_numpy(bad).cuda())
    r = torch.full((b.batch,), -7, dtype=torch.int32, device="cuda")
    fz.check(fz.fusion_merge_router(fz.FUSION_F32, rg, db.x, db.dim, torch.from_numpy(rs.w).cuda(), rs.beta,
                                    rs.tau_tgt, rs.tau_ref, r, None, f.status))
    torch.cuda.synchronize()
    assert int(f.status.item()) & fz.FUSION_DEV_BAD_OFFSETS


def test_merge_driven_by_router():
    """fusion_merge_router -> fusion_stage (merge) equals the oracle's router -> merge."""
    w = make_workload("deit_s_chain12_bf16_b256", batch=48)
    b = w.batch
    rs = make_router(np.random.default_rng(10), b.dim, "bf16")
    f = runner.Fusion(b.batch, 1)
    db = P.device_batch(b)
    ro = f.merge_router(db, torch.from_numpy(rs.w.view(np.int16).copy()).cuda(), rs.beta, rs.tau_tgt, rs.tau_ref)
    ref = oracle.merge_router("bf16", b.offsets, b.x, rs.w, rs.beta, rs.tau_tgt, rs.tau_ref)
    assert not (ref["r_gap"] < NEAR).any()
    g = P.to_host(f.stage(db, fz.FUSION_STAGE_MERGE, ro["r"]), "bf16")
    torch.cuda.synchronize()
    assert int(f.status.item()) == 0
    o = oracle.stage(b, StageSpec(True, False, False, r=ref["r"]))
    rep = P.Report()
    ids = np.arange(b.batch)
    nb = int(g["batch"][0])
    P.compare_tokens(rep, "bf16", b.offsets, ids, b.offsets, ids, g, o, g["ids"][:nb], o["ids"])
    print(f"[router -> merge] {rep.summary()}")
    rep.check()
