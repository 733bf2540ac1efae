"""CUDA path vs the CPU oracle on the seeded workloads (GPU only).

Reduced batches span many CTAs and ragged tails and finish in seconds on the
oracle; the full-size checks run the GPU at the benchmark's sizes and compare a
seeded sample of images against the oracle run on those images alone (images
are independent apart from compaction order, which is compared through ids).
"""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle  # noqa: E402
import parity as P  # noqa: E402
from paper_2607_02612_gb300 import runner  # noqa: E402
from workloads import Batch, make_workload  # noqa: E402

pytestmark = pytest.mark.gpu

CASES = [
    ("deit_s_stage_f32_b8", None),
    ("deit_s_chain12_bf16_b256", None),
    ("deit_b_stage_bf16_b512", 96),
    ("vit_l16_384_stage_bf16_b128", 12),
    ("ragged_b8192_n65_chain4_f32", 512),
    ("ragged_b8192_n65_chain4_bf16", 512),
]
IDS = [c[0] for c in CASES]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_02612_gb300 import build
    build()
    assert torch.cuda.is_available()


def _first(w, attr):
    for s in w.stages:
        if getattr(s, attr):
            return s
    raise AssertionError(attr)


def _report(rep, label):
    print(f"[{label}] {rep.summary()}")
    rep.check()


@pytest.mark.parametrize("name,B", CASES, ids=IDS)
def test_merge_parity(name, B):
    w = make_workload(name, batch=B)
    b, spec = w.batch, w.stages[0]
    fz = runner.Fusion(b.batch)
    db = P.device_batch(b)
    g = P.to_host(fz.merge(db, torch.from_numpy(spec.r).cuda()), b.dtype)
    assert int(fz.status.item()) == 0
    o = oracle.merge(b.dtype, b.offsets, b.x, b.keys, b.sizes, b.scores, spec.r)
    np.testing.assert_array_equal(g["offsets"], o["offsets"])
    rep = P.Report()
    P.count_decision_near_ties(rep, o)
    ids = np.arange(b.batch)
    P.compare_tokens(rep, b.dtype, b.offsets, ids, b.offsets, ids, g, o, ids, ids, a_match_gpu=g["a_match"])
    for i in range(b.batch):
        if i in rep.excluded:
            continue
        a0, a1 = b.offsets[i], b.offsets[i + 1]
        assert np.array_equal(g["dst_map"][a0:a1], o["dst_map"][a0:a1]), f"dst_map of sample {i}"
    _report(rep, f"merge {name}")


@pytest.mark.parametrize("name,B", CASES, ids=IDS)
def test_exit_parity(name, B):
    w = make_workload(name, batch=B)
    b, spec = w.batch, _first(w, "exit")
    fz = runner.Fusion(b.batch, spec.head.classes)
    g = P.to_host(fz.exit_check(P.device_batch(b), runner.head_tensors(spec.head, b.dtype)), b.dtype)
    assert int(fz.status.item()) == 0
    o = oracle.exit_check(b.dtype, b.offsets, b.x, spec.head)
    rep = P.Report()
    P.compare_exit(rep, b.dtype, np.arange(b.batch), g["exit_mask"], g["logits"], g["max_prob"], o)
    _report(rep, f"exit {name}")


@pytest.mark.parametrize("name,B", CASES, ids=IDS)
def test_prune_parity(name, B):
    w = make_workload(name, batch=B)
    b, spec = w.batch, _first(w, "prune")
    fz = runner.Fusion(b.batch)
    g = P.to_host(fz.prune(P.device_batch(b), torch.from_numpy(spec.rho).cuda()), b.dtype)
    assert int(fz.status.item()) == 0
    o = oracle.prune(b.dtype, b.offsets, b.x, b.sizes, b.scores, spec.rho)
    np.testing.assert_array_equal(g["offsets"], o["offsets"])
    t = int(o["offsets"][-1])
    np.testing.assert_array_equal(g["keep_idx"][:t], o["keep_idx"])
    np.testing.assert_array_equal(g["x"][:t], o["x"])
    np.testing.assert_array_equal(g["sizes"][:t], o["sizes"])
    np.testing.assert_array_equal(g["scores"][:t], o["scores"])


@pytest.mark.parametrize("name,B", CASES[:2] + CASES[4:], ids=IDS[:2] + IDS[4:])
def test_compact_parity(name, B):
    w = make_workload(name, batch=B)
    b = w.batch
    mask = (np.random.default_rng(17).random(b.batch) < 0.45).astype(np.uint8)
    fz = runner.Fusion(b.batch)
    g = P.to_host(fz.compact(P.device_batch(b), torch.from_numpy(mask).cuda()), b.dtype)
    assert int(fz.status.item()) == 0
    o = oracle.compact(b.dtype, b.offsets, b.x, b.sizes, b.scores, mask)
    nb = int(g["batch"][0])
    assert nb == o["n_out"]
    np.testing.assert_array_equal(g["offsets"][:nb + 1], o["offsets"])
    np.testing.assert_array_equal(g["ids"][:nb], o["ids"])
    t = int(o["offsets"][-1])
    np.testing.assert_array_equal(g["keep_idx"][:t], o["keep_idx"])
    np.testing.assert_array_equal(g["x"][:t], o["x"])


@pytest.mark.parametrize("name,B", CASES, ids=IDS)
def test_fused_stage_parity(name, B):
    """merge -> exit -> prune -> compact in one call equals the oracle's composition."""
    w = make_workload(name, batch=B)
    b, spec = w.batch, _first(w, "exit")
    fz = runner.Fusion(b.batch, spec.head.classes)
    r, rho, head = P.stage_tensors(spec, b.dtype)
    g = P.to_host(fz.stage(P.device_batch(b), P.flags_of(spec), r, rho, head, a_match=True), b.dtype)
    assert int(fz.status.item()) == 0
    o = oracle.stage(b, spec)
    rep = P.Report()
    P.count_decision_near_ties(rep, o)
    ids = np.arange(b.batch)
    P.compare_exit(rep, b.dtype, ids, g["exit_mask"], g["logits"], g["max_prob"], o)
    nb = int(g["batch"][0])
    P.compare_tokens(rep, b.dtype, b.offsets, ids, b.offsets, ids, g, o, g["ids"][:nb], o["ids"],
                     a_match_gpu=g["a_match"])
    _report(rep, f"stage {name}")


@pytest.mark.parametrize("name,B,graph", [
    ("deit_s_chain12_bf16_b256", None, True),
    ("ragged_b8192_n65_chain4_bf16", 1024, False),
    ("ragged_b8192_n65_chain4_f32", 1024, True),
])
def test_chain_parity(name, B, graph):
    """Every stage of a chained schedule (compaction between blocks, no host sync)."""
    w = make_workload(name, batch=B)
    g_outs, status = P.chain_on_gpu(w, graph=graph)
    assert status == 0
    o_outs = oracle.chain(w)
    rep = P.Report()
    P.compare_chain(rep, w, g_outs, o_outs)
    assert rep.compared_samples > 0
    _report(rep, f"chain {name}")


def test_chain_host_results():
    """The serving loop of the end-to-end measurement: pinned host inputs copied in, the chain
    replayed as a CUDA graph, the results fetched into pinned host buffers (survivor count
    first, then the survivors' exact extent).  On two consecutive replays the device outputs
    match the oracle's chain and the fetched host copies equal the device outputs."""
    w = make_workload("deit_s_chain12_bf16_b256", batch=64)
    b = w.batch
    fzr = runner.Fusion(b.batch, max(s.head.classes for s in w.stages if s.head is not None))
    db = P.device_batch(b)
    stages = [runner.ChainStage(P.flags_of(s), *P.stage_tensors(s, b.dtype)) for s in w.stages]
    ch = runner.Chain(fzr, db, stages)
    hr = ch.host_results()
    xh = torch.from_numpy(np.ascontiguousarray(b.x).view(np.int16)).pin_memory()
    ch.run()
    torch.cuda.synchronize()
    g = ch.capture()
    o_outs = oracle.chain(w)
    for rep_i in range(2):
        db.x.view(torch.int16).copy_(xh, non_blocking=True)
        g.replay()
        res, nbytes = hr.fetch()
        assert int(fzr.status.item()) == 0
        d_outs = [P.to_host(o, b.dtype) for o in ch.outs]
        rep = P.Report()
        P.compare_chain(rep, w, d_outs, o_outs)
        assert rep.compared_samples > 0
        _report(rep, f"host results, replay {rep_i}")
        last = d_outs[-1]
        nb = int(last["batch"][0])
        rows = int(last["offsets"][nb])
        assert res["batch"] == nb
        np.testing.assert_array_equal(res["offsets"].numpy(), last["offsets"][:nb + 1])
        np.testing.assert_array_equal(res["ids"].numpy(), last["ids"][:nb])
        np.testing.assert_array_equal(res["sizes"].numpy(), last["sizes"][:rows])
        np.testing.assert_array_equal(res["x"].view(torch.int16).numpy().view(np.uint16), last["x"][:rows])
        entering = [b.batch] + [int(o["batch"][0]) for o in d_outs[:-1]]
        exits = [(o, n) for o, n in zip(d_outs, entering) if o["exit_mask"] is not None]
        assert len(res["exits"]) == len(exits) == sum(1 for s in w.stages if s.exit)
        for (hm, hp), (o, n) in zip(res["exits"], exits):
            assert len(hm) == len(hp) == n
            np.testing.assert_array_equal(hm.numpy(), o["exit_mask"][:n])
            np.testing.assert_array_equal(hp.numpy(), o["max_prob"][:n])
        assert nbytes >= res["x"].numel() * 2


def _np(t: torch.Tensor) -> np.ndarray:
    return (t.view(torch.int16) if t.dtype == torch.bfloat16 else t).numpy().copy()


def _host_copy(res):
    r = {k: (_np(v) if isinstance(v, torch.Tensor) else v) for k, v in res.items() if k != "exits"}
    r["exits"] = [(_np(m), _np(p)) for m, p in res["exits"]]
    return r


@pytest.mark.parametrize("name,B", [("deit_s_chain12_bf16_b256", 64), ("ragged_b8192_n65_chain4_f32", 256)])
def test_pipeline_overlapped_steps(name, B):
    """Steps submitted back to back through the two-slot pipeline (input copies overlapping the
    previous step's kernels, results one step late) give, step by step, the results of the same
    inputs run one at a time; those match the oracle's chain for both inputs.  The DeiT-S bf16
    schedule and the float32 65-token schedule with an exit check at every block."""
    wa = make_workload(name, batch=B)
    wb = type(wa)(wa.spec, make_workload(name, batch=B, seed_offset=1).batch, wa.stages)
    b = wa.batch
    assert np.array_equal(b.offsets, wb.batch.offsets)
    bf = b.dtype == "bf16"
    fzr = runner.Fusion(b.batch, max(s.head.classes for s in wa.stages if s.head is not None))
    stages = [runner.ChainStage(P.flags_of(s), *P.stage_tensors(s, b.dtype)) for s in wa.stages]
    ch = runner.Chain(fzr, P.device_batch(b), stages)

    def pinned(bb):
        return {"x": torch.from_numpy(np.ascontiguousarray(bb.x).view(np.int16) if bf else bb.x).pin_memory(),
                "sizes": torch.from_numpy(bb.sizes).pin_memory(),
                "scores": torch.from_numpy(bb.scores).pin_memory(),
                "offsets": torch.from_numpy(bb.offsets).pin_memory()}
    hosts = [pinned(wa.batch), pinned(wb.batch)]
    # one at a time, on a separate chain
    solo = ch.clone()
    hr = solo.host_results()
    want = []
    for i, w in enumerate((wa, wb)):
        db = solo.inp
        (db.x.view(torch.int16) if bf else db.x).copy_(hosts[i]["x"])
        db.sizes.copy_(hosts[i]["sizes"])
        db.scores.copy_(hosts[i]["scores"])
        db.offsets.copy_(hosts[i]["offsets"])
        solo.run()
        want.append(_host_copy(hr.fetch()[0]))
        assert want[-1]["status"] == 0
        rep = P.Report()
        P.compare_chain(rep, w, [P.to_host(o, b.dtype) for o in solo.outs], oracle.chain(w), fresh_logits=(i == 0))
        assert rep.compared_samples > 0
        _report(rep, f"pipeline reference input {i}")
    pipe = runner.Pipeline(ch)
    seq = [0, 1, 1, 0, 1, 0, 0]
    got = []
    for i in seq:
        r = pipe.submit(hosts[i])
        if r is not None:
            got.append(_host_copy(r[0]))
    got.append(_host_copy(pipe.finish()[0]))
    assert pipe.status() == 0
    assert len(got) == len(seq)
    for k, (i, g) in enumerate(zip(seq, got)):
        e = want[i]
        assert g["batch"] == e["batch"] and g["status"] == 0, (k, i)
        for name in ("offsets", "ids", "sizes", "x"):
            np.testing.assert_array_equal(g[name], e[name], err_msg=f"step {k} input {i} {name}")
        assert len(g["exits"]) == len(e["exits"]) == sum(1 for s in wa.stages if s.exit)
        for (gm, gp), (em, ep) in zip(g["exits"], e["exits"]):
            np.testing.assert_array_equal(gm, em)
            np.testing.assert_array_equal(gp, ep)
    assert want[0]["batch"] != want[1]["batch"] or not np.array_equal(want[0]["ids"], want[1]["ids"])


def _mlp_heads_at(w, placement, seed, tau_mode="gap"):
    """Put MLP exit heads on the given exit stages ({stage index: pool}) and set each tau from the
    oracle's max_prob values of that stage's merged tokens (what the head reads, Sec. III-B):
    "gap" puts tau in the widest gap around the median, so that about half the images exit and
    none sits at the threshold; "drawn" draws tau uniformly between the 25th and 75th
    percentiles with the seeded generator, wherever it falls.  Returns the oracle's chain."""
    from workloads import make_mlp_head
    b = w.batch
    rng = np.random.default_rng(seed)
    outs = []
    bb = b
    for si, spec in enumerate(w.stages):
        if si in placement:
            head = make_mlp_head(rng, placement[si], b.dim, 2 * b.dim, 1000, b.dtype)
            T = int(bb.offsets[-1])
            ids = np.arange(bb.batch, dtype=np.int32) if bb.ids is None else np.asarray(bb.ids, np.int32)
            if spec.merge:
                m = oracle.merge(b.dtype, bb.offsets, bb.x[:T], bb.keys[:T], bb.sizes[:T], bb.scores[:T],
                                 spec.r[ids])
                offs, xs, szs = m["offsets"], m["x"], m["sizes"]
            else:
                offs, xs, szs = bb.offsets, bb.x[:T], bb.sizes[:T]
            mp = np.sort(oracle.exit_mlp(b.dtype, offs, xs, szs, head)["max_prob"])
            if tau_mode == "gap":
                lo = max(0, len(mp) // 2 - 5)
                k = lo + int(np.argmax(np.diff(mp[lo:lo + 11])))
                head.tau = float(np.float32(0.5 * (mp[k] + mp[k + 1])))
            else:
                head.tau = float(np.float32(rng.uniform(np.percentile(mp, 25), np.percentile(mp, 75))))
            spec.mlp_head = head
            spec.head = None
        res = oracle.stage(bb, spec)
        outs.append(res)
        bb = oracle.next_batch(bb, res)
    return outs


@pytest.mark.parametrize("graph,tau_mode", [(True, "gap"), (False, "gap"), (True, "drawn")])
def test_chain_with_mlp_heads(graph, tau_mode):
    """The DeiT-S schedule with the paper's MLP exit heads inside the fused stage: SpatialPool
    at block 8, CLS-only at block 10 (the linear head at blocks 4 and 6); every stage against
    the oracle, whose MLP exit check reads the merged tokens as stored.  Exit decisions must
    agree wherever the oracle's margin |c - tau| is at least 1e-6 (closer ones are counted); one
    case draws tau from the generator instead of placing it in a gap."""
    from workloads import POOL_CLS, POOL_SPATIAL
    w = make_workload("deit_s_chain12_bf16_b256", batch=64)
    o_outs = _mlp_heads_at(w, {7: POOL_SPATIAL, 9: POOL_CLS}, 21, tau_mode)
    g_outs, status = P.chain_on_gpu(w, graph=graph)
    assert status == 0
    rep = P.Report()
    P.compare_chain(rep, w, g_outs, o_outs)
    assert rep.compared_samples > 0
    for si in (7, 9):
        n = int(o_outs[si]["exit_mask"].sum())
        assert 0 < n < len(o_outs[si]["exit_mask"]), (si, n)
    _report(rep, f"chain with MLP heads, graph={graph}, tau {tau_mode}")


@pytest.mark.parametrize("pool", [0, 1])
def test_stage_mlp_f32(pool):
    """One fused float32 stage (merge, MLP exit check on the merged tokens, prune) on the
    65-token schedule, tau drawn from the generator."""
    w = make_workload("ragged_b8192_n65_chain4_f32", batch=300, seed_offset=3)
    w = type(w)(w.spec, w.batch, w.stages[:1])
    w.stages[0].prune = True
    w.stages[0].rho = np.full(w.batch.batch, 0.7, np.float32)
    o_outs = _mlp_heads_at(w, {0: pool}, 31 + pool, "drawn")
    g_outs, status = P.chain_on_gpu(w)
    assert status == 0
    rep = P.Report()
    P.compare_chain(rep, w, g_outs, o_outs)
    assert rep.compared_samples > 0
    _report(rep, f"f32 MLP stage pool {pool}")


def _subset(batch: Batch, idx: np.ndarray) -> Batch:
    """The images idx of a batch, repacked (ids keep the original image numbers)."""
    counts = np.diff(batch.offsets)[idx]
    offs = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    rows = np.concatenate([np.arange(batch.offsets[i], batch.offsets[i + 1]) for i in idx])
    x = batch.x[rows]
    keys = x if batch.keys_alias else batch.keys[rows]
    return Batch(batch.dtype, offs, x, keys, batch.sizes[rows], batch.scores[rows], ids=idx.astype(np.int32))


@pytest.mark.parametrize("name", ["deit_b_stage_bf16_b512", "vit_l16_384_stage_bf16_b128",
                                  "ragged_b8192_n65_chain4_bf16", "ragged_b8192_n65_chain4_f32",
                                  "deit_s_chain12_bf16_b256"])
def test_full_size_sampled(name):
    """Full batch on the GPU in the benchmark's configuration (CUDA graph); the oracle
    recomputes a seeded sample of images one by one and every stage of theirs must match."""
    w = make_workload(name)
    g_outs, status = P.chain_on_gpu(w, graph=True)
    assert status == 0
    n = 48 if w.batch.batch > 48 else w.batch.batch
    idx = np.sort(np.random.default_rng(99).choice(w.batch.batch, n, replace=False))
    w_sub = type(w)(w.spec, _subset(w.batch, idx), w.stages)
    o_outs = oracle.chain(w_sub)
    rep = P.Report()
    # per stage, compare the sampled ids only
    o_ids_in = idx.astype(np.int32)
    o_off_in = w_sub.batch.offsets
    g_ids_in = np.arange(w.batch.batch, dtype=np.int32)
    g_off_in = w.batch.offsets
    for s, (g, o) in enumerate(zip(g_outs, o_outs)):
        spec = w.stages[s]
        P.count_decision_near_ties(rep, o)
        g_nb = int(g["batch"][0])
        if spec.exit:
            gpos = {int(t): i for i, t in enumerate(g_ids_in)}
            for i, t in enumerate(o_ids_in):
                t = int(t)
                if t in rep.excluded:
                    continue
                ig = gpos[t]
                if g["exit_mask"][ig] != o["exit_mask"][i]:
                    if o["exit_gap"][i] < P.NEAR_TIE:
                        rep.near_tie_mismatch["exit"] += 1
                        rep.excluded.add(t)
                    else:
                        rep.fail(f"stage {s}: exit differs for image {t}")
        P.compare_tokens(rep, w.batch.dtype, o_off_in, o_ids_in, g_off_in, g_ids_in, g, o, g["ids"][:g_nb],
                         o["ids"])
        o_ids_in, o_off_in = o["ids"], o["offsets"]
        g_ids_in, g_off_in = g["ids"][:g_nb], g["offsets"][:g_nb + 1]
    assert rep.compared_samples > 0
    _report(rep, f"full {name}")
