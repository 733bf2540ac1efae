"""Edge cases and device-side error reporting of the CUDA path (GPU only).

Degenerate samples (P = 0, 1, 2), clamped merge counts, keep ratios 0 and 1, all or
no samples exiting, exact ties (identical keys), zero-norm keys, signed-zero
scores, keys separate from or aliased to the tokens, an empty batch, a device batch
count below the host bound, the largest supported sample, and malformed inputs
that must raise status bits without touching memory out of bounds.
"""
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
from workloads import Batch, Head, StageSpec, f32_to_bf16_bits  # noqa: E402

pytestmark = pytest.mark.gpu


def make_batch(counts, dim, dtype, seed=0, keys="alias", kdim=None, same_keys=False, zero_key=False,
               signed_zero_scores=False, sizes="ones"):
    rng = np.random.default_rng(seed)
    counts = np.asarray(counts)
    offs = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    T = int(offs[-1])
    x32 = rng.standard_normal((T, dim)).astype(np.float32)
    if same_keys:
        x32[:] = rng.standard_normal(dim).astype(np.float32)
    if zero_key and T > 3:
        x32[3] = 0.0
    sz = np.ones(T, np.float32) if sizes == "ones" else rng.integers(1, 5, T).astype(np.float32)
    sc = rng.random(T).astype(np.float32)
    if signed_zero_scores:
        sc[::2] = -0.0
        sc[1::2] = 0.0
    x = f32_to_bf16_bits(x32) if dtype == "bf16" else x32
    if keys == "alias":
        k = x
    else:
        k32 = rng.standard_normal((T, kdim or dim)).astype(np.float32)
        k = f32_to_bf16_bits(k32) if dtype == "bf16" else k32
    return Batch(dtype, offs, x, k, sz, sc)


def make_head(dim, C, dtype, tau, seed=1, scale=1.0):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((C, dim)) * scale).astype(np.float32)
    rd = (lambda a: f32_to_bf16_bits(a)) if dtype == "bf16" else (lambda a: a)
    return Head(rd(np.ones(dim, np.float32)), rd(np.zeros(dim, np.float32)), 1e-6, rd(W),
                np.zeros(C, np.float32), tau)


def run_stage_and_compare(b, spec, label):
    classes = spec.head.classes if spec.head is not None else 1
    f = runner.Fusion(b.batch, classes)
    r, rho, head = P.stage_tensors(spec, b.dtype)
    g = P.to_host(f.stage(P.device_batch(b), P.flags_of(spec), r, rho, head, a_match=spec.merge), b.dtype)
    assert int(f.status.item()) == 0, label
    o = oracle.stage(b, spec)
    rep = P.Report()
    ids = np.arange(b.batch)
    if spec.exit:
        P.compare_exit(rep, b.dtype, ids, g["exit_mask"], g["logits"], g["max_prob"], o)
    nb = int(g["batch"][0])
    assert nb == o["n_out"], label
    P.compare_tokens(rep, b.dtype, b.offsets, ids, b.offsets, ids, g, o, g["ids"][:nb], o["ids"],
                     a_match_gpu=g.get("a_match"))
    print(f"[{label}] {rep.summary()}")
    rep.check()
    return g, o


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("keys", ["alias", "separate"])
def test_degenerate_and_ragged_samples(dtype, keys):
    counts = [1, 2, 3, 4, 5, 6, 17, 64, 65, 1, 33, 2]
    b = make_batch(counts, 48, dtype, keys=keys, kdim=32, sizes="u1to4")
    B = len(counts)
    r = np.array([0, 3, 1, 1, 2, 99, 8, -4, 40, 5, 16, 0], np.int32)
    rho = np.array([0.0, 1.0, 0.5, 0.3, 1.0, 0.0, 0.61, 0.9, 0.25, 1.0, 0.99, 0.5], np.float32)
    for flags in [(True, False, False), (False, False, True), (True, False, True), (True, True, True)]:
        m, e, p = flags
        head = make_head(48, 10, dtype, 0.45, scale=0.15) if e else None
        spec = StageSpec(m, e, p, r=r, rho=rho, head=head)
        run_stage_and_compare(b, spec, f"{dtype}/{keys}/{flags}")
    assert B == len(r)


@pytest.mark.parametrize("dim,classes", [(16, 1), (80, 127), (208, 129), (384, 1000), (1024, 1000), (48, 640)])
def test_exit_head_widths(dim, classes):
    """The linear exit head over widths that end inside a 64-dim weight chunk (16, 80, 208),
    class counts below, at and past a 128-class tile, and heads of one to eight tiles; tau in
    the widest gap between the oracle's max_prob values around the median, so that about half
    the samples exit and none sits at the threshold."""
    rng = np.random.default_rng(dim + classes)
    counts = rng.integers(1, 24, 41)
    b = make_batch(counts, dim, "bf16", seed=dim, sizes="u1to4")
    head = make_head(dim, classes, "bf16", 0.5, seed=classes, scale=2.0 / np.sqrt(dim))
    spec = StageSpec(False, True, False, head=head)
    o = oracle.stage(b, spec)
    mp = np.sort(o["max_prob"])
    lo = len(mp) // 2 - 5
    k = lo + int(np.argmax(np.diff(mp[lo:lo + 11])))
    head.tau = float(np.float32(0.5 * (mp[k] + mp[k + 1]))) if mp[k + 1] > mp[k] else float(mp[k])
    run_stage_and_compare(b, StageSpec(False, True, False, head=head), f"exit head dim {dim} classes {classes}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_identical_keys_zero_norm_and_signed_zero(dtype):
    b = make_batch([33, 20, 9], 32, dtype, same_keys=True, signed_zero_scores=True)
    spec = StageSpec(True, False, True, r=np.array([5, 9, 4], np.int32), rho=np.array([0.5, 0.7, 0.34], np.float32))
    g, o = run_stage_and_compare(b, spec, f"ties {dtype}")
    b2 = make_batch([17, 17], 32, dtype, zero_key=True, seed=4)
    spec2 = StageSpec(True, False, False, r=np.array([8, 8], np.int32))
    run_stage_and_compare(b2, spec2, f"zero-key {dtype}")


def _grid_batch(counts, dim, seed, scale=1.0):
    """bf16 tokens on a coarse grid (multiples of 2^-5 in [-4, 4), times `scale`), so that
    size-weighted means land exactly on, or right next to, bf16 rounding midpoints; sizes
    mix integers and halves (power-of-two and other sums); keys are unit vectors that send
    A token a to B token f(a), with one, two or three sources per destination."""
    rng = np.random.default_rng(seed)
    counts = np.asarray(counts)
    offs = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    T = int(offs[-1])
    x32 = (rng.integers(-128, 128, (T, dim)) / 32.0 * scale).astype(np.float32)
    k32 = np.zeros((T, dim), np.float32)
    for i in range(len(counts)):
        N = int(counts[i]); base = int(offs[i]); nB = N // 2
        for pos in range(1, N):
            if pos % 2 == 1:
                k32[base + pos, ((pos - 1) // 2) % dim] = 1.0
            else:
                a = (pos - 2) // 2
                dest = a if a < nB // 3 else (a // 2 if a < 2 * nB // 3 else a // 3)
                k32[base + pos, min(dest, nB - 1) % dim] = 1.0
        k32[base, :] = 1.0
    sz = rng.choice(np.array([1, 1, 1, 2, 3, 0.5, 1.5, 7], np.float32), T).astype(np.float32)
    sc = rng.random(T).astype(np.float32)
    return Batch("bf16", offs, f32_to_bf16_bits(x32), f32_to_bf16_bits(k32), sz, sc)


@pytest.mark.parametrize("scale", [1.0, 2.0 ** -100, 2.0 ** -110])
def test_merged_mean_rounding_ties_and_near_ties(scale):
    """bf16 merged tokens must be the exactly rounded weighted mean, ties to even, whatever
    path the kernel takes (two-term power-of-two sums, the bounded float path, the exact
    float-float path for three sources or near-midpoint and tiny values)."""
    b = _grid_batch([65, 129, 97, 33, 65], 64, seed=21, scale=scale)
    r = np.array([32, 64, 40, 16, 20], np.int32)
    run_stage_and_compare(b, StageSpec(True, False, False, r=r), f"grid means scale={scale}")


@pytest.mark.parametrize("tau", [0.0, 2.0])
def test_all_or_no_samples_exit(tau):
    b = make_batch([10] * 37, 64, "bf16", seed=3)
    spec = StageSpec(True, True, True, r=np.full(37, 3, np.int32), rho=np.full(37, 0.5, np.float32),
                     head=make_head(64, 130, "bf16", tau))
    g, o = run_stage_and_compare(b, spec, f"tau={tau}")
    assert int(g["batch"][0]) == (0 if tau == 0.0 else 37)
    assert g["offsets"][0] == 0


@pytest.mark.parametrize("dtype,classes", [("bf16", 1100), ("f32", 1100), ("bf16", 300), ("f32", 7)])
def test_exit_check_head_sizes(dtype, classes):
    """Heads of up to 8 class tiles run as one cluster per sample tile, larger ones (1100
    classes: 9 tiles) on the kernel with a global last-CTA merge; both against the oracle."""
    b = make_batch([9, 17, 33, 5, 12, 40, 7, 21, 3, 30], 64, dtype, seed=13)
    r, rho = np.full(10, 3, np.int32), np.full(10, 0.6, np.float32)
    # tau halfway between the 5th and 6th largest max-probability: half the samples exit
    probe = oracle.stage(b, StageSpec(True, True, True, r=r, rho=rho, head=make_head(64, classes, dtype, 2.0, scale=0.5)))
    mp = np.sort(probe["max_prob"])
    spec = StageSpec(True, True, True, r=r, rho=rho, head=make_head(64, classes, dtype, float(mp[4] + mp[5]) / 2, scale=0.5))
    g, o = run_stage_and_compare(b, spec, f"head {dtype} C={classes}")
    assert int(g["batch"][0]) == 5


def test_empty_batch_and_device_count():
    b = make_batch([5, 7, 9, 11], 32, "f32", seed=8)
    db = P.device_batch(b)
    f = runner.Fusion(4, 3)
    spec = StageSpec(True, True, True, r=np.full(4, 2, np.int32), rho=np.full(4, 0.5, np.float32),
                     head=make_head(32, 3, "f32", 2.0))
    r, rho, head = P.stage_tensors(spec, "f32")
    # device count 0: nothing survives, nothing is written
    db.batch = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = P.to_host(f.stage(db, 7, r, rho, head), "f32")
    assert int(f.status.item()) == 0
    assert int(g["batch"][0]) == 0 and g["offsets"][0] == 0
    assert np.all(g["keep_idx"] == -1)
    # device count 2 of a bound of 4: only the first two samples are processed
    db.batch = torch.full((1,), 2, dtype=torch.int32, device="cuda")
    g = P.to_host(f.stage(db, 7, r, rho, head), "f32")
    sub = Batch("f32", b.offsets[:3], b.x, b.keys, b.sizes, b.scores)
    o = oracle.stage(sub, StageSpec(True, True, True, r=spec.r, rho=spec.rho, head=spec.head))
    assert int(g["batch"][0]) == o["n_out"] == 2
    np.testing.assert_array_equal(g["offsets"][:3], o["offsets"])
    np.testing.assert_array_equal(g["keep_idx"][:o["offsets"][-1]], o["keep_idx"])


@pytest.mark.parametrize("dtype,classes", [("bf16", 10), ("bf16", 1000), ("f32", 10), ("bf16", 4000)])
def test_host_batch_bound_zero(dtype, classes):
    """A host batch bound of 0 is a legal empty call: the exit check (cluster kernel up to 1024
    classes, the general one above) and the fused stage with the exit flag return FUSION_OK, raise
    no status bit, touch no exit output, and the stage writes a batch count of 0 and offsets [0]."""
    b = make_batch([5, 7], 32, dtype, seed=3)
    db = P.device_batch(b)
    db.max_batch = 0
    f = runner.Fusion(0, classes)
    head = runner.head_tensors(make_head(32, classes, dtype, 0.5), dtype)
    mask = torch.full((1,), 7, dtype=torch.uint8, device="cuda")
    logits = torch.full((1, classes), 3.0, dtype=torch.float32, device="cuda")
    maxp = torch.full((1,), -1.0, dtype=torch.float32, device="cuda")
    fz.check(fz.fusion_exit_check(runner.DTYPE_CODE[dtype], db.ragged(), db.x, db.dim, head.c_struct(), mask,
                                  logits, maxp, f.workspace, f.ws_bytes, f.status))
    torch.cuda.synchronize()
    assert int(f.status.item()) == 0
    assert int(mask.item()) == 7 and float(maxp.item()) == -1.0 and bool(torch.all(logits == 3.0))
    o = f.stage_outputs(db, 7, head)
    o.update(exit_mask=mask, logits=logits, max_prob=maxp,   # non-null, one row: the call must not touch them
             ids=torch.full((1,), 5, dtype=torch.int32, device="cuda"))
    for k in ("offsets", "batch"):
        o[k] = torch.full_like(o[k], 5)
    r = torch.full((1,), 2, dtype=torch.int32, device="cuda")
    rho = torch.full((1,), 0.5, dtype=torch.float32, device="cuda")
    g = P.to_host(f.stage(db, 7, r, rho, head, out=o), dtype)
    assert int(f.status.item()) == 0
    assert int(g["batch"][0]) == 0 and int(g["offsets"][0]) == 0
    assert int(mask.item()) == 7 and float(maxp.item()) == -1.0 and bool(torch.all(logits == 3.0))


def test_ids_index_router_outputs():
    """With ids, r and rho are read at the original image number."""
    b = make_batch([9, 11, 13], 32, "f32", seed=5)
    b.ids = np.array([2, 0, 1], np.int32)
    spec = StageSpec(True, False, True, r=np.array([3, 1, 2], np.int32), rho=np.array([0.2, 0.6, 0.9], np.float32))
    g, o = run_stage_and_compare(b, spec, "ids")
    np.testing.assert_array_equal(g["ids"][:3], b.ids)


def test_prune_keep_count_is_exact():
    """k = ceil(rho * P) on the exact product, including rho one float step either side of
    k/P (where a rounded product would land on the integer)."""
    rng = np.random.default_rng(12)
    counts, rhos = [], []
    for P in (1, 2, 3, 5, 7, 10, 64, 96, 196, 576, 1023):
        for kk in sorted({0, 1, P // 3, P // 2, P - 1, P}):
            base = np.float32(kk / P)
            for r in (np.nextafter(base, np.float32(0)), base, np.nextafter(base, np.float32(2))):
                counts.append(P + 1)
                rhos.append(r)
    counts += [6, 11, 197]
    rhos += [np.float32(0.4), np.float32(0.1), np.float32(0.7)]
    b = make_batch(counts, 16, "f32", seed=13)
    b.scores = rng.random(len(b.scores)).astype(np.float32)
    spec = StageSpec(False, False, True, r=np.zeros(len(counts), np.int32), rho=np.array(rhos, np.float32))
    g, o = run_stage_and_compare(b, spec, "keep counts")
    np.testing.assert_array_equal(g["offsets"][:len(counts) + 1], o["offsets"])


def test_largest_sample():
    b = make_batch([fz.FUSION_MAX_TOKENS, 3], 16, "bf16", seed=6)
    spec = StageSpec(True, False, True, r=np.array([300, 1], np.int32), rho=np.array([0.37, 1.0], np.float32))
    run_stage_and_compare(b, spec, "max tokens")


# ---------------------------------------------------------------------------
# malformed inputs: status bits, no out-of-bounds access, no token writes
# ---------------------------------------------------------------------------
def _stage_raw(b, db, offsets=None, batch=None, ids=None, keys=None):
    f = runner.Fusion(db.max_batch, 1)
    o = f.stage_outputs(db, 5, None)
    o["x"].fill_(7)
    o["keep_idx"].fill_(-5)
    rr = torch.full((db.max_batch,), 2, dtype=torch.int32, device="cuda")
    rho = torch.full((db.max_batch,), 0.5, dtype=torch.float32, device="cuda")
    rg = fz.ragged(db.max_batch, db.max_tokens, db.max_rows, offsets if offsets is not None else db.offsets,
                   batch, ids)
    fz.check(fz.fusion_stage(fz.FUSION_F32, 5, rg, db.x, db.dim, keys if keys is not None else db.keys,
                             db.key_dim, db.sizes, db.scores, rr, rho, None, None, None, None, o["x"],
                             o["sizes"], o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"], None,
                             f.workspace, f.ws_bytes, f.status))
    torch.cuda.synchronize()
    return int(f.status.item()), o


def test_bad_offsets_raise_status_and_write_nothing():
    b = make_batch([8, 8, 8], 16, "f32", seed=7)
    db = P.device_batch(b)
    for bad in ([0, 8, 4, 24], [0, 8, 16, 99], [-3, 8, 16, 24], [0, 0, 16, 24], [0, 8, 16, 24 + 0]):
        offs = torch.tensor(bad, dtype=torch.int32, device="cuda")
        st, o = _stage_raw(b, db, offsets=offs)
        if bad == [0, 8, 16, 24]:
            assert st == 0
            continue
        assert st & fz.FUSION_DEV_BAD_OFFSETS, bad
        assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7), bad


def test_bad_batch_and_ids_raise_status():
    b = make_batch([8, 8], 16, "f32", seed=9)
    db = P.device_batch(b)
    st, o = _stage_raw(b, db, batch=torch.full((1,), 3, dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_BATCH
    assert torch.all(o["keep_idx"] == -5)
    st, o = _stage_raw(b, db, ids=torch.tensor([0, 7], dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_IDS
    assert torch.all(o["keep_idx"] == -5)


def _stage_raw_exit(db, offsets=None, batch=None, ids=None):
    """bf16 merge + exit + prune on the tcgen05 per-sample kernel, with malformed inputs."""
    head = runner.head_tensors(make_head(db.dim, 10, "bf16", 0.5), "bf16")
    f = runner.Fusion(db.max_batch, 10)
    o = f.stage_outputs(db, 7, head)
    o["x"].fill_(7)
    o["keep_idx"].fill_(-5)
    rr = torch.full((db.max_batch,), 2, dtype=torch.int32, device="cuda")
    rho = torch.full((db.max_batch,), 0.5, dtype=torch.float32, device="cuda")
    rg = fz.ragged(db.max_batch, db.max_tokens, db.max_rows, offsets if offsets is not None else db.offsets,
                   batch, ids)
    fz.check(fz.fusion_stage(fz.FUSION_BF16, 7, rg, db.x, db.dim, db.keys, db.key_dim, db.sizes, db.scores, rr,
                             rho, head.c_struct(), o["exit_mask"], o["logits"], o["max_prob"], o["x"], o["sizes"],
                             o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"], None, f.workspace,
                             f.ws_bytes, f.status))
    torch.cuda.synchronize()
    return int(f.status.item()), o


def test_malformed_inputs_with_exit_check_write_nothing():
    b = make_batch([20, 20, 20], 64, "bf16", seed=11)
    db = P.device_batch(b)
    st, o = _stage_raw_exit(db)
    assert st == 0
    for bad in ([0, 20, 10, 60], [0, 20, 40, 99], [-3, 20, 40, 60], [0, 0, 40, 60]):
        st, o = _stage_raw_exit(db, offsets=torch.tensor(bad, dtype=torch.int32, device="cuda"))
        assert st & fz.FUSION_DEV_BAD_OFFSETS, bad
        assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7), bad
        assert int(o["batch"][0]) == 0 and int(o["offsets"][0]) == 0, bad
    st, o = _stage_raw_exit(db, batch=torch.full((1,), 4, dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_BATCH
    assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7)
    st, o = _stage_raw_exit(db, ids=torch.tensor([0, 9, 1], dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_IDS
    assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7)


def _stage_raw_mlp(db, offsets=None, batch=None, ids=None):
    """bf16 merge + MLP exit (SpatialPool) + prune through fusion_stage_mlp, malformed inputs."""
    from workloads import POOL_SPATIAL, make_mlp_head
    head = runner.mlp_head_tensors(make_mlp_head(np.random.default_rng(4), POOL_SPATIAL, db.dim, 2 * db.dim, 10,
                                                 "bf16", tau=0.5), "bf16")
    f = runner.Fusion(db.max_batch, 10)
    o = f.stage_outputs(db, 7, None, mlp_head=head)
    o["x"].fill_(7)
    o["keep_idx"].fill_(-5)
    ws, nbytes = f.mlp_workspace(db, head)
    rr = torch.full((db.max_batch,), 2, dtype=torch.int32, device="cuda")
    rho = torch.full((db.max_batch,), 0.5, dtype=torch.float32, device="cuda")
    rg = fz.ragged(db.max_batch, db.max_tokens, db.max_rows, offsets if offsets is not None else db.offsets,
                   batch, ids)
    fz.check(fz.fusion_stage_mlp(fz.FUSION_BF16, 7, rg, db.x, db.dim, db.keys, db.key_dim, db.sizes, db.scores, rr,
                                 rho, head.c_struct(), o["exit_mask"], o["logits"], o["max_prob"], o["x"],
                                 o["sizes"], o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"], None,
                                 ws, nbytes, f.status))
    torch.cuda.synchronize()
    return int(f.status.item()), o


def test_malformed_inputs_with_mlp_exit_write_nothing():
    """The fused stage with an MLP exit head on malformed offsets, device batch count and ids:
    the status bit is raised and no token row or keep index is written."""
    b = make_batch([20, 20, 20], 64, "bf16", seed=11, sizes="u1to4")
    db = P.device_batch(b)
    st, o = _stage_raw_mlp(db)
    assert st == 0
    for bad in ([0, 20, 10, 60], [0, 20, 40, 99], [-3, 20, 40, 60], [0, 0, 40, 60]):
        st, o = _stage_raw_mlp(db, offsets=torch.tensor(bad, dtype=torch.int32, device="cuda"))
        assert st & fz.FUSION_DEV_BAD_OFFSETS, bad
        assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7), bad
        assert int(o["batch"][0]) == 0 and int(o["offsets"][0]) == 0, bad
    st, o = _stage_raw_mlp(db, batch=torch.full((1,), 4, dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_BATCH
    assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7)
    st, o = _stage_raw_mlp(db, ids=torch.tensor([0, 9, 1], dtype=torch.int32, device="cuda"))
    assert st & fz.FUSION_DEV_BAD_IDS
    assert torch.all(o["keep_idx"] == -5) and torch.all(o["x"] == 7)


def test_nonfinite_keys_raise_status():
    b = make_batch([9, 9], 16, "f32", seed=10, keys="separate")
    db = P.device_batch(b)
    k = db.keys.clone()
    k[2, 3] = float("nan")
    st, _ = _stage_raw(b, db, keys=k)
    assert st & fz.FUSION_DEV_NONFINITE
