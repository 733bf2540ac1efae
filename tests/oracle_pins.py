"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Every function raises AssertionError when the oracle disagrees with:
* the hand-worked examples in tests/golden/worked_examples.json;
* brute force on tiny inputs (exhaustive pair search, subset enumeration);
* library routines (torch float64 layer_norm / linear / softmax, numpy stable argsort,
  numpy cumsum, torch's float32 -> bfloat16 conversion);
* invariants and special cases that follow from the definitions (conservation of
  size-weighted mass, r = 0 identity, cosine scale invariance, W = 0 -> max-prob 1/C, ...).

They are plain functions so that tests/test_oracle_mutants.py can run the whole set
against oracle builds with a planted mistake and check that some pin fails.
"""
from __future__ import annotations

import itertools
import json
import math
import os

import numpy as np
import torch

import oracle
from workloads import POOL_CLS, POOL_SPATIAL, Head, MlpHead, bf16_bits_to_f32, f32_to_bf16_bits

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "worked_examples.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _num(v):
    if isinstance(v, str):
        if v == "inf":
            return math.inf
        return float(eval(v, {"sqrt": math.sqrt, "__builtins__": {}}))  # noqa: S307
    return float(v)


def _one(x):
    """Offsets of a single-sample batch."""
    return np.array([0, len(x)], np.int32)


# ---------------------------------------------------------------------------
# brute-force references (tiny inputs only)
# ---------------------------------------------------------------------------
def brute_merge(keys, x, sizes, scores, r):
    """Exhaustive merge of one sample: cosine via numpy norms, argmax by scanning every B
    candidate, top-r by enumerating all r-subsets of A (largest exact sum, then the
    lexicographically smallest index set), outputs via a dense assignment matrix."""
    keys = np.asarray(keys, np.float64)
    x = np.asarray(x, np.float64)
    N = len(x)
    A = [p for p in range(2, N, 2)]
    Bp = [p for p in range(1, N, 2)]
    kn = keys / np.maximum(np.linalg.norm(keys, axis=1, keepdims=True), 1e-12)
    S = kn[A] @ kn[Bp].T if A and Bp else np.zeros((len(A), len(Bp)))
    match, sbest = [], []
    for m in range(len(A)):
        cand = sorted(range(len(Bp)), key=lambda n: (-S[m, n], n))
        match.append(cand[0])
        sbest.append(S[m, cand[0]])
    r_eff = min(max(int(r), 0), len(A))
    best_set = None
    for comb in itertools.combinations(range(len(A)), r_eff):
        key = (math.fsum(sbest[m] for m in comb), tuple(-m for m in comb))
        if best_set is None or key > best_set[0]:
            best_set = (key, comb)
    chosen = set(best_set[1]) if best_set else set()
    kept = [p for p in range(N) if not (p in A and A.index(p) in chosen)]
    dest = {}
    for p in range(N):
        if p in A and A.index(p) in chosen:
            dest[p] = kept.index(Bp[match[A.index(p)]])
        else:
            dest[p] = kept.index(p)
    M = np.zeros((len(kept), N))
    for p in range(N):
        M[dest[p], p] = sizes[p]
    Ind = (M > 0).astype(np.float64)
    x_out = (M @ x) / M.sum(axis=1, keepdims=True)
    return dict(x=x_out, sizes=M.sum(axis=1), scores=Ind @ np.asarray(scores, np.float64),
                keep_idx=np.array(kept), dst_map=np.array([dest[p] for p in range(N)]),
                a_match=np.array([Bp[match[A.index(p)]] if p in A else -1 for p in range(N)]),
                sbest=np.array(sbest), chosen=sorted(chosen))


def brute_prune_keep(scores, rho):
    """Positions kept by pruning one sample: all k-subsets of the patches, largest exact
    score sum, then the lexicographically smallest set; CLS always kept."""
    P = len(scores) - 1
    k = math.ceil(float(np.float32(rho)) * P)
    k = min(max(k, 0), P)
    best = None
    for comb in itertools.combinations(range(1, P + 1), k):
        key = (math.fsum(float(scores[p]) for p in comb), tuple(-p for p in comb))
        if best is None or key > best[0]:
            best = (key, comb)
    return [0] + sorted(best[1])


# ---------------------------------------------------------------------------
# conversions
# ---------------------------------------------------------------------------
def pin_bf16_rounding_table():
    """Round-to-nearest-even at the bf16 grid: exact midpoints go to the even neighbour."""
    cases = {
        1.0: 0x3F80, -1.0: 0xBF80, 0.0: 0x0000,
        1.0 + 2 ** -8: 0x3F80,            # midpoint 1 | 1+2^-7 -> even (1.0)
        1.0 + 3 * 2 ** -8: 0x3F82,        # midpoint 1+2^-7 | 1+2^-6 -> even (1+2^-6)
        1.0 + 2 ** -8 + 2 ** -30: 0x3F81,  # just above a midpoint -> up
        1.0 + 2 ** -7: 0x3F81,
        2.0 ** 128: 0x7F80,               # overflow -> +inf
        -(2.0 ** 128): 0xFF80,
        2.0 ** -133: 0x0001,              # smallest bf16 subnormal
        2.0 ** -134: 0x0000,              # half of it: tie -> even (0)
        3 * 2.0 ** -135: 0x0001,          # 0.75 of the smallest subnormal -> up
        2.0 ** -133 + 2.0 ** -134: 0x0002,  # 1.5 subnormal steps: tie -> even (2 steps)
        5 * 2.0 ** -135: 0x0001,          # 1.25 steps -> 1
        7 * 2.0 ** -135: 0x0002,          # 1.75 steps -> 2
    }
    for v, bits in cases.items():
        got = oracle.double_to_bf16(v)
        assert got == bits, f"bf16({v!r}) = {got:#06x}, expected {bits:#06x}"
    assert oracle.double_to_bf16(-0.0) == 0x8000
    for bits in (0x3F80, 0x0001, 0x7F7F, 0xC2F7):
        v = oracle.bf16_to_double(bits)
        assert oracle.double_to_bf16(v) == bits


def pin_bf16_rounding_vs_torch():
    """On float32 inputs the oracle's rounding equals torch's float32 -> bfloat16 cast."""
    rng = np.random.default_rng(11)
    v = np.concatenate([rng.standard_normal(4000).astype(np.float32),
                        (rng.standard_normal(2000) * 1e-30).astype(np.float32),
                        (rng.standard_normal(2000) * 1e30).astype(np.float32),
                        (rng.standard_normal(2000) * 1e-39).astype(np.float32)])
    # exact midpoints between neighbouring bf16 values
    b = rng.integers(0x0080, 0x7F00, 1000).astype(np.uint32)
    mids = ((b << 16) | 0x8000).view(np.float32)
    v = np.concatenate([v, mids, -mids])
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.double_to_bf16(float(t)) for t in v], np.uint16)
    bad = np.nonzero(got != ref)[0]
    assert len(bad) == 0, f"{len(bad)} mismatches, first {v[bad[0]]!r}: {got[bad[0]]:#06x} vs {ref[bad[0]]:#06x}"


# ---------------------------------------------------------------------------
# merge
# ---------------------------------------------------------------------------
def pin_merge_worked_examples():
    for ex in _golden()["merge"]:
        keys = np.array(ex["keys"], np.float32)
        x = np.array(ex["x"], np.float32)
        sizes = np.array(ex["sizes"], np.float32)
        scores = np.linspace(0.01, 0.07, len(x)).astype(np.float32)
        for case in ex["cases"]:
            m = oracle.merge("f32", _one(x), x, keys, sizes, scores, np.array([case["r"]], np.int32))
            exp_x = np.array([[_num(v) for v in row] for row in case["x_out"]], np.float32)
            assert m["x"].shape == exp_x.shape, (ex["name"], case["r"], m["x"].shape)
            np.testing.assert_array_equal(m["x"], exp_x, err_msg=f"{ex['name']} r={case['r']}")
            np.testing.assert_array_equal(m["sizes"], np.array(case["sizes_out"], np.float32))
            np.testing.assert_array_equal(m["keep_idx"], case["keep_idx"])
            np.testing.assert_array_equal(m["dst_map"], case["dst_map"])
            np.testing.assert_array_equal(m["a_match"], ex["a_match"])
            g = _num(case["topr_gap"])
            if math.isinf(g):
                assert math.isinf(m["topr_gap"][0])
            else:
                assert abs(m["topr_gap"][0] - g) < 1e-6, (ex["name"], m["topr_gap"][0], g)
        for pos, expr in ex.get("argmax_gap", {}).items():
            m = oracle.merge("f32", _one(x), x, keys, sizes, scores, np.array([0], np.int32))
            assert abs(m["argmax_gap"][int(pos)] - _num(expr)) < 1e-12


def _tiny_case(rng, N, dk, d, dtype="f32", dup=False):
    keys = rng.standard_normal((N, dk)).astype(np.float32)
    if dup and N > 4:
        keys[3] = keys[1]          # exact duplicate B tokens -> exact ties
        keys[4] = keys[1] * 2.0    # same direction, other scale
    x = rng.standard_normal((N, d)).astype(np.float32)
    sizes = rng.integers(1, 5, N).astype(np.float32)
    sizes[0] = 1
    scores = rng.random(N).astype(np.float32)
    return keys, x, sizes, scores


def pin_merge_brute_force():
    """Exhaustive search on every N in 1..17 and several r."""
    rng = np.random.default_rng(5)
    for N in range(1, 18):
        for trial in range(3):
            keys, x, sizes, scores = _tiny_case(rng, N, 5, 3, dup=(trial == 2))
            nA = (N - 1) // 2
            for r in sorted({0, 1, nA // 2, nA, nA + 3}):
                m = oracle.merge("f32", _one(x), x, keys, sizes, scores, np.array([r], np.int32))
                bf = brute_merge(keys, x, sizes, scores, r)
                np.testing.assert_array_equal(m["a_match"], bf["a_match"], err_msg=f"N={N} r={r}")
                np.testing.assert_array_equal(m["keep_idx"], bf["keep_idx"], err_msg=f"N={N} r={r}")
                np.testing.assert_array_equal(m["dst_map"], bf["dst_map"], err_msg=f"N={N} r={r}")
                np.testing.assert_allclose(m["x"], bf["x"], rtol=1e-6, atol=1e-6)
                np.testing.assert_array_equal(m["sizes"], bf["sizes"].astype(np.float32))
                np.testing.assert_allclose(m["scores"], bf["scores"], rtol=1e-6)
                # argmax gap: best minus runner-up over B
                for p in range(2, N, 2):
                    Bp = list(range(1, N, 2))
                    kk = keys.astype(np.float64)
                    kn = kk / np.linalg.norm(kk, axis=1, keepdims=True)
                    s = np.sort(kn[Bp] @ kn[p])[::-1]
                    gap = s[0] - s[1] if len(s) > 1 else math.inf
                    assert (math.isinf(gap) and math.isinf(m["argmax_gap"][p])) or \
                        abs(m["argmax_gap"][p] - gap) < 1e-12


def pin_merge_invariants():
    """Conservation: per sample, sum(size*x) and sum(size) are unchanged by merging; CLS is
    untouched; the sample loses exactly r_eff tokens; every input row has a destination."""
    rng = np.random.default_rng(7)
    counts = np.array([1, 2, 3, 17, 64, 197, 33])
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    T = int(offsets[-1])
    x = rng.standard_normal((T, 24)).astype(np.float32)
    keys = rng.standard_normal((T, 16)).astype(np.float32)
    sizes = rng.integers(1, 5, T).astype(np.float32)
    scores = rng.random(T).astype(np.float32)
    r = np.array([3, 0, 1, 5, 40, 24, 100], np.int32)
    m = oracle.merge("f32", offsets, x, keys, sizes, scores, r)
    for i in range(len(counts)):
        a, b = offsets[i], offsets[i + 1]
        oa, ob = m["offsets"][i], m["offsets"][i + 1]
        r_eff = min(max(int(r[i]), 0), (counts[i] - 1) // 2)
        assert ob - oa == counts[i] - r_eff
        mass_in = (sizes[a:b, None].astype(np.float64) * x[a:b]).sum(0)
        mass_out = (m["sizes"][oa:ob, None].astype(np.float64) * m["x"][oa:ob]).sum(0)
        scale = np.abs(sizes[a:b, None] * x[a:b]).sum(0).max()
        assert np.max(np.abs(mass_out - mass_in)) <= 1e-5 * scale
        assert m["sizes"][oa:ob].sum() == sizes[a:b].sum()
        s_in = scores[a:b].astype(np.float64).sum()
        assert abs(m["scores"][oa:ob].astype(np.float64).sum() - s_in) <= 1e-6 * s_in + 1e-12
        np.testing.assert_array_equal(m["x"][oa], x[a])          # CLS untouched
        assert m["keep_idx"][oa] == a
        assert np.all((m["dst_map"][a:b] >= oa) & (m["dst_map"][a:b] < ob))
        assert np.all(np.diff(m["keep_idx"][oa:ob]) > 0)          # ascending positions


def pin_merge_identity_and_equal_keys():
    """r = 0 is the identity; with all keys equal every A token picks the first B token and
    the r lowest A positions merge into it (closed-form mean)."""
    rng = np.random.default_rng(3)
    N, d = 15, 6
    x = rng.standard_normal((N, d)).astype(np.float32)
    sizes = np.ones(N, np.float32)
    scores = rng.random(N).astype(np.float32)
    keys = rng.standard_normal((N, 4)).astype(np.float32)
    m = oracle.merge("f32", _one(x), x, keys, sizes, scores, np.array([0], np.int32))
    np.testing.assert_array_equal(m["x"], x)
    np.testing.assert_array_equal(m["dst_map"], np.arange(N))
    same = np.tile(np.array([[0.5, -1.0, 2.0, 0.25]], np.float32), (N, 1))
    for r in (1, 3, 7):
        m = oracle.merge("f32", _one(x), x, same, sizes, scores, np.array([r], np.int32))
        merged_pos = [2 + 2 * q for q in range(r)]
        for p in range(2, N, 2):
            assert m["a_match"][p] == 1
        expect = (x[1].astype(np.float64) + x[merged_pos].astype(np.float64).sum(0)) / (1 + r)
        np.testing.assert_allclose(m["x"][1], expect, rtol=1e-6)
        assert m["sizes"][1] == 1 + r
        assert list(m["keep_idx"]) == [p for p in range(N) if p not in merged_pos]


def pin_merge_scale_invariance():
    """Cosine similarity ignores each key's length: rescaling keys by positive factors must not
    change any decision (a path that skips the normalisation fails this)."""
    rng = np.random.default_rng(9)
    N = 41
    keys, x, sizes, scores = _tiny_case(rng, N, 8, 4)
    factors = np.exp2(rng.integers(-6, 7, N)).astype(np.float32)   # exact power-of-two scales
    r = np.array([9], np.int32)
    a = oracle.merge("f32", _one(x), x, keys, sizes, scores, r)
    b = oracle.merge("f32", _one(x), x, keys * factors[:, None], sizes, scores, r)
    np.testing.assert_array_equal(a["a_match"], b["a_match"])
    np.testing.assert_array_equal(a["dst_map"], b["dst_map"])
    np.testing.assert_array_equal(a["x"], b["x"])


def pin_merge_orthogonal_pairs():
    """Hand-built one-hot keys give a known matching: A token m points at B token pi(m)."""
    nA = 6
    perm = [4, 0, 5, 2, 1, 3]
    N = 1 + 2 * nA
    keys = np.zeros((N, nA + 1), np.float32)
    keys[0, nA] = 1.0
    for n in range(nA):
        keys[1 + 2 * n, n] = 1.0
    for m in range(nA):
        keys[2 + 2 * m, perm[m]] = 1.0 + 0.1 * m
        keys[2 + 2 * m, nA] = 0.05 * (m + 1)    # unequal best similarities
    x = np.arange(N * 2, dtype=np.float32).reshape(N, 2)
    m = oracle.merge("f32", _one(x), x, keys, np.ones(N, np.float32), np.zeros(N, np.float32),
                     np.array([2], np.int32))
    for q in range(nA):
        assert m["a_match"][2 + 2 * q] == 1 + 2 * perm[q]
    # the two A tokens with the smallest side component have the largest cosines: m = 0, 1
    assert list(m["keep_idx"]) == [p for p in range(N) if p not in (2, 4)]


def pin_merge_bf16_rounding_point():
    """bf16: the weighted mean is rounded to bf16 once, from the exact mean; keys enter the
    dot products as stored."""
    x32 = np.array([[0, 0], [1.0, 3.0], [1.0 + 2 ** -6, 3.0 + 2 ** -6]], np.float32)
    xb = f32_to_bf16_bits(x32)
    keys = f32_to_bf16_bits(np.array([[1, 1], [1, 0], [1, 0]], np.float32))
    m = oracle.merge("bf16", _one(xb), xb, keys, np.ones(3, np.float32), np.zeros(3, np.float32),
                     np.array([1], np.int32))
    # mean of 1 and 1+2^-6 is 1+2^-7 (exact, representable); mean of 3 and 3+2^-6 = 3+2^-7 lies
    # halfway between the bf16 neighbours 3 and 3+2^-6 -> ties to even -> 3.0
    got = bf16_bits_to_f32(m["x"][1])
    np.testing.assert_array_equal(got, np.array([1.0 + 2 ** -7, 3.0], np.float32))


# ---------------------------------------------------------------------------
# exit check
# ---------------------------------------------------------------------------
def _torch_exit(x_cls64, gamma, beta, eps, W, b, dtype):
    u = torch.nn.functional.layer_norm(torch.from_numpy(x_cls64), (x_cls64.shape[1],),
                                       torch.from_numpy(gamma), torch.from_numpy(beta), eps)
    if dtype == "bf16":
        u = u.float().bfloat16().double()
    lg = torch.nn.functional.linear(u, torch.from_numpy(W), torch.from_numpy(b))
    p = torch.softmax(lg, dim=1)
    return u.numpy(), lg.numpy(), p.max(dim=1).values.numpy()


def pin_exit_vs_torch():
    """LayerNorm(CLS) -> Linear -> softmax max against torch float64 library routines."""
    rng = np.random.default_rng(21)
    for dtype in ("f32", "bf16"):
        B, N, d, C = 9, 5, 48, 37
        x32 = (rng.standard_normal((B * N, d)) * 2 + 0.5).astype(np.float32)
        W32 = (rng.standard_normal((C, d)) * 0.3).astype(np.float32)
        g32 = (1 + 0.1 * rng.standard_normal(d)).astype(np.float32)
        b32 = (0.1 * rng.standard_normal(d)).astype(np.float32)
        bias = (0.2 * rng.standard_normal(C)).astype(np.float32)
        if dtype == "bf16":
            xs, Ws, gs, bs = (f32_to_bf16_bits(a) for a in (x32, W32, g32, b32))
            xf, Wf, gf, bf = (bf16_bits_to_f32(a) for a in (xs, Ws, gs, bs))
        else:
            xs, Ws, gs, bs = x32, W32, g32, b32
            xf, Wf, gf, bf = x32, W32, g32, b32
        offsets = np.arange(0, B * N + 1, N, dtype=np.int32)
        head = Head(gs, bs, 1e-6, Ws, bias, 0.5)
        e = oracle.exit_check(dtype, offsets, xs, head)
        u, lg, c = _torch_exit(xf[offsets[:-1]].astype(np.float64), gf.astype(np.float64),
                               bf.astype(np.float64), 1e-6, Wf.astype(np.float64),
                               bias.astype(np.float64), dtype)
        if dtype == "bf16":
            # the bf16 rounding of the LayerNorm output is the (separately pinned) oracle rounding
            # applied to torch's float64 LayerNorm
            u_ref = np.array([[oracle.bf16_to_double(oracle.double_to_bf16(v)) for v in row] for row in u])
            np.testing.assert_array_equal(e["u"], u_ref)
            lg = torch.nn.functional.linear(torch.from_numpy(u_ref), torch.from_numpy(Wf.astype(np.float64)),
                                            torch.from_numpy(bias.astype(np.float64))).numpy()
            c = torch.softmax(torch.from_numpy(lg), dim=1).max(dim=1).values.numpy()
        else:
            np.testing.assert_allclose(e["u"], u, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(e["logits"], lg, rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(e["max_prob"], c, rtol=1e-6)
        clear = np.abs(c - 0.5) > 1e-9
        np.testing.assert_array_equal(e["exit_mask"][clear], (c[clear] >= 0.5).astype(np.uint8))
        np.testing.assert_allclose(e["exit_gap"], np.abs(c - 0.5), atol=1e-9)


def pin_exit_special_cases():
    """W = 0, b = 0 -> max-prob exactly 1/C; the rule is c >= tau (equality exits);
    tau <= 1/C -> all exit; tau > 1 -> none; one dominant logit -> c ~ 1;
    constant CLS (zero variance) -> u = beta."""
    rng = np.random.default_rng(2)
    B, d, C = 6, 16, 4
    x = rng.standard_normal((B, d)).astype(np.float32)
    offsets = np.arange(B + 1, dtype=np.int32)
    ones, zeros = np.ones(d, np.float32), np.zeros(d, np.float32)
    W0 = np.zeros((C, d), np.float32)
    e = oracle.exit_check("f32", offsets, x, Head(ones, zeros, 1e-6, W0, np.zeros(C, np.float32), 0.25))
    np.testing.assert_array_equal(e["max_prob"], np.full(B, 0.25, np.float32))
    assert e["exit_mask"].all()                       # c == tau exits
    e = oracle.exit_check("f32", offsets, x, Head(ones, zeros, 1e-6, W0, np.zeros(C, np.float32),
                                                 float(np.nextafter(np.float32(0.25), np.float32(1)))))
    assert not e["exit_mask"].any()
    W = (rng.standard_normal((C, d)) * 0.1).astype(np.float32)
    e = oracle.exit_check("f32", offsets, x, Head(ones, zeros, 1e-6, W, np.zeros(C, np.float32), 0.2))
    assert e["exit_mask"].all()                       # max-prob >= 1/C always
    e = oracle.exit_check("f32", offsets, x, Head(ones, zeros, 1e-6, W, np.zeros(C, np.float32), 1.0001))
    assert not e["exit_mask"].any()
    bias = np.array([0, 60, 0, 0], np.float32)
    e = oracle.exit_check("f32", offsets, x, Head(ones, zeros, 1e-6, W, bias, 0.999))
    assert e["exit_mask"].all() and np.all(e["max_prob"] > 0.999)
    xc = np.full((B, d), 3.5, np.float32)
    beta = rng.standard_normal(d).astype(np.float32)
    e = oracle.exit_check("f32", offsets, xc, Head(ones, beta, 1e-6, W, np.zeros(C, np.float32), 0.5))
    np.testing.assert_allclose(e["u"], np.tile(beta, (B, 1)), rtol=0, atol=0)


# ---------------------------------------------------------------------------
# prune
# ---------------------------------------------------------------------------
def pin_prune_worked_examples():
    for ex in _golden()["prune"]:
        s = np.array(ex["scores"], np.float32)
        N = len(s)
        x = np.arange(N * 3, dtype=np.float32).reshape(N, 3)
        sizes = np.arange(1, N + 1, dtype=np.float32)
        p = oracle.prune("f32", _one(x), x, sizes, s, np.array([ex["rho"]], np.float32))
        assert list(p["keep_idx"]) == ex["keep_idx"], (ex["name"], p["keep_idx"])
        np.testing.assert_array_equal(p["x"], x[ex["keep_idx"]])
        np.testing.assert_array_equal(p["sizes"], sizes[ex["keep_idx"]])
        if "rho_one_keep_idx" in ex:
            p = oracle.prune("f32", _one(x), x, sizes, s, np.array([1.0], np.float32))
            assert list(p["keep_idx"]) == ex["rho_one_keep_idx"]


def pin_prune_brute_force_and_argsort():
    """Subset enumeration (P <= 16) and numpy's stable argsort agree with the oracle's keep set
    and count k = ceil(rho * P)."""
    rng = np.random.default_rng(13)
    for P in range(0, 17):
        for trial in range(4):
            N = P + 1
            s = rng.random(N).astype(np.float32)
            if trial == 1:
                s = np.round(s * 4).astype(np.float32) / 4     # many exact ties
            rho = np.float32(rng.random()) if trial < 3 else np.float32(1.0)
            x = rng.standard_normal((N, 2)).astype(np.float32)
            p = oracle.prune("f32", _one(x), x, np.ones(N, np.float32), s, np.array([rho], np.float32))
            expect = brute_prune_keep(s, rho)
            assert list(p["keep_idx"]) == expect, (P, trial, p["keep_idx"], expect)
            k = min(max(math.ceil(float(rho) * P), 0), P)
            order = np.argsort(-s[1:].astype(np.float64), kind="stable")[:k] + 1
            assert list(p["keep_idx"]) == [0] + sorted(order.tolist())


# ---------------------------------------------------------------------------
# compact and the composed stage
# ---------------------------------------------------------------------------
def pin_compact_examples():
    for ex in _golden()["compact"]:
        off = np.array(ex["offsets"], np.int32)
        T = int(off[-1])
        x = np.arange(T * 2, dtype=np.float32).reshape(T, 2)
        c = oracle.compact("f32", off, x, np.ones(T, np.float32), np.zeros(T, np.float32),
                           np.array(ex["exit_mask"], np.uint8))
        assert list(c["offsets"]) == ex["offsets_out"]
        assert list(c["ids"]) == ex["ids_out"]
        assert list(c["keep_idx"]) == ex["keep_idx"]
        np.testing.assert_array_equal(c["x"], x[ex["keep_idx"]])
    rng = np.random.default_rng(4)
    counts = rng.integers(1, 9, 50)
    off = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    T = int(off[-1])
    x = rng.standard_normal((T, 3)).astype(np.float32)
    for mask in (np.zeros(50, np.uint8), np.ones(50, np.uint8), (rng.random(50) < 0.4).astype(np.uint8)):
        ids = rng.permutation(1000)[:50].astype(np.int32)
        c = oracle.compact("f32", off, x, np.ones(T, np.float32), None, mask, ids)
        surv = np.nonzero(mask == 0)[0]
        np.testing.assert_array_equal(c["offsets"], np.concatenate([[0], np.cumsum(counts[surv])]))
        np.testing.assert_array_equal(c["ids"], ids[surv])
        assert c["n_out"] == len(surv)


def pin_stage_exit_sees_merged_cls():
    """Merging never moves CLS, so the exit check on merged tokens equals the exit check on
    the stage input bit for bit (the CUDA path relies on this identity)."""
    from workloads import make_workload
    w = make_workload("ragged_b8192_n65_chain4_bf16", batch=64)
    b, spec = w.batch, w.stages[0]
    m = oracle.merge("bf16", b.offsets, b.x, b.keys, b.sizes, b.scores, spec.r)
    e1 = oracle.exit_check("bf16", m["offsets"], m["x"], spec.head)
    e0 = oracle.exit_check("bf16", b.offsets, b.x, spec.head)
    for k in ("exit_mask", "logits", "max_prob"):
        np.testing.assert_array_equal(e0[k], e1[k])
    assert 0 < e0["exit_mask"].sum() < 64


def pin_stage_composition():
    """The stage equals merge -> exit -> (drop exited) -> prune, and every output row that no
    merge touched is a verbatim copy of its input row."""
    from workloads import make_workload
    w = make_workload("ragged_b8192_n65_chain4_f32", batch=40)
    b, spec = w.batch, w.stages[0]
    res = oracle.stage(b, spec)
    m = oracle.merge("f32", b.offsets, b.x, b.keys, b.sizes, b.scores, spec.r)
    surv = np.nonzero(res["exit_mask"] == 0)[0]
    assert res["n_out"] == len(surv)
    np.testing.assert_array_equal(res["ids"], surv)
    k = 0
    for j, i in enumerate(surv):
        n_merged = m["offsets"][i + 1] - m["offsets"][i]
        kk = min(max(math.ceil(float(spec.rho[i]) * (n_merged - 1)), 0), n_merged - 1)
        assert res["offsets"][j + 1] - res["offsets"][j] == 1 + kk
        k += 1 + kk
    assert res["offsets"][-1] == k
    untouched = res["sizes"] == b.sizes[res["keep_idx"]]
    np.testing.assert_array_equal(res["x"][untouched], b.x[res["keep_idx"][untouched]])


# ---------------------------------------------------------------------------
# merge router with profile scaling (Sec. III-C, Eq. 4-5)
# ---------------------------------------------------------------------------
def _router_batch(cls, Ns):
    """One sample per N, each with `cls` as its CLS row and zero patch rows."""
    d = len(cls)
    offs = np.concatenate([[0], np.cumsum(Ns)]).astype(np.int32)
    x = np.zeros((int(offs[-1]), d), np.float32)
    x[offs[:-1]] = np.asarray(cls, np.float32)
    return offs, x


def pin_router_worked_examples():
    for ex in _golden()["router"]:
        Ns = [c["N"] for c in ex["cases"]]
        offs, x = _router_batch(ex["cls"], Ns)
        o = oracle.merge_router("f32", offs, x, np.array(ex["w"], np.float32), ex["beta"], ex["tau_tgt"], ex["tau_ref"])
        np.testing.assert_array_equal(o["r"], [c["r"] for c in ex["cases"]], err_msg=ex["name"])
        assert np.all(np.abs(o["mt"] - ex["mt"]) < 1e-7), (ex["name"], o["mt"])


def pin_router_special_cases():
    Ns = [1, 2, 3, 8, 65, 197, 577]
    offs, x = _router_batch([0.7, -1.3, 2.0], Ns)
    w0 = np.zeros(3, np.float32)
    # w = 0, beta = 0, equal profiles: mt = 1/2, r = floor(N / 4)
    o = oracle.merge_router("f32", offs, x, w0, 0.0, 0.3, 0.3)
    np.testing.assert_array_equal(o["r"], [N // 4 for N in Ns])
    # a saturated sigmoid merges every pair (floor(N / 2)) or none
    o = oracle.merge_router("f32", offs, x, w0, 60.0, 0.3, 0.3)
    np.testing.assert_array_equal(o["r"], [N // 2 for N in Ns])
    o = oracle.merge_router("f32", offs, x, w0, -60.0, 0.3, 0.3)
    np.testing.assert_array_equal(o["r"], [0] * len(Ns))
    # r grows with beta and with the profile's merge budget (lower target keep ratio)
    w = np.array([0.3, 0.1, -0.2], np.float32)
    prev = None
    for beta in np.linspace(-6, 6, 25):
        r = oracle.merge_router("f32", offs, x, w, float(beta), 0.5, 0.5)["r"]
        assert prev is None or np.all(r >= prev), beta
        prev = r
    prev = None
    for tt in np.linspace(1.0, 0.0, 11):
        r = oracle.merge_router("f32", offs, x, w, 0.5, float(tt), 0.4)["r"]
        assert prev is None or np.all(r >= prev), tt
        prev = r
    # bf16 inputs: values exactly representable in bf16 give the same counts as float32
    xb, wb = f32_to_bf16_bits(x), f32_to_bf16_bits(w)
    np.testing.assert_array_equal(oracle.merge_router("bf16", offs, xb, wb, 0.5, 0.25, 0.4)["r"],
                                  oracle.merge_router("f32", offs, x, w, 0.5, 0.25, 0.4)["r"])
    # outputs land at the original sample id
    ids = np.array([6, 0, 5, 1, 4, 2, 3], np.int32)
    o1 = oracle.merge_router("f32", offs, x, w, 0.5, 0.25, 0.4)
    o2 = oracle.merge_router("f32", offs, x, w, 0.5, 0.25, 0.4, ids=ids)
    np.testing.assert_array_equal(o2["r"][ids], o1["r"])


def _scores_batch(Ns, d, rng, lo=-9, hi=10, lead=0, tail=0):
    offs = (lead + np.concatenate([[0], np.cumsum(Ns)])).astype(np.int32)
    x = rng.integers(lo, hi, size=(int(offs[-1]) + tail, d)).astype(np.float32)
    return offs, x


def pin_scores_integer_brute_force():
    """Linear pruning-router scores (Eq. 8) on integer-valued tokens and weights are exact:
    each one equals Python's integer dot product plus the bias, row by row.  Rows before
    offsets[0] and after offsets[B] keep their initial zero (a legitimate score here ends in
    .5, never 0)."""
    rng = np.random.default_rng(31)
    d = 7
    offs, x = _scores_batch([1, 3, 2, 5, 1], d, rng, lead=2, tail=3)
    w = rng.integers(-5, 6, size=d).astype(np.float32)
    b = -3.5
    s = oracle.token_scores("f32", offs, x, w, b)
    for t in range(x.shape[0]):
        if offs[0] <= t < offs[-1]:
            exact = sum(int(w[j]) * int(x[t, j]) for j in range(d)) + b
            assert s[t] == exact, (t, s[t], exact)
        else:
            assert s[t] == 0.0, t


def pin_scores_correctly_rounded():
    """Real-valued float32 tokens: each product is exact in double, so math.fsum of the
    products and the bias (the correctly rounded double of the exact sum), rounded to
    float32, is the score to the last bit; the oracle agrees on every row of this draw."""
    rng = np.random.default_rng(32)
    T, d = 300, 384
    x = rng.standard_normal((T, d)).astype(np.float32)
    w = (rng.standard_normal(d) / np.sqrt(d)).astype(np.float32)
    b = float(np.float32(0.37))
    offs = np.array([0, 100, 197, 300], np.int32)
    s = oracle.token_scores("f32", offs, x, w, b)
    wd = [float(v) for v in w]
    for t in range(T):
        ref = np.float32(math.fsum([wd[j] * float(x[t, j]) for j in range(d)] + [b]))
        assert s[t] == ref, (t, s[t], ref)


def pin_scores_special_cases():
    """A one-hot head reads one coordinate (s = x[t, j] + b rounded once); values exactly
    representable in bf16 score the same in both element types; an empty batch scores
    nothing."""
    rng = np.random.default_rng(33)
    T, d = 40, 16
    x = rng.standard_normal((T, d)).astype(np.float32)
    offs = np.array([0, 17, 40], np.int32)
    for j in (0, 5, d - 1):
        w = np.zeros(d, np.float32)
        w[j] = 1.0
        s = oracle.token_scores("f32", offs, x, w, 0.25)
        np.testing.assert_array_equal(s, (x[:, j].astype(np.float64) + 0.25).astype(np.float32))
    xr = bf16_bits_to_f32(f32_to_bf16_bits(x))
    wr = bf16_bits_to_f32(f32_to_bf16_bits(rng.standard_normal(d).astype(np.float32)))
    np.testing.assert_array_equal(
        oracle.token_scores("bf16", offs, f32_to_bf16_bits(xr), f32_to_bf16_bits(wr), -1.5),
        oracle.token_scores("f32", offs, xr, wr, -1.5))
    s = oracle.token_scores("f32", np.array([0], np.int32), x, wr, 3.0)
    assert not s.any()


def _mlp_case(rng, dtype, pool, B=7, d=32, H=48, C=29, Ns=(1, 2, 5, 9, 4, 3, 6)):
    """A small ragged batch with sizes in {1..4} and an MLP head, as stored and as float64."""
    offsets = np.concatenate([[0], np.cumsum(Ns[:B])]).astype(np.int32)
    T = int(offsets[-1])
    x32 = (rng.standard_normal((T, d)) * 1.5 + 0.3).astype(np.float32)
    sizes = rng.integers(1, 5, T).astype(np.float32)
    parts = dict(g=1 + 0.1 * rng.standard_normal(d), b=0.1 * rng.standard_normal(d),
                 w1=rng.standard_normal((H, d)) / np.sqrt(d), w2=rng.standard_normal((C, H)) * 2 / np.sqrt(H))
    parts = {k: v.astype(np.float32) for k, v in parts.items()}
    b1 = (0.1 * rng.standard_normal(H)).astype(np.float32)
    b2 = (0.1 * rng.standard_normal(C)).astype(np.float32)
    if dtype == "bf16":
        xs = f32_to_bf16_bits(x32)
        st = {k: f32_to_bf16_bits(v) for k, v in parts.items()}
        fl = {k: bf16_bits_to_f32(v).astype(np.float64) for k, v in st.items()}
        xf = bf16_bits_to_f32(xs).astype(np.float64)
    else:
        xs, st = x32, parts
        fl = {k: v.astype(np.float64) for k, v in parts.items()}
        xf = x32.astype(np.float64)
    head = MlpHead(pool, st["g"], st["b"], 1e-6, st["w1"], b1, st["w2"], b2, 0.08)
    return offsets, xs, xf, sizes, head, fl, b1.astype(np.float64), b2.astype(np.float64)


def pin_exit_mlp_vs_torch():
    """MLP exit heads (pool -> LayerNorm -> W1, GELU -> W2 -> softmax max) against torch
    float64 library routines: weighted mean, layer_norm, linear, gelu (erf form), softmax.
    For bf16 the oracle's separately pinned rounding is applied to torch's LayerNorm output
    and hidden activations."""
    rng = np.random.default_rng(41)
    T_ = torch.from_numpy
    F = torch.nn.functional
    rnd = np.vectorize(lambda v: oracle.bf16_to_double(oracle.double_to_bf16(v)))
    for dtype in ("f32", "bf16"):
        for pool in (POOL_CLS, POOL_SPATIAL):
            offsets, xs, xf, sizes, head, fl, b1, b2 = _mlp_case(rng, dtype, pool)
            e = oracle.exit_mlp(dtype, offsets, xs, sizes, head)
            for i in range(len(offsets) - 1):
                o, n = offsets[i], offsets[i + 1] - offsets[i]
                if pool == POOL_CLS or n < 2:
                    z = T_(xf[o])
                else:
                    w = T_(sizes[o + 1:o + n].astype(np.float64))
                    z = (w[:, None] * T_(xf[o + 1:o + n])).sum(0) / w.sum()
                np.testing.assert_allclose(e["pool"][i], z.numpy(), rtol=1e-13, atol=1e-13)
                u = F.layer_norm(z[None], (z.shape[0],), T_(fl["g"]), T_(fl["b"]), eps=1e-6)
                if dtype == "bf16":
                    u = T_(rnd(u.numpy()))
                h = F.gelu(F.linear(u, T_(fl["w1"]), T_(b1)))
                if dtype == "bf16":
                    h_ref = rnd(h.numpy())
                    # a pre-rounding value this close to a bf16 midpoint may round either way
                    near = np.abs(h.numpy() - h_ref) > 0.5 * np.abs(h_ref) * 2.0 ** -8 * (1 - 1e-9)
                    ok = (e["hidden"][i] == h_ref[0]) | near[0]
                    assert ok.all(), (dtype, pool, i)
                    h = T_(e["hidden"][i][None])
                else:
                    np.testing.assert_allclose(e["hidden"][i], h.numpy()[0], rtol=1e-12, atol=1e-12)
                lg = F.linear(h, T_(fl["w2"]), T_(b2))
                c = torch.softmax(lg, dim=1).max().item()
                np.testing.assert_allclose(e["logits"][i], lg.numpy()[0], rtol=1e-6, atol=1e-6)
                np.testing.assert_allclose(e["max_prob"][i], c, rtol=1e-6)
                assert e["exit_mask"][i] == (c >= float(np.float32(head.tau))) or abs(c - head.tau) < 1e-9


def pin_exit_mlp_special_cases():
    """Closed forms of the MLP heads: SpatialPool weights by size and skips CLS (a two-patch
    sample pools to (a + 3 b) / 4); it pools the CLS row when there is no patch; equal patch
    tokens pool to themselves; with W1 = I and b1 = +40 the GELU is the identity (in double)
    and the head reduces to the separately pinned linear exit head; with b1 = -40 the hidden
    layer is 0 and the logits are b2."""
    rng = np.random.default_rng(42)
    d, C = 16, 11
    x = rng.standard_normal((4 + 3, d)).astype(np.float32)
    offsets = np.array([0, 3, 4, 7], np.int32)           # [CLS a b], [CLS], [CLS v v]
    sizes = np.array([1, 1, 3, 2, 1, 4, 2], np.float32)
    x[5] = x[6] = rng.standard_normal(d).astype(np.float32)
    g, b = np.ones(d, np.float32), np.zeros(d, np.float32)
    W2 = (rng.standard_normal((C, d)) * 0.7).astype(np.float32)
    b2 = (0.3 * rng.standard_normal(C)).astype(np.float32)
    eye = np.eye(d, dtype=np.float32)
    head = MlpHead(POOL_SPATIAL, g, b, 1e-6, eye, np.full(d, 40.0, np.float32), W2, b2, 0.3)
    e = oracle.exit_mlp("f32", offsets, x, sizes, head)
    np.testing.assert_allclose(e["pool"][0], (x[1].astype(np.float64) + 3 * x[2].astype(np.float64)) / 4,
                               rtol=1e-15, atol=1e-15)
    np.testing.assert_array_equal(e["pool"][1], x[3].astype(np.float64))
    np.testing.assert_array_equal(e["pool"][2], x[5].astype(np.float64))
    # identity first layer: head == LayerNorm -> W2 with bias b2 + 40 W2 1, the linear head
    # (samples 1 and 2, whose pools are float32 values the linear head can take as CLS rows)
    shifted = (b2.astype(np.float64) + 40.0 * W2.astype(np.float64).sum(1))
    cls_rows = np.stack([e["pool"][i] for i in (1, 2)]).astype(np.float32)
    lin = oracle.exit_check("f32", np.arange(3, dtype=np.int32), cls_rows,
                            Head(g, b, 1e-6, W2, shifted.astype(np.float32), 0.3))
    lin_logits = lin["logits"].astype(np.float64) - (shifted - shifted.astype(np.float32).astype(np.float64))
    np.testing.assert_allclose(e["logits"][1:], lin_logits, rtol=1e-6, atol=1e-5)
    np.testing.assert_allclose(e["hidden"][1:], lin["u"] + 40.0, rtol=1e-15, atol=1e-13)
    # saturated-negative hidden layer
    head.b1 = np.full(d, -40.0, np.float32)
    e = oracle.exit_mlp("f32", offsets, x, sizes, head)
    assert not e["hidden"].any()
    np.testing.assert_array_equal(e["logits"], np.tile(b2, (3, 1)))
    # CLS-only head reads the CLS row only
    head.pool = POOL_CLS
    e = oracle.exit_mlp("f32", offsets, x, sizes, head)
    np.testing.assert_array_equal(e["pool"], x[offsets[:-1]].astype(np.float64))


def pin_attention_vs_torch():
    """Size-aware attention against torch float64 scaled_dot_product_attention with log(sizes)
    as the additive mask (the logit bias of ToMe's proportional attention), per sample and
    head, both dtypes, with and without sizes."""
    rng = np.random.default_rng(51)
    F = torch.nn.functional
    H, dh = 3, 16
    Ns = [1, 5, 17, 2, 33]
    offsets = np.concatenate([[0], np.cumsum(Ns)]).astype(np.int32)
    T = int(offsets[-1])
    q32 = (rng.standard_normal((T, 3 * H * dh)) * 1.5).astype(np.float32)
    sizes = rng.integers(1, 6, T).astype(np.float32)
    for dtype in ("f32", "bf16"):
        qs = f32_to_bf16_bits(q32) if dtype == "bf16" else q32
        qf = (bf16_bits_to_f32(qs) if dtype == "bf16" else q32).astype(np.float64)
        for sz in (sizes, None):
            got = oracle.attention(dtype, offsets, qs, H, sz)
            for i in range(len(Ns)):
                o, n = offsets[i], offsets[i + 1] - offsets[i]
                blk = torch.from_numpy(qf[o:o + n].reshape(n, 3, H, dh)).permute(1, 2, 0, 3)   # [3, H, n, dh]
                mask = torch.zeros(n, n, dtype=torch.float64) if sz is None else \
                    torch.log(torch.from_numpy(sz[o:o + n].astype(np.float64)))[None, :].expand(n, n)
                ref = F.scaled_dot_product_attention(blk[0], blk[1], blk[2], attn_mask=mask)   # [H, n, dh]
                np.testing.assert_allclose(got[o:o + n], ref.permute(1, 0, 2).reshape(n, H * dh).numpy(),
                                           rtol=1e-12, atol=1e-12)


def pin_attention_closed_forms():
    """A zero query sees equal logits, so proportional attention returns the size-weighted
    mean of the values; a token present twice with size 1 attends and is attended exactly
    like one token of size 2 (the property that makes merged tokens of size s stand for the
    s tokens they replaced); a one-token sample returns its value; no sizes means sizes 1."""
    rng = np.random.default_rng(52)
    H, dh = 2, 8
    x = rng.standard_normal((4, 3 * H * dh)).astype(np.float32)
    sizes = np.array([1, 3, 2, 5], np.float32)
    x0 = x.copy()
    x0[:, :H * dh] = 0.0                                   # q = 0
    got = oracle.attention("f32", np.array([0, 4], np.int32), x0, H, sizes)
    v = x0[:, 2 * H * dh:].astype(np.float64)
    mean = (sizes[:, None].astype(np.float64) * v).sum(0) / sizes.sum()
    np.testing.assert_allclose(got, np.tile(mean, (4, 1)), rtol=1e-14, atol=1e-14)
    dup = np.stack([x[0], x[1], x[1]])                     # [t0, t1, t1] sizes 1 vs [t0, t1] sizes (1, 2)
    a = oracle.attention("f32", np.array([0, 3], np.int32), dup, H, np.ones(3, np.float32))
    b = oracle.attention("f32", np.array([0, 2], np.int32), x[:2], H, np.array([1, 2], np.float32))
    np.testing.assert_allclose(a[:2], b, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(a[2], b[1], rtol=1e-13, atol=1e-13)
    one = oracle.attention("f32", np.array([0, 1], np.int32), x[:1], H, sizes[:1])
    np.testing.assert_array_equal(one[0], x[0, 2 * H * dh:].astype(np.float64))
    np.testing.assert_array_equal(oracle.attention("f32", np.array([0, 4], np.int32), x, H, None),
                                  oracle.attention("f32", np.array([0, 4], np.int32), x, H, np.ones(4, np.float32)))


def pin_spatial_pool_merge_invariant():
    """Merging keeps sum s_t x_t and sum s_t over the patch rows (Sec. III-C), so the SpatialPool
    of a sample's input equals that of its merged tokens up to the rounding of the merged means
    as stored: float32, a relative 2^-24 per merged element; bf16, 2^-9 (checked for both), and
    the CLS row is unchanged.  An oracle stage with an MLP head takes its exit decision from the
    merged tokens as stored (Sec. III-B): the same mask as exit_mlp on the merged batch."""
    import dataclasses
    from workloads import make_mlp_head, make_workload
    for name, batch, bound in (("deit_s_stage_f32_b8", None, 4 * 2.0 ** -24),
                               ("deit_s_chain12_bf16_b256", 8, 2.0 ** -9)):
        w = make_workload(name, batch=batch)
        b, spec = w.batch, w.stages[0]
        T = int(b.offsets[-1])
        m = oracle.merge(b.dtype, b.offsets, b.x[:T], b.keys[:T], b.sizes[:T], b.scores[:T], spec.r)
        assert int(m["offsets"][-1]) < T   # tokens were merged
        head = make_mlp_head(np.random.default_rng(5), POOL_SPATIAL, b.dim, 2 * b.dim, 10, b.dtype)
        pin_ = oracle.exit_mlp(b.dtype, b.offsets, b.x[:T], b.sizes[:T], head)["pool"]
        pm = oracle.exit_mlp(b.dtype, m["offsets"], m["x"], m["sizes"], head)["pool"]
        xf = b.x[:T] if b.dtype == "f32" else bf16_bits_to_f32(b.x[:T])
        scale = np.abs(xf).max()
        assert np.abs(pin_ - pm).max() <= bound * scale, (name, np.abs(pin_ - pm).max() / scale)
        if b.dtype == "bf16":   # the rounding of the merged means does show in the pool
            assert np.abs(pin_ - pm).max() > 0.0
        for i in range(b.batch):   # CLS rows untouched
            np.testing.assert_array_equal(m["x"][m["offsets"][i]], b.x[b.offsets[i]])
        ch = make_mlp_head(np.random.default_rng(6), POOL_CLS, b.dim, 2 * b.dim, 10, b.dtype)
        np.testing.assert_array_equal(oracle.exit_mlp(b.dtype, b.offsets, b.x[:T], b.sizes[:T], ch)["pool"],
                                      oracle.exit_mlp(b.dtype, m["offsets"], m["x"], m["sizes"], ch)["pool"])
        e_m = oracle.exit_mlp(b.dtype, m["offsets"], m["x"], m["sizes"], head)
        head.tau = float(np.float32(np.median(e_m["max_prob"])))
        res = oracle.stage(b, dataclasses.replace(spec, head=None, mlp_head=head, exit=True))
        e_m = oracle.exit_mlp(b.dtype, m["offsets"], m["x"], m["sizes"], head)
        np.testing.assert_array_equal(res["exit_mask"], e_m["exit_mask"])
        np.testing.assert_array_equal(res["max_prob"], e_m["max_prob"])


ALL_PINS = [
    pin_bf16_rounding_table,
    pin_bf16_rounding_vs_torch,
    pin_merge_worked_examples,
    pin_merge_brute_force,
    pin_merge_invariants,
    pin_merge_identity_and_equal_keys,
    pin_merge_scale_invariance,
    pin_merge_orthogonal_pairs,
    pin_merge_bf16_rounding_point,
    pin_exit_vs_torch,
    pin_exit_special_cases,
    pin_prune_worked_examples,
    pin_prune_brute_force_and_argsort,
    pin_compact_examples,
    pin_stage_exit_sees_merged_cls,
    pin_stage_composition,
    pin_router_worked_examples,
    pin_router_special_cases,
    pin_scores_integer_brute_force,
    pin_scores_correctly_rounded,
    pin_scores_special_cases,
    pin_exit_mlp_vs_torch,
    pin_exit_mlp_special_cases,
    pin_attention_vs_torch,
    pin_attention_closed_forms,
    pin_spatial_pool_merge_invariant,
]
