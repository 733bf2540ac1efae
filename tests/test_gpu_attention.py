"""Size-aware attention over a ragged batch (the block consuming a compacted batch, Algorithm 1
Block_b, with ToMe's proportional attention) on the GPU against the oracle.

Tolerance from the arithmetic: q k^T is exact in bf16 products with float32 accumulation; the
probabilities are rounded to bf16 for the second product (relative 2^-9 each) and the output
is rounded to bf16 (2^-9), so |out - oracle| <= 2^-8 max_j |v_j| per sample, head and dim; the
test allows 2^-7 max_j |v_j| (+ 1e-6)."""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle  # noqa: E402
import paper_2607_02612_gb300 as fz  # noqa: E402
from workloads import bf16_bits_to_f32, f32_to_bf16_bits, make_workload  # noqa: E402

pytestmark = pytest.mark.gpu

DH = 64
SENTINEL = 0x7F7F   # a bf16 bit pattern no output row can hold here (3.39e38)


def _case(Ns, H, seed, lead=0, tail=0, scale=1.0):
    rng = np.random.default_rng(seed)
    offsets = (lead + np.concatenate([[0], np.cumsum(Ns)])).astype(np.int32)
    rows = int(offsets[-1]) + tail
    qkv = f32_to_bf16_bits((rng.standard_normal((rows, 3 * H * DH)) * scale).astype(np.float32))
    sizes = rng.integers(1, 5, rows).astype(np.float32)
    return offsets, qkv, sizes


def _run(offsets, qkv, H, sizes, batch=None, max_tokens=None, max_batch=None):
    rows = qkv.shape[0]
    dev = "cuda"
    B = len(offsets) - 1
    mt = int(np.max(np.diff(offsets))) if max_tokens is None else max_tokens
    offs = torch.from_numpy(np.asarray(offsets, np.int32)).to(dev)
    bt = None if batch is None else torch.full((1,), batch, dtype=torch.int32, device=dev)
    rg = fz.ragged(B if max_batch is None else max_batch, mt, rows, offs, bt)
    q = torch.from_numpy(qkv.view(np.int16)).to(dev).view(torch.bfloat16)
    sz = None if sizes is None else torch.from_numpy(sizes).to(dev)
    out = torch.full((rows, H * DH), 0, dtype=torch.int16, device=dev)
    out.fill_(SENTINEL)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    fz.check(fz.fusion_attention(fz.FUSION_BF16, rg, q, H, DH, sz, out.view(torch.bfloat16), st))
    torch.cuda.synchronize()
    return out.cpu().numpy().view(np.uint16), int(st.item())


def _check(offsets, qkv, H, sizes, label, nb=None, **kw):
    g, st = _run(offsets, qkv, H, sizes, batch=nb, **kw)
    nb = len(offsets) - 1 if nb is None else nb
    ref = oracle.attention("bf16", offsets[:nb + 1], qkv, H, sizes)
    gf = bf16_bits_to_f32(g).astype(np.float64)
    v = bf16_bits_to_f32(qkv[:, 2 * H * DH:]).astype(np.float64)
    worst = 0.0
    for i in range(nb):
        o, e = int(offsets[i]), int(offsets[i + 1])
        vmax = np.abs(v[o:e]).reshape(e - o, H, DH).max(axis=0).reshape(H * DH)   # per head and dim
        tol = 2.0 ** -7 * vmax + 1e-6
        err = np.abs(gf[o:e] - ref[o:e])
        assert (err <= tol).all(), (label, i, float((err / tol).max()))
        worst = max(worst, float((err / tol).max()))
    inside = np.zeros(qkv.shape[0], bool)
    for i in range(nb):
        inside[offsets[i]:offsets[i + 1]] = True
    assert (g[~inside] == SENTINEL).all(), label
    print(f"[{label}] {nb} samples, {int(inside.sum())} rows x {H} heads, max err / tolerance {worst:.3f}")
    return st


@pytest.mark.parametrize("sizes", [True, False])
def test_attention_tile_boundaries(sizes):
    """Sample lengths on both sides of every boundary of the resident-sample kernel: 8-row TMA boxes,
    16-key MMA granularity, 64-key K-blocks, the 128-row query tile, the 256-token bound."""
    Ns = [1, 2, 7, 8, 9, 15, 16, 17, 63, 64, 65, 127, 128, 129, 130, 191, 192, 200, 255, 256]
    offsets, qkv, sz = _case(Ns, 3, 61, lead=3, tail=5)
    st = _check(offsets, qkv, 3, sz if sizes else None, f"boundaries sizes={sizes}")
    assert st == 0


def test_attention_deit_s_shapes():
    """DeiT-S: 6 heads of 64, 197 tokens, the step's input batch (sizes of the workload), 64 images."""
    w = make_workload("deit_s_chain12_bf16_b256", batch=64)
    b = w.batch
    _, qkv, _ = _case([int(b.offsets[-1])], 6, 62)
    st = _check(b.offsets, qkv, 6, b.sizes, "DeiT-S b64")
    assert st == 0


def test_attention_large_logits_and_count():
    """Logits of a few tens (peaked softmax), 12 heads (DeiT-B width), and a device batch count
    below the bound: samples past it stay unwritten."""
    Ns = [197, 5, 150, 33, 197, 64]
    offsets, qkv, sz = _case(Ns, 12, 63, scale=2.5)
    st = _check(offsets, qkv, 12, sz, "scale 2.5, 12 heads, count 4", nb=4, max_batch=6)
    assert st == 0


@pytest.mark.parametrize("sizes", [True, False])
def test_attention_long_samples(sizes):
    """Samples past 256 tokens stream key blocks of 128 (the ViT-L/16@384 length, 577, and the
    1024-token bound), mixed with short ones in the same call and around the block edges."""
    Ns = [577, 1, 300, 129, 1024, 256, 257, 385, 640]
    offsets, qkv, sz = _case(Ns, 2, 65, lead=2, tail=3)
    st = _check(offsets, qkv, 2, sz if sizes else None, f"long samples sizes={sizes}")
    assert st == 0


def test_attention_vit_l_shapes():
    """ViT-L/16@384: 16 heads of 64, 577 tokens, a few images."""
    offsets, qkv, sz = _case([577, 577, 400], 16, 66)
    st = _check(offsets, qkv, 16, sz, "ViT-L 16 heads")
    assert st == 0


def test_attention_malformed():
    offsets, qkv, sz = _case([10, 20, 30], 2, 64)
    bad = offsets.copy()
    bad[2] = bad[1] - 1                    # a decreasing pair: that sample is not written
    g, st = _run(bad, qkv, 2, sz, max_tokens=64)
    assert st & fz.FUSION_DEV_BAD_OFFSETS
    long = np.array([0, 10, 300, 310], np.int32)   # longer than max_tokens
    qkv2 = np.zeros((310, qkv.shape[1]), np.uint16)
    g, st = _run(long, qkv2, 2, None, max_tokens=256)
    assert st & fz.FUSION_DEV_BAD_OFFSETS
    assert (g[10:300] == SENTINEL).all()
    g, st = _run(long, qkv2, 2, None, max_tokens=280)   # the key-block kernel checks the same
    assert st & fz.FUSION_DEV_BAD_OFFSETS
    assert (g[10:300] == SENTINEL).all()
