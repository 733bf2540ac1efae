"""The C-ABI library on the host: it loads, exports every function include/fusion.h
declares, and rejects bad arguments before enqueueing anything.  No GPU needed:
every call here fails a host-side check, so no CUDA call is made."""
import ctypes
import os
import re

import pytest

import paper_2607_02612_gb300 as fz
from paper_2607_02612_gb300 import _binding as fb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fusion.h")

FAKE = 0x100000   # never dereferenced: every call below fails a host check first


@pytest.fixture(scope="module")
def lib():
    fz.build()
    return fb.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fusion_[a-z_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert set(names) == set(fb.EXPORTED), names
    raw = ctypes.CDLL(fb.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), n


def test_status_strings_and_version(lib):
    assert fz.fusion_status_string(0) == "ok"
    for code in (-1, -2, -3, -4, -5, 1, 2, 4, 8, 16):
        assert fz.fusion_status_string(code) != "unknown status"
    assert "sm_103a" in fz.fusion_version()


def test_workspace_size_grows_with_batch_and_classes(lib):
    a = fz.fusion_workspace_size(256, 1000)
    assert a > 0 and a % 256 == 0
    assert fz.fusion_workspace_size(8192, 1000) > a
    assert fz.fusion_workspace_size(256, 4000) > a
    assert fz.fusion_workspace_size(0, 1) > 0


def _r(max_batch=4, max_tokens=197, max_rows=800, offsets=FAKE):
    return fz.ragged(max_batch, max_tokens, max_rows, offsets)


def _merge(**kw):
    args = dict(dtype=fz.FUSION_BF16, in_=_r(), x=FAKE, dim=384, keys=FAKE, key_dim=384, sizes=FAKE,
                scores=FAKE, r=FAKE, x_out=FAKE, sizes_out=FAKE, scores_out=FAKE, offsets_out=FAKE,
                keep_idx=None, dst_map=None, a_match=None, workspace=FAKE,
                workspace_bytes=fz.fusion_workspace_size(4, 1), dev_status=FAKE, stream=0)
    args.update(kw)
    return fz.fusion_merge(*args.values())


@pytest.mark.parametrize("kw,code", [
    (dict(dtype=7), fz.FUSION_ERR_DTYPE),
    (dict(dim=17), fz.FUSION_ERR_SHAPE),
    (dict(dim=0), fz.FUSION_ERR_SHAPE),
    (dict(dim=2048), fz.FUSION_ERR_SHAPE),
    (dict(key_dim=8), fz.FUSION_ERR_SHAPE),
    (dict(x=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(keys=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(r=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(x=FAKE + 8), fz.FUSION_ERR_INVALID_ARG),
    (dict(x_out=FAKE + 4), fz.FUSION_ERR_INVALID_ARG),
    (dict(scores_out=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(in_=_r(max_tokens=0)), fz.FUSION_ERR_SHAPE),
    (dict(in_=_r(max_tokens=5000)), fz.FUSION_ERR_SHAPE),
    (dict(in_=_r(max_batch=-1)), fz.FUSION_ERR_SHAPE),
    (dict(in_=_r(offsets=None)), fz.FUSION_ERR_INVALID_ARG),
    (dict(workspace=None), fz.FUSION_ERR_WORKSPACE),
    (dict(workspace_bytes=16), fz.FUSION_ERR_WORKSPACE),
])
def test_merge_rejects_bad_arguments(lib, kw, code):
    assert _merge(**kw) == code


def _head(**kw):
    h = dict(gamma=FAKE, beta=FAKE, eps=1e-6, weight=FAKE, bias=FAKE, classes=1000, tau=0.9)
    h.update(kw)
    return fz.exit_head(*h.values())


def _stage(**kw):
    args = dict(dtype=fz.FUSION_BF16, flags=7, in_=_r(), x=FAKE, dim=384, keys=FAKE, key_dim=384, sizes=FAKE,
                scores=FAKE, r=FAKE, rho=FAKE, head=_head(), exit_mask=FAKE, logits=FAKE, max_prob=FAKE,
                x_out=FAKE, sizes_out=FAKE, scores_out=FAKE, offsets_out=FAKE, ids_out=FAKE, batch_out=FAKE,
                keep_idx=None, a_match=None, workspace=FAKE, workspace_bytes=fz.fusion_workspace_size(4, 1000),
                dev_status=FAKE, stream=0)
    args.update(kw)
    return fz.fusion_stage(*args.values())


@pytest.mark.parametrize("kw,code", [
    (dict(flags=8), fz.FUSION_ERR_INVALID_ARG),
    (dict(flags=-1), fz.FUSION_ERR_INVALID_ARG),
    (dict(head=_head(classes=0)), fz.FUSION_ERR_SHAPE),
    (dict(head=_head(weight=None)), fz.FUSION_ERR_INVALID_ARG),
    (dict(head=_head(gamma=FAKE + 2)), fz.FUSION_ERR_INVALID_ARG),
    (dict(exit_mask=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(rho=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(ids_out=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(batch_out=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(flags=6, a_match=FAKE), fz.FUSION_ERR_INVALID_ARG),
    (dict(workspace_bytes=fz.fusion_workspace_size(4, 1)), fz.FUSION_ERR_WORKSPACE),
    (dict(scores=None, scores_out=None), fz.FUSION_ERR_INVALID_ARG),   # prune needs scores
])
def test_stage_rejects_bad_arguments(lib, kw, code):
    assert _stage(**kw) == code


def test_other_calls_reject_bad_arguments(lib):
    ws = fz.fusion_workspace_size(4, 1000)
    assert fz.fusion_exit_check(fz.FUSION_F32, _r(), FAKE, 384, _head(classes=0), FAKE, None, None, FAKE, ws,
                                FAKE, 0) == fz.FUSION_ERR_SHAPE
    assert fz.fusion_exit_check(fz.FUSION_F32, _r(), FAKE, 384, _head(), None, None, None, FAKE, ws,
                                FAKE, 0) == fz.FUSION_ERR_INVALID_ARG
    assert fz.fusion_prune(fz.FUSION_F32, _r(), FAKE, 384, FAKE, None, FAKE, FAKE, FAKE, FAKE, FAKE, None,
                           FAKE, ws, FAKE, 0) == fz.FUSION_ERR_INVALID_ARG
    assert fz.fusion_compact(fz.FUSION_F32, _r(), FAKE, 384, FAKE, None, None, FAKE, FAKE, None, FAKE, FAKE,
                             FAKE, None, FAKE, ws, FAKE, 0) == fz.FUSION_ERR_INVALID_ARG
    assert fz.fusion_compact(2, _r(), FAKE, 384, FAKE, None, FAKE, FAKE, FAKE, None, FAKE, FAKE,
                             FAKE, None, FAKE, ws, FAKE, 0) == fz.FUSION_ERR_DTYPE


def test_binding_refuses_host_tensors(lib):
    import torch
    with pytest.raises(fz.FusionError):
        fb._ptr(torch.zeros(4))


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(fz.FusionError):
        fb.load(str(tmp_path / "libfusion.so"))


def test_binding_constants_match_header():
    """The Python mirrors of the header's #define values stay in step with it."""
    with open(os.path.join(ROOT, "include", "fusion.h")) as f:
        text = f.read()
    defs = dict(re.findall(r"#define\s+(FUSION_[A-Z0-9_]+)\s+(-?\d+)", text))
    for name in ("FUSION_MAX_TOKENS", "FUSION_MAX_DIM", "FUSION_FUSED_PLAN_MAX_BATCH", "FUSION_STAGE_MERGE",
                 "FUSION_STAGE_EXIT", "FUSION_STAGE_PRUNE", "FUSION_DEV_TIMEOUT", "FUSION_POOL_CLS",
                 "FUSION_POOL_SPATIAL", "FUSION_ATTN_HEAD_DIM", "FUSION_ATTN_MAX_TOKENS"):
        assert int(defs[name]) == getattr(fb, name), name


def test_merge_router_rejects_bad_arguments(lib):
    def call(**kw):
        args = dict(dtype=fz.FUSION_BF16, in_=_r(), x=FAKE, dim=384, w=FAKE, beta=0.0, tau_tgt=0.5, tau_ref=0.3,
                    r_out=FAKE, m_out=None, dev_status=FAKE, stream=0)
        args.update(kw)
        return fz.fusion_merge_router(*args.values())
    assert call(dtype=3) == fz.FUSION_ERR_DTYPE
    assert call(dim=20) == fz.FUSION_ERR_SHAPE
    assert call(in_=_r(offsets=None)) == fz.FUSION_ERR_INVALID_ARG
    for kw in (dict(x=None), dict(w=None), dict(r_out=None), dict(tau_ref=1.0), dict(tau_ref=1.5),
               dict(beta=float("nan")), dict(tau_tgt=float("inf"))):
        assert call(**kw) == fz.FUSION_ERR_INVALID_ARG, kw


def test_token_scores_rejects_bad_arguments(lib):
    def call(**kw):
        args = dict(dtype=fz.FUSION_BF16, in_=_r(), x=FAKE, dim=384, w=FAKE, b=0.0, scores_out=FAKE,
                    dev_status=FAKE, stream=0)
        args.update(kw)
        return fz.fusion_token_scores(*args.values())
    assert call(dtype=5) == fz.FUSION_ERR_DTYPE
    assert call(dim=24) == fz.FUSION_ERR_SHAPE
    assert call(in_=_r(max_tokens=0)) == fz.FUSION_ERR_SHAPE
    assert call(in_=_r(offsets=None)) == fz.FUSION_ERR_INVALID_ARG
    for kw in (dict(x=None), dict(w=None), dict(scores_out=None), dict(x=FAKE + 4), dict(w=FAKE + 8),
               dict(b=float("nan")), dict(b=float("-inf"))):
        assert call(**kw) == fz.FUSION_ERR_INVALID_ARG, kw


def test_exit_check_mlp_rejects_bad_arguments(lib):
    ws = fz.fusion_exit_mlp_workspace_size(4, 384, 768, 1000)
    assert ws > fz.fusion_workspace_size(4, 1000)
    assert fz.fusion_exit_mlp_workspace_size(8, 384, 768, 1000) > ws
    assert fz.fusion_exit_mlp_workspace_size(4, 384, 1024, 1000) > ws

    def head(**kw):
        h = dict(pool=fz.FUSION_POOL_SPATIAL, gamma=FAKE, beta=FAKE, eps=1e-6, w1=FAKE, b1=FAKE, hidden=768,
                 w2=FAKE, b2=FAKE, classes=1000, tau=0.5)
        h.update(kw)
        return fz.mlp_head(*h.values())

    def call(**kw):
        args = dict(dtype=fz.FUSION_BF16, in_=_r(), x=FAKE, dim=384, sizes=FAKE, head=head(), exit_mask=FAKE,
                    logits=None, max_prob=None, workspace=FAKE, workspace_bytes=ws, dev_status=FAKE, stream=0)
        args.update(kw)
        return fz.fusion_exit_check_mlp(*args.values())
    assert call(dtype=4) == fz.FUSION_ERR_DTYPE
    assert call(dim=100) == fz.FUSION_ERR_SHAPE
    assert call(head=head(hidden=100)) == fz.FUSION_ERR_SHAPE
    assert call(head=head(hidden=2048)) == fz.FUSION_ERR_SHAPE
    assert call(head=head(classes=0)) == fz.FUSION_ERR_SHAPE
    for kw in (dict(head=head(pool=2)), dict(sizes=None), dict(x=None), dict(exit_mask=None), dict(x=FAKE + 8),
               dict(head=head(w1=None)), dict(head=head(b2=None)), dict(head=head(w2=FAKE + 4))):
        assert call(**kw) == fz.FUSION_ERR_INVALID_ARG, kw
    assert call(sizes=None, head=head(pool=fz.FUSION_POOL_CLS), workspace=None) == fz.FUSION_ERR_WORKSPACE
    assert call(workspace_bytes=ws - 1) == fz.FUSION_ERR_WORKSPACE


def _mlp_head(**kw):
    h = dict(pool=fz.FUSION_POOL_SPATIAL, gamma=FAKE, beta=FAKE, eps=1e-6, w1=FAKE, b1=FAKE, hidden=768,
             w2=FAKE, b2=FAKE, classes=1000, tau=0.5)
    h.update(kw)
    return fz.mlp_head(*h.values())


def _stage_mlp(**kw):
    args = dict(dtype=fz.FUSION_BF16, flags=7, in_=_r(), x=FAKE, dim=384, keys=FAKE, key_dim=384, sizes=FAKE,
                scores=FAKE, r=FAKE, rho=FAKE, head=_mlp_head(), exit_mask=FAKE, logits=FAKE, max_prob=FAKE,
                x_out=FAKE, sizes_out=FAKE, scores_out=FAKE, offsets_out=FAKE, ids_out=FAKE, batch_out=FAKE,
                keep_idx=None, a_match=None, workspace=FAKE,
                workspace_bytes=fz.fusion_exit_mlp_workspace_size(4, 384, 768, 1000), dev_status=FAKE, stream=0)
    args.update(kw)
    return fz.fusion_stage_mlp(*args.values())


@pytest.mark.parametrize("kw,code", [
    (dict(dtype=4), fz.FUSION_ERR_DTYPE),
    (dict(flags=8), fz.FUSION_ERR_INVALID_ARG),
    (dict(head=_mlp_head(hidden=100)), fz.FUSION_ERR_SHAPE),
    (dict(head=_mlp_head(classes=0)), fz.FUSION_ERR_SHAPE),
    (dict(head=_mlp_head(pool=2)), fz.FUSION_ERR_INVALID_ARG),
    (dict(head=_mlp_head(w1=None)), fz.FUSION_ERR_INVALID_ARG),
    (dict(head=_mlp_head(w2=FAKE + 4)), fz.FUSION_ERR_INVALID_ARG),
    (dict(exit_mask=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(sizes=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(rho=None), fz.FUSION_ERR_INVALID_ARG),
    (dict(flags=6, a_match=FAKE), fz.FUSION_ERR_INVALID_ARG),
    (dict(workspace=None), fz.FUSION_ERR_WORKSPACE),
    (dict(workspace=FAKE + 8), fz.FUSION_ERR_WORKSPACE),
    # the linear head's scratch is too small for the MLP head's
    (dict(workspace_bytes=fz.fusion_workspace_size(4, 1000)), fz.FUSION_ERR_WORKSPACE),
    (dict(workspace_bytes=fz.fusion_exit_mlp_workspace_size(4, 384, 768, 1000) - 1), fz.FUSION_ERR_WORKSPACE),
    # without the exit check the stage's own scratch is enough, and a bad head is not read
    (dict(flags=5, head=_mlp_head(pool=2), workspace_bytes=fz.fusion_workspace_size(4, 1) - 1),
     fz.FUSION_ERR_WORKSPACE),
])
def test_stage_mlp_rejects_bad_arguments(lib, kw, code):
    assert _stage_mlp(**kw) == code


def test_attention_rejects_bad_arguments(lib):
    def call(**kw):
        args = dict(dtype=fz.FUSION_BF16, in_=_r(max_tokens=197), qkv=FAKE, heads=6, head_dim=64, sizes=None,
                    out=FAKE, dev_status=FAKE, stream=0)
        args.update(kw)
        return fz.fusion_attention(*args.values())
    assert call(dtype=fz.FUSION_F32) == fz.FUSION_ERR_DTYPE
    assert call(dtype=9) == fz.FUSION_ERR_DTYPE
    assert call(head_dim=32) == fz.FUSION_ERR_SHAPE
    assert call(heads=0) == fz.FUSION_ERR_SHAPE
    assert call(in_=_r(offsets=None)) == fz.FUSION_ERR_INVALID_ARG
    for kw in (dict(qkv=None), dict(out=None), dict(qkv=FAKE + 2), dict(out=FAKE + 8)):
        assert call(**kw) == fz.FUSION_ERR_INVALID_ARG, kw
