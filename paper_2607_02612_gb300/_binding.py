"""ctypes binding of the C ABI declared in include/fusion.h.

Argument marshalling only: torch tensors become device pointers, the current
torch stream becomes the cudaStream_t.  Every computation happens in
libfusion.so; if that library is missing this module raises instead of falling
back to anything else.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libfusion.so")

# return codes and flags (mirror include/fusion.h)
FUSION_OK = 0
FUSION_ERR_INVALID_ARG = -1
FUSION_ERR_SHAPE = -2
FUSION_ERR_DTYPE = -3
FUSION_ERR_WORKSPACE = -4
FUSION_ERR_CUDA = -5
FUSION_DEV_BAD_OFFSETS = 1
FUSION_DEV_BAD_BATCH = 2
FUSION_DEV_NONFINITE = 4
FUSION_DEV_INTERNAL = 8
FUSION_DEV_BAD_IDS = 16
FUSION_DEV_TIMEOUT = 32
FUSION_F32 = 0
FUSION_BF16 = 1
FUSION_STAGE_MERGE = 1
FUSION_STAGE_EXIT = 2
FUSION_STAGE_PRUNE = 4
FUSION_MAX_TOKENS = 1024
FUSION_FUSED_PLAN_MAX_BATCH = 1024
FUSION_MAX_DIM = 1024
FUSION_ATTN_HEAD_DIM = 64
FUSION_ATTN_MAX_TOKENS = 1024
FUSION_POOL_CLS = 0
FUSION_POOL_SPATIAL = 1

EXPORTED = ("fusion_status_string", "fusion_version", "fusion_profile_next", "fusion_workspace_size",
            "fusion_merge", "fusion_exit_check", "fusion_exit_check_noalloc", "fusion_prune", "fusion_compact",
            "fusion_stage", "fusion_merge_router", "fusion_token_scores", "fusion_exit_mlp_workspace_size",
            "fusion_exit_check_mlp", "fusion_attention", "fusion_stage_mlp",
            "fusion_stage_mlp_workspace_size", "fusion_set_launch_gate")


class FusionError(RuntimeError):
    pass


class fusion_ragged(ctypes.Structure):
    _fields_ = [("max_batch", ctypes.c_int32), ("max_tokens", ctypes.c_int32),
                ("max_rows", ctypes.c_int64), ("offsets", ctypes.c_void_p),
                ("batch", ctypes.c_void_p), ("ids", ctypes.c_void_p)]


class fusion_mlp_head(ctypes.Structure):
    _fields_ = [("pool", ctypes.c_int32), ("ln_gamma", ctypes.c_void_p), ("ln_beta", ctypes.c_void_p),
                ("ln_eps", ctypes.c_float), ("w1", ctypes.c_void_p), ("b1", ctypes.c_void_p),
                ("hidden", ctypes.c_int32), ("w2", ctypes.c_void_p), ("b2", ctypes.c_void_p),
                ("classes", ctypes.c_int32), ("tau", ctypes.c_float)]


class fusion_exit_head(ctypes.Structure):
    _fields_ = [("ln_gamma", ctypes.c_void_p), ("ln_beta", ctypes.c_void_p),
                ("ln_eps", ctypes.c_float), ("weight", ctypes.c_void_p),
                ("bias", ctypes.c_void_p), ("classes", ctypes.c_int32), ("tau", ctypes.c_float)]


_lib = None


def load(path: Optional[str] = None):
    """Load libfusion.so (built in-tree by build()); raise if it is absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if path is None:
        from .build import build as _build, _stale
        if _stale():
            _build()   # sources changed since the last build: rebuild (needs nvcc)
    if not os.path.exists(p):
        raise FusionError(f"{p} is missing: build the CUDA library first "
                          "(python -m paper_2607_02612_gb300.build)")
    lib = ctypes.CDLL(p)
    V, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    F = ctypes.c_float
    R, H = fusion_ragged, fusion_exit_head
    lib.fusion_status_string.argtypes = [ctypes.c_int]
    lib.fusion_status_string.restype = ctypes.c_char_p
    lib.fusion_version.argtypes = []
    lib.fusion_version.restype = ctypes.c_char_p
    lib.fusion_profile_next.argtypes = [V, V, V]
    lib.fusion_profile_next.restype = ctypes.c_int
    lib.fusion_set_launch_gate.argtypes = [V, I64]
    lib.fusion_set_launch_gate.restype = ctypes.c_int
    lib.fusion_workspace_size.argtypes = [I32, I32]
    lib.fusion_workspace_size.restype = SZ
    lib.fusion_merge.argtypes = [ctypes.c_int, R, V, I32, V, I32, V, V, V, V, V, V, V, V, V, V, V, SZ, V, V]
    lib.fusion_exit_check.argtypes = [ctypes.c_int, R, V, I32, H, V, V, V, V, SZ, V, V]
    lib.fusion_exit_check_noalloc.argtypes = [ctypes.c_int, R, V, I32, H, V, V, V, V, V]
    lib.fusion_prune.argtypes = [ctypes.c_int, R, V, I32, V, V, V, V, V, V, V, V, V, SZ, V, V]
    lib.fusion_compact.argtypes = [ctypes.c_int, R, V, I32, V, V, V, V, V, V, V, V, V, V, V, SZ, V, V]
    lib.fusion_stage.argtypes = [ctypes.c_int, ctypes.c_int, R, V, I32, V, I32, V, V, V, V, H, V, V, V,
                                 V, V, V, V, V, V, V, V, V, SZ, V, V]
    lib.fusion_merge_router.argtypes = [ctypes.c_int, R, V, I32, V, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                        V, V, V, V]
    lib.fusion_token_scores.argtypes = [ctypes.c_int, R, V, I32, V, ctypes.c_float, V, V, V]
    lib.fusion_exit_mlp_workspace_size.argtypes = [I32, I32, I32, I32]
    lib.fusion_exit_mlp_workspace_size.restype = SZ
    lib.fusion_stage_mlp_workspace_size.argtypes = [I32, I64, I32, I32, I32]
    lib.fusion_stage_mlp_workspace_size.restype = SZ
    lib.fusion_exit_check_mlp.argtypes = [ctypes.c_int, R, V, I32, V, fusion_mlp_head, V, V, V, V, SZ, V, V]
    lib.fusion_attention.argtypes = [ctypes.c_int, R, V, I32, I32, V, V, V, V]
    lib.fusion_stage_mlp.argtypes = [ctypes.c_int, ctypes.c_int, R, V, I32, V, I32, V, V, V, V, fusion_mlp_head, V,
                                     V, V, V, V, V, V, V, V, V, V, V, SZ, V, V]
    for name in ("fusion_merge", "fusion_exit_check", "fusion_exit_check_noalloc", "fusion_prune",
                 "fusion_compact", "fusion_stage", "fusion_merge_router", "fusion_token_scores",
                 "fusion_exit_check_mlp", "fusion_attention", "fusion_stage_mlp",
            "fusion_stage_mlp_workspace_size", "fusion_set_launch_gate"):
        getattr(lib, name).restype = ctypes.c_int
    del I64, F
    if path is None:
        _lib = lib
    return lib


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, torch.Tensor):
        if not t.is_cuda:
            raise FusionError("device tensor expected")
        if not t.is_contiguous():
            raise FusionError("contiguous tensor expected")
        return t.data_ptr()
    raise TypeError(f"cannot pass {type(t)} as a device pointer")


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def ragged(max_batch: int, max_tokens: int, max_rows: int, offsets, batch=None, ids=None) -> fusion_ragged:
    return fusion_ragged(int(max_batch), int(max_tokens), int(max_rows), _ptr(offsets), _ptr(batch), _ptr(ids))


def exit_head(gamma, beta, eps: float, weight, bias, classes: int, tau: float) -> fusion_exit_head:
    return fusion_exit_head(_ptr(gamma), _ptr(beta), float(eps), _ptr(weight), _ptr(bias), int(classes),
                            float(tau))


def mlp_head(pool: int, gamma, beta, eps: float, w1, b1, hidden: int, w2, b2, classes: int,
             tau: float) -> fusion_mlp_head:
    return fusion_mlp_head(int(pool), _ptr(gamma), _ptr(beta), float(eps), _ptr(w1), _ptr(b1), int(hidden),
                           _ptr(w2), _ptr(b2), int(classes), float(tau))


def check(rc: int) -> None:
    if rc != FUSION_OK:
        raise FusionError(f"fusion call failed: {rc} ({fusion_status_string(rc)})")


# ---------------------------------------------------------------------------
# the C ABI, same names and argument order
# ---------------------------------------------------------------------------
def fusion_status_string(code: int) -> str:
    return load().fusion_status_string(int(code)).decode()


def fusion_version() -> str:
    return load().fusion_version().decode()


def _event(e) -> Optional[int]:
    if e is None:
        return None
    if isinstance(e, torch.cuda.Event):
        if not e.cuda_event:   # torch creates the CUDA event lazily, at its first record()
            e.record()
        return e.cuda_event
    return int(e)


def fusion_profile_next(start=None, mid=None, end=None) -> int:
    """Arm the next call of this thread to record torch.cuda.Event objects around its kernels."""
    return load().fusion_profile_next(_event(start), _event(mid), _event(end))


def fusion_set_launch_gate(flag=None, polls: int = 0) -> int:
    """Make the following calls' per-sample kernels wait (bounded) for a device int32 flag to
    become nonzero; flag None clears the gate."""
    return int(load().fusion_set_launch_gate(_ptr(flag), int(polls)))


def fusion_workspace_size(max_batch: int, classes: int) -> int:
    return int(load().fusion_workspace_size(int(max_batch), int(classes)))


def fusion_merge(dtype, in_, x, dim, keys, key_dim, sizes, scores, r, x_out, sizes_out, scores_out,
                 offsets_out, keep_idx, dst_map, a_match, workspace, workspace_bytes, dev_status,
                 stream=None) -> int:
    return load().fusion_merge(int(dtype), in_, _ptr(x), int(dim), _ptr(keys), int(key_dim), _ptr(sizes),
                               _ptr(scores), _ptr(r), _ptr(x_out), _ptr(sizes_out), _ptr(scores_out),
                               _ptr(offsets_out), _ptr(keep_idx), _ptr(dst_map), _ptr(a_match),
                               _ptr(workspace), int(workspace_bytes), _ptr(dev_status), _stream(stream))


def fusion_exit_check(dtype, in_, x, dim, head, exit_mask, logits, max_prob, workspace, workspace_bytes,
                      dev_status, stream=None) -> int:
    return load().fusion_exit_check(int(dtype), in_, _ptr(x), int(dim), head, _ptr(exit_mask), _ptr(logits),
                                    _ptr(max_prob), _ptr(workspace), int(workspace_bytes), _ptr(dev_status),
                                    _stream(stream))


def fusion_exit_check_noalloc(dtype, in_, x, dim, head, exit_mask, logits, max_prob, dev_status,
                              stream=None) -> int:
    """fusion_exit_check with the library's built-in scratch (for callers that cannot allocate)."""
    return load().fusion_exit_check_noalloc(int(dtype), in_, _ptr(x), int(dim), head, _ptr(exit_mask),
                                            _ptr(logits), _ptr(max_prob), _ptr(dev_status), _stream(stream))


def fusion_merge_router(dtype, in_, x, dim, w, beta, tau_tgt, tau_ref, r_out, m_out, dev_status,
                        stream=None) -> int:
    """Merge counts from the router with profile scaling (Sec. III-C, Eq. 4-5), by original id."""
    return load().fusion_merge_router(int(dtype), in_, _ptr(x), int(dim), _ptr(w), float(beta), float(tau_tgt),
                                      float(tau_ref), _ptr(r_out), _ptr(m_out), _ptr(dev_status), _stream(stream))


def fusion_token_scores(dtype, in_, x, dim, w, b, scores_out, dev_status, stream=None) -> int:
    """Prune scores from a linear pruning router, s = w . z + b per token row (Sec. III-E, Eq. 8)."""
    return load().fusion_token_scores(int(dtype), in_, _ptr(x), int(dim), _ptr(w), float(b), _ptr(scores_out),
                                      _ptr(dev_status), _stream(stream))


def fusion_stage_mlp_workspace_size(max_batch: int, max_rows: int, dim: int, hidden: int, classes: int) -> int:
    return int(load().fusion_stage_mlp_workspace_size(int(max_batch), int(max_rows), int(dim), int(hidden),
                                                       int(classes)))


def fusion_exit_mlp_workspace_size(max_batch: int, dim: int, hidden: int, classes: int) -> int:
    return int(load().fusion_exit_mlp_workspace_size(int(max_batch), int(dim), int(hidden), int(classes)))


def fusion_exit_check_mlp(dtype, in_, x, dim, sizes, head, exit_mask, logits, max_prob, workspace, workspace_bytes,
                          dev_status, stream=None) -> int:
    """Exit check with an MLP exit head (SpatialPool or CLS-only; Sec. III-D, Eq. 6-7)."""
    return load().fusion_exit_check_mlp(int(dtype), in_, _ptr(x), int(dim), _ptr(sizes), head, _ptr(exit_mask),
                                        _ptr(logits), _ptr(max_prob), _ptr(workspace), int(workspace_bytes),
                                        _ptr(dev_status), _stream(stream))


def fusion_attention(dtype, in_, qkv, heads, head_dim, sizes, out, dev_status, stream=None) -> int:
    """Size-aware attention per sample and head over a ragged batch (ToMe proportional attention)."""
    return load().fusion_attention(int(dtype), in_, _ptr(qkv), int(heads), int(head_dim), _ptr(sizes), _ptr(out),
                                   _ptr(dev_status), _stream(stream))


def fusion_prune(dtype, in_, x, dim, sizes, scores, rho, x_out, sizes_out, scores_out, offsets_out,
                 keep_idx, workspace, workspace_bytes, dev_status, stream=None) -> int:
    return load().fusion_prune(int(dtype), in_, _ptr(x), int(dim), _ptr(sizes), _ptr(scores), _ptr(rho),
                               _ptr(x_out), _ptr(sizes_out), _ptr(scores_out), _ptr(offsets_out),
                               _ptr(keep_idx), _ptr(workspace), int(workspace_bytes), _ptr(dev_status),
                               _stream(stream))


def fusion_compact(dtype, in_, x, dim, sizes, scores, exit_mask, x_out, sizes_out, scores_out, offsets_out,
                   ids_out, batch_out, keep_idx, workspace, workspace_bytes, dev_status, stream=None) -> int:
    return load().fusion_compact(int(dtype), in_, _ptr(x), int(dim), _ptr(sizes), _ptr(scores),
                                 _ptr(exit_mask), _ptr(x_out), _ptr(sizes_out), _ptr(scores_out),
                                 _ptr(offsets_out), _ptr(ids_out), _ptr(batch_out), _ptr(keep_idx),
                                 _ptr(workspace), int(workspace_bytes), _ptr(dev_status), _stream(stream))


def fusion_stage(dtype, flags, in_, x, dim, keys, key_dim, sizes, scores, r, rho, head, exit_mask, logits,
                 max_prob, x_out, sizes_out, scores_out, offsets_out, ids_out, batch_out, keep_idx, a_match,
                 workspace, workspace_bytes, dev_status, stream=None) -> int:
    if head is None:
        head = fusion_exit_head()
    return load().fusion_stage(int(dtype), int(flags), in_, _ptr(x), int(dim), _ptr(keys), int(key_dim),
                               _ptr(sizes), _ptr(scores), _ptr(r), _ptr(rho), head, _ptr(exit_mask),
                               _ptr(logits), _ptr(max_prob), _ptr(x_out), _ptr(sizes_out), _ptr(scores_out),
                               _ptr(offsets_out), _ptr(ids_out), _ptr(batch_out), _ptr(keep_idx),
                               _ptr(a_match), _ptr(workspace), int(workspace_bytes), _ptr(dev_status),
                               _stream(stream))


def fusion_stage_mlp(dtype, flags, in_, x, dim, keys, key_dim, sizes, scores, r, rho, head, exit_mask, logits,
                     max_prob, x_out, sizes_out, scores_out, offsets_out, ids_out, batch_out, keep_idx, a_match,
                     workspace, workspace_bytes, dev_status, stream=None) -> int:
    if head is None:
        head = fusion_mlp_head()
    return load().fusion_stage_mlp(int(dtype), int(flags), in_, _ptr(x), int(dim), _ptr(keys), int(key_dim),
                                   _ptr(sizes), _ptr(scores), _ptr(r), _ptr(rho), head, _ptr(exit_mask),
                                   _ptr(logits), _ptr(max_prob), _ptr(x_out), _ptr(sizes_out), _ptr(scores_out),
                                   _ptr(offsets_out), _ptr(ids_out), _ptr(batch_out), _ptr(keep_idx),
                                   _ptr(a_match), _ptr(workspace), int(workspace_bytes), _ptr(dev_status),
                                   _stream(stream))
