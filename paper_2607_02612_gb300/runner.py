"""Python-side plumbing around the C ABI: device buffers, output allocation,
stage chains and CUDA-graph capture.  torch provides memory and streams only;
every step of the computation runs in libfusion.so.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np
import torch

from . import _binding as fb

DTYPE_CODE = {"f32": fb.FUSION_F32, "bf16": fb.FUSION_BF16}
TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


def tokens_to_torch(a: np.ndarray, dtype: str, device) -> torch.Tensor:
    """float32 array or bf16 bit patterns (uint16) -> device tensor of the storage dtype."""
    a = np.ascontiguousarray(a)
    if dtype == "bf16":
        return torch.from_numpy(a.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(a.astype(np.float32, copy=False)).to(device)


def tokens_to_numpy(t: torch.Tensor, dtype: str) -> np.ndarray:
    """Device tensor -> float32 array or bf16 bit patterns (uint16)."""
    if dtype == "bf16":
        return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return t.float().cpu().numpy()


@dataclass
class DeviceBatch:
    """A ragged token batch on the device plus the host-side bounds the C ABI needs."""
    dtype: str
    dim: int
    max_batch: int
    max_tokens: int
    max_rows: int
    x: torch.Tensor
    keys: torch.Tensor
    sizes: torch.Tensor
    scores: Optional[torch.Tensor]
    offsets: torch.Tensor
    batch: Optional[torch.Tensor] = None
    ids: Optional[torch.Tensor] = None

    @property
    def key_dim(self) -> int:
        return int(self.keys.shape[1])

    def ragged(self) -> fb.fusion_ragged:
        return fb.ragged(self.max_batch, self.max_tokens, self.max_rows, self.offsets, self.batch, self.ids)


def device_batch(dtype: str, offsets, x, keys, sizes, scores, ids=None, max_tokens=None,
                 device="cuda") -> DeviceBatch:
    offsets = np.asarray(offsets, np.int32)
    B = len(offsets) - 1
    xt = tokens_to_torch(x, dtype, device)
    kt = xt if keys is x else tokens_to_torch(keys, dtype, device)
    if max_tokens is None:
        max_tokens = int(np.max(np.diff(offsets))) if B > 0 else 1
    return DeviceBatch(
        dtype=dtype, dim=int(xt.shape[1]), max_batch=B, max_tokens=int(max_tokens), max_rows=int(xt.shape[0]),
        x=xt, keys=kt, sizes=torch.from_numpy(np.asarray(sizes, np.float32)).to(device),
        scores=None if scores is None else torch.from_numpy(np.asarray(scores, np.float32)).to(device),
        offsets=torch.from_numpy(offsets).to(device),
        ids=None if ids is None else torch.from_numpy(np.asarray(ids, np.int32)).to(device))


@dataclass
class HeadTensors:
    gamma: torch.Tensor
    beta: torch.Tensor
    eps: float
    weight: torch.Tensor
    bias: torch.Tensor
    tau: float

    @property
    def classes(self) -> int:
        return int(self.weight.shape[0])

    def c_struct(self) -> fb.fusion_exit_head:
        return fb.exit_head(self.gamma, self.beta, self.eps, self.weight, self.bias, self.classes, self.tau)


def head_tensors(head, dtype: str, device="cuda") -> HeadTensors:
    return HeadTensors(tokens_to_torch(head.gamma, dtype, device), tokens_to_torch(head.beta, dtype, device),
                       float(head.eps), tokens_to_torch(head.weight, dtype, device),
                       torch.from_numpy(np.asarray(head.bias, np.float32)).to(device), float(head.tau))


@dataclass
class MlpHeadTensors:
    """An MLP exit head on the device (fusion_mlp_head)."""
    pool: int
    gamma: torch.Tensor
    beta: torch.Tensor
    eps: float
    w1: torch.Tensor
    b1: torch.Tensor
    w2: torch.Tensor
    b2: torch.Tensor
    tau: float

    @property
    def hidden(self) -> int:
        return int(self.w1.shape[0])

    @property
    def classes(self) -> int:
        return int(self.w2.shape[0])

    def c_struct(self) -> fb.fusion_mlp_head:
        return fb.mlp_head(self.pool, self.gamma, self.beta, self.eps, self.w1, self.b1, self.hidden, self.w2,
                           self.b2, self.classes, self.tau)


def mlp_head_tensors(head, dtype: str, device="cuda") -> MlpHeadTensors:
    f32 = lambda a: torch.from_numpy(np.asarray(a, np.float32)).to(device)   # noqa: E731
    return MlpHeadTensors(int(head.pool), tokens_to_torch(head.gamma, dtype, device),
                          tokens_to_torch(head.beta, dtype, device), float(head.eps),
                          tokens_to_torch(head.w1, dtype, device), f32(head.b1),
                          tokens_to_torch(head.w2, dtype, device), f32(head.b2), float(head.tau))


class Fusion:
    """Owns a zero-initialised workspace and a device status word; each method
    allocates its outputs and enqueues one C-ABI call on the current stream."""

    def __init__(self, max_batch: int, classes: int = 1, device="cuda"):
        self.device = torch.device(device)
        self.ws_bytes = fb.fusion_workspace_size(max_batch, classes)
        self.workspace = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self._mlp_ws: Optional[torch.Tensor] = None   # scratch of exit_check_mlp, sized at first use
        self.max_batch = max_batch
        self.classes = classes

    def _outputs(self, b: DeviceBatch, with_scores: bool) -> Dict[str, torch.Tensor]:
        dev = self.device
        return dict(
            x=torch.empty((b.max_rows, b.dim), dtype=TORCH_DTYPE[b.dtype], device=dev),
            sizes=torch.empty(b.max_rows, dtype=torch.float32, device=dev),
            scores=torch.empty(b.max_rows, dtype=torch.float32, device=dev) if with_scores else None,
            offsets=torch.zeros(b.max_batch + 1, dtype=torch.int32, device=dev),
            keep_idx=torch.full((b.max_rows,), -1, dtype=torch.int32, device=dev))

    def merge(self, b: DeviceBatch, r: torch.Tensor, *, dst_map=True, a_match=True) -> Dict[str, torch.Tensor]:
        o = self._outputs(b, b.scores is not None)
        o["dst_map"] = torch.full((b.max_rows,), -1, dtype=torch.int32, device=self.device) if dst_map else None
        o["a_match"] = torch.full((b.max_rows,), -1, dtype=torch.int32, device=self.device) if a_match else None
        fb.check(fb.fusion_merge(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, b.keys, b.key_dim, b.sizes,
                                 b.scores, r, o["x"], o["sizes"], o["scores"], o["offsets"], o["keep_idx"],
                                 o["dst_map"], o["a_match"], self.workspace, self.ws_bytes, self.status))
        return o

    def merge_router(self, b: DeviceBatch, w: torch.Tensor, beta: float, tau_tgt: float, tau_ref: float,
                     out: Optional[Dict[str, torch.Tensor]] = None) -> Dict[str, torch.Tensor]:
        """Merge counts r (by original id) from the router with profile scaling (Eq. 4-5)."""
        o = out if out is not None else dict(
            r=torch.zeros(b.max_batch, dtype=torch.int32, device=self.device),
            m=torch.zeros(b.max_batch, dtype=torch.float32, device=self.device))
        fb.check(fb.fusion_merge_router(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, w, beta, tau_tgt, tau_ref,
                                        o["r"], o["m"], self.status))
        return o

    def token_scores(self, b: DeviceBatch, w: torch.Tensor, bias: float,
                     out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """Prune scores s = w . z + bias of every token row from a linear pruning router (Eq. 8)."""
        o = out if out is not None else torch.zeros(b.max_rows, dtype=torch.float32, device=self.device)
        fb.check(fb.fusion_token_scores(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, w, bias, o, self.status))
        return o

    def exit_check_mlp(self, b: DeviceBatch, head: "MlpHeadTensors") -> Dict[str, torch.Tensor]:
        """Exit check with an MLP exit head (SpatialPool or CLS-only), its own scratch."""
        dev = self.device
        o = dict(exit_mask=torch.zeros(b.max_batch, dtype=torch.uint8, device=dev),
                 logits=torch.zeros((b.max_batch, head.classes), dtype=torch.float32, device=dev),
                 max_prob=torch.zeros(b.max_batch, dtype=torch.float32, device=dev))
        ws, nbytes = self.mlp_workspace(b, head)
        fb.check(fb.fusion_exit_check_mlp(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, b.sizes, head.c_struct(),
                                          o["exit_mask"], o["logits"], o["max_prob"], ws, nbytes, self.status))
        return o

    def mlp_workspace(self, b: DeviceBatch, head: "MlpHeadTensors"):
        """The zero-filled scratch of the MLP-head calls (it grows to the largest head seen;
        a Chain sizes it for all its stages before any graph capture)."""
        # the stage's size covers the exit check alone too (its layout starts with the same scratch)
        nbytes = fb.fusion_stage_mlp_workspace_size(b.max_batch, b.max_rows, b.dim, head.hidden, head.classes)
        if self._mlp_ws is None or self._mlp_ws.numel() < nbytes:
            self._mlp_ws = torch.zeros(nbytes, dtype=torch.uint8, device=self.device)
        return self._mlp_ws, nbytes

    def attention(self, b: DeviceBatch, qkv: torch.Tensor, heads: int, sizes: Optional[torch.Tensor] = None,
                  out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """Size-aware attention of the batch's samples: qkv [max_rows, 3 * heads * 64] bf16, sizes
        [max_rows] (None: plain attention); returns [max_rows, heads * 64] bf16."""
        o = out if out is not None else torch.zeros((b.max_rows, heads * fb.FUSION_ATTN_HEAD_DIM),
                                                    dtype=torch.bfloat16, device=self.device)
        fb.check(fb.fusion_attention(DTYPE_CODE["bf16"], b.ragged(), qkv, heads, fb.FUSION_ATTN_HEAD_DIM, sizes, o,
                                     self.status))
        return o

    def exit_check(self, b: DeviceBatch, head: HeadTensors) -> Dict[str, torch.Tensor]:
        dev = self.device
        o = dict(exit_mask=torch.zeros(b.max_batch, dtype=torch.uint8, device=dev),
                 logits=torch.zeros((b.max_batch, head.classes), dtype=torch.float32, device=dev),
                 max_prob=torch.zeros(b.max_batch, dtype=torch.float32, device=dev))
        fb.check(fb.fusion_exit_check(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, head.c_struct(),
                                      o["exit_mask"], o["logits"], o["max_prob"], self.workspace, self.ws_bytes,
                                      self.status))
        return o

    def prune(self, b: DeviceBatch, rho: torch.Tensor) -> Dict[str, torch.Tensor]:
        o = self._outputs(b, True)
        fb.check(fb.fusion_prune(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, b.sizes, b.scores, rho, o["x"],
                                 o["sizes"], o["scores"], o["offsets"], o["keep_idx"], self.workspace,
                                 self.ws_bytes, self.status))
        return o

    def compact(self, b: DeviceBatch, exit_mask: torch.Tensor) -> Dict[str, torch.Tensor]:
        o = self._outputs(b, b.scores is not None)
        o["ids"] = torch.zeros(b.max_batch, dtype=torch.int32, device=self.device)
        o["batch"] = torch.zeros(1, dtype=torch.int32, device=self.device)
        fb.check(fb.fusion_compact(DTYPE_CODE[b.dtype], b.ragged(), b.x, b.dim, b.sizes, b.scores, exit_mask,
                                   o["x"], o["sizes"], o["scores"], o["offsets"], o["ids"], o["batch"],
                                   o["keep_idx"], self.workspace, self.ws_bytes, self.status))
        return o

    def stage(self, b: DeviceBatch, flags: int, r=None, rho=None, head: Optional[HeadTensors] = None,
              a_match: bool = False, out: Optional[Dict[str, torch.Tensor]] = None,
              mlp_head: Optional["MlpHeadTensors"] = None) -> Dict[str, torch.Tensor]:
        """One fused stage; the exit check uses `head` (linear) or `mlp_head` (an MLP exit head)."""
        o = out if out is not None else self.stage_outputs(b, flags, head, a_match, mlp_head=mlp_head)
        if mlp_head is not None:
            ws, nbytes = self.mlp_workspace(b, mlp_head)
            fb.check(fb.fusion_stage_mlp(
                DTYPE_CODE[b.dtype], flags, b.ragged(), b.x, b.dim, b.keys, b.key_dim, b.sizes, b.scores, r, rho,
                mlp_head.c_struct(), o["exit_mask"], o["logits"], o["max_prob"], o["x"], o["sizes"], o["scores"],
                o["offsets"], o["ids"], o["batch"], o["keep_idx"], o.get("a_match"), ws, nbytes, self.status))
            return o
        fb.check(fb.fusion_stage(
            DTYPE_CODE[b.dtype], flags, b.ragged(), b.x, b.dim, b.keys, b.key_dim, b.sizes, b.scores, r, rho,
            head.c_struct() if head is not None else None, o["exit_mask"], o["logits"], o["max_prob"], o["x"],
            o["sizes"], o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"], o.get("a_match"),
            self.workspace, self.ws_bytes, self.status))
        return o

    def stage_outputs(self, b: DeviceBatch, flags: int, head: Optional[HeadTensors], a_match: bool = False,
                      mlp_head: Optional["MlpHeadTensors"] = None):
        dev = self.device
        o = self._outputs(b, b.scores is not None)
        o["ids"] = torch.zeros(b.max_batch, dtype=torch.int32, device=dev)
        o["batch"] = torch.zeros(1, dtype=torch.int32, device=dev)
        has_exit = bool(flags & fb.FUSION_STAGE_EXIT)
        o["exit_mask"] = torch.zeros(b.max_batch, dtype=torch.uint8, device=dev) if has_exit else None
        classes = (mlp_head or head).classes if has_exit else 0
        o["logits"] = torch.zeros((b.max_batch, classes), dtype=torch.float32, device=dev) if has_exit else None
        o["max_prob"] = torch.zeros(b.max_batch, dtype=torch.float32, device=dev) if has_exit else None
        o["a_match"] = torch.full((b.max_rows,), -1, dtype=torch.int32, device=dev) if a_match else None
        return o


def output_batch(b: DeviceBatch, o: Dict[str, torch.Tensor]) -> DeviceBatch:
    """The batch a stage hands to the next block (keys alias the new tokens)."""
    return DeviceBatch(dtype=b.dtype, dim=b.dim, max_batch=b.max_batch, max_tokens=b.max_tokens,
                       max_rows=b.max_rows, x=o["x"], keys=o["x"], sizes=o["sizes"], scores=o["scores"],
                       offsets=o["offsets"], batch=o["batch"], ids=o["ids"])


@dataclass
class ChainStage:
    flags: int
    r: Optional[torch.Tensor] = None
    rho: Optional[torch.Tensor] = None
    head: Optional[HeadTensors] = None
    mlp_head: Optional[MlpHeadTensors] = None   # an MLP exit head in place of `head`


@dataclass
class Chain:
    """A schedule of stages over pre-allocated buffers; stage s+1 reads what stage s wrote.
    run() enqueues every stage on the current stream with no host synchronisation."""
    fusion: Fusion
    inp: DeviceBatch
    stages: List[ChainStage]
    outs: List[Dict[str, torch.Tensor]] = field(default_factory=list)
    batches: List[DeviceBatch] = field(default_factory=list)

    def __post_init__(self):
        b = self.inp
        for st in self.stages:
            o = self.fusion.stage_outputs(b, st.flags, st.head, mlp_head=st.mlp_head)
            if st.mlp_head is not None:
                self.fusion.mlp_workspace(b, st.mlp_head)   # sized before any capture
            self.outs.append(o)
            self.batches.append(b)
            b = output_batch(b, o)

    def run_stage(self, s: int, stream=None):
        st, b, o = self.stages[s], self.batches[s], self.outs[s]
        if st.mlp_head is not None:
            ws, nbytes = self.fusion.mlp_workspace(b, st.mlp_head)
            fb.check(fb.fusion_stage_mlp(
                DTYPE_CODE[b.dtype], st.flags, b.ragged(), b.x, b.dim, b.keys, b.key_dim, b.sizes, b.scores, st.r,
                st.rho, st.mlp_head.c_struct(), o["exit_mask"], o["logits"], o["max_prob"], o["x"], o["sizes"],
                o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"], None, ws, nbytes, self.fusion.status,
                stream))
            return
        fb.check(fb.fusion_stage(
            DTYPE_CODE[b.dtype], st.flags, b.ragged(), b.x, b.dim, b.keys, b.key_dim, b.sizes, b.scores, st.r,
            st.rho, st.head.c_struct() if st.head is not None else None, o["exit_mask"], o["logits"],
            o["max_prob"], o["x"], o["sizes"], o["scores"], o["offsets"], o["ids"], o["batch"], o["keep_idx"],
            None, self.fusion.workspace, self.fusion.ws_bytes, self.fusion.status, stream))

    def run(self, stream=None):
        for s in range(len(self.stages)):
            self.run_stage(s, stream)

    def capture(self) -> torch.cuda.CUDAGraph:
        """Capture the whole chain as one CUDA graph (run() once before, eagerly)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run()
        return g

    def host_results(self) -> "HostResults":
        """Pinned host buffers sized for this chain's results (see HostResults)."""
        return HostResults(self)

    def clone(self) -> "Chain":
        """The same schedule over its own input, output and scratch buffers (the stage
        parameters, read only, are shared); the inputs start as a copy of this chain's."""
        b = self.inp
        x = b.x.clone()
        keys = x if b.keys is b.x else b.keys.clone()
        cp = lambda t: None if t is None else t.clone()   # noqa: E731
        inp = DeviceBatch(dtype=b.dtype, dim=b.dim, max_batch=b.max_batch, max_tokens=b.max_tokens,
                          max_rows=b.max_rows, x=x, keys=keys, sizes=b.sizes.clone(), scores=cp(b.scores),
                          offsets=b.offsets.clone(), batch=cp(b.batch), ids=cp(b.ids))
        fus = Fusion(self.fusion.max_batch, self.fusion.classes, self.fusion.device)
        return Chain(fus, inp, list(self.stages))


class HostResults:
    """Pinned host copies of a chain's results: the survivors of the last stage (count,
    offsets, ids, sizes, token rows), every exit check's mask and max probability over the
    images entering it, and the device status word.

    fetch() runs on the current stream after the chain was enqueued: one asynchronous copy
    of the fixed-size parts (the count, the offsets bound, the exit outputs), one host wait,
    then copies of the survivors' exact extent and a second wait.  Returns host views
    (valid until the next fetch) and the number of bytes copied."""

    def __init__(self, chain: Chain):
        last = chain.outs[-1]
        self._last = last
        self._exits = [(o["exit_mask"], o["max_prob"]) for o in chain.outs if o["exit_mask"] is not None]
        # images entering each exit check (None: the whole input batch)
        self._exit_in = [b.batch for b, o in zip(chain.batches, chain.outs) if o["exit_mask"] is not None]
        self._exit_max = [b.max_batch for b, o in zip(chain.batches, chain.outs) if o["exit_mask"] is not None]
        pin = lambda t: torch.empty(t.shape, dtype=t.dtype).pin_memory()   # noqa: E731
        self.batch = pin(last["batch"])
        self.offsets = pin(last["offsets"])
        self.ids = pin(last["ids"])
        self.sizes = pin(last["sizes"])
        self.x = pin(last["x"])
        self.exits = [(pin(m), pin(p)) for m, p in self._exits]
        self.exit_in = [None if t is None else pin(t) for t in self._exit_in]
        self._status = chain.fusion.status
        self.status = pin(self._status)

    def fetch(self):
        self.fetch_fixed()
        torch.cuda.current_stream().synchronize()
        self.fetch_exact()
        torch.cuda.current_stream().synchronize()
        return self.result()

    def fetch_fixed(self):
        """Enqueue (current stream) the copies whose size the host knows: the survivor count,
        the offsets bound and the exit outputs."""
        last = self._last
        self.batch.copy_(last["batch"], non_blocking=True)
        self.offsets.copy_(last["offsets"], non_blocking=True)
        self.status.copy_(self._status, non_blocking=True)
        self._n = self.batch.numel() * 4 + self.offsets.numel() * 4 + 4
        for (hm, hp), (m, p), hc, c in zip(self.exits, self._exits, self.exit_in, self._exit_in):
            hm.copy_(m, non_blocking=True)
            hp.copy_(p, non_blocking=True)
            self._n += hm.numel() * hm.element_size() + hp.numel() * hp.element_size()
            if hc is not None:
                hc.copy_(c, non_blocking=True)
                self._n += 4

    def fetch_exact(self):
        """Enqueue (current stream) the survivors' rows; the fixed copies must have landed."""
        last = self._last
        self._nb = int(self.batch[0])
        self._rows = int(self.offsets[self._nb])
        for name, k in (("ids", self._nb), ("sizes", self._rows), ("x", self._rows)):
            h = getattr(self, name)
            h[:k].copy_(last[name][:k], non_blocking=True)
            self._n += h[:k].numel() * h.element_size()

    def result(self):
        nb, rows = self._nb, self._rows
        res = {"batch": nb, "offsets": self.offsets[:nb + 1], "ids": self.ids[:nb], "sizes": self.sizes[:rows],
               "x": self.x[:rows], "status": int(self.status[0]), "exits": []}
        for (hm, hp), hc, mx in zip(self.exits, self.exit_in, self._exit_max):
            n = mx if hc is None else int(hc[0])
            res["exits"].append((hm[:n], hp[:n]))
        return res, self._n


class Pipeline:
    """Back-to-back steps of one schedule with host inputs and host results, the copies
    overlapped with the computation: step k runs on slot k % 2 (a chain with its own
    buffers, replayed as a CUDA graph), its inputs are copied on one copy stream while step
    k - 1 computes, and its results come back on another.  The survivors' exact extent is
    known only once the host has read their count, so submit() of step k returns the results
    of step k - 1 (None for the first) and finish() those of the last step; host results stay
    valid until the next call.  Slots are not reused before their results are on the host."""

    def __init__(self, chain: Chain):
        self.chains = [chain, chain.clone()]
        self.graphs = []
        for ch in self.chains:
            ch.run()
            torch.cuda.synchronize()
            self.graphs.append(ch.capture())
        self.hr = [ch.host_results() for ch in self.chains]
        self.s_h2d, self.s_cmp, self.s_d2h = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        ev = lambda: [torch.cuda.Event(), torch.cuda.Event()]   # noqa: E731
        self.ev_h2d, self.ev_cmp, self.ev_cnt, self.ev_res = ev(), ev(), ev(), ev()
        self.k = 0
        self.pending: Optional[int] = None

    def _inputs(self, slot: int) -> Dict[str, torch.Tensor]:
        b = self.chains[slot].inp
        d = {"x": b.x.view(torch.int16) if b.dtype == "bf16" else b.x, "sizes": b.sizes, "offsets": b.offsets}
        if b.keys is not b.x:
            d["keys"] = b.keys.view(torch.int16) if b.dtype == "bf16" else b.keys
        if b.scores is not None:
            d["scores"] = b.scores
        return d

    def submit(self, host: Dict[str, torch.Tensor]):
        """host: pinned tensors named after the input fields (x as int16 bits for bf16)."""
        c = self.k % 2
        dst = self._inputs(c)
        with torch.cuda.stream(self.s_h2d):
            if self.k >= 2:
                self.s_h2d.wait_event(self.ev_cmp[c])   # the slot's previous replay read its inputs
            for name, t in host.items():
                dst[name].copy_(t, non_blocking=True)
            self.ev_h2d[c].record(self.s_h2d)
        with torch.cuda.stream(self.s_cmp):
            self.s_cmp.wait_event(self.ev_h2d[c])
            if self.k >= 2:
                self.s_cmp.wait_event(self.ev_res[c])   # the slot's previous results are on the host
            self.graphs[c].replay()
            self.ev_cmp[c].record(self.s_cmp)
        prev = self._complete()
        with torch.cuda.stream(self.s_d2h):
            self.s_d2h.wait_event(self.ev_cmp[c])
            self.hr[c].fetch_fixed()
            self.ev_cnt[c].record(self.s_d2h)
        self.pending = c
        self.k += 1
        return prev

    def _complete(self):
        p = self.pending
        if p is None:
            return None
        self.pending = None
        self.ev_cnt[p].synchronize()
        with torch.cuda.stream(self.s_d2h):
            self.hr[p].fetch_exact()
            self.ev_res[p].record(self.s_d2h)
        self.ev_res[p].synchronize()
        return self.hr[p].result()

    def finish(self):
        """Results of the last submitted step (None if there is none)."""
        return self._complete()

    def status(self) -> int:
        """OR of the slots' device status words (synchronises)."""
        torch.cuda.synchronize()
        return int(self.chains[0].fusion.status.item()) | int(self.chains[1].fusion.status.item())
