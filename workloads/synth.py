"""Seeded synthetic workloads with the shapes and value distributions of the
paper's DeiT-S / DeiT-B / ViT-L token tensors (Sec. III-A: one CLS token plus
N patch tokens of width d; Table I schedule for DeiT-S).

The paper's datasets (ImageNet-1k and friends) and trained timm checkpoints are
not available, so every tensor here is drawn from a seeded generator:

* tokens: per image, K cluster centres ~ N(0, I_d); each patch token picks a
  centre uniformly and adds N(0, noise^2 I_d); the CLS token is N(0, I_d);
* CLS-attention scores: softmax over the image's patches of N(0, 1) logits
  (the CLS entry is 0 and never used);
* token sizes: all 1, or integers uniform in {1..4} (CLS size 1);
* router outputs: merge counts r_i integer-uniform, keep ratios rho_i uniform;
* exit heads: W ~ N(0, 0.02^2) * alpha, b = 0, LayerNorm gamma = 1, beta = 0.

Values stored as bf16 are rounded from float32 with round-to-nearest-even;
both the oracle and the CUDA path receive the same bf16 bit patterns.
No merge / exit / prune / compact arithmetic lives in this module.
"""
from __future__ import annotations

import json
import os
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
EXIT_SCALE_FILE = os.path.join(_HERE, "exit_scale.json")


# --------------------------------------------------------------------------
# storage-dtype helpers (data preparation only)
# --------------------------------------------------------------------------
def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); return uint16 bit patterns."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    rounded = (u + 0x7FFF + lsb) >> 16
    out = rounded.astype(np.uint16)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns (uint16) to float32 exactly."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# workload description
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class ConfigSpec:
    name: str
    dtype: str                      # "f32" or "bf16"
    batch: int                      # B
    tokens: int                     # N incl. CLS
    dim: int                        # d (keys have the same width)
    clusters: int                   # cluster centres per image
    noise: float                    # std of the per-token noise
    classes: int                    # exit-head classes C
    tau: float                      # exit threshold
    r_range: Tuple[int, int]        # inclusive merge-count range
    rho_range: Tuple[float, float]  # keep-ratio range (lo == hi -> fixed)
    sizes: str                      # "ones" or "u1to4"
    keys: str                       # "alias" (keys are x) or "separate"
    blocks: int                     # number of stages in the schedule
    exit_blocks: Tuple[int, ...]    # 1-based blocks with exit-check + prune
    seed: int
    note: str = ""


CONFIGS: Dict[str, ConfigSpec] = {
    # DeiT-S-shaped single stage, FP32
    "deit_s_stage_f32_b8": ConfigSpec(
        "deit_s_stage_f32_b8", "f32", 8, 197, 384, 12, 0.3, 1000, 0.9,
        (16, 16), (0.7, 0.7), "ones", "separate", 1, (1,), 2607 * 10 + 1),
    # DeiT-S full 12-block schedule of stages, BF16 (the throughput workload)
    "deit_s_chain12_bf16_b256": ConfigSpec(
        "deit_s_chain12_bf16_b256", "bf16", 256, 197, 384, 12, 0.3, 1000, 0.85,
        (0, 24), (0.5, 1.0), "ones", "alias", 12, (4, 6, 8, 10), 2607 * 10 + 2),
    # DeiT-B-shaped single stage, BF16, non-uniform input sizes
    "deit_b_stage_bf16_b512": ConfigSpec(
        "deit_b_stage_bf16_b512", "bf16", 512, 197, 768, 12, 0.3, 1000, 0.9,
        (8, 32), (0.4, 0.9), "u1to4", "separate", 1, (1,), 2607 * 10 + 3),
    # ViT-L/16 at 384x384, BF16, 32 clusters per image
    "vit_l16_384_stage_bf16_b128": ConfigSpec(
        "vit_l16_384_stage_bf16_b128", "bf16", 128, 577, 1024, 32, 0.3, 1000, 0.9,
        (16, 64), (0.5, 0.9), "ones", "alias", 1, (1,), 2607 * 10 + 4),
    # Ragged high-exit stress, 4 chained full stages, FP32 and BF16
    "ragged_b8192_n65_chain4_f32": ConfigSpec(
        "ragged_b8192_n65_chain4_f32", "f32", 8192, 65, 384, 12, 0.3, 100, 0.6,
        (0, 16), (0.3, 1.0), "ones", "alias", 4, (1, 2, 3, 4), 2607 * 10 + 5),
    "ragged_b8192_n65_chain4_bf16": ConfigSpec(
        "ragged_b8192_n65_chain4_bf16", "bf16", 8192, 65, 384, 12, 0.3, 100, 0.6,
        (0, 16), (0.3, 1.0), "ones", "alias", 4, (1, 2, 3, 4), 2607 * 10 + 5),
}


@dataclass
class Head:
    """Exit head parameters: LayerNorm(CLS) -> Linear(d -> C) -> softmax, threshold tau."""
    gamma: np.ndarray   # [d] f32 or bf16 bits
    beta: np.ndarray    # [d]
    eps: float
    weight: np.ndarray  # [C, d] row-major
    bias: np.ndarray    # [C] f32
    tau: float

    @property
    def classes(self) -> int:
        return int(self.weight.shape[0])


@dataclass
class StageSpec:
    merge: bool
    exit: bool
    prune: bool
    r: Optional[np.ndarray] = None     # [B_orig] int32, indexed by original image id
    rho: Optional[np.ndarray] = None   # [B_orig] f32, indexed by original image id
    head: Optional[Head] = None
    mlp_head: Optional["MlpHead"] = None   # an MLP exit head in place of `head`


@dataclass
class Batch:
    """A ragged packed token batch: sample i owns rows offsets[i]..offsets[i+1]-1, CLS first."""
    dtype: str
    offsets: np.ndarray      # [B+1] int32
    x: np.ndarray            # [T, d] f32 or uint16 (bf16 bits)
    keys: np.ndarray         # [T, dk]; the same object as x when keys alias x
    sizes: np.ndarray        # [T] f32
    scores: np.ndarray       # [T] f32
    ids: Optional[np.ndarray] = None  # [B] int32 original image ids (None = identity)

    @property
    def batch(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def dim(self) -> int:
        return int(self.x.shape[1])

    @property
    def keys_alias(self) -> bool:
        return self.keys is self.x


@dataclass
class Workload:
    spec: ConfigSpec
    batch: Batch
    stages: List[StageSpec] = field(default_factory=list)


def _load_exit_scale(name: str) -> float:
    try:
        with open(EXIT_SCALE_FILE) as f:
            return float(json.load(f).get(name, 1.0))
    except FileNotFoundError:
        return 1.0


def _round(a: np.ndarray, dtype: str) -> np.ndarray:
    a = np.ascontiguousarray(a, dtype=np.float32)
    return f32_to_bf16_bits(a) if dtype == "bf16" else a


def make_tokens(rng: np.random.Generator, counts: np.ndarray, dim: int, clusters: int,
                noise: float) -> np.ndarray:
    """Cluster-plus-noise tokens, CLS first per image, packed [sum(counts), dim] float32."""
    counts = np.asarray(counts, dtype=np.int64)
    total = int(counts.sum())
    out = np.empty((total, dim), dtype=np.float32)
    row = 0
    uniform = bool(np.all(counts == counts[0])) if len(counts) else True
    chunk = 256
    for i0 in range(0, len(counts), chunk):
        cs = counts[i0:i0 + chunk]
        nb = len(cs)
        centres = rng.standard_normal((nb, clusters, dim), dtype=np.float32)
        if uniform:
            n = int(cs[0])
            cls = rng.standard_normal((nb, dim), dtype=np.float32)
            pick = rng.integers(0, clusters, size=(nb, n - 1))
            pt = centres[np.arange(nb)[:, None], pick]
            pt += np.float32(noise) * rng.standard_normal((nb, n - 1, dim), dtype=np.float32)
            blk = np.concatenate([cls[:, None, :], pt], axis=1).reshape(nb * n, dim)
            out[row:row + nb * n] = blk
            row += nb * n
        else:
            for j in range(nb):
                n = int(cs[j])
                out[row] = rng.standard_normal(dim, dtype=np.float32)
                pick = rng.integers(0, clusters, size=n - 1)
                out[row + 1:row + n] = centres[j, pick] + np.float32(noise) * rng.standard_normal(
                    (n - 1, dim), dtype=np.float32)
                row += n
    return out


def make_scores(rng: np.random.Generator, counts: np.ndarray) -> np.ndarray:
    """Per image: CLS entry 0, patches = softmax of N(0,1) logits over that image's patches."""
    out = np.zeros(int(np.sum(counts)), dtype=np.float32)
    row = 0
    for n in counts:
        n = int(n)
        if n > 1:
            z = rng.standard_normal(n - 1)
            e = np.exp(z - z.max())
            out[row + 1:row + n] = (e / e.sum()).astype(np.float32)
        row += n
    return out


def make_head(rng: np.random.Generator, classes: int, dim: int, tau: float, alpha: float,
              dtype: str) -> Head:
    w = (rng.standard_normal((classes, dim)) * 0.02 * alpha).astype(np.float32)
    return Head(gamma=_round(np.ones(dim, np.float32), dtype),
                beta=_round(np.zeros(dim, np.float32), dtype),
                eps=1e-6,
                weight=_round(w, dtype),
                bias=np.zeros(classes, dtype=np.float32),
                tau=float(tau))


@dataclass
class RouterSpec:
    """Merge-router parameters (Sec. III-C, Eq. 4-5): weight w [dim] (the tokens' dtype),
    bias beta, target keep ratio tau_tgt of the operating profile and tau_ref of the
    reference profile."""
    w: np.ndarray
    beta: float
    tau_tgt: float
    tau_ref: float


def make_router(rng: np.random.Generator, dim: int, dtype: str, tau_tgt: float = 0.5,
                tau_ref: float = 0.3) -> RouterSpec:
    """Random router weights with w . z of unit scale for unit-variance CLS rows (no trained
    router exists here): w ~ N(0, 1/dim), beta ~ N(0, 0.25^2)."""
    w = (rng.standard_normal(dim) / np.sqrt(dim)).astype(np.float32)
    return RouterSpec(_round(w, dtype), float(np.float32(rng.normal(0.0, 0.25))), tau_tgt, tau_ref)


@dataclass
class ScoreHeadSpec:
    """Linear pruning-router scoring head (Sec. III-E, Eq. 8): weight w [dim] (the tokens'
    dtype) and bias b; a token's score is w . z + b."""
    w: np.ndarray
    b: float


def make_score_head(rng: np.random.Generator, dim: int, dtype: str) -> ScoreHeadSpec:
    """Random scoring-head weights with scores of unit scale for unit-variance tokens (no
    trained head exists here): w ~ N(0, 1/dim), b ~ N(0, 0.25^2)."""
    w = (rng.standard_normal(dim) / np.sqrt(dim)).astype(np.float32)
    return ScoreHeadSpec(_round(w, dtype), float(np.float32(rng.normal(0.0, 0.25))))


POOL_CLS = 0       # CLS-only exit head
POOL_SPATIAL = 1   # SpatialPool exit head: size-weighted mean of the patch tokens


@dataclass
class MlpHead:
    """An exit head as a 2-layer MLP (the paper's SpatialPool and CLS-only heads):
    pool -> LayerNorm -> Linear(d -> H) -> GELU -> Linear(H -> C) -> softmax, threshold tau."""
    pool: int
    gamma: np.ndarray   # [d] f32 or bf16 bits
    beta: np.ndarray    # [d]
    eps: float
    w1: np.ndarray      # [H, d] row-major
    b1: np.ndarray      # [H] f32
    w2: np.ndarray      # [C, H] row-major
    b2: np.ndarray      # [C] f32
    tau: float

    @property
    def hidden(self) -> int:
        return int(self.w1.shape[0])

    @property
    def classes(self) -> int:
        return int(self.w2.shape[0])


def make_mlp_head(rng: np.random.Generator, pool: int, dim: int, hidden: int, classes: int, dtype: str,
                  tau: float = 0.05, logit_scale: float = 3.0) -> MlpHead:
    """Random MLP exit head (no trained head exists here): LayerNorm affine near identity,
    W1 ~ N(0, 1/d), b1 ~ N(0, 0.1^2), W2 ~ N(0, s^2 / H) so that the logits have standard
    deviation about s (softmax maxima spread over a useful range), b2 ~ N(0, 0.1^2)."""
    gamma = (1.0 + 0.1 * rng.standard_normal(dim)).astype(np.float32)
    beta = (0.1 * rng.standard_normal(dim)).astype(np.float32)
    w1 = (rng.standard_normal((hidden, dim)) / np.sqrt(dim)).astype(np.float32)
    b1 = (0.1 * rng.standard_normal(hidden)).astype(np.float32)
    w2 = (rng.standard_normal((classes, hidden)) * logit_scale / np.sqrt(hidden)).astype(np.float32)
    b2 = (0.1 * rng.standard_normal(classes)).astype(np.float32)
    return MlpHead(int(pool), _round(gamma, dtype), _round(beta, dtype), 1e-6, _round(w1, dtype), b1,
                   _round(w2, dtype), b2, float(tau))


def ragged_counts_from_sizes(rng: np.random.Generator, batch: int, max_tokens: int):
    """Ragged variant of the non-uniform-size config: draw patch sizes uniform in {1..4}
    until the next one would push the image's total (CLS included) past max_tokens."""
    counts, sizes = [], []
    for _ in range(batch):
        s = [1.0]
        total = 1
        while True:
            v = int(rng.integers(1, 5))
            if total + v > max_tokens:
                break
            s.append(float(v))
            total += v
        counts.append(len(s))
        sizes.extend(s)
    return np.asarray(counts, np.int64), np.asarray(sizes, np.float32)


def make_workload(name: str, batch: Optional[int] = None, *, alpha: Optional[float] = None,
                  ragged_sizes: bool = False, seed_offset: int = 0) -> Workload:
    """Build the seeded workload `name` (a key of CONFIGS).

    batch overrides B (reduced-size parity runs); alpha overrides the exit-weight scale;
    ragged_sizes builds the ragged token counts of the non-uniform-size config."""
    spec = CONFIGS[name]
    B = spec.batch if batch is None else int(batch)
    seed = spec.seed + seed_offset
    rng_tok = np.random.default_rng([seed, 0])
    rng_aux = np.random.default_rng([seed, 1])
    if ragged_sizes:
        counts, sizes = ragged_counts_from_sizes(rng_aux, B, spec.tokens)
    else:
        counts = np.full(B, spec.tokens, dtype=np.int64)
        sizes = np.ones(int(counts.sum()), dtype=np.float32)
        if spec.sizes == "u1to4":
            sizes = rng_aux.integers(1, 5, size=int(counts.sum())).astype(np.float32)
            starts = np.concatenate([[0], np.cumsum(counts)[:-1]])
            sizes[starts] = 1.0
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    x32 = make_tokens(rng_tok, counts, spec.dim, spec.clusters, spec.noise)
    scores = make_scores(rng_aux, counts)
    x = _round(x32, spec.dtype)
    if spec.keys == "alias":
        keys = x
    else:
        # separate keys: the tokens plus a small independent perturbation, so that a
        # path which confuses keys with x is caught
        k32 = x32 + np.float32(0.1) * np.random.default_rng([seed, 2]).standard_normal(
            x32.shape, dtype=np.float32)
        keys = _round(k32, spec.dtype)
    b = Batch(spec.dtype, offsets, x, keys, sizes, scores)
    a = _load_exit_scale(name) if alpha is None else float(alpha)
    stages: List[StageSpec] = []
    for blk in range(1, spec.blocks + 1):
        rs = np.random.default_rng([seed, 100 + blk])
        lo, hi = spec.r_range
        r = rs.integers(lo, hi + 1, size=B).astype(np.int32)
        full = blk in spec.exit_blocks
        rho = head = None
        if full:
            rlo, rhi = spec.rho_range
            rho = (np.full(B, rlo, np.float32) if rlo == rhi
                   else rs.uniform(rlo, rhi, size=B).astype(np.float32))
            head = make_head(np.random.default_rng([seed, 200 + blk]), spec.classes, spec.dim,
                             spec.tau, a, spec.dtype)
        stages.append(StageSpec(merge=True, exit=full, prune=full, r=r, rho=rho, head=head))
    return Workload(spec, b, stages)
