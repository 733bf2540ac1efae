"""Find the exit-head weight scale alpha of the high-exit workloads, using only the oracle.

The workloads draw exit-head weights W ~ N(0, 0.02^2) * alpha.  Two of them ask
for a target exit rate instead of a fixed alpha:

* deit_s_chain12_bf16_b256: about 30 % of samples exit over the four checks
  (blocks 4, 6, 8, 10) together;
* ragged_b8192_n65_chain4_{f32,bf16}: about 60 % of the samples reaching a
  check exit there.

The exit decision only reads the CLS token, which merging and pruning never
change, so the rate is measured on the stage-1 CLS tokens with each block's
head.  alpha is found by bisection on log(alpha) with a calibration seed that no
test or benchmark uses, and written to workloads/exit_scale.json.

Run:  python -m oracle.calibrate_exit_scale
"""
from __future__ import annotations

import json
import math
import os
import sys

import numpy as np

_ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if _ROOT not in sys.path:
    sys.path.insert(0, _ROOT)

import oracle  # noqa: E402
from workloads import synth  # noqa: E402

CALIBRATION_SEED_OFFSET = 7919
CALIBRATION_BATCH = 1024

TARGETS = {
    "deit_s_chain12_bf16_b256": ("cumulative", 0.30),
    "ragged_b8192_n65_chain4_f32": ("per_check", 0.60),
    "ragged_b8192_n65_chain4_bf16": ("per_check", 0.60),
}


def _cls_batch(name: str):
    spec = synth.CONFIGS[name]
    seed = spec.seed + CALIBRATION_SEED_OFFSET
    rng = np.random.default_rng([seed, 0])
    counts = np.ones(CALIBRATION_BATCH, np.int64)  # CLS rows only
    x = synth.make_tokens(rng, counts, spec.dim, spec.clusters, spec.noise)
    xs = synth._round(x, spec.dtype)
    offsets = np.arange(CALIBRATION_BATCH + 1, dtype=np.int32)
    return spec, seed, xs, offsets


def exit_rate(name: str, alpha: float) -> float:
    spec, seed, x, offsets = _cls_batch(name)
    mode, _ = TARGETS[name]
    masks = []
    for blk in spec.exit_blocks:
        head = synth.make_head(np.random.default_rng([seed, 200 + blk]), spec.classes, spec.dim,
                               spec.tau, alpha, spec.dtype)
        masks.append(oracle.exit_check(spec.dtype, offsets, x, head)["exit_mask"].astype(bool))
    if mode == "cumulative":
        return float(np.mean(np.logical_or.reduce(masks)))
    return float(np.mean([m.mean() for m in masks]))


def calibrate(name: str, iters: int = 24) -> float:
    _, target = TARGETS[name]
    lo, hi = math.log(1.0), math.log(2000.0)
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if exit_rate(name, math.exp(mid)) < target:
            lo = mid
        else:
            hi = mid
    return float(math.exp(0.5 * (lo + hi)))


def main() -> None:
    out = {}
    for name in TARGETS:
        a = calibrate(name)
        out[name] = round(a, 6)
        print(f"{name}: alpha={a:.6f} rate={exit_rate(name, a):.4f}", flush=True)
    with open(synth.EXIT_SCALE_FILE, "w") as f:
        json.dump(out, f, indent=1, sort_keys=True)
        f.write("\n")


if __name__ == "__main__":
    main()
