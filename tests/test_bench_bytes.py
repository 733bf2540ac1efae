"""bench.py's algorithmic bytes per stage (the roofline's numerator), on hand-counted cases (CPU).

Per stage: the exit check reads every input CLS row, the head (W, bias, gamma, beta) and writes
mask and max-prob per input image and logits per image that exits; the plan reads offsets and
r/rho and writes the output offsets, ids and slots.  Per surviving image the per-sample kernel
reads all its keys when it merges (every key takes part in the decision), else only the rows it
keeps, plus sizes and scores of every input row and a few scalars, and writes each output row with
its size and score (and its input row id when the caller asks for it).  An exited image costs
nothing in the per-sample kernel.
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from workloads import StageSpec  # noqa: E402


def test_stage_bytes_hand_counted():
    d, C, eb = 16, 10, 2
    # image 0: 5 tokens, exits; image 1: 3 tokens, merges 1 pair (r = 5 clamps to (3-1)//2 = 1),
    # keeps 2 rows; image 2: 4 tokens, r = 0 (no merge), keeps 3 rows
    spec = StageSpec(True, True, True, r=np.array([2, 5, 0], np.int32), rho=np.ones(3, np.float32))
    in_off = np.array([0, 5, 8, 12], np.int32)
    in_ids = np.array([0, 1, 2], np.int32)
    out_off = np.array([0, 2, 5], np.int32)
    out_ids = np.array([1, 2], np.int32)
    first, image = bench.stage_bytes(spec, "bf16", d, in_off, in_ids, out_off, out_ids, C, row_ids=True)
    exit_bytes = 3 * 32 + C * 32 + C * 4 + 2 * 32 + 1 * C * 4 + 3 * (1 + 4)   # CLS rows, W, b, gamma+beta;
    #                                                                         logits of the 1 exit, mask, c
    plan_bytes = 4 * 4 + 3 * 8 + 2 * 12 + 4                                # offsets, r+rho, per output, count
    assert first == exit_bytes + plan_bytes == 575 + 68
    img1 = 3 * 32 + 3 * 8 + 16 + 2 * (32 + 12)     # all 3 keys read (it merges), 2 rows written
    img2 = 3 * 32 + 4 * 8 + 16 + 3 * (32 + 12)     # no merge: only the 3 kept rows read
    assert image == img1 + img2 == 224 + 276
    # without row ids (the timed chain does not ask for them): 4 bytes fewer per output row
    _, image2 = bench.stage_bytes(spec, "bf16", d, in_off, in_ids, out_off, out_ids, C)
    assert image2 == image - 5 * 4


def test_stage_bytes_without_exit():
    d = 32
    spec = StageSpec(True, False, False, r=np.array([1], np.int32))
    first, image = bench.stage_bytes(spec, "f32", d, np.array([0, 7], np.int32), np.array([0], np.int32),
                                     np.array([0, 6], np.int32), np.array([0], np.int32), 0)
    assert first == 2 * 4 + 8 + 12 + 4
    assert image == 7 * 128 + 7 * 8 + 16 + 6 * (128 + 8)
