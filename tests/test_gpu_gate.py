"""A bounded device wait that runs out (GPU only): failure detection without a GPU fault.

The launch gate (fusion_set_launch_gate) makes the per-sample kernels wait, before they read
any input, for a device flag.  With a flag that nothing sets and a short poll limit, every CTA
gives up: the call raises FUSION_DEV_TIMEOUT in the status word, writes none of the stage's
outputs, and leaves the context usable; the same call with the flag set matches the oracle.
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
from workloads import make_workload  # noqa: E402

pytestmark = pytest.mark.gpu


def _stage(f, db, spec, flags, head, out, flag, polls):
    try:
        assert fz.fusion_set_launch_gate(flag, polls) == fz.FUSION_OK
        f.stage(db, flags, torch.from_numpy(spec.r).cuda(), torch.from_numpy(spec.rho).cuda(), head, out=out)
        torch.cuda.synchronize()
    finally:
        fz.fusion_set_launch_gate(None, 0)


def test_gate_wait_runs_out_then_the_stage_matches_the_oracle():
    w = make_workload("deit_s_chain12_bf16_b256", batch=32)
    b = w.batch
    spec = next(s for s in w.stages if s.exit)
    flags = fz.FUSION_STAGE_MERGE | fz.FUSION_STAGE_EXIT | fz.FUSION_STAGE_PRUNE
    head = runner.head_tensors(spec.head, b.dtype)
    f = runner.Fusion(b.batch, head.classes)
    db = P.device_batch(b)
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")   # nothing sets it

    out = f.stage_outputs(db, flags, head)
    out["x"].fill_(7.0)
    out["offsets"].fill_(-7)
    out["batch"].fill_(-7)
    _stage(f, db, spec, flags, head, out, flag, 100)
    st = int(f.status.item())
    assert st & fz.FUSION_DEV_TIMEOUT, st
    assert st & ~fz.FUSION_DEV_TIMEOUT == 0, st
    assert int(out["batch"].item()) == -7                      # no output written
    assert bool(torch.all(out["offsets"] == -7))
    assert bool(torch.all(out["x"] == 7.0))

    f.status.zero_()
    flag.fill_(1)                                                 # the producer sets the flag
    out2 = f.stage_outputs(db, flags, head)
    _stage(f, db, spec, flags, head, out2, flag, 100)
    assert int(f.status.item()) == 0
    ref = oracle.stage(b, spec)
    nb = int(out2["batch"].item())
    assert nb == ref["n_out"]
    np.testing.assert_array_equal(out2["offsets"][:nb + 1].cpu().numpy(), ref["offsets"])
    decided = ref["exit_gap"] >= P.NEAR_TIE
    np.testing.assert_array_equal(out2["exit_mask"].cpu().numpy()[decided], ref["exit_mask"][decided])
    t = int(ref["offsets"][-1])
    assert np.array_equal(runner.tokens_to_numpy(out2["x"][:t], b.dtype), ref["x"])


def test_gate_with_negative_polls_is_rejected():
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert fz.fusion_set_launch_gate(flag, -1) == fz.FUSION_ERR_INVALID_ARG
    assert fz.fusion_set_launch_gate(None, 0) == fz.FUSION_OK
