"""fusion_exit_check_noalloc against fusion_exit_check and the oracle (GPU only).

The no-allocation variant serves callers that cannot call cudaMalloc (plugin hosts
that pass only inputs and outputs, programs without a device allocator).  It must
give the same exit decisions, logits and max-probabilities as the workspace-based
call and as the oracle, on two calls in a row that share the built-in scratch, and
it must refuse a batch whose scratch would not fit.  Logits are written only for the
samples that exit; the other rows keep what the caller put there.  This file is
collected last.
"""
import ctypes
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle  # noqa: E402
import parity as P  # noqa: E402
import paper_2607_02612_gb300 as fz  # noqa: E402
from paper_2607_02612_gb300 import _binding as fb  # noqa: E402
from paper_2607_02612_gb300 import runner  # noqa: E402
from workloads import make_workload  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,B", [("deit_s_chain12_bf16_b256", None), ("ragged_b8192_n65_chain4_f32", 2048)])
def test_noalloc_matches_workspace_call_twice(name, B):
    fz.build()
    lib = fb.load()
    w = make_workload(name, batch=B)
    b = w.batch
    spec = next(s for s in w.stages if s.exit)
    db = P.device_batch(b)
    head = runner.head_tensors(spec.head, b.dtype)
    dt = runner.DTYPE_CODE[b.dtype]
    f = runner.Fusion(b.batch, head.classes)
    ref = f.exit_check(db, head)
    torch.cuda.synchronize()
    assert int(f.status.item()) == 0
    orc = oracle.exit_check(b.dtype, b.offsets, b.x, spec.head)
    ref_mask = ref["exit_mask"].cpu().numpy()
    decided = orc["exit_gap"] >= P.NEAR_TIE   # decisions with an oracle margin below 1e-6 are only counted
    assert np.array_equal(ref_mask[decided], orc["exit_mask"][decided]), "workspace call differs from the oracle"
    ex = ref_mask == 1
    for call in range(2):
        mask = torch.full((b.batch,), 7, dtype=torch.uint8, device="cuda")
        logits = torch.full((b.batch, head.classes), float("nan"), dtype=torch.float32, device="cuda")
        maxp = torch.full((b.batch,), -1.0, dtype=torch.float32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        rc = lib.fusion_exit_check_noalloc(dt, db.ragged(), db.x.data_ptr(), db.dim, head.c_struct(),
                                           mask.data_ptr(), logits.data_ptr(), maxp.data_ptr(),
                                           status.data_ptr(), torch.cuda.current_stream().cuda_stream)
        assert rc == fz.FUSION_OK, fz.fusion_status_string(rc)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert torch.equal(mask, ref["exit_mask"]), f"call {call}: exit masks differ"
        tol = P.TOL[b.dtype]
        lg = logits.cpu().numpy()
        if ex.any():
            e = P.rel_err_rows(lg[ex], ref["logits"].cpu().numpy()[ex])
            assert e.max() <= tol, f"call {call}: logits off by {e.max()}"
            eo = P.rel_err_rows(lg[ex], orc["logits"][ex])
            assert eo.max() <= tol, f"call {call}: logits off the oracle's by {eo.max()}"
        assert np.all(np.isnan(lg[~ex])), f"call {call}: logits written for samples that continue"
        mp = maxp.cpu().numpy()
        ep = np.abs(mp - ref["max_prob"].cpu().numpy()) / ref["max_prob"].cpu().numpy()
        assert ep.max() <= tol, f"call {call}: max_prob off by {ep.max()}"
        epo = np.abs(mp.astype(np.float64) - orc["max_prob"]) / orc["max_prob"]
        assert epo.max() <= tol, f"call {call}: max_prob off the oracle's by {epo.max()}"


def test_noalloc_rejects_batches_beyond_its_scratch():
    lib = fb.load()
    big = fz.ragged(1 << 20, 197, 1 << 28, 0x100000)
    head = fz.exit_head(0x100000, 0x100000, 1e-6, 0x100000, 0x100000, 1000, 0.9)
    rc = lib.fusion_exit_check_noalloc(fz.FUSION_BF16, big, 0x100000, 384, head, 0x100000, None, None, None, None)
    assert rc == fz.FUSION_ERR_WORKSPACE
    assert fz.fusion_workspace_size(1 << 20, 1000) > (1 << 20)


@pytest.mark.parametrize("classes", [10, 4000])
def test_noalloc_batch_bound_zero(classes):
    """A host batch bound of 0 is an empty call: FUSION_OK, no status bit, outputs untouched."""
    x = torch.zeros((4, 32), dtype=torch.bfloat16, device="cuda")
    offsets = torch.zeros(1, dtype=torch.int32, device="cuda")
    rg = fz.ragged(0, 4, 4, offsets)
    gamma = torch.ones(32, dtype=torch.bfloat16, device="cuda")
    beta = torch.zeros(32, dtype=torch.bfloat16, device="cuda")
    W = torch.ones((classes, 32), dtype=torch.bfloat16, device="cuda")
    bias = torch.zeros(classes, dtype=torch.float32, device="cuda")
    head = fz.exit_head(gamma, beta, 1e-6, W, bias, classes, 0.5)
    mask = torch.full((1,), 7, dtype=torch.uint8, device="cuda")
    logits = torch.full((1, classes), 3.0, dtype=torch.float32, device="cuda")
    maxp = torch.full((1,), -1.0, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rc = fz.fusion_exit_check_noalloc(fz.FUSION_BF16, rg, x, 32, head, mask, logits, maxp, status)
    assert rc == fz.FUSION_OK, fz.fusion_status_string(rc)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert int(mask.item()) == 7 and float(maxp.item()) == -1.0 and bool(torch.all(logits == 3.0))
