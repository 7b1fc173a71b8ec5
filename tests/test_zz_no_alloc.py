"""sdad_lsq_grad_noalloc: least squares for callers that cannot allocate.

Callers running under a device allocator they do not own (a framework's
caching pool, a host that reserves all device memory at start-up) cannot call
cudaMalloc or provide a workspace.  The library serves them with a built-in
8 MiB scratch array.  This file checks, through the C ABI, that calls in a
row (with a call on a problem of another size between them) give the results
of the workspace entry point sdad_lsq_grad: bit for bit in the deterministic
column-pass mode, within the parity tolerance with the atomic scatter.  It
also checks that a problem too large for the array is refused.
It is collected last so that a failure here leaves every other test run.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import runner as R
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W
from tests.parity import GRAD_TOL, LOSS_TOL, grad_err, loss_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def _noalloc(run, tmode):
    """One sdad_lsq_grad_noalloc call on a LsqRun's device operands."""
    loss = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
    dx = torch.full((run.p.n,), float("nan"), dtype=torch.float32, device="cuda")
    dA = torch.full((run.A.nnz,), float("nan"), dtype=torch.float32, device="cuda")
    desc = run.A.desc()
    code = S.lib().sdad_lsq_grad_noalloc(ctypes.byref(desc), run.x.data_ptr(), run.y.data_ptr(),
                                         loss.data_ptr(), dx.data_ptr(), dA.data_ptr(), tmode,
                                         torch.cuda.current_stream().cuda_stream)
    assert code == S.SDAD_OK, S.STATUS_NAMES.get(code, code)
    torch.cuda.synchronize()
    return {"loss": float(loss.item()), "dx": dx.cpu().numpy(), "dA": dA.cpu().numpy()}


def _reference(run):
    run.step()
    torch.cuda.synchronize()
    run.check()
    return run.outputs()


@pytest.mark.parametrize("tmode", [S.SDAD_T_CSC, S.SDAD_T_ATOMIC])
def test_noalloc_matches_workspace_entry_point_twice(tmode):
    big = R.LsqRun(W.make("lsq", "full"), tmode=tmode)     # 2000 x 2000, about 20k keys
    small = R.LsqRun(W.make("lsq", "small"), tmode=tmode)  # another size: another layout
    ref_big, ref_small = _reference(big), _reference(small)
    # the scratch keeps what the previous call left in it: the second call on
    # the large problem runs on the small problem's leftovers
    for run, ref in ((big, ref_big), (small, ref_small), (big, ref_big)):
        got = _noalloc(run, tmode)
        if tmode == S.SDAD_T_CSC:
            # the column pass has a fixed summation order: equal bit for bit
            assert got["loss"] == ref["loss"]
            np.testing.assert_array_equal(got["dx"], ref["dx"])
            np.testing.assert_array_equal(got["dA"], ref["dA"])
        else:
            assert loss_err(got["loss"], ref["loss"]) <= LOSS_TOL
            assert grad_err(got["dx"], ref["dx"]) <= GRAD_TOL
            assert grad_err(got["dA"], ref["dA"]) <= GRAD_TOL


def test_noalloc_refuses_problems_beyond_its_scratch():
    # 4M rows need more than the 8 MiB built-in scratch (one float per row)
    rowptr = torch.zeros(4_000_001, dtype=torch.int32, device="cuda")
    x = torch.zeros(4, dtype=torch.float32, device="cuda")
    y = torch.zeros(4_000_000, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    desc = S.sdad_csr(4_000_000, 4, 0, rowptr.data_ptr(), 0, 0, 0, 0, 0)
    code = S.lib().sdad_lsq_grad_noalloc(ctypes.byref(desc), x.data_ptr(), y.data_ptr(),
                                         loss.data_ptr(), None, None, S.SDAD_T_AUTO, None)
    assert code == -6   # SDAD_ERR_WORKSPACE
    assert np.isfinite(loss.item())
