"""Failure detection on the GPU: a bounded device wait that runs out.

Every wait of the library's kernels on an mbarrier (bulk copies landing in
shared memory, tensor-core MMAs finishing) polls a bounded number of times.
Here the limit is set to zero through sdad_workspace_set_wait_limit, so the
first such wait gives up at once: the call must still return, the kernels must
end (each waits, with the default limit, for the copies and MMAs it issued
itself), and sdad_check must report SDAD_ERR_TIMEOUT.  Nothing is made to
hang or fault.  With the default limit restored, the same workspace must give
the oracle's results again.
"""

import pytest
import torch

from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import runner as R
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W
from tests.parity import COMPARED, assert_close, oracle_for

pytestmark = pytest.mark.gpu

SDAD_ERR_TIMEOUT = -8


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


# the graph loss waits in its tensor-core projections (TMA tiles, MMAs); MF
# and CP's sorted per-mode passes wait in the streaming engine (bulk copies)
@pytest.mark.parametrize("name,kw", [("gnn", {}), ("mf", {}), ("cp3", {"tmode": 1})])
def test_wait_that_runs_out_is_reported_and_the_workspace_recovers(name, kw):
    p = W.make(name, "small")
    run = R.RUNS[name](p, **kw)
    S.sdad_workspace_set_wait_limit(run.ws.view, 0)
    run.step()
    torch.cuda.synchronize()
    assert S.sdad_check(run.ws.view) == SDAD_ERR_TIMEOUT
    # the status word was cleared by the check; the limit stays until reset
    run.step()
    assert S.sdad_check(run.ws.view) == SDAD_ERR_TIMEOUT
    S.sdad_workspace_set_wait_limit(run.ws.view, -1)
    run.step()
    torch.cuda.synchronize()
    assert S.sdad_check(run.ws.view) == 0
    assert_close(run.outputs(), oracle_for(name, p), COMPARED[name])


def test_wait_limit_argument_checks():
    ws = S.Workspace(4096)
    L = S.lib()
    assert L.sdad_workspace_set_wait_limit(None, 0, None) == -1            # NULL
    assert L.sdad_workspace_set_wait_limit(ws.view.data_ptr() + 16, 0, None) == -4   # ALIGN
    assert L.sdad_workspace_set_wait_limit(ws.view.data_ptr(), 1 << 40, None) == -2  # SHAPE
    assert L.sdad_workspace_set_wait_limit(ws.view.data_ptr(), 5, None) == 0
    torch.cuda.synchronize()
    hdr = ws.view[:12].cpu().view(torch.int32)
    assert int(hdr[2]) == 6   # stored as polls + 1
