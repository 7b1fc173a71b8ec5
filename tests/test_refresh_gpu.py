"""Value refresh of the twins on the device (sdad_gather_by_perm).

A CSR matrix carries value copies in its other physical formats: the CSC
twin's val_csc = val[perm] and the row-blocked twin's bcsc_val = val[bperm]
(0 on padding keys).  When a step changes A's values on the device, the
copies are gathered again there.  Checked: the gather's own contract (padding
and out-of-range entries give 0; bit-exact against a host gather), and the
loss and gradients after a device-side change of the values, against the
oracle of the changed matrix, in the column-pass layouts that read the
copies (plain CSC twin, row-blocked twin, split).
"""

import numpy as np
import pytest
import torch

from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import runner as R
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W
from tests.parity import COMPARED, assert_close, oracle_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def test_gather_contract():
    rng = np.random.default_rng(3)
    src = rng.standard_normal(1000).astype(np.float32)
    perm = rng.integers(-1, 1000, 3001).astype(np.int32)
    perm[::7] = -1
    perm[5] = 1000          # out of range reads as 0 as well
    out = torch.full((perm.size,), float("nan"), dtype=torch.float32, device="cuda")
    S.sdad_gather_by_perm(torch.from_numpy(src).cuda(), torch.from_numpy(perm).cuda(), out)
    torch.cuda.synchronize()
    want = np.where((perm >= 0) & (perm < src.size), src[np.clip(perm, 0, src.size - 1)], 0)
    np.testing.assert_array_equal(out.cpu().numpy(), want.astype(np.float32))
    ints = torch.arange(50, dtype=torch.int32, device="cuda") * 3
    p2 = torch.tensor([49, 0, 7, -1], dtype=torch.int32, device="cuda")
    got = S.sdad_gather_by_perm(ints, p2, torch.empty(4, dtype=torch.int32, device="cuda"))
    assert got.cpu().tolist() == [147, 0, 21, 0]


@pytest.mark.parametrize("kw", [{}, {"blocked": 9}, {"split": (9, 4.0)}])
def test_values_changed_on_the_device(kw):
    p = W.make("logreg", "small")
    kw = dict(kw)
    if "split" in kw:
        lg, per_block = kw.pop("split")
        kw.update(blocked=lg, block_cols=S.split_columns(p.col, p.n, p.m, lg, per_block))
    r = R.LogregRun(p, tmode=S.SDAD_T_CSC, ranked=True, **kw)
    r.step()
    torch.cuda.synchronize()
    r.check()
    # a device-side update of A's values (CSR order), then the twins' copies
    A = r.X
    A.val.mul_(-0.5).add_(0.25)
    A.refresh_values()
    r.step()
    torch.cuda.synchronize()
    r.check()
    q = W.SparseMatrixProblem(p.name, p.m, p.n, p.row, p.col,
                              (p.val * np.float32(-0.5) + np.float32(0.25)).astype(np.float32),
                              p.dense, p.params)
    assert_close(r.outputs(), oracle_for("logreg", q), COMPARED["logreg"])
