"""Least squares over a COO operand in entry order (sdad_lsq_coo_grad).

The same expression as sdad_lsq_grad over another storage of the same
dictionary: entries in any order, repeated keys adding their values.  Checked
against the fp64 oracle: loss, dx and dA in the entries' order (each entry of
a repeated key gets the key's gradient), on shuffled, duplicated, empty and
hub-row inputs; an entry out of range is skipped and reported by the kernel's
own bounds check as SDAD_ERR_INDEX.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W
from tests.parity import GRAD_TOL, LOSS_TOL, grad_err, loss_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_coo(m, n, row, col, val, x, y):
    t = [dev(np.asarray(a, np.int32)) for a in (row, col)] + [dev(np.asarray(val, np.float32))]
    A = S.sdad_coo(m, n, int(len(row)), *(a.data_ptr() if a.numel() else None for a in t))
    ws = S.Workspace(S.sdad_workspace_bytes(S.SDAD_EXPR_LSQ, m, n, len(row), 0))
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    dx = torch.full((n,), float("nan"), dtype=torch.float32, device="cuda")
    dA = torch.full((max(len(row), 1),), float("nan"), dtype=torch.float32, device="cuda")
    S.sdad_lsq_coo_grad(A, dev(x), dev(y), loss, dx, dA, ws)
    torch.cuda.synchronize()
    code = S.sdad_check(ws)
    return code, float(loss.item()), dx.cpu().numpy(), dA.cpu().numpy()[:len(row)]


def reference(m, n, row, col, val, x, y):
    """The oracle on the deduplicated dictionary; dA read back per entry."""
    key = np.asarray(row, np.int64) * n + np.asarray(col, np.int64)
    uk, inv = np.unique(key, return_inverse=True)
    uval = np.zeros(uk.size, np.float64)
    np.add.at(uval, inv, np.asarray(val, np.float64))
    o = oracle.lsq(m, n, (uk // n).astype(np.int32), (uk % n).astype(np.int32),
                   uval.astype(np.float32), x, y)
    return o["loss"], o["dx"], np.asarray(o["dA"])[inv]


@pytest.mark.parametrize("case", ["shuffled", "duplicates", "hub_row"])
def test_coo_against_oracle(case):
    rng = np.random.default_rng(21)
    p = W.make("lsq", "small")
    row, col, val = p.row.copy(), p.col.copy(), p.val.copy()
    m, n = p.m, p.n
    if case == "duplicates":   # every third key split into two entries of half the value
        d = np.arange(0, row.size, 3)
        val = val.copy()
        val[d] *= np.float32(0.5)
        row, col, val = np.concatenate([row, row[d]]), np.concatenate([col, col[d]]), \
            np.concatenate([val, val[d]])
    if case == "hub_row":      # row 0 holds every column (many lanes add to one z entry)
        row = np.concatenate([row, np.zeros(n, np.int32)])
        col = np.concatenate([col, np.arange(n, dtype=np.int32)])
        val = np.concatenate([val, rng.standard_normal(n).astype(np.float32)])
    order = rng.permutation(row.size)
    row, col, val = row[order], col[order], val[order]
    code, L, dx, dA = run_coo(m, n, row, col, val, p.dense["x"], p.dense["y"])
    assert code == 0
    rL, rdx, rdA = reference(m, n, row, col, val, p.dense["x"], p.dense["y"])
    assert loss_err(L, rL) <= LOSS_TOL
    assert grad_err(dx, rdx) <= GRAD_TOL
    assert grad_err(dA, rdA) <= GRAD_TOL


def test_coo_empty_and_out_of_range():
    rng = np.random.default_rng(22)
    x = rng.standard_normal(5).astype(np.float32)
    y = rng.standard_normal(7).astype(np.float32)
    code, L, dx, _ = run_coo(7, 5, [], [], [], x, y)
    assert code == 0 and abs(L - 0.5 * float((y.astype(np.float64) ** 2).sum())) <= 1e-6 * L
    assert np.all(dx == 0)
    # one entry with a column past n: skipped, reported as SDAD_ERR_INDEX (-3)
    code, L, dx, dA = run_coo(7, 5, [1, 2], [3, 5], [1.0, 2.0], x, y)
    assert code == -3
    rL, rdx, rdA = reference(7, 5, [1], [3], [1.0], x, y)
    assert loss_err(L, rL) <= LOSS_TOL and grad_err(dx, rdx) <= GRAD_TOL
