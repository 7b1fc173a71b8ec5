"""Least squares and logistic regression with ranked column ids
(sdad_csr_rank_columns), against the fp64 oracle through the C ABI.

The ranked numbering changes only how the library stores and reads the
matrix: every output must match the oracle of the original matrix.  Cases
cover both transposed-product modes, many columns used by few rows, a column
present in every row (the first rank; its CSC column spans many chunks),
empty operands and repeated calls.
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

MODES = [S.SDAD_T_AUTO, S.SDAD_T_CSC, S.SDAD_T_ATOMIC]


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def run(name, p, **kw):
    r = R.RUNS[name](p, ranked=True, **kw)
    r.step()
    torch.cuda.synchronize()
    r.check()
    return r, r.outputs()


@pytest.mark.parametrize("tmode", MODES)
def test_lsq_ranked(tmode):
    p = W.make("lsq", "small")
    r, out = run("lsq", p, tmode=tmode)
    assert np.array_equal(r.A.host["rankcol"][r.A.host["rcolidx"]], p.col)
    assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


@pytest.mark.parametrize("tmode", MODES)
def test_logreg_ranked(tmode):
    p = W.make("logreg", "small")
    _, out = run("logreg", p, tmode=tmode, want_dX=True)
    assert_close(out, oracle_for("logreg", p), ["dw", "dX"])


@pytest.mark.parametrize("tmode", MODES)
def test_logreg_ranked_many_columns(tmode):
    # 30,000 Zipf columns, most of them used by a few rows only
    p = W.make("logreg", "small", m=6000, n=30000)
    assert np.unique(p.col).size > 20000
    _, out = run("logreg", p, tmode=tmode, want_dX=True)
    assert_close(out, oracle_for("logreg", p), ["dw", "dX"])


def test_lsq_ranked_column_in_every_row_and_ragged_tail():
    rng = np.random.default_rng(11)
    m, n = 9000, 5000
    row = np.concatenate([np.arange(m), rng.integers(0, m, 30001)])
    col = np.concatenate([np.full(m, 4321), rng.integers(0, n, 30001)])
    key = np.unique(row.astype(np.int64) * n + col)
    row, col = key // n, key % n
    p = W.SparseMatrixProblem("lsq", m, n, row.astype(np.int32), col.astype(np.int32),
                              rng.standard_normal(row.size).astype(np.float32),
                              {"x": rng.standard_normal(n).astype(np.float32),
                               "y": rng.standard_normal(m).astype(np.float32)}, {})
    for tmode in MODES:
        r, out = run("lsq", p, tmode=tmode)
        assert r.A.host["rankcol"][0] == 4321
        assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


def test_ranked_empty_operands():
    e = np.zeros(0, np.int32)
    for m, n in ((5, 7), (3, 0)):
        p = W.SparseMatrixProblem("lsq", m, n, e, e, np.zeros(0, np.float32),
                                  {"x": np.ones(n, np.float32),
                                   "y": np.arange(m, dtype=np.float32)}, {})
        for tmode in MODES:
            _, out = run("lsq", p, tmode=tmode)
            assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


def test_ranked_csc_is_bit_reproducible_and_atomic_loss_is_stable():
    p = W.make("logreg", "small", m=6000, n=30000)
    r = R.LogregRun(p, tmode=S.SDAD_T_CSC, ranked=True)
    outs = []
    for _ in range(3):
        r.step()
        outs.append(r.outputs())
    for o in outs[1:]:
        assert o["loss"] == outs[0]["loss"] and np.array_equal(o["dw"], outs[0]["dw"])
    # the atomic path fixes the order of the loss sum (the dw additions are not ordered)
    q = R.LogregRun(p, tmode=S.SDAD_T_ATOMIC, ranked=True)
    losses = []
    for _ in range(3):
        q.step()
        losses.append(q.outputs()["loss"])
    q.check()
    assert losses[1] == losses[0] and losses[2] == losses[0]


# A larger instance (70,000 rows, 60,000 Zipf columns), in every mode, with
# dX (the emitting variant of the row pass) and without.
@pytest.mark.parametrize("tmode", MODES)
@pytest.mark.parametrize("want_dX", [False, True])
def test_logreg_ranked_larger(tmode, want_dX):
    p = W.make("logreg", "small", m=70000, n=60000, mean_row=20.0)
    _, out = run("logreg", p, tmode=tmode, want_dX=want_dX)
    assert_close(out, oracle_for("logreg", p), ["dw", "dX"] if want_dX else ["dw"])


def test_lsq_ranked_larger():
    p = W.lsq_problem(m=70000, n=50000, draws=800000, seed=99)
    _, out = run("lsq", p, tmode=S.SDAD_T_CSC)
    assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])
