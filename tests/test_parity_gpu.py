"""GPU path against the fp64 oracle, element by element, through the C ABI.

Bar: sparse patterns bit-exact (the gradient arrays line up with the
operand's own keys), loss within 1e-4 relative, every gradient within
max_i |g_i - g*_i| / ||g*||_2 <= 1e-4.  Sizes span many chunks and end in a
ragged tail; edge cases cover empty operands, empty rows and columns, rows
and columns far longer than a chunk, and repeated calls on one workspace.
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


def run(name, p, **kw):
    r = R.RUNS[name](p, **kw)
    r.step()
    torch.cuda.synchronize()
    r.check()
    return r, r.outputs()


def matrix(name, m, n, row, col, val, dense, params=None):
    key = np.asarray(row, np.int64) * n + np.asarray(col, np.int64)
    order = np.argsort(key, kind="stable")
    return W.SparseMatrixProblem(name, m, n, np.asarray(row, np.int32)[order],
                                 np.asarray(col, np.int32)[order],
                                 np.asarray(val, np.float32)[order], dense, params or {})


def pattern_matches(run_obj, p):
    A = getattr(run_obj, "A", None) or getattr(run_obj, "X", None) or getattr(run_obj, "R", None)
    h = A.host
    assert np.array_equal(h["colidx"], p.col)
    cnt = np.bincount(p.row, minlength=p.m)
    assert np.array_equal(h["rowptr"], np.concatenate([[0], np.cumsum(cnt)]).astype(np.int32))


# ----------------------------------------------------------------------------
# generated workloads (scaled-down configurations)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("tmode", [S.SDAD_T_CSC, S.SDAD_T_ATOMIC])
def test_lsq_small(tmode):
    p = W.make("lsq", "small")
    r, out = run("lsq", p, tmode=tmode)
    pattern_matches(r, p)
    assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


def test_lsq_configuration_size():
    p = W.make("lsq", "full")       # 2000 x 2000, about 20k keys
    _, out = run("lsq", p)
    assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


def test_lsq_many_chunks():
    p = W.lsq_problem(m=3000, n=2500, draws=60001, seed=77)
    _, out = run("lsq", p)
    assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


@pytest.mark.parametrize("tmode", [S.SDAD_T_CSC, S.SDAD_T_ATOMIC])
def test_logreg_small(tmode):
    p = W.make("logreg", "small")
    r, out = run("logreg", p, tmode=tmode, want_dX=True)
    pattern_matches(r, p)
    ref = oracle_for("logreg", p)
    assert_close(out, ref, ["dw", "dX"])


# the two-pass path over the CSC twin, the one-pass atomic scatter (with and
# without the ranked numbering that sums the hot columns in shared memory),
# and AUTO (both timed on the first call, the faster kept)
@pytest.mark.parametrize("kw", [{"tmode": S.SDAD_T_CSC}, {"tmode": S.SDAD_T_ATOMIC},
                                {"tmode": S.SDAD_T_ATOMIC, "ranked": True},
                                {"tmode": S.SDAD_T_AUTO, "ranked": True}])
def test_mf_small(kw):
    p = W.make("mf", "small")
    r, out = run("mf", p, want_dR=True, **kw)
    pattern_matches(r, p)
    assert_close(out, oracle_for("mf", p), ["dU", "dV", "dR"])
    if kw["tmode"] == S.SDAD_T_AUTO:   # the kept choice on a second call
        r.step()
        torch.cuda.synchronize()
        r.check()
        assert_close(r.outputs(), oracle_for("mf", p), ["dU", "dV", "dR"])


def test_mf_atomic_without_csc_twin():
    # AUTO on a matrix without its CSC twin takes the one-pass scatter
    p = W.make("mf", "small")
    r = R.MfRun(p)
    r.desc.colptr = r.desc.rowidx = r.desc.val_csc = None
    r.step()
    torch.cuda.synchronize()
    r.check()
    assert_close(r.outputs(), oracle_for("mf", p), ["dU", "dV"])


@pytest.mark.parametrize("tmode", [S.SDAD_T_CSC, S.SDAD_T_ATOMIC])
def test_cp3_small(tmode):
    p = W.make("cp3", "small")
    _, out = run("cp3", p, tmode=tmode, want_dT=True)
    assert_close(out, oracle_for("cp3", p), ["dA", "dB", "dC", "dT"])


# dA in the column walk (transpose permutation) or in the forward walk; G by
# the column walk, scattered from the CSR (atomic), or as AUTO measures
@pytest.mark.parametrize("kw", [{"with_perm": True, "tmode": S.SDAD_T_CSC},
                                {"with_perm": False, "tmode": S.SDAD_T_CSC},
                                {"with_perm": True, "tmode": S.SDAD_T_ATOMIC},
                                {"with_perm": True, "tmode": S.SDAD_T_AUTO}])
def test_gnn_small(kw):
    p = W.make("gnn", "small")
    r, out = run("gnn", p, **kw)
    pattern_matches(r, p)
    assert_close(out, oracle_for("gnn", p), COMPARED["gnn"])


def test_gnn_without_csc_twin():
    # AUTO on a graph without its CSC twin scatters G from the CSR
    p = W.make("gnn", "small")
    r = R.GnnRun(p, with_perm=False)
    r.desc.colptr = r.desc.rowidx = r.desc.val_csc = None
    r.step()
    torch.cuda.synchronize()
    r.check()
    assert_close(r.outputs(), oracle_for("gnn", p), COMPARED["gnn"])


# ----------------------------------------------------------------------------
# edge cases
# ----------------------------------------------------------------------------

def test_lsq_empty_matrix():
    rng = np.random.default_rng(1)
    p = matrix("lsq", 7, 5, [], [], [], {"x": rng.standard_normal(5).astype(np.float32),
                                         "y": rng.standard_normal(7).astype(np.float32)})
    for tmode in (S.SDAD_T_CSC, S.SDAD_T_ATOMIC):
        _, out = run("lsq", p, tmode=tmode)
        ref = oracle_for("lsq", p)
        assert abs(out["loss"] - ref["loss"]) <= 1e-6 * ref["loss"]
        assert not out["dx"].any()


def test_lsq_long_rows_empty_rows_ragged_tail():
    # row 1 spans several chunks (WHOLE rows read past the staged chunk),
    # rows 0, 3 and the trailing rows are empty, nnz is not a multiple of 4
    rng = np.random.default_rng(2)
    n = 9000
    long_cols = rng.choice(n, size=7001, replace=False)
    rows = [np.full(7001, 1)]
    cols = [long_cols]
    for i in (2, 4, 5, 6):
        c = rng.choice(n, size=13, replace=False)
        rows.append(np.full(13, i))
        cols.append(c)
    row = np.concatenate(rows)
    col = np.concatenate(cols)
    m = 10
    p = matrix("lsq", m, n, row, col, rng.standard_normal(row.size),
               {"x": rng.standard_normal(n).astype(np.float32),
                "y": rng.standard_normal(m).astype(np.float32)})
    assert p.nnz % 4 != 0
    for tmode in (S.SDAD_T_CSC, S.SDAD_T_ATOMIC):
        _, out = run("lsq", p, tmode=tmode)
        assert_close(out, oracle_for("lsq", p), COMPARED["lsq"])


def test_logreg_hot_column_across_chunks():
    # column 0 is stored in every row: its CSC column spans many chunks
    rng = np.random.default_rng(3)
    m, n = 12000, 300
    row = np.concatenate([np.arange(m), rng.integers(0, m, 20000)])
    col = np.concatenate([np.zeros(m, np.int64), rng.integers(1, n, 20000)])
    key = np.unique(row * n + col)
    row, col = key // n, key % n
    p = matrix("logreg", m, n, row, col, rng.lognormal(size=row.size),
               {"w": (0.3 * rng.standard_normal(n)).astype(np.float32),
                "y": (rng.random(m) < 0.5).astype(np.float32)})
    for tmode in (S.SDAD_T_CSC, S.SDAD_T_ATOMIC):
        _, out = run("logreg", p, tmode=tmode, want_dX=True)
        assert_close(out, oracle_for("logreg", p), ["dw", "dX"])


@pytest.mark.parametrize("kw", [{"tmode": S.SDAD_T_CSC},
                                {"tmode": S.SDAD_T_ATOMIC, "ranked": True}])
def test_mf_hub_row_and_column(kw):
    rng = np.random.default_rng(4)
    m, n, k = 400, 6000, 64
    row = np.concatenate([np.zeros(5500, np.int64), rng.integers(0, m, 9000),
                          rng.integers(0, m, 3000)])
    col = np.concatenate([rng.choice(n, 5500, replace=False), rng.integers(0, n, 9000),
                          np.full(3000, 17)])
    key = np.unique(row * n + col)
    row, col = key // n, key % n
    p = matrix("mf", m, n, row, col, rng.integers(1, 6, row.size),
               {"U": (0.1 * rng.standard_normal((m, k))).astype(np.float32),
                "V": (0.1 * rng.standard_normal((n, k))).astype(np.float32)},
               {"k": k, "lam": 0.01})
    _, out = run("mf", p, want_dR=True, **kw)
    assert_close(out, oracle_for("mf", p), ["dU", "dV", "dR"])


def test_cp3_hub_index():
    rng = np.random.default_rng(5)
    dims, R_ = (50, 4000, 300), 32
    nn = 12000
    i = np.concatenate([np.zeros(6000, np.int64), rng.integers(0, dims[0], nn - 6000)])
    j = rng.integers(0, dims[1], nn)
    k = rng.integers(0, dims[2], nn)
    key = np.unique((i * dims[1] + j) * dims[2] + k)
    kk = key % dims[2]
    ij = key // dims[2]
    p = W.SparseTensor3Problem("cp3", dims, (ij // dims[1]).astype(np.int32),
                               (ij % dims[1]).astype(np.int32), kk.astype(np.int32),
                               rng.standard_normal(key.size).astype(np.float32),
                               {c: (0.2 * rng.standard_normal((d, R_))).astype(np.float32)
                                for c, d in zip("ABC", dims)}, {"rank": R_})
    for tmode in (S.SDAD_T_CSC, S.SDAD_T_ATOMIC):
        _, out = run("cp3", p, tmode=tmode, want_dT=True)
        assert_close(out, oracle_for("cp3", p), ["dA", "dB", "dC", "dT"])


@pytest.mark.parametrize("kw", [{"with_perm": True}, {"with_perm": False},
                                {"with_perm": True, "tmode": S.SDAD_T_ATOMIC}])
def test_gnn_hub_rows_columns_and_empty_rows(kw):
    # row 0 holds 3000 keys (> one chunk), column 5 holds every even row
    # (a long column part), rows in the upper half with odd index are empty
    rng = np.random.default_rng(6)
    nv = 3000
    row = np.concatenate([np.zeros(3000, np.int64), rng.integers(0, nv // 2, 8000),
                          np.arange(0, nv, 2)])
    col = np.concatenate([np.arange(3000), rng.integers(0, nv, 8000), np.full(nv // 2, 5)])
    key = np.unique(row * nv + col)
    row, col = key // nv, key % nv
    p = matrix("gnn", nv, nv, row, col, rng.random(row.size),
               {"H": rng.standard_normal((nv, 128)).astype(np.float32),
                "W": (0.1 * rng.standard_normal((128, 64))).astype(np.float32),
                "Z": rng.standard_normal((nv, 64)).astype(np.float32)},
               {"f_in": 128, "f_out": 64})
    assert (np.bincount(row, minlength=nv) == 0).any()
    _, out = run("gnn", p, **kw)
    assert_close(out, oracle_for("gnn", p), COMPARED["gnn"])


# ----------------------------------------------------------------------------
# reproducibility and repeated calls
# ----------------------------------------------------------------------------

def test_csc_paths_are_bit_reproducible():
    p = W.make("logreg", "small")
    r = R.LogregRun(p, tmode=S.SDAD_T_CSC)
    outs = []
    for _ in range(3):
        r.step()
        torch.cuda.synchronize()
        outs.append(r.outputs())
    r.check()
    for o in outs[1:]:
        assert o["loss"] == outs[0]["loss"]
        assert np.array_equal(o["dw"], outs[0]["dw"])
    q = W.make("lsq", "small")
    r = R.LsqRun(q, tmode=S.SDAD_T_CSC)
    r.step()
    a = r.outputs()
    r.step()
    b = r.outputs()
    assert a["loss"] == b["loss"] and np.array_equal(a["dx"], b["dx"])
    assert np.array_equal(a["dA"], b["dA"])


def test_repeated_calls_share_one_workspace():
    p = W.make("gnn", "small")
    r = R.GnnRun(p)
    losses = []
    for _ in range(3):
        r.step()
        losses.append(r.outputs()["loss"])
    r.check()
    ref = oracle_for("gnn", p)["loss"]
    for v in losses:
        assert abs(v - ref) <= 1e-4 * abs(ref)


def test_check_reports_ok():
    p = W.make("cp3", "small")
    r = R.Cp3Run(p)
    r.step()
    assert S.sdad_check(r.ws) == 0


def test_gnn_dA_alone_through_the_column_walk():
    # dA requested without dH, dW: with the permutation the column walk still runs
    p = W.make("gnn", "small")
    r = R.GnnRun(p)
    r.dH = r.dW = None
    r.step()
    torch.cuda.synchronize()
    r.check()
    out = {"loss": float(r.loss.item()), "dA": r.dA.cpu().numpy()}
    assert_close(out, oracle_for("gnn", p), ["dA"])
