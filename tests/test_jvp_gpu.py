"""Forward mode on the GPU (sdad_lsq_jvp, sdad_logreg_jvp): the loss and its
directional derivative along a tangent of the dense vector and of the
sparse operand's values, against the fp64 oracle's forward mode, and against
the GPU's own reverse-mode gradient by the adjoint identity
<grad L, t> = dL[t] (a second, independent check of both paths)."""

import numpy as np
import pytest
import torch

import oracle
from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import runner as R
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W

pytestmark = pytest.mark.gpu
TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def dev(a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()


class Jvp:
    """One problem's device operands; run(vt, valt) -> (L, L')."""

    def __init__(self, name, p):
        self.name, self.p = name, p
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=False)
        self.v = dev(p.dense["x" if name == "lsq" else "w"])
        self.y = dev(p.dense["y"])
        expr = S.SDAD_EXPR_LSQ if name == "lsq" else S.SDAD_EXPR_LOGREG
        self.ws = S.Workspace(S.sdad_workspace_bytes(expr, p.m, p.n, self.A.nnz, 0))
        self.out = torch.zeros(2, dtype=torch.float64, device="cuda")

    def run(self, vt=None, valt=None):
        fn = S.sdad_lsq_jvp if self.name == "lsq" else S.sdad_logreg_jvp
        fn(self.A, self.v, self.y, self.out[0:], self.out[1:], dev(vt), dev(valt), self.ws)
        torch.cuda.synchronize()
        assert S.sdad_check(self.ws) == 0
        o = self.out.cpu().numpy()
        return float(o[0]), float(o[1])

    def oracle(self, vt=None, valt=None):
        p, d = self.p, self.p.dense
        if self.name == "lsq":
            return oracle.lsq_jvp(p.m, p.n, p.row, p.col, p.val, d["x"], d["y"], vt, valt)
        return oracle.logreg_jvp(p.m, p.n, p.row, p.col, p.val, d["w"], d["y"], vt, valt)


def tangents(rng, p):
    return (rng.standard_normal(p.n).astype(np.float32),
            rng.standard_normal(p.nnz).astype(np.float32))


def bound(g, vt, valt):
    """sum |grad| |tangent|: the scale of the directional derivative's rounding."""
    s = float(np.abs(g[0]) @ np.abs(vt)) if vt is not None else 0.0
    if valt is not None:
        s += float(np.abs(g[1]) @ np.abs(valt))
    return s


def oracle_grad(name, p):
    d = p.dense
    if name == "lsq":
        o = oracle.lsq(p.m, p.n, p.row, p.col, p.val, d["x"], d["y"])
        return o["dx"], o["dA"]
    o = oracle.logreg(p.m, p.n, p.row, p.col, p.val, d["w"], d["y"])
    return o["dw"], o["dX"]


@pytest.mark.parametrize("parts", ["both", "vector", "values"])
@pytest.mark.parametrize("name", ["lsq", "logreg"])
def test_jvp_against_oracle(name, parts):
    p = W.make(name, "small")
    rng = np.random.default_rng(5)
    vt, valt = tangents(rng, p)
    vt = vt if parts in ("both", "vector") else None
    valt = valt if parts in ("both", "values") else None
    j = Jvp(name, p)
    L, Lt = j.run(vt, valt)
    ref = j.oracle(vt, valt)
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * bound(oracle_grad(name, p), vt, valt)


@pytest.mark.parametrize("name", ["lsq", "logreg"])
def test_adjoint_identity_between_gpu_forward_and_reverse(name):
    p = W.make(name, "small")
    rng = np.random.default_rng(6)
    vt, valt = tangents(rng, p)
    _, Lt = Jvp(name, p).run(vt, valt)
    r = R.RUNS[name](p, tmode=S.SDAD_T_CSC, **({"want_dX": True} if name == "logreg" else {}))
    r.step()
    torch.cuda.synchronize()
    r.check()
    o = r.outputs()
    g = (o["dx"], o["dA"]) if name == "lsq" else (o["dw"], o["dX"])
    dot = float(g[0].astype(np.float64) @ vt) + float(g[1].astype(np.float64) @ valt)
    assert abs(Lt - dot) <= TOL * bound(g, vt, valt)


@pytest.mark.parametrize("name", ["lsq", "logreg"])
def test_zero_tangent_and_reproducibility(name):
    p = W.make(name, "small")
    j = Jvp(name, p)
    L0, Lt0 = j.run(None, None)
    assert Lt0 == 0.0
    rng = np.random.default_rng(7)
    vt, valt = tangents(rng, p)
    a = j.run(vt, valt)
    for _ in range(2):
        assert j.run(vt, valt) == a
    assert a[0] == L0


def test_empty_rows_and_empty_matrix():
    rng = np.random.default_rng(8)
    e = np.zeros(0, np.int32)
    p = W.SparseMatrixProblem("lsq", 50, 7, e, e, np.zeros(0, np.float32),
                              {"x": rng.standard_normal(7).astype(np.float32),
                               "y": rng.standard_normal(50).astype(np.float32)}, {})
    L, Lt = Jvp("lsq", p).run(rng.standard_normal(7).astype(np.float32), None)
    ref = oracle.lsq_jvp(50, 7, e, e, np.zeros(0, np.float32), p.dense["x"], p.dense["y"])
    assert abs(L - ref["loss"]) <= 1e-6 * ref["loss"] and Lt == 0.0


@pytest.mark.full
def test_logreg_full_size():
    p = W.make("logreg", "full")
    rng = np.random.default_rng(9)
    vt, valt = tangents(rng, p)
    j = Jvp("logreg", p)
    L, Lt = j.run(vt, valt)
    ref = j.oracle(vt, valt)
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * bound(oracle_grad("logreg", p), vt, valt)


# ----------------------------------------------------------------------------
# matrix factorisation and CP
# ----------------------------------------------------------------------------

def _jvp_mf(run, valt, Ut, Vt):
    out = torch.zeros(2, dtype=torch.float64, device="cuda")
    S.sdad_mf_jvp(run.desc, run.U, run.V, run.k, run.lam, out[0:], out[1:], dev(valt), dev(Ut),
                  dev(Vt), run.ws)
    torch.cuda.synchronize()
    run.check()
    o = out.cpu().numpy()
    return float(o[0]), float(o[1])


def _jvp_cp(run, tt, At, Bt, Ct):
    out = torch.zeros(2, dtype=torch.float64, device="cuda")
    S.sdad_cp3_jvp(run.desc, run.A, run.B, run.C, run.R, out[0:], out[1:], dev(tt), dev(At),
                   dev(Bt), dev(Ct), run.ws)
    torch.cuda.synchronize()
    run.check()
    o = out.cpu().numpy()
    return float(o[0]), float(o[1])


def _sbound(pairs):
    return sum(float(np.abs(np.asarray(g, np.float64)).ravel() @ np.abs(t).ravel())
               for g, t in pairs if t is not None)


def test_mf_jvp_against_oracle_and_reverse_mode():
    p = W.make("mf", "small")
    rng = np.random.default_rng(12)
    valt = rng.standard_normal(p.nnz).astype(np.float32)
    Ut = rng.standard_normal(p.dense["U"].shape).astype(np.float32)
    Vt = rng.standard_normal(p.dense["V"].shape).astype(np.float32)
    run = R.MfRun(p, want_dR=True)
    L, Lt = _jvp_mf(run, valt, Ut, Vt)
    ref = oracle.mf_jvp(p.m, p.n, p.row, p.col, p.val, p.dense["U"], p.dense["V"],
                        p.params["lam"], valt, Ut, Vt)
    g = oracle.mf(p.m, p.n, p.row, p.col, p.val, p.dense["U"], p.dense["V"], p.params["lam"])
    b = _sbound([(g["dR"], valt), (g["dU"], Ut), (g["dV"], Vt)])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * b
    run.step()
    torch.cuda.synchronize()
    o = run.outputs()
    dot = float(o["dR"].astype(np.float64) @ valt + (o["dU"].astype(np.float64) * Ut).sum() +
                (o["dV"].astype(np.float64) * Vt).sum())
    assert abs(Lt - dot) <= TOL * b
    L0, Lt0 = _jvp_mf(run, None, None, None)
    assert Lt0 == 0.0 and L0 == L
    assert _jvp_mf(run, valt, Ut, Vt) == (L, Lt)   # reproducible


def test_cp3_jvp_against_oracle_and_reverse_mode():
    p = W.make("cp3", "small")
    rng = np.random.default_rng(13)
    tt = rng.standard_normal(p.nnz).astype(np.float32)
    Ft = [rng.standard_normal(p.dense[x].shape).astype(np.float32) for x in ("A", "B", "C")]
    run = R.Cp3Run(p, want_dT=True)
    L, Lt = _jvp_cp(run, tt, *Ft)
    ref = oracle.cp3_jvp(p.dims, p.i, p.j, p.k, p.val, p.dense["A"], p.dense["B"], p.dense["C"],
                         tt, *Ft)
    g = oracle.cp3(p.dims, p.i, p.j, p.k, p.val, p.dense["A"], p.dense["B"], p.dense["C"])
    b = _sbound([(g["dT"], tt), (g["dA"], Ft[0]), (g["dB"], Ft[1]), (g["dC"], Ft[2])])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * b
    run.step()
    torch.cuda.synchronize()
    o = run.outputs()
    dot = float(o["dT"].astype(np.float64) @ tt + sum(
        (o[n].astype(np.float64) * t).sum() for n, t in zip(("dA", "dB", "dC"), Ft)))
    assert abs(Lt - dot) <= TOL * b
    L0, Lt0 = _jvp_cp(run, None, None, None, None)
    assert Lt0 == 0.0 and L0 == L
    # only the factor A moves
    La, Lta = _jvp_cp(run, None, Ft[0], None, None)
    refa = oracle.cp3_jvp(p.dims, p.i, p.j, p.k, p.val, p.dense["A"], p.dense["B"],
                          p.dense["C"], None, Ft[0], None, None)
    assert abs(Lta - refa["loss_t"]) <= TOL * _sbound([(g["dA"], Ft[0])])


@pytest.mark.full
def test_mf_cp3_jvp_full_size():
    rng = np.random.default_rng(14)
    p = W.make("mf", "full")
    Ut = rng.standard_normal(p.dense["U"].shape).astype(np.float32)
    run = R.MfRun(p)
    L, Lt = _jvp_mf(run, None, Ut, None)
    ref = oracle.mf_jvp(p.m, p.n, p.row, p.col, p.val, p.dense["U"], p.dense["V"],
                        p.params["lam"], None, Ut, None)
    g = oracle.mf(p.m, p.n, p.row, p.col, p.val, p.dense["U"], p.dense["V"], p.params["lam"])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * _sbound([(g["dU"], Ut)])
    del run, g
    p = W.make("cp3", "full")
    tt = rng.standard_normal(p.nnz).astype(np.float32)
    run = R.Cp3Run(p)
    L, Lt = _jvp_cp(run, tt, None, None, None)
    ref = oracle.cp3_jvp(p.dims, p.i, p.j, p.k, p.val, p.dense["A"], p.dense["B"], p.dense["C"],
                         tt)
    g = oracle.cp3(p.dims, p.i, p.j, p.k, p.val, p.dense["A"], p.dense["B"], p.dense["C"])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * _sbound([(g["dT"], tt)])


# ----------------------------------------------------------------------------
# graph propagation: P' = H' W + H W' on the tensor cores (one two-source product), Y' = A' P + A P'
# ----------------------------------------------------------------------------

def _jvp_gnn(run, valt, Ht, Wt):
    out = torch.zeros(2, dtype=torch.float64, device="cuda")
    S.sdad_gnn_jvp(run.desc, run.H, run.W, run.Z, run.f_in, run.f_out, out[0:], out[1:],
                   dev(valt), dev(Ht), dev(Wt), run.ws)
    torch.cuda.synchronize()
    run.check()
    o = out.cpu().numpy()
    return float(o[0]), float(o[1])


def _gnn_tangents(rng, p):
    return (rng.standard_normal(p.nnz).astype(np.float32),
            rng.standard_normal(p.dense["H"].shape).astype(np.float32),
            (0.1 * rng.standard_normal(p.dense["W"].shape)).astype(np.float32))


@pytest.mark.parametrize("parts", ["all", "values", "H", "W"])
def test_gnn_jvp_against_oracle_and_reverse_mode(parts):
    p = W.make("gnn", "small")
    rng = np.random.default_rng(15)
    valt, Ht, Wt = _gnn_tangents(rng, p)
    valt = valt if parts in ("all", "values") else None
    Ht = Ht if parts in ("all", "H") else None
    Wt = Wt if parts in ("all", "W") else None
    run = R.GnnRun(p)
    L, Lt = _jvp_gnn(run, valt, Ht, Wt)
    d = p.dense
    ref = oracle.gnn_jvp(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"], valt, Ht, Wt)
    g = oracle.gnn(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"])
    b = _sbound([(g["dA"], valt), (g["dH"], Ht), (g["dW"], Wt)])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * b
    # adjoint identity with the GPU's reverse mode
    run.step()
    torch.cuda.synchronize()
    run.check()
    o = run.outputs()
    dot = sum(float((o[k].astype(np.float64) * t).sum())
              for k, t in (("dA", valt), ("dH", Ht), ("dW", Wt)) if t is not None)
    assert abs(Lt - dot) <= TOL * b
    assert _jvp_gnn(run, valt, Ht, Wt) == (L, Lt)   # reproducible


def test_gnn_jvp_zero_tangent_and_empty_rows():
    p = W.make("gnn", "small")
    run = R.GnnRun(p)
    L0, Lt0 = _jvp_gnn(run, None, None, None)
    d = p.dense
    ref = oracle.gnn_jvp(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"])
    assert Lt0 == 0.0 and abs(L0 - ref["loss"]) <= TOL * abs(ref["loss"])
    # a matrix without keys: L = 1/2 |Z|^2, L' = 0 whatever the tangent
    e = np.zeros(0, np.int32)
    q = W.SparseMatrixProblem("gnn", p.m, p.n, e, e, np.zeros(0, np.float32), p.dense, p.params)
    run0 = R.GnnRun(q)
    rng = np.random.default_rng(16)
    _, Ht, Wt = _gnn_tangents(rng, p)
    L, Lt = _jvp_gnn(run0, None, Ht, Wt)
    z = d["Z"].astype(np.float64)
    assert abs(L - 0.5 * (z * z).sum()) <= 1e-6 * L and Lt == 0.0


@pytest.mark.full
def test_gnn_jvp_full_size():
    p = W.make("gnn", "full")
    rng = np.random.default_rng(17)
    valt, Ht, Wt = _gnn_tangents(rng, p)
    run = R.GnnRun(p)
    # every tangent: P' = H' W + H W' as one two-source product
    L, Lt = _jvp_gnn(run, valt, Ht, Wt)
    d = p.dense
    ref = oracle.gnn_jvp(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"], valt, Ht, Wt)
    g = oracle.gnn(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"])
    assert abs(L - ref["loss"]) <= TOL * abs(ref["loss"])
    assert abs(Lt - ref["loss_t"]) <= TOL * _sbound([(g["dA"], valt), (g["dH"], Ht), (g["dW"], Wt)])
