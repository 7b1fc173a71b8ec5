"""Shared helpers of the parity tests: tolerances and oracle runs."""

import numpy as np

import oracle

# Two gates on every gradient (fp32 path against the fp64 oracle), both 1e-4:
#   elementwise  max_i |g_i - g*_i| / ||g*||_2
#   normwise     ||g - g*||_2 / ||g*||_2
# Since ||d||_2 >= max_i |d_i|, the normwise gate implies the elementwise one;
# grad_err reports the larger of the two, so one comparison checks both.
GRAD_TOL = 1e-4
LOSS_TOL = 1e-4


def grad_errs(got, ref):
    """(elementwise, normwise) errors of a gradient, both normalised by ||g*||_2."""
    got = np.asarray(got, dtype=np.float64).reshape(-1)
    ref = np.asarray(ref, dtype=np.float64).reshape(-1)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0, 0.0
    nrm = float(np.linalg.norm(ref))
    d = got - ref
    mx = float(np.max(np.abs(d)))
    nw = float(np.linalg.norm(d))
    if not np.isfinite(mx):
        return float("inf"), float("inf")
    return (mx / nrm, nw / nrm) if nrm > 0 else (mx, nw)


def grad_err(got, ref):
    return max(grad_errs(got, ref))


def loss_err(got, ref):
    return abs(got - ref) / abs(ref) if ref != 0 else abs(got)


def assert_close(out, ref, keys, tol=GRAD_TOL, ltol=LOSS_TOL):
    errs = {"loss": loss_err(out["loss"], ref["loss"])}
    for k in keys:
        errs[k] = grad_err(out[k], ref[k])
    bad = {k: v for k, v in errs.items() if v > (ltol if k == "loss" else tol)}
    assert not bad, "tolerance exceeded: %s (all: %s)" % (bad, errs)
    return errs


def oracle_for(name, p):
    d = p.dense
    if name == "lsq":
        return oracle.lsq(p.m, p.n, p.row, p.col, p.val, d["x"], d["y"])
    if name == "logreg":
        return oracle.logreg(p.m, p.n, p.row, p.col, p.val, d["w"], d["y"])
    if name == "mf":
        return oracle.mf(p.m, p.n, p.row, p.col, p.val, d["U"], d["V"], p.params["lam"])
    if name == "cp3":
        return oracle.cp3(p.dims, p.i, p.j, p.k, p.val, d["A"], d["B"], d["C"])
    if name == "gnn":
        return oracle.gnn(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"])
    if name == "smvm":
        o = oracle.smvm(p.m, p.n, p.row, p.col, p.val, d["X"])
        return {"loss": o["f"], "dX": o["dX"]}
    if name == "smmm":
        o = oracle.smmm(p.m, p.n, p.n, (p.row, p.col, p.val), p.params["B"])
        return {"loss": o["f"], "dB": o["dB"]}
    if name == "batax":
        o = oracle.batax(p.m, p.n, p.row, p.col, p.val, d["X"], p.params["beta"])
        return {"loss": 0.0, "f": o["f"], "J": o["jval"], "jrow": o["jrow"], "jcol": o["jcol"]}
    raise KeyError(name)


# outputs compared for each loss (runner output name -> oracle output name)
COMPARED = {
    "lsq": ["dx", "dA"],
    "logreg": ["dw"],
    "mf": ["dU", "dV"],
    "cp3": ["dA", "dB", "dC"],
    "gnn": ["dA", "dH", "dW"],
    "smvm": ["dX"],
    "smmm": ["dB"],
    "batax": ["f", "J"],
}
