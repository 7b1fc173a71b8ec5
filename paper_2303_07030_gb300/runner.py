"""Device-side set-up and one call of each loss, for tests and the benchmark.

A ``*Run`` object uploads a generated problem (see ``workloads``), builds the
physical formats with the library's host builders, allocates outputs and the
workspace, and ``step()`` enqueues one loss-and-gradient evaluation through the
C ABI.  Nothing here computes any part of a loss.
"""

from __future__ import annotations

import numpy as np
import torch

from . import sdad as S


def _dev(a, device):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


class _Base:
    expr = 0
    tmode = S.SDAD_T_AUTO

    def _workspace(self, rows, cols, nnz, width):
        # lsq/logreg: width = rb_log2 of the row-blocked CSC twin (0: none)
        self.ws = S.Workspace(S.sdad_workspace_bytes(self.expr, rows, cols, nnz, width),
                              device=self.device)

    def check(self, stream=None):
        code = S.sdad_check(self.ws, stream)
        if code != 0:
            raise S.SdadError(code, "device status")

    def host_bytes_in(self):
        return 0

    def step_inputs(self):
        """Device tensors one step reads (the inputs an end-to-end step copies in)."""
        raise NotImplementedError


def _csr_inputs(A, csc, ranked):
    ts = [A.rowptr, A.rcolidx if ranked else A.colidx, A.val]
    if ranked:
        ts.append(A.rankcol)
    if csc and A.bcsc_log2:
        ts += [A.bcsc_ptr, A.bcsc_key, A.bcsc_val]
        if A.bcsc_cols is not None:   # split: the blocked columns plus the rest's CSC
            ts += [A.bcsc_cols, A.colptr, A.rowidx, A.val_csc]
    elif csc:
        ts += [A.colptr, A.rowidx, A.val_csc]
    return [t for t in ts if t is not None and t.numel()]


class LsqRun(_Base):
    expr = S.SDAD_EXPR_LSQ

    def __init__(self, p, tmode=S.SDAD_T_AUTO, want_dA=True, want_dx=True, ranked=False,
                 blocked=0, block_cols=None, device="cuda"):
        self.p, self.tmode, self.device, self.ranked = p, tmode, device, ranked
        self.csc = want_dx and tmode != S.SDAD_T_ATOMIC
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, ranked=ranked,
                             blocked=blocked, block_cols=block_cols, device=device)
        self.desc = self.A.desc()
        self.x = _dev(p.dense["x"], device)
        self.y = _dev(p.dense["y"], device)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dx = torch.empty(p.n, dtype=torch.float32, device=device) if want_dx else None
        self.dA = torch.empty(self.A.nnz, dtype=torch.float32, device=device) if want_dA else None
        self._workspace(p.m, p.n, self.A.nnz, blocked)

    def step(self, stream=None):
        S.sdad_lsq_grad(self.desc, self.x, self.y, self.loss, self.dx, self.dA, self.tmode,
                        self.ws, stream)

    def step_inputs(self):
        return _csr_inputs(self.A, self.csc, self.ranked) + [self.x, self.y]

    def outputs(self):
        out = {"loss": float(self.loss.item())}
        if self.dx is not None:
            out["dx"] = self.dx.cpu().numpy()
        if self.dA is not None:
            out["dA"] = self.dA.cpu().numpy()
        return out


class LogregRun(_Base):
    expr = S.SDAD_EXPR_LOGREG

    def __init__(self, p, tmode=S.SDAD_T_AUTO, want_dX=False, ranked=False, blocked=0,
                 block_cols=None, device="cuda"):
        self.p, self.tmode, self.device, self.ranked = p, tmode, device, ranked
        self.csc = tmode != S.SDAD_T_ATOMIC
        self.X = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, ranked=ranked,
                             blocked=blocked, block_cols=block_cols, device=device)
        self.desc = self.X.desc()
        self.w = _dev(p.dense["w"], device)
        self.y = _dev(p.dense["y"], device)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dw = torch.empty(p.n, dtype=torch.float32, device=device)
        self.dX = torch.empty(self.X.nnz, dtype=torch.float32, device=device) if want_dX else None
        self._workspace(p.m, p.n, self.X.nnz, blocked)

    def step(self, stream=None):
        S.sdad_logreg_grad(self.desc, self.w, self.y, self.loss, self.dw, self.dX, self.tmode,
                           self.ws, stream)

    def step_inputs(self):
        return _csr_inputs(self.X, self.csc, self.ranked) + [self.w, self.y]

    def outputs(self):
        out = {"loss": float(self.loss.item()), "dw": self.dw.cpu().numpy()}
        if self.dX is not None:
            out["dX"] = self.dX.cpu().numpy()
        return out


class MfRun(_Base):
    expr = S.SDAD_EXPR_MF

    def __init__(self, p, want_dR=False, tmode=S.SDAD_T_AUTO, ranked=False, device="cuda"):
        """tmode: SDAD_T_CSC (row pass + column pass over the CSC twin), SDAD_T_ATOMIC
        (one pass, dV scattered with atomics; with ranked columns the most used
        columns are summed in shared memory first) or AUTO (measured)."""
        self.p, self.device, self.tmode, self.ranked = p, device, tmode, ranked
        self.k = int(p.params["k"])
        self.lam = float(p.params["lam"])
        self.R = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, ranked=ranked,
                             device=device)
        self.desc = self.R.desc()
        self.U = _dev(p.dense["U"], device)
        self.V = _dev(p.dense["V"], device)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dU = torch.empty_like(self.U)
        self.dV = torch.empty_like(self.V)
        self.dR = torch.empty(self.R.nnz, dtype=torch.float32, device=device) if want_dR else None
        self._workspace(p.m, p.n, self.R.nnz, self.k)

    def step(self, stream=None):
        S.sdad_mf_grad(self.desc, self.U, self.V, self.k, self.lam, self.loss, self.dU, self.dV,
                       self.dR, self.tmode, self.ws, stream)

    def step_inputs(self):
        csc = self.dV is not None and self.tmode != S.SDAD_T_ATOMIC
        ts = _csr_inputs(self.R, csc, False)
        if self.ranked:   # the atomic scatter reads the ranks beside the column ids
            ts += [t for t in (self.R.rcolidx, self.R.rankcol) if t is not None and t.numel()]
        return ts + [self.U, self.V]

    def outputs(self):
        out = {"loss": float(self.loss.item()), "dU": self.dU.cpu().numpy(),
               "dV": self.dV.cpu().numpy()}
        if self.dR is not None:
            out["dR"] = self.dR.cpu().numpy()
        return out


class Cp3Run(_Base):
    expr = S.SDAD_EXPR_CP3

    def __init__(self, p, tmode=S.SDAD_T_AUTO, want_dT=False, device="cuda"):
        self.p, self.tmode, self.device = p, tmode, device
        self.R = int(p.params["rank"])
        # AUTO is the one-pass atomic scatter for this loss (the sorted copies are not read)
        self.atomic = tmode in (S.SDAD_T_AUTO, S.SDAD_T_ATOMIC)
        modes = () if self.atomic else (0, 1, 2)
        self.T = S.Coo3Device(p.dims, p.i, p.j, p.k, p.val, modes=modes, device=device)
        self.desc = self.T.desc()
        self.A = _dev(p.dense["A"], device)
        self.B = _dev(p.dense["B"], device)
        self.C = _dev(p.dense["C"], device)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dA = torch.empty_like(self.A)
        self.dB = torch.empty_like(self.B)
        self.dC = torch.empty_like(self.C)
        self.dT = torch.empty(p.nnz, dtype=torch.float32, device=device) if want_dT else None
        dmax = max(p.dims)
        self._workspace(dmax, dmax, p.nnz, self.R)

    def step(self, stream=None):
        S.sdad_cp3_grad(self.desc, self.A, self.B, self.C, self.R, self.loss, self.dA, self.dB,
                        self.dC, self.dT, self.tmode, self.ws, stream)

    def step_inputs(self):
        T = self.T
        if self.atomic:
            ts = T.idx + [T.val]
        else:
            ts = []
            for m in range(3):
                ts += T.sidx[m] + [T.sval[m], T.segptr[m]]
                if self.dT is not None:
                    ts.append(T.sperm[m])
        return [t for t in ts if t is not None and t.numel()] + [self.A, self.B, self.C]

    def outputs(self):
        out = {"loss": float(self.loss.item()), "dA": self.dA.cpu().numpy(),
               "dB": self.dB.cpu().numpy(), "dC": self.dC.cpu().numpy()}
        if self.dT is not None:
            out["dT"] = self.dT.cpu().numpy()
        return out


class GnnRun(_Base):
    expr = S.SDAD_EXPR_GNN

    def __init__(self, p, want_dA=True, with_perm=True, tmode=S.SDAD_T_AUTO, device="cuda"):
        """tmode: SDAD_T_CSC (G = A^T D by the column walk over the CSC twin),
        SDAD_T_ATOMIC (G scattered from the CSR) or AUTO (measured)."""
        self.p, self.device, self.tmode = p, device, tmode
        self.f_in, self.f_out = int(p.params["f_in"]), int(p.params["f_out"])
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, with_perm=with_perm,
                             device=device)
        self.desc = self.A.desc()
        self.H = _dev(p.dense["H"], device)
        self.W = _dev(p.dense["W"], device)
        self.Z = _dev(p.dense["Z"], device)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dA = torch.empty(self.A.nnz, dtype=torch.float32, device=device) if want_dA else None
        self.dH = torch.empty_like(self.H)
        self.dW = torch.empty_like(self.W)
        self._workspace(p.m, p.n, self.A.nnz, self.f_out)

    def step(self, stream=None):
        S.sdad_gnn_grad(self.desc, self.H, self.W, self.Z, self.f_in, self.f_out, self.loss,
                        self.dA, self.dH, self.dW, self.tmode, self.ws, stream)

    def step_inputs(self):
        extra = [self.A.perm] if self.A.with_perm else []
        return _csr_inputs(self.A, True, False) + extra + [self.H, self.W, self.Z]

    def outputs(self):
        out = {"loss": float(self.loss.item()), "dH": self.dH.cpu().numpy(),
               "dW": self.dW.cpu().numpy()}
        if self.dA is not None:
            out["dA"] = self.dA.cpu().numpy()
        return out


class SmvmRun(_Base):
    """SMVM f = sum A(i,j) X(j); df/dX = A^T 1."""
    expr = S.SDAD_EXPR_SMVM

    def __init__(self, p, device="cuda"):
        self.p, self.device = p, device
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, device=device)
        self.desc = self.A.desc()
        self.X = _dev(p.dense["X"], device)
        self.f = torch.zeros(1, dtype=torch.float64, device=device)
        self.dX = torch.empty(p.n, dtype=torch.float32, device=device)
        self._workspace(p.m, p.n, self.A.nnz, 0)

    def step(self, stream=None):
        S.sdad_smvm_grad(self.desc, self.X, self.f, self.dX, self.ws, stream)

    def step_inputs(self):
        return [t for t in (self.A.rowptr, self.A.colptr, self.A.val_csc, self.X) if t.numel()]

    def outputs(self):
        return {"loss": float(self.f.item()), "dX": self.dX.cpu().numpy()}


class SmmmRun(_Base):
    """SMMM f = sum A(i,k) B(k,j); df/dB on B's keys."""
    expr = S.SDAD_EXPR_SMMM

    def __init__(self, p, device="cuda"):
        self.p, self.device = p, device
        brow, bcol, bval = p.params["B"]
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, device=device)
        self.B = S.CsrDevice(p.n, p.n, brow, bcol, bval, csc=False, device=device)
        self.descA, self.descB = self.A.desc(), self.B.desc()
        self.f = torch.zeros(1, dtype=torch.float64, device=device)
        self.dB = torch.empty(self.B.nnz, dtype=torch.float32, device=device)
        self._workspace(p.m, p.n, self.A.nnz, 0)

    def step(self, stream=None):
        S.sdad_smmm_grad(self.descA, self.descB, self.f, self.dB, self.ws, stream)

    def step_inputs(self):
        ts = [self.A.colptr, self.A.val_csc, self.B.rowptr, self.B.colidx, self.B.val]
        return [t for t in ts if t.numel()]

    def outputs(self):
        return {"loss": float(self.f.item()), "dB": self.dB.cpu().numpy()}


class BataxRun(_Base):
    """BATAX f = beta A^T A X; df/dX = beta A^T A on the pattern of A^T A."""
    expr = S.SDAD_EXPR_BATAX

    def __init__(self, p, want_f=True, device="cuda"):
        self.p, self.device = p, device
        self.beta = float(p.params["beta"])
        self.A = S.CsrDevice(p.m, p.n, p.row, p.col, p.val, csc=True, device=device)
        self.desc = self.A.desc()
        jr, jc = S.sdad_csr_gram_pattern(p.m, p.n, self.A.host["rowptr"], self.A.host["colidx"])
        self.jnnz = int(jc.size)
        self.host_pattern = (jr, jc)
        self.jrowptr, self.jcolidx = _dev(jr, device), _dev(jc, device)
        self.X = _dev(p.dense["X"], device)
        self.f = torch.empty(p.n, dtype=torch.float32, device=device) if want_f else None
        self.J = torch.empty(max(self.jnnz, 1), dtype=torch.float32, device=device)
        self._workspace(p.m, p.n, self.A.nnz, 0)

    def step(self, stream=None):
        S.sdad_batax_grad(self.desc, self.X, self.beta, self.f, self.jrowptr, self.jcolidx,
                          self.jnnz, self.J, self.ws, stream)

    def step_inputs(self):
        ts = [self.A.rowptr, self.A.colidx, self.A.val, self.A.colptr, self.A.rowidx,
              self.A.val_csc, self.jrowptr, self.jcolidx, self.X]
        return [t for t in ts if t.numel()]

    def outputs(self):
        out = {"loss": 0.0, "J": self.J.cpu().numpy()[:self.jnnz]}
        if self.f is not None:
            out["f"] = self.f.cpu().numpy()
        return out


RUNS = {"lsq": LsqRun, "logreg": LogregRun, "mf": MfRun, "cp3": Cp3Run, "gnn": GnnRun,
        "smvm": SmvmRun, "smmm": SmmmRun, "batax": BataxRun}
