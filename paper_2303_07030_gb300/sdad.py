"""Python binding of libsdad (ctypes).  Argument marshalling only.

Functions carry the C names (``sdad_lsq_grad`` ...) and take torch tensors
(or None for NULL); every step of the computation runs in the library's CUDA
kernels.  PyTorch is used for device memory and streams.  The library must
have been built (``paper_2303_07030_gb300.build.build()``); if it is missing
the import of this module's ``lib()`` raises -- there is no CPU fallback.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libsdad.so")

SDAD_OK = 0
STATUS_NAMES = {
    0: "SDAD_OK", -1: "SDAD_ERR_NULL", -2: "SDAD_ERR_SHAPE", -3: "SDAD_ERR_INDEX",
    -4: "SDAD_ERR_ALIGN", -5: "SDAD_ERR_OVERFLOW", -6: "SDAD_ERR_WORKSPACE",
    -7: "SDAD_ERR_CUDA", -8: "SDAD_ERR_TIMEOUT", -9: "SDAD_ERR_UNSUPPORTED",
}
SDAD_T_AUTO, SDAD_T_CSC, SDAD_T_ATOMIC = 0, 1, 2
SDAD_EXPR_LSQ, SDAD_EXPR_LOGREG, SDAD_EXPR_MF, SDAD_EXPR_CP3, SDAD_EXPR_GNN = 1, 2, 3, 4, 5
SDAD_EXPR_SMVM, SDAD_EXPR_SMMM, SDAD_EXPR_BATAX = 6, 7, 8

# every symbol include/sdad.h declares
EXPORTS = [
    "sdad_status_string", "sdad_version", "sdad_csr_from_coo", "sdad_csr_transpose",
    "sdad_csr_rank_columns", "sdad_csr_block_transpose", "sdad_csr_transpose_rest",
    "sdad_coo3_mode_index", "sdad_workspace_bytes", "sdad_workspace_init", "sdad_check",
    "sdad_workspace_set_wait_limit",
    "sdad_lsq_grad", "sdad_logreg_grad", "sdad_mf_grad", "sdad_cp3_grad", "sdad_gnn_grad",
    "sdad_lsq_grad_noalloc", "sdad_lsq_jvp", "sdad_logreg_jvp", "sdad_mf_jvp", "sdad_cp3_jvp",
    "sdad_smvm_grad", "sdad_smmm_grad", "sdad_csr_gram_pattern",
    "sdad_batax_grad",
    "sdad_timing_enable", "sdad_timing_reset", "sdad_timing_count", "sdad_timing_get",
    "sdad_probe_fma", "sdad_gather_by_perm", "sdad_gnn_jvp", "sdad_lsq_coo_grad",
]


class SdadError(RuntimeError):
    def __init__(self, code, what):
        self.code = code
        super().__init__("%s: %s (%d)" % (what, STATUS_NAMES.get(code, "?"), code))


class sdad_csr(ctypes.Structure):
    _fields_ = [
        ("m", ctypes.c_int32), ("n", ctypes.c_int32), ("nnz", ctypes.c_int64),
        ("rowptr", ctypes.c_void_p), ("colidx", ctypes.c_void_p), ("val", ctypes.c_void_p),
        ("colptr", ctypes.c_void_p), ("rowidx", ctypes.c_void_p), ("val_csc", ctypes.c_void_p),
        ("rcolidx", ctypes.c_void_p), ("rankcol", ctypes.c_void_p),
        ("bcsc_log2", ctypes.c_int32), ("bcsc_nnz", ctypes.c_int64),
        ("bcsc_ptr", ctypes.c_void_p), ("bcsc_key", ctypes.c_void_p), ("bcsc_val", ctypes.c_void_p),
        ("bcsc_ncols", ctypes.c_int32), ("bcsc_cols", ctypes.c_void_p),
        ("bcsc_rest_nnz", ctypes.c_int64), ("csc_perm", ctypes.c_void_p),
    ]


class sdad_coo(ctypes.Structure):
    _fields_ = [
        ("m", ctypes.c_int32), ("n", ctypes.c_int32), ("nnz", ctypes.c_int64),
        ("row", ctypes.c_void_p), ("col", ctypes.c_void_p), ("val", ctypes.c_void_p),
    ]


class sdad_coo3(ctypes.Structure):
    _fields_ = [
        ("dims", ctypes.c_int32 * 3), ("nnz", ctypes.c_int64),
        ("idx", ctypes.c_void_p * 3), ("val", ctypes.c_void_p),
        ("sidx", (ctypes.c_void_p * 3) * 3), ("sval", ctypes.c_void_p * 3),
        ("sperm", ctypes.c_void_p * 3), ("segptr", ctypes.c_void_p * 3),
    ]


_lib = None


def lib():
    """The loaded libsdad.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libsdad.so not built (run paper_2303_07030_gb300.build.build())")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                 ctypes.c_float, ctypes.c_size_t)
        P = ctypes.POINTER
        sigs = {
            "sdad_status_string": ([i32], ctypes.c_char_p),
            "sdad_version": ([], i32),
            "sdad_csr_from_coo": ([i32, i32, i64, vp, vp, vp, vp, vp, vp, P(i64)], i32),
            "sdad_csr_transpose": ([i32, i32, i64, vp, vp, vp, vp, vp], i32),
            "sdad_csr_rank_columns": ([i32, i64, vp, vp, vp], i32),
            "sdad_csr_block_transpose": ([i32, i32, i64, vp, vp, i32, i32, vp, vp, vp, vp,
                                          P(i64)], i32),
            "sdad_csr_transpose_rest": ([i32, i32, i64, vp, vp, i32, vp, vp, vp, vp, P(i64)],
                                        i32),
            "sdad_coo3_mode_index": ([i64, vp, vp, vp, vp, i32, vp, vp], i32),
            "sdad_workspace_bytes": ([i32, i32, i32, i64, i32, P(sz)], i32),
            "sdad_workspace_init": ([vp, vp], i32),
            "sdad_check": ([vp, vp], i32),
            "sdad_workspace_set_wait_limit": ([vp, i64, vp], i32),
            "sdad_lsq_grad": ([P(sdad_csr), vp, vp, vp, vp, vp, i32, vp, sz, vp], i32),
            "sdad_logreg_grad": ([P(sdad_csr), vp, vp, vp, vp, vp, i32, vp, sz, vp], i32),
            "sdad_mf_grad": ([P(sdad_csr), vp, vp, i32, f32, vp, vp, vp, vp, i32, vp, sz, vp],
                             i32),
            "sdad_cp3_grad": ([P(sdad_coo3), vp, vp, vp, i32, vp, vp, vp, vp, vp, i32, vp, sz,
                               vp], i32),
            "sdad_gnn_grad": ([P(sdad_csr), vp, vp, vp, i32, i32, vp, vp, vp, vp, i32, vp, sz,
                               vp], i32),
            "sdad_lsq_grad_noalloc": ([P(sdad_csr), vp, vp, vp, vp, vp, i32, vp], i32),
            "sdad_lsq_jvp": ([P(sdad_csr), vp, vp, vp, vp, vp, vp, vp, sz, vp], i32),
            "sdad_logreg_jvp": ([P(sdad_csr), vp, vp, vp, vp, vp, vp, vp, sz, vp], i32),
            "sdad_mf_jvp": ([P(sdad_csr), vp, vp, i32, f32, vp, vp, vp, vp, vp, vp, sz, vp], i32),
            "sdad_cp3_jvp": ([P(sdad_coo3), vp, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, sz, vp],
                             i32),
            "sdad_smvm_grad": ([P(sdad_csr), vp, vp, vp, vp, sz, vp], i32),
            "sdad_smmm_grad": ([P(sdad_csr), P(sdad_csr), vp, vp, vp, sz, vp], i32),
            "sdad_csr_gram_pattern": ([i32, i32, i64, vp, vp, vp, vp, P(i64)], i32),
            "sdad_batax_grad": ([P(sdad_csr), vp, f32, vp, vp, vp, i64, vp, vp, sz, vp], i32),
            "sdad_timing_enable": ([i32], i32),
            "sdad_timing_reset": ([], i32),
            "sdad_timing_count": ([], i32),
            "sdad_timing_get": ([i32, P(ctypes.c_char_p), P(ctypes.c_float)], i32),
            "sdad_probe_fma": ([vp, i32, i32, P(ctypes.c_double), vp], i32),
            "sdad_gather_by_perm": ([vp, i64, vp, i64, vp, vp], i32),
            "sdad_gnn_jvp": ([P(sdad_csr), vp, vp, vp, i32, i32, vp, vp, vp, vp, vp, vp, sz, vp],
                             i32),
            "sdad_lsq_coo_grad": ([P(sdad_coo), vp, vp, vp, vp, vp, vp, sz, vp], i32),
        }
        for name, (args, res) in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _ptr(t):
    """Device or host address of a tensor / numpy array, or None."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def _check(code, what):
    if code != SDAD_OK:
        raise SdadError(code, what)


# ----------------------------------------------------------------------------
# host builders (numpy in, numpy out)
# ----------------------------------------------------------------------------

def sdad_csr_from_coo(m, n, row, col, val=None):
    row = np.ascontiguousarray(row, dtype=np.int32)
    col = np.ascontiguousarray(col, dtype=np.int32)
    v = None if val is None else np.ascontiguousarray(val, dtype=np.float32)
    nnz = row.size
    rowptr = np.zeros(m + 1, np.int32)
    colidx = np.zeros(max(nnz, 1), np.int32)
    vout = np.zeros(max(nnz, 1), np.float32) if v is not None else None
    nout = ctypes.c_int64(0)
    _check(lib().sdad_csr_from_coo(m, n, nnz, _ptr(row), _ptr(col), _ptr(v), _ptr(rowptr),
                                   _ptr(colidx), _ptr(vout), ctypes.byref(nout)),
           "sdad_csr_from_coo")
    k = nout.value
    return rowptr, colidx[:k].copy(), (vout[:k].copy() if vout is not None else None)


def sdad_csr_transpose(m, n, rowptr, colidx):
    rowptr = np.ascontiguousarray(rowptr, dtype=np.int32)
    colidx = np.ascontiguousarray(colidx, dtype=np.int32)
    nnz = colidx.size
    colptr = np.zeros(n + 1, np.int32)
    rowidx = np.zeros(max(nnz, 1), np.int32)
    perm = np.zeros(max(nnz, 1), np.int32)
    _check(lib().sdad_csr_transpose(m, n, nnz, _ptr(rowptr), _ptr(colidx), _ptr(colptr),
                                    _ptr(rowidx), _ptr(perm)), "sdad_csr_transpose")
    return colptr, rowidx[:nnz].copy(), perm[:nnz].copy()


def sdad_csr_rank_columns(n, colidx):
    colidx = np.ascontiguousarray(colidx, dtype=np.int32)
    nnz = colidx.size
    rcol = np.zeros(max(nnz, 1), np.int32)
    rankcol = np.zeros(max(n, 1), np.int32)
    _check(lib().sdad_csr_rank_columns(n, nnz, _ptr(colidx), _ptr(rcol), _ptr(rankcol)),
           "sdad_csr_rank_columns")
    return rcol[:nnz].copy(), rankcol[:n].copy()


BCSC_CHUNK = 1024


def sdad_csr_block_transpose(m, n, rowptr, colidx, rb_log2, cols=None):
    """Row-blocked CSC twin of the columns `cols` (all when None)."""
    rowptr = np.ascontiguousarray(rowptr, dtype=np.int32)
    colidx = np.ascontiguousarray(colidx, dtype=np.int32)
    nnz = colidx.size
    if cols is not None:
        cols = np.ascontiguousarray(cols, dtype=np.int32)
    ncols = n if cols is None else cols.size
    cnt = ctypes.c_int64(0)
    _check(lib().sdad_csr_block_transpose(m, n, nnz, _ptr(rowptr), _ptr(colidx), rb_log2, ncols,
                                          _ptr(cols), None, None, None, ctypes.byref(cnt)),
           "sdad_csr_block_transpose")
    nb = (m + (1 << rb_log2) - 1) >> rb_log2
    blkptr = np.zeros(nb + 1, np.int32)
    bkey = np.zeros(max(cnt.value, 1), np.uint32)
    bperm = np.zeros(max(cnt.value, 1), np.int32)
    _check(lib().sdad_csr_block_transpose(m, n, nnz, _ptr(rowptr), _ptr(colidx), rb_log2, ncols,
                                          _ptr(cols), _ptr(blkptr), _ptr(bkey), _ptr(bperm),
                                          ctypes.byref(cnt)), "sdad_csr_block_transpose")
    return blkptr, bkey[:cnt.value].copy(), bperm[:cnt.value].copy()


def sdad_csr_transpose_rest(m, n, rowptr, colidx, cols):
    """CSC twin of the keys whose column is not in `cols`: (colptr, rowidx, perm)."""
    rowptr = np.ascontiguousarray(rowptr, dtype=np.int32)
    colidx = np.ascontiguousarray(colidx, dtype=np.int32)
    cols = np.ascontiguousarray(cols, dtype=np.int32)
    nnz = colidx.size
    colptr = np.zeros(n + 1, np.int32)
    rowidx = np.zeros(max(nnz, 1), np.int32)
    perm = np.zeros(max(nnz, 1), np.int32)
    cnt = ctypes.c_int64(0)
    _check(lib().sdad_csr_transpose_rest(m, n, nnz, _ptr(rowptr), _ptr(colidx), cols.size,
                                         _ptr(cols), _ptr(colptr), _ptr(rowidx), _ptr(perm),
                                         ctypes.byref(cnt)), "sdad_csr_transpose_rest")
    return colptr, rowidx[:cnt.value].copy(), perm[:cnt.value].copy()


def split_columns(colidx, n, m, rb_log2, min_per_block):
    """The columns with at least `min_per_block` keys per row block on
    average (ascending ids): the ones a split column pass reads from the
    row-blocked twin."""
    nb = max(1, (m + (1 << rb_log2) - 1) >> rb_log2)
    cnt = np.bincount(np.asarray(colidx, dtype=np.int64), minlength=n)
    return np.flatnonzero(cnt >= min_per_block * nb).astype(np.int32)


def sdad_coo3_mode_index(i, j, k, dims, mode):
    i, j, k = (np.ascontiguousarray(a, dtype=np.int32) for a in (i, j, k))
    d = np.ascontiguousarray(dims, dtype=np.int32)
    nnz = i.size
    perm = np.zeros(max(nnz, 1), np.int32)
    seg = np.zeros(int(d[mode]) + 1 if 0 <= mode < 3 else 1, np.int32)
    _check(lib().sdad_coo3_mode_index(nnz, _ptr(i), _ptr(j), _ptr(k), _ptr(d), mode, _ptr(perm),
                                      _ptr(seg)), "sdad_coo3_mode_index")
    return perm[:nnz].copy(), seg


# ----------------------------------------------------------------------------
# workspace
# ----------------------------------------------------------------------------

def sdad_workspace_bytes(expr, rows, cols, nnz, width):
    out = ctypes.c_size_t(0)
    _check(lib().sdad_workspace_bytes(expr, rows, cols, nnz, width, ctypes.byref(out)),
           "sdad_workspace_bytes")
    return out.value


def sdad_workspace_init(ws, stream=None):
    _check(lib().sdad_workspace_init(_ptr(ws), _stream(stream)), "sdad_workspace_init")


def sdad_check(ws, stream=None):
    return lib().sdad_check(_ptr(ws), _stream(stream))


def sdad_workspace_set_wait_limit(ws, polls, stream=None):
    """polls < 0: the default limit; otherwise every bounded wait polls that often."""
    _check(lib().sdad_workspace_set_wait_limit(_ptr(ws), int(polls), _stream(stream)),
           "sdad_workspace_set_wait_limit")


class Workspace:
    """Device workspace: a zero-initialised torch byte buffer, 256-byte aligned."""

    def __init__(self, nbytes, device="cuda"):
        import torch
        self.buf = torch.zeros(nbytes + 256, dtype=torch.uint8, device=device)
        off = (-self.buf.data_ptr()) % 256
        self.view = self.buf[off:off + nbytes]
        self.nbytes = nbytes

    def data_ptr(self):
        return self.view.data_ptr()


# ----------------------------------------------------------------------------
# per-kernel timing
# ----------------------------------------------------------------------------

def sdad_timing_enable(on=True):
    _check(lib().sdad_timing_enable(1 if on else 0), "sdad_timing_enable")


def sdad_timing_reset():
    _check(lib().sdad_timing_reset(), "sdad_timing_reset")


def sdad_timing_count():
    return int(lib().sdad_timing_count())


def sdad_timing_get(i):
    name = ctypes.c_char_p()
    ms = ctypes.c_float(0)
    _check(lib().sdad_timing_get(i, ctypes.byref(name), ctypes.byref(ms)), "sdad_timing_get")
    return name.value.decode(), float(ms.value)


def sdad_timing_records():
    """All (kernel name, milliseconds) records since the last reset."""
    return [sdad_timing_get(i) for i in range(sdad_timing_count())]


def sdad_gather_by_perm(src, perm, out, stream=None):
    """out[q] = src[perm[q]] (0 where perm[q] is out of range), on the device; 4-byte dtypes."""
    assert src.element_size() == 4 and out.element_size() == 4 and perm.numel() == out.numel()
    _check(lib().sdad_gather_by_perm(_ptr(src), src.numel(), _ptr(perm), perm.numel(), _ptr(out),
                                     _stream(stream)), "sdad_gather_by_perm")
    return out


def sdad_probe_fma(out, blocks, iters, stream=None):
    """Enqueues the FP32 FMA probe; returns the FLOPs it performs."""
    fl = ctypes.c_double(0.0)
    _check(lib().sdad_probe_fma(_ptr(out), int(blocks), int(iters), ctypes.byref(fl),
                                _stream(stream)), "sdad_probe_fma")
    return fl.value


# ----------------------------------------------------------------------------
# device operands
# ----------------------------------------------------------------------------

class CsrDevice:
    """CSR matrix (plus optional CSC twin) in device memory, built from a
    sorted, duplicate-free or arbitrary host COO with the library's builders."""

    def __init__(self, m, n, row, col, val, csc=True, ranked=False, blocked=0, block_cols=None,
                 with_perm=False, device="cuda"):
        """blocked: rb_log2 of a row-blocked CSC twin (0: none).  block_cols:
        the columns it holds (None: all); the CSC twin then holds the others.
        with_perm: pass the CSC twin's transpose permutation (csc_perm)."""
        self.with_perm = bool(with_perm and csc)
        import torch
        rowptr, colidx, v = sdad_csr_from_coo(m, n, row, col, val)
        self.m, self.n, self.nnz = int(m), int(n), int(colidx.size)
        dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.rowptr, self.colidx, self.val = dev(rowptr), dev(colidx), dev(v)
        self.host = {"rowptr": rowptr, "colidx": colidx, "val": v}
        split = bool(blocked) and block_cols is not None
        self.colptr = self.rowidx = self.val_csc = self.perm = None
        self.bcsc_rest_nnz = 0
        if csc or split:
            if split:
                colptr, rowidx, perm = sdad_csr_transpose_rest(m, n, rowptr, colidx, block_cols)
                self.bcsc_rest_nnz = int(rowidx.size)
            else:
                colptr, rowidx, perm = sdad_csr_transpose(m, n, rowptr, colidx)
            self.colptr, self.rowidx, self.perm = dev(colptr), dev(rowidx), dev(perm)
            self.val_csc = torch.empty(perm.size, dtype=torch.float32, device=device)
            sdad_gather_by_perm(self.val, self.perm, self.val_csc)
            self.host.update(colptr=colptr, rowidx=rowidx, perm=perm)
        self.bcsc_log2, self.bcsc_nnz, self.bcsc_ncols = 0, 0, 0
        self.bcsc_ptr = self.bcsc_key = self.bcsc_val = self.bcsc_cols = self.bperm = None
        if blocked:
            # row-blocked CSC twin with 2^blocked rows per block
            bp, bk, bperm = sdad_csr_block_transpose(m, n, rowptr, colidx, blocked, block_cols)
            self.bcsc_log2, self.bcsc_nnz = int(blocked), int(bk.size)
            self.bcsc_ptr, self.bcsc_key, self.bperm = dev(bp), dev(bk.view(np.int32)), dev(bperm)
            self.bcsc_val = torch.empty(bk.size, dtype=torch.float32, device=device)
            sdad_gather_by_perm(self.val, self.bperm, self.bcsc_val)
            self.host.update(bcsc_ptr=bp, bcsc_key=bk, bcsc_perm=bperm)
            if split:
                bc = np.ascontiguousarray(block_cols, dtype=np.int32)
                self.bcsc_ncols = int(bc.size)
                self.bcsc_cols = dev(bc) if bc.size else dev(np.zeros(1, np.int32))
                self.host.update(bcsc_cols=bc)
        self.rcolidx = self.rankcol = None
        if ranked:
            rcol, rankcol = sdad_csr_rank_columns(n, colidx)
            self.rcolidx, self.rankcol = dev(rcol), dev(rankcol)
            self.host.update(rcolidx=rcol, rankcol=rankcol)

    def refresh_values(self, stream=None):
        """After self.val changed on the device: the twins' value copies again
        (val_csc = val[perm], bcsc_val = val[bperm]), gathered on the device."""
        if self.val_csc is not None and self.perm is not None:
            sdad_gather_by_perm(self.val, self.perm, self.val_csc, stream)
        if self.bcsc_val is not None and self.bperm is not None:
            sdad_gather_by_perm(self.val, self.bperm, self.bcsc_val, stream)

    def desc(self):
        return sdad_csr(self.m, self.n, self.nnz, _ptr(self.rowptr), _ptr(self.colidx),
                        _ptr(self.val), _ptr(self.colptr), _ptr(self.rowidx), _ptr(self.val_csc),
                        _ptr(self.rcolidx), _ptr(self.rankcol), self.bcsc_log2, self.bcsc_nnz,
                        _ptr(self.bcsc_ptr), _ptr(self.bcsc_key), _ptr(self.bcsc_val),
                        self.bcsc_ncols, _ptr(self.bcsc_cols), self.bcsc_rest_nnz,
                        _ptr(self.perm) if self.with_perm else None)


class Coo3Device:
    """3-way COO tensor in device memory with one mode-sorted copy per mode."""

    def __init__(self, dims, i, j, k, val, modes=(0, 1, 2), device="cuda"):
        import torch
        dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.dims = tuple(int(d) for d in dims)
        self.nnz = int(np.asarray(i).size)
        host_idx = [np.ascontiguousarray(a, dtype=np.int32) for a in (i, j, k)]
        host_val = np.ascontiguousarray(val, dtype=np.float32)
        self.idx = [dev(a) for a in host_idx]
        self.val = dev(host_val)
        self.sidx = [[None] * 3 for _ in range(3)]
        self.sval = [None] * 3
        self.sperm = [None] * 3
        self.segptr = [None] * 3
        for m in modes:
            perm, seg = sdad_coo3_mode_index(host_idx[0], host_idx[1], host_idx[2], self.dims, m)
            self.sperm[m] = dev(perm)
            self.segptr[m] = dev(seg)
            # the sorted copies, gathered on the device through the mode's permutation
            for c in range(3):
                self.sidx[m][c] = sdad_gather_by_perm(self.idx[c], self.sperm[m],
                                                      torch.empty_like(self.idx[c]))
            self.sval[m] = sdad_gather_by_perm(self.val, self.sperm[m], torch.empty_like(self.val))

    def desc(self):
        d = sdad_coo3()
        for c in range(3):
            d.dims[c] = self.dims[c]
            d.idx[c] = _ptr(self.idx[c])
        d.nnz = self.nnz
        d.val = _ptr(self.val)
        for m in range(3):
            for c in range(3):
                d.sidx[m][c] = _ptr(self.sidx[m][c])
            d.sval[m] = _ptr(self.sval[m])
            d.sperm[m] = _ptr(self.sperm[m])
            d.segptr[m] = _ptr(self.segptr[m])
        return d


# ----------------------------------------------------------------------------
# entry points (same names as the C ABI)
# ----------------------------------------------------------------------------

def _ws(ws):
    return (ws.data_ptr(), ws.nbytes) if ws is not None else (None, 0)


def sdad_lsq_grad(A, x, y, loss, dx=None, dA_val=None, tmode=SDAD_T_AUTO, ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_lsq_grad(ctypes.byref(d), _ptr(x), _ptr(y), _ptr(loss), _ptr(dx),
                               _ptr(dA_val), tmode, wp, wb, _stream(stream)), "sdad_lsq_grad")


def sdad_lsq_grad_noalloc(A, x, y, loss, dx=None, dA_val=None, tmode=SDAD_T_AUTO, stream=None):
    """Least squares without a workspace (built-in 8 MiB scratch; see sdad.h)."""
    d = A.desc() if hasattr(A, "desc") else A
    _check(lib().sdad_lsq_grad_noalloc(ctypes.byref(d), _ptr(x), _ptr(y), _ptr(loss), _ptr(dx),
                                       _ptr(dA_val), tmode, _stream(stream)),
           "sdad_lsq_grad_noalloc")


def sdad_logreg_grad(X, w, y, loss, dw=None, dX_val=None, tmode=SDAD_T_AUTO, ws=None,
                     stream=None):
    d = X.desc() if hasattr(X, "desc") else X
    wp, wb = _ws(ws)
    _check(lib().sdad_logreg_grad(ctypes.byref(d), _ptr(w), _ptr(y), _ptr(loss), _ptr(dw),
                                  _ptr(dX_val), tmode, wp, wb, _stream(stream)),
           "sdad_logreg_grad")


def sdad_mf_grad(R, U, V, k, lam, loss, dU=None, dV=None, dR_val=None, tmode=SDAD_T_AUTO,
                 ws=None, stream=None):
    d = R.desc() if hasattr(R, "desc") else R
    wp, wb = _ws(ws)
    _check(lib().sdad_mf_grad(ctypes.byref(d), _ptr(U), _ptr(V), k, lam, _ptr(loss), _ptr(dU),
                              _ptr(dV), _ptr(dR_val), tmode, wp, wb, _stream(stream)),
           "sdad_mf_grad")


def sdad_cp3_grad(T, A, B, C, rank, loss, dA=None, dB=None, dC=None, dT_val=None,
                  tmode=SDAD_T_AUTO, ws=None, stream=None):
    d = T.desc() if hasattr(T, "desc") else T
    wp, wb = _ws(ws)
    _check(lib().sdad_cp3_grad(ctypes.byref(d), _ptr(A), _ptr(B), _ptr(C), rank, _ptr(loss),
                               _ptr(dA), _ptr(dB), _ptr(dC), _ptr(dT_val), tmode, wp, wb,
                               _stream(stream)), "sdad_cp3_grad")


def sdad_lsq_jvp(A, x, y, loss, loss_t, x_t=None, A_t_val=None, ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_lsq_jvp(ctypes.byref(d), _ptr(x), _ptr(y), _ptr(x_t), _ptr(A_t_val),
                              _ptr(loss), _ptr(loss_t), wp, wb, _stream(stream)), "sdad_lsq_jvp")


def sdad_logreg_jvp(X, w, y, loss, loss_t, w_t=None, X_t_val=None, ws=None, stream=None):
    d = X.desc() if hasattr(X, "desc") else X
    wp, wb = _ws(ws)
    _check(lib().sdad_logreg_jvp(ctypes.byref(d), _ptr(w), _ptr(y), _ptr(w_t), _ptr(X_t_val),
                                 _ptr(loss), _ptr(loss_t), wp, wb, _stream(stream)),
           "sdad_logreg_jvp")


def sdad_mf_jvp(R, U, V, k, lam, loss, loss_t, R_t_val=None, U_t=None, V_t=None, ws=None,
                stream=None):
    d = R.desc() if hasattr(R, "desc") else R
    wp, wb = _ws(ws)
    _check(lib().sdad_mf_jvp(ctypes.byref(d), _ptr(U), _ptr(V), k, float(lam), _ptr(R_t_val),
                             _ptr(U_t), _ptr(V_t), _ptr(loss), _ptr(loss_t), wp, wb,
                             _stream(stream)), "sdad_mf_jvp")


def sdad_lsq_coo_grad(A, x, y, loss, dx=None, dA_val=None, ws=None, stream=None):
    """A: an sdad_coo (device row, col, val in entry order)."""
    wp, wb = _ws(ws)
    _check(lib().sdad_lsq_coo_grad(ctypes.byref(A), _ptr(x), _ptr(y), _ptr(loss), _ptr(dx),
                                   _ptr(dA_val), wp, wb, _stream(stream)), "sdad_lsq_coo_grad")


def sdad_gnn_jvp(A, H, W, Z, f_in, f_out, loss, loss_t, A_t_val=None, H_t=None, W_t=None,
                 ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_gnn_jvp(ctypes.byref(d), _ptr(H), _ptr(W), _ptr(Z), f_in, f_out,
                              _ptr(A_t_val), _ptr(H_t), _ptr(W_t), _ptr(loss), _ptr(loss_t), wp,
                              wb, _stream(stream)), "sdad_gnn_jvp")


def sdad_cp3_jvp(T, A, B, C, rank, loss, loss_t, T_t_val=None, A_t=None, B_t=None, C_t=None,
                 ws=None, stream=None):
    d = T.desc() if hasattr(T, "desc") else T
    wp, wb = _ws(ws)
    _check(lib().sdad_cp3_jvp(ctypes.byref(d), _ptr(A), _ptr(B), _ptr(C), rank, _ptr(T_t_val),
                              _ptr(A_t), _ptr(B_t), _ptr(C_t), _ptr(loss), _ptr(loss_t), wp, wb,
                              _stream(stream)), "sdad_cp3_jvp")


def sdad_smvm_grad(A, X, f, dX=None, ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_smvm_grad(ctypes.byref(d), _ptr(X), _ptr(f), _ptr(dX), wp, wb,
                                _stream(stream)), "sdad_smvm_grad")


def sdad_smmm_grad(A, B, f, dB_val=None, ws=None, stream=None):
    da = A.desc() if hasattr(A, "desc") else A
    db = B.desc() if hasattr(B, "desc") else B
    wp, wb = _ws(ws)
    _check(lib().sdad_smmm_grad(ctypes.byref(da), ctypes.byref(db), _ptr(f), _ptr(dB_val), wp,
                                wb, _stream(stream)), "sdad_smmm_grad")


def sdad_csr_gram_pattern(m, n, rowptr, colidx):
    """Pattern of A^T A: (jrowptr, jcolidx)."""
    rowptr = np.ascontiguousarray(rowptr, dtype=np.int32)
    colidx = np.ascontiguousarray(colidx, dtype=np.int32)
    jrowptr = np.zeros(n + 1, np.int32)
    cnt = ctypes.c_int64(0)
    _check(lib().sdad_csr_gram_pattern(m, n, colidx.size, _ptr(rowptr), _ptr(colidx),
                                       _ptr(jrowptr), None, ctypes.byref(cnt)),
           "sdad_csr_gram_pattern")
    jcolidx = np.zeros(max(cnt.value, 1), np.int32)
    _check(lib().sdad_csr_gram_pattern(m, n, colidx.size, _ptr(rowptr), _ptr(colidx),
                                       _ptr(jrowptr), _ptr(jcolidx), ctypes.byref(cnt)),
           "sdad_csr_gram_pattern")
    return jrowptr, jcolidx[:cnt.value].copy()


def sdad_batax_grad(A, X, beta, f=None, jrowptr=None, jcolidx=None, jnnz=0, J_val=None,
                    ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_batax_grad(ctypes.byref(d), _ptr(X), float(beta), _ptr(f), _ptr(jrowptr),
                                 _ptr(jcolidx), int(jnnz), _ptr(J_val), wp, wb,
                                 _stream(stream)), "sdad_batax_grad")


def sdad_gnn_grad(A, H, W, Z, f_in, f_out, loss, dA_val=None, dH=None, dW=None,
                  tmode=SDAD_T_AUTO, ws=None, stream=None):
    d = A.desc() if hasattr(A, "desc") else A
    wp, wb = _ws(ws)
    _check(lib().sdad_gnn_grad(ctypes.byref(d), _ptr(H), _ptr(W), _ptr(Z), f_in, f_out,
                               _ptr(loss), _ptr(dA_val), _ptr(dH), _ptr(dW), tmode, wp, wb,
                               _stream(stream)), "sdad_gnn_grad")
