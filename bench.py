#!/usr/bin/env python3
"""Benchmark: loss + full gradient of sparse losses on one GB300 per rank.

Headline workload (the largest): graph propagation Y = A (H W), L = 1/2
|Y - Z|^2 on an R-MAT graph of 2^22 vertices and 2^26 edges (a, b, c = .57,
.19, .19), H 2^22 x 128, W 128 x 64; one step = one call of sdad_gnn_grad
(loss, dA on A's keys, dH, dW) with every input resident in HBM.  The line
also carries, under "configs", the same measurement of every other workload
(least squares, logistic regression, matrix factorisation, CP, and the
paper's SMVM, SMMM and BATAX kernels), each at full size, and the FP32 FMA
rate measured in the same run ("fp32_fma_peak"), against which the
arithmetic-bound kernels are reported.  ``--config`` picks another headline;
``--others none`` measures the headline alone.

Prints one JSON line (rank 0).  Timing: W warm-up steps, then K steps, each
bracketed by CUDA events on the launching stream; the inputs of the large
workloads exceed the 129 MB L2, the small workloads flush L2 (a 256 MB write)
between timed steps.  Per-kernel times come from a second pass of the same
K steps with every library kernel bracketed by events on its stream.

``--impl reference`` times the fp64 CPU oracle instead (host cores, bounded
sample of the same workload); under torchrun only rank 0 runs it.
"""

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "nnz·iter/s for loss+full gradient; achieved HBM GB/s vs GB300 peak"
UNIT = "nnz·iter/s"

WORKLOAD_NAMES = {
    "lsq": "least squares 0.5|Ax-y|^2, A 2000x2000 uniform 0.5% (~20k nnz), grads dx, dA",
    "logreg": "logistic regression, X 1e6x1e5 CSR, Poisson(50) keys/row, Zipf(1.1) columns, "
              "lognormal values; loss + dw",
    "mf": "matrix factorisation, R 5e5x2e5, 5e7 keys, Zipf(1.2) rows and columns, k=64; "
          "loss + dU + dV",
    "cp3": "CP decomposition, 1e4^3 tensor, 1e7 uniform keys, rank 32; loss + dA + dB + dC",
    "gnn": "graph propagation A(HW), R-MAT 2^22 nodes 2^26 edges, 128->64; loss + dA + dH + dW",
    "smvm": "SMVM f = sum A(i,j) X(j), df/dX; A a banded stand-in for Table 1 consph "
            "(83,000^2, 3.05M keys)",
    "smmm": "SMMM f = sum A(i,k) B(k,j), df/dB on B's keys; A, B banded stand-ins for Table 1 "
            "consph (83,000^2, 3.05M keys each)",
    "batax": "BATAX f = beta A^T A X, f and df/dX = beta A^T A (on the pattern of A^T A); A a "
             "banded stand-in for Table 1 consph (83,000^2, 3.05M keys)",
}


ALL_CONFIGS = ["gnn", "logreg", "mf", "cp3", "lsq", "smvm", "smmm", "batax"]
SMALL_CONFIGS = ("lsq", "smvm", "smmm", "batax")   # inputs below L2: flushed between steps


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="gnn", choices=list(WORKLOAD_NAMES),
                    help="the headline workload (default: the largest, graph propagation)")
    ap.add_argument("--others", default="all", choices=["all", "none"],
                    help="all: also measure every other workload under the line's 'configs'")
    ap.add_argument("--tmode", default="auto", choices=["auto", "csc", "atomic"])
    ap.add_argument("--transpose", default="auto", choices=["auto", "csc", "blocked", "split"],
                    help="lsq/logreg: column pass over the plain CSC twin; over a row-blocked "
                         "CSC twin of every column (r gathered from shared memory); or split: "
                         "the columns with at least --block-min keys per row block from a "
                         "row-blocked twin, the others from a plain CSC twin.  auto: blocked "
                         "for the 1e6-row logistic matrix, CSC for the 2000-row least squares")
    ap.add_argument("--block-log2", type=int, default=15,
                    help="rows per block (log2) of the row-blocked twin")
    ap.add_argument("--block-min", type=float, default=32.0,
                    help="split: keys per row block a column needs to be blocked")
    ap.add_argument("--columns", default="auto", choices=["auto", "ranked", "plain"],
                    help="lsq/logreg: column numbering of the matrix (ranked by key count, "
                         "built once on the host, or as generated; auto: ranked for the "
                         "Zipf-skewed logistic columns, as generated for the uniform lsq ones)")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the benchmark line: the density / dimension sweep of the "
                         "library's own passes (least squares at fixed dimension and at fixed "
                         "keys per row, logistic regression by keys per row, R-MAT graphs by "
                         "scale); one JSON line with a point per instance")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-jvp", action="store_true", help="skip the forward-mode timing")
    ap.add_argument("--override", action="append", default=[], metavar="KEY=VALUE",
                    help="change a generator parameter of the headline workload (profiling of "
                         "a smaller instance, e.g. m=400000); the line then says so")
    return ap.parse_args()


def overrides(args):
    out = {}
    for kv in args.override:
        k, v = kv.split("=", 1)
        try:
            out[k] = int(v) if v.lstrip("-").isdigit() else float(v)
        except ValueError:
            out[k] = v   # a name (e.g. matrix=pdb1HYS)
    return out


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ----------------------------------------------------------------------------
# algorithmic bytes per launch of each kernel (compulsory traffic: every array
# moved once per pass; gathered vectors counted once)
# ----------------------------------------------------------------------------

def kernel_bytes(cfg, p, nnz, tmode_csc, want_extra, ranked=False, blocked=0, split=None):
    """split: (H, keys of the H blocked columns) when only some columns are blocked."""
    m, n = p.m if hasattr(p, "m") else 0, p.n if hasattr(p, "n") else 0
    b = {}
    if cfg in ("lsq", "logreg"):
        rowk = "lsq_row" if cfg == "lsq" else "logreg_row"
        b[rowk] = 8 * nnz + 4 * (m + 1) + 4 * m + 4 * n
        if cfg == "lsq" or want_extra:
            b[rowk] += 4 * nnz                  # dA / dX written
        if tmode_csc:
            b[rowk] += 4 * m                    # r kept for the column pass
            if blocked:   # per-block column sums, summed over the blocks afterwards
                h, hk = split if split is not None else (n, nnz)
                if split is not None:   # the other columns' plain pass
                    b["scalar_col"] = 8 * (nnz - hk) + 4 * (n + 1) + 4 * m + 4 * n
                # compulsory traffic only: the per-block sums P (nb x h floats, in L2)
                # are this design's own
                b["scalar_bcol"] = 8 * hk + 4 * m
                b["bcol_combine"] = 4 * h + (4 * h if split is not None else 0)
            else:
                b["scalar_col"] = 8 * nnz + 4 * (n + 1) + 4 * m + 4 * n
        else:
            b[rowk] += 4 * n                    # dw / dx accumulated once
            b["zero"] = 4 * n
        if ranked:
            b["rank_prep"] = 4 * n * 4          # rankcol, v gathered, v' written, acc zeroed
            b["rank_finish"] = 4 * n * 3        # rankcol, acc, dw written (per-CTA blocks not counted)
    elif cfg == "mf":
        k = 64
        b["mf_row"] = 8 * nnz + 4 * (m + 1) + 4 * k * (m + n) + 4 * k * m
        b["mf_col"] = 8 * nnz + 4 * (n + 1) + 4 * k * (m + n) + 4 * k * n
        # one pass: column ids, ranks and values of the keys; U, V read; dU, dV written
        b["mf_atomic"] = 12 * nnz + 4 * (m + 1) + 2 * 4 * k * (m + n)
        b["mf_init"] = 2 * 4 * k * (m + n)
    elif cfg == "cp3":
        d = sum(p.dims)
        b["cp_mode"] = 12 * nnz + 4 * (max(p.dims) + 1) + 4 * 32 * d + 4 * 32 * max(p.dims)
        b["cp_atomic"] = 16 * nnz + 2 * 4 * 32 * d   # entries; factors read, gradients written
    elif cfg == "smvm":
        b["col_sums"] = 4 * nnz + 4 * (n + 1) + 4 * n
        b["smvm_dot"] = 8 * n
    elif cfg == "smmm":
        nb = int(p.params["B"][0].size)
        na = nnz - nb
        b["col_sums"] = 4 * na + 4 * (n + 1) + 4 * n
        b["smmm_row"] = 8 * nb + 4 * (n + 1) + 4 * n + 4 * nb
    elif cfg == "batax":
        b["batax_row"] = 8 * nnz + 4 * (m + 1) + 4 * n + 4 * m
        b["scalar_col"] = 8 * nnz + 4 * (n + 1) + 4 * m + 4 * n
        jnnz = p.params.get("jnnz", 0)
        # A's CSR and CSC once, the Jacobian's pattern read and its values written
        b["batax_gram"] = 16 * nnz + 8 * (n + 1) + 8 * jnnz
    elif cfg == "gnn":
        f_in, f_out = 128, 64
        # rows and columns that hold keys: only their Z, D, P and G rows are walked
        mr = int(np.count_nonzero(np.bincount(p.row, minlength=m)))
        nc = int(np.count_nonzero(np.bincount(p.col, minlength=n)))
        row = 4 * f_out
        b["proj_fwd"] = 4 * n * f_in + 4 * n * f_out + 4 * f_in * f_out
        # pointers; Z of the rows without keys read, G of the columns without keys zeroed
        b["gnn_empty"] = 4 * (m + 1) + 4 * (n + 1) + row * (m - mr) + row * (n - nc)
        # keys (index, value); P of each column with keys once; Z read and D written per row with keys
        b["gnn_fwd"] = 8 * nnz + 4 * (m + 1) + row * nc + 2 * row * mr
        # keys (index, value, transpose permutation) and dA; D once per row with keys;
        # P read and G written once per column with keys
        b["gnn_col"] = 12 * nnz + 4 * nnz + 4 * (n + 1) + row * mr + 2 * row * nc
        b["proj_bwd"] = 4 * n * f_in * 2 + 4 * n * f_out
    return b


def kernel_flops(cfg, p, nnz):
    """FP32 arithmetic per launch of the kernels bound by it rather than by HBM."""
    f = {}
    if cfg == "mf":
        f["mf_row"] = 256 * nnz       # per key: 64-wide dot (128) + 64-wide axpy (128)
        f["mf_col"] = 256 * nnz
        f["mf_atomic"] = 384 * nnz    # dot + two axpys (dU in registers, dV scattered)
    elif cfg == "cp3":
        f["cp_atomic"] = 384 * nnz    # e: 32 x 3; three 32-wide gradient terms: 3 x 32 x 3
        f["cp_mode"] = 192 * nnz      # e and one mode's gradient term
    return f


# ----------------------------------------------------------------------------
# measured DRAM traffic (ncu dram__bytes_read.sum + dram__bytes_write.sum) of
# some kernels, per key, each from one capture of a reduced instance of its
# workload in the benchmark's layout, scaled to a launch by its keys (traffic
# grows with the keys at fixed density).  A figure belongs to the kernel
# source it was taken on: when that file changes, or the layout differs, the
# traffic is reported as null until it is captured again.
# ----------------------------------------------------------------------------
NCU_TRAFFIC = {
    "gnn": {
        # the full workload itself (2^22 vertices, 2^26 edges): dram__bytes_read.sum +
        # dram__bytes_write.sum of one launch each, a 1-pass ncu capture; per kernel the
        # source file it was taken on
        "nnz": 67108864,
        "bytes_per_launch": {
            "gnn_col": ("paper_2303_07030_gb300/csrc/k_gnn.cu",
                        "dd3221af39633b7b53b0c1a2bd68e53ef5b27e88", 7699289856 + 1921465088),
            "gnn_fwd": ("paper_2303_07030_gb300/csrc/k_gnn.cu",
                        "dd3221af39633b7b53b0c1a2bd68e53ef5b27e88", 5900874496 + 521272832),
            "gnn_empty": ("paper_2303_07030_gb300/csrc/k_gnn.cu",
                          "dd3221af39633b7b53b0c1a2bd68e53ef5b27e88", 602373888 + 490958592),
            "proj_bwd": ("paper_2303_07030_gb300/csrc/k_dense.cu",
                         "b83192d0b63745197114a081c7ba70ebb98cbf5d", 3229915904 + 2096727040),
            "proj_fwd": ("paper_2303_07030_gb300/csrc/k_dense.cu",
                         "b83192d0b63745197114a081c7ba70ebb98cbf5d", 2150839552 + 1033744128),
        },
        "capture": "ncu 1-pass dram bytes of the full workload (one launch per kernel)",
    },
    "logreg": {
        # the full workload (49,997,656 keys); ranked columns, 2^15-row blocked twin
        "layout": {"ranked": True, "blocked": 15, "split": False},
        "nnz": 49997656,
        "bytes_per_launch": {
            "logreg_row": ("paper_2303_07030_gb300/csrc/k_scalar.cu",
                           "27511a24b3fadccf241b92a0236303fc2a5a640e", 416612352 + 8102912),
            "scalar_bcol": ("paper_2303_07030_gb300/csrc/k_scalar.cu",
                            "27511a24b3fadccf241b92a0236303fc2a5a640e", 416723200 + 9714944),
        },
        "capture": "ncu 1-pass dram bytes of the full workload (one launch per kernel)",
    },
}


def _sha1(rel):
    import hashlib
    try:
        with open(os.path.join(ROOT, rel), "rb") as f:
            return hashlib.sha1(f.read()).hexdigest()
    except OSError:
        return None


def measured_traffic(cfg, kernel, nnz, layout=None):
    """DRAM bytes per launch of `kernel` from an ncu capture of this very workload
    (same key count and layout), or (None, None) when none was taken or the
    kernel's source has changed since (SHA-1 of the file)."""
    ent = NCU_TRAFFIC.get(cfg)
    if ent is None or (ent.get("layout") is not None and layout != ent["layout"]):
        return None, None
    got = ent["bytes_per_launch"].get(kernel)
    if ent.get("nnz") != nnz or got is None or _sha1(got[0]) != got[1]:
        return None, None
    return int(got[2]), ent["capture"]


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                 "--format=csv,noheader,nounits", "-lms", "200", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        out = {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        if not self.proc:
            return out
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        try:
            rows = [l.split(",") for l in open(self.path).read().strip().splitlines() if l.strip()]
            os.unlink(self.path)
        except Exception:
            return out
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except Exception:
                continue
            for nm, v in zip(names, r[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if sm:
            out = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                   "reasons": sorted(reasons), "samples": len(sm)}
        return out


# ----------------------------------------------------------------------------
# oracle timing (CPU baseline and the reference arm)
# ----------------------------------------------------------------------------

def row_sample(p, max_rows):
    """The first rows of a matrix problem (a bounded sample of the workload)."""
    from paper_2303_07030_gb300 import workloads as W
    r = min(p.m, max_rows)
    k = int(np.searchsorted(p.row, r))
    dense = dict(p.dense)
    for key in ("y", "Z", "U"):
        if key in dense:
            dense[key] = dense[key][:r]
    return W.SparseMatrixProblem(p.name, r, p.n, p.row[:k], p.col[:k], p.val[:k], dense,
                                 p.params), k


def oracle_call(cfg, p):
    import oracle
    d = p.dense
    if cfg == "lsq":
        return oracle.lsq(p.m, p.n, p.row, p.col, p.val, d["x"], d["y"])
    if cfg == "logreg":
        return oracle.logreg(p.m, p.n, p.row, p.col, p.val, d["w"], d["y"])
    if cfg == "mf":
        return oracle.mf(p.m, p.n, p.row, p.col, p.val, d["U"], d["V"], p.params["lam"])
    if cfg == "cp3":
        return oracle.cp3(p.dims, p.i, p.j, p.k, p.val, d["A"], d["B"], d["C"])
    if cfg == "smvm":
        return oracle.smvm(p.m, p.n, p.row, p.col, p.val, d["X"])
    if cfg == "smmm":
        return oracle.smmm(p.m, p.n, p.n, (p.row, p.col, p.val), p.params["B"])
    if cfg == "batax":
        return oracle.batax(p.m, p.n, p.row, p.col, p.val, d["X"], p.params["beta"])
    return oracle.gnn(p.m, p.n, p.row, p.col, p.val, d["H"], d["W"], d["Z"])


def step_keys(cfg, p):
    """Keys one step processes (the metric's unit): A's, plus B's for SMMM."""
    return p.nnz + (int(p.params["B"][0].size) if cfg == "smmm" else 0)


def oracle_sample(cfg, p, target_s):
    """Picks a bounded sample whose oracle call takes about target_s seconds."""
    if cfg == "cp3":
        from paper_2303_07030_gb300 import workloads as W
        k = min(p.nnz, 2_000_000)
        q = W.SparseTensor3Problem(p.name, p.dims, p.i[:k], p.j[:k], p.k[:k], p.val[:k],
                                   p.dense, p.params)
        return q, k, "first %d of %d entries" % (k, p.nnz)
    if cfg == "lsq":
        return p, p.nnz, "whole workload"
    rows = max(1, p.m // 200)
    q, k = row_sample(p, rows)
    t0 = time.perf_counter()
    oracle_call(cfg, q)
    dt = max(time.perf_counter() - t0, 1e-3)
    rows = int(min(p.m, rows * max(1.0, target_s / dt)))
    q, k = row_sample(p, rows)
    if cfg == "smmm":   # B whole
        nb = int(p.params["B"][0].size)
        return q, k + nb, "first %d of %d rows of A (%d of %d keys) and all %d keys of B" % (
            q.m, p.m, k, p.nnz, nb)
    return q, k, "first %d of %d rows (%d of %d keys)" % (q.m, p.m, k, p.nnz)


def busy_cores(cpu_s, wall_s):
    """Cores the process kept busy on average (its CPU time over the wall time,
    every thread counted: a threaded BLAS under the oracle's matrix products shows
    up here)."""
    return max(1.0, round(cpu_s / max(wall_s, 1e-9), 1))


def cpu_baseline(cfg, p, budget_s=15.0):
    import oracle  # noqa: F401  (builds the oracle library on first use)
    q, k, desc = oracle_sample(cfg, p, target_s=budget_s / 3)
    n, t, c = 0, 0.0, 0.0
    while t < budget_s and n < 50:
        t0, c0 = time.perf_counter(), time.process_time()
        oracle_call(cfg, q)
        t += time.perf_counter() - t0
        c += time.process_time() - c0
        n += 1
    cores = busy_cores(c, t)
    return {"value": k * n / t, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": desc + ", %d calls in %.1f s, fp64 oracle (%.1f s CPU time)" % (n, t, c)}


# ----------------------------------------------------------------------------

def transpose_name(blocked, split):
    if not blocked:
        return "CSC"
    if split is None:
        return "row-blocked CSC, 2^%d rows per block" % blocked
    return ("split: %d columns (%d keys) row-blocked, 2^%d rows per block; the rest CSC"
            % (split[0], split[1], blocked))


def make_run(cfg, p, tmode, ranked, blocked=0, block_cols=None):
    from paper_2303_07030_gb300 import runner as R
    from paper_2303_07030_gb300 import sdad as S
    tm = {"auto": S.SDAD_T_AUTO, "csc": S.SDAD_T_CSC, "atomic": S.SDAD_T_ATOMIC}[tmode]
    if cfg == "lsq":
        return R.LsqRun(p, tmode=tm, ranked=ranked, blocked=blocked, block_cols=block_cols)
    if cfg == "logreg":
        return R.LogregRun(p, tmode=tm, ranked=ranked, blocked=blocked, block_cols=block_cols)
    if cfg == "mf":   # ranked columns: the atomic scatter sums the hot ones in shared memory
        return R.MfRun(p, tmode=tm, ranked=True)
    if cfg == "cp3":
        return R.Cp3Run(p, tmode=tm)
    if cfg in ("smvm", "smmm", "batax"):
        return R.RUNS[cfg](p)
    return R.GnnRun(p)


def host_inputs(run, cfg):
    """(device tensor, pinned host copy) pairs of every input a step reads."""
    return [(t, t.cpu().pin_memory()) for t in run.step_inputs()]


def host_outputs(run, cfg):
    outs = {"lsq": ("loss", "dx", "dA"), "logreg": ("loss", "dw"), "mf": ("loss", "dU", "dV"),
            "cp3": ("loss", "dA", "dB", "dC"), "gnn": ("loss", "dA", "dH", "dW"),
            "smvm": ("f", "dX"), "smmm": ("f", "dB"), "batax": ("f", "J")}[cfg]
    pairs = []
    for name in outs:
        t = getattr(run, name, None)
        if cfg == "cp3" and name in ("dA", "dB", "dC"):
            t = getattr(run, name)
        if t is not None:
            pairs.append((t, torch_empty_pinned_like(t)))
    return pairs


def torch_empty_pinned_like(t):
    import torch
    return torch.empty(t.shape, dtype=t.dtype, pin_memory=True)


def fp32_fma_peak(S, torch, stream):
    """FP32 FMA rate of this GPU (TFLOP/s): best of five probe launches."""
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    blocks, iters = sms * 8, 8192
    out = torch.empty(blocks * 256, dtype=torch.float32, device="cuda")
    S.sdad_probe_fma(out, blocks, iters, stream)   # warm-up
    best = None
    for _ in range(5):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fl = S.sdad_probe_fma(out, blocks, iters, stream)
        b.record(stream)
        torch.cuda.synchronize()
        t = a.elapsed_time(b) * 1e-3
        best = t if best is None else min(best, t)
    return {"tflops": round(fl / best / 1e12, 2), "how": "%d CTAs x 256 threads, 16 independent "
            "FMA chains of %d steps per thread, best of 5 (CUDA events)" % (blocks, iters)}


def layout_for(cfg, p, args, S):
    """(ranked, blocked, block_cols, split, transpose) of a workload's matrix."""
    ranked = cfg in ("lsq", "logreg") and (
        args.columns == "ranked" or (args.columns == "auto" and cfg == "logreg"))
    blocked, block_cols, split = 0, None, None
    transpose = args.transpose
    if transpose == "auto":
        transpose = "blocked" if cfg == "logreg" else "csc"
    if cfg in ("lsq", "logreg") and transpose in ("blocked", "split"):
        # at most one block on small matrices
        blocked = min(args.block_log2, max(4, (p.m - 1).bit_length()))
        if transpose == "split":
            block_cols = S.split_columns(p.col, p.n, p.m, blocked, args.block_min)
            split = (int(block_cols.size), int(np.isin(p.col, block_cols).sum()))
    return ranked, blocked, block_cols, split, transpose


def jvp_closure(cfg, run, torch):
    """One forward-mode call of the workload's loss along a seeded tangent of every
    dense operand and of the sparse values (None for the paper's matrix kernels)."""
    from paper_2303_07030_gb300 import sdad as S
    g = torch.Generator(device="cuda")
    g.manual_seed(20230313)

    def like(t):
        return torch.randn(t.shape, generator=g, device=t.device, dtype=t.dtype)

    def vals(n):
        return torch.randn(int(n), generator=g, device="cuda", dtype=torch.float32)

    lt = torch.zeros(1, dtype=torch.float64, device="cuda")
    if cfg == "lsq":
        xt, at = like(run.x), vals(run.A.nnz)
        return lambda: S.sdad_lsq_jvp(run.desc, run.x, run.y, run.loss, lt, xt, at, run.ws)
    if cfg == "logreg":
        wt, at = like(run.w), vals(run.X.nnz)
        return lambda: S.sdad_logreg_jvp(run.desc, run.w, run.y, run.loss, lt, wt, at, run.ws)
    if cfg == "mf":
        ut, vt, rt = like(run.U), like(run.V), vals(run.R.nnz)
        return lambda: S.sdad_mf_jvp(run.desc, run.U, run.V, run.k, run.lam, run.loss, lt, rt,
                                     ut, vt, run.ws)
    if cfg == "cp3":
        at, bt, ct, tt = like(run.A), like(run.B), like(run.C), vals(run.p.nnz)
        return lambda: S.sdad_cp3_jvp(run.desc, run.A, run.B, run.C, run.R, run.loss, lt, tt,
                                      at, bt, ct, run.ws)
    if cfg == "gnn":
        ht, wt, at = like(run.H), like(run.W), vals(run.A.nnz)
        return lambda: S.sdad_gnn_jvp(run.desc, run.H, run.W, run.Z, run.f_in, run.f_out,
                                      run.loss, lt, at, ht, wt, run.ws)
    return None


def time_jvp(cfg, run, nnz, steps, torch, S):
    """Forward mode (Sec. 4.2): ms per call and keys per second over `steps` calls
    after three warm-up calls, with the per-kernel times of a bracketed pass."""
    fn = jvp_closure(cfg, run, torch)
    if fn is None:
        return None
    for _ in range(3):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    S.sdad_timing_reset()
    S.sdad_timing_enable(True)
    for _ in range(steps):
        fn()
    torch.cuda.synchronize()
    S.sdad_timing_enable(False)
    per = {}
    for k, t in S.sdad_timing_records():
        per.setdefault(k, []).append(t)
    run.check()
    return {"ms_per_call": round(ms, 5), "value": nnz / (ms * 1e-3), "unit": UNIT,
            "tangent": "every dense operand and the sparse values",
            "kernels": {k: round(sum(v) / len(v), 5) for k, v in per.items()}}


def measure(cfg, args, ov, dist, world, local, headline, fma):
    """One workload: timed steps, per-kernel times, rooflines; e2e for the headline."""
    import torch
    from paper_2303_07030_gb300 import sdad as S
    from paper_2303_07030_gb300 import workloads as W

    p = W.make(cfg, "full", **ov)
    ranked, blocked, block_cols, split, transpose = layout_for(cfg, p, args, S)
    tmode = args.tmode if headline else "auto"
    run = make_run(cfg, p, tmode, ranked, blocked, block_cols)
    if cfg == "batax":
        p.params["jnnz"] = run.jnnz
    nnz = step_keys(cfg, p)
    stream = torch.cuda.current_stream()
    flush = None
    if cfg in SMALL_CONFIGS:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(max(args.warmup, 0)):
        run.step()
    torch.cuda.synchronize()
    run.check()

    # ---------------- timed region (inputs resident in HBM) ----------------
    clk = ClockSampler(local)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    clk.start()
    time.sleep(0.3)
    for i in range(args.steps):
        if flush is not None:
            flush.fill_(i & 0xff)
        starts[i].record(stream)
        run.step()
        ends[i].record(stream)
    torch.cuda.synchronize()
    barrier()
    clocks = clk.stop()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    run.check()

    # ---------------- per-kernel durations ----------------------------------
    # the same K steps again with every library kernel bracketed by CUDA events
    # on its launch stream; the brackets add a few microseconds per launch, so
    # the step time above is taken without them
    S.sdad_timing_reset()
    S.sdad_timing_enable(True)
    k0 = torch.cuda.Event(enable_timing=True)
    k1 = torch.cuda.Event(enable_timing=True)
    k0.record(stream)
    for i in range(args.steps):
        if flush is not None:
            flush.fill_(i & 0xff)
        run.step()
    k1.record(stream)
    torch.cuda.synchronize()
    S.sdad_timing_enable(False)
    recs = S.sdad_timing_records()
    bracketed_ms = k0.elapsed_time(k1) / max(args.steps, 1)
    run.check()
    ms = sum(step_ms) / len(step_ms)
    if dist is not None:
        t = torch.tensor([ms], device="cuda", dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    value = world * nnz / (ms * 1e-3)

    # per-kernel roofline
    per = {}
    for name, kms in recs:
        a = per.setdefault(name, [0, 0.0])
        a[0] += 1
        a[1] += kms
    csc = getattr(run, "csc", tmode != "atomic")
    kb = kernel_bytes(cfg, p, nnz, csc, False, ranked, blocked, split)
    kf = kernel_flops(cfg, p, nnz)
    dom = max((k for k in per if k in kb), key=lambda k: per[k][1], default=None)
    hbm, src = peaks()
    roofline = None
    if dom is not None:
        avg_ms = per[dom][1] / per[dom][0]
        ach = kb[dom] / (avg_ms * 1e-3) / 1e9
        layout = {"ranked": ranked, "blocked": blocked, "split": split is not None}
        traffic, tsrc = measured_traffic(cfg, dom, nnz, layout)
        roofline = {"bound": "hbm", "kernel": dom, "achieved": round(ach, 1), "peak": hbm,
                    "peak_source": src, "unit": "GB/s", "frac": round(ach / hbm, 4),
                    "traffic": traffic, "traffic_source": tsrc,
                    "algorithmic_bytes": kb[dom], "avg_launch_ms": round(avg_ms, 5)}
    tot_ms = max(sum(x[1] for x in per.values()), 1e-12)
    kernels = {}
    for k, v in per.items():
        e = {"launches": v[0], "ms_per_launch": round(v[1] / v[0], 5),
             "share": round(v[1] / tot_ms, 4)}
        if k in kb:
            gbs = kb[k] / (v[1] / v[0] * 1e-3) / 1e9
            e["hbm_frac"] = round(gbs / hbm, 4)
        if k in kf and fma:
            tf = kf[k] / (v[1] / v[0] * 1e-3) / 1e12
            e["fp32_tflops"] = round(tf, 2)
            e["fp32_frac"] = round(tf / fma["tflops"], 4)
        kernels[k] = e

    # ---------------- end to end: host buffers, copies inside the timing ----
    # Every step copies its inputs in from pinned host memory, runs, and copies
    # its loss and gradients back.  Two buffer sets and three streams: while
    # step s computes, step s + 1's inputs copy in and step s - 1's outputs copy
    # out (the host link carries both directions at once).  The serial figure
    # (one stream: in, step, out) is reported beside it.
    e2e = None
    if headline and not args.no_e2e:
        ins = host_inputs(run, cfg)
        host_in = [h for _, h in ins]
        run2 = make_run(cfg, p, tmode, ranked, blocked, block_cols)
        runs = [run, run2]
        dev_in = [[d for d, _ in ins], list(run2.step_inputs())]
        outs = [host_outputs(r, cfg) for r in runs]
        h2d = sum(h.numel() * h.element_size() for h in host_in)
        d2h = sum(h.numel() * h.element_size() for _, h in outs[0])
        # serial: one stream
        for _ in range(2):
            for d, h in ins:
                d.copy_(h, non_blocking=True)
            run.step()
            for d, h in outs[0]:
                h.copy_(d, non_blocking=True)
        torch.cuda.synchronize()
        barrier()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            for d, h in ins:
                d.copy_(h, non_blocking=True)
            run.step()
            for d, h in outs[0]:
                h.copy_(d, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        serial_ms = e0.elapsed_time(e1) / args.steps
        # double-buffered
        s_in, s_cmp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        ev_in = [torch.cuda.Event() for _ in runs]
        ev_cmp = [torch.cuda.Event() for _ in runs]
        ev_out = [torch.cuda.Event() for _ in runs]

        def pipelined(first, count):
            for st in range(first, first + count):
                b = st % 2
                if st >= 2:   # step st - 2 has read this set's inputs
                    s_in.wait_event(ev_cmp[b])
                with torch.cuda.stream(s_in):
                    for d, h in zip(dev_in[b], host_in):
                        d.copy_(h, non_blocking=True)
                ev_in[b].record(s_in)
                s_cmp.wait_event(ev_in[b])
                if st >= 2:   # ... and its outputs are copied out
                    s_cmp.wait_event(ev_out[b])
                runs[b].step(s_cmp)
                ev_cmp[b].record(s_cmp)
                s_out.wait_event(ev_cmp[b])
                with torch.cuda.stream(s_out):
                    for d, h in outs[b]:
                        h.copy_(d, non_blocking=True)
                ev_out[b].record(s_out)

        pipelined(0, 2)
        torch.cuda.synchronize()
        barrier()
        e0.record(s_in)
        pipelined(2, args.steps)
        e1.record(s_out)   # after the last copy out, which waits for everything before it
        torch.cuda.synchronize()
        for r in runs:
            r.check()
        ems = e0.elapsed_time(e1) / args.steps
        if dist is not None:
            t = torch.tensor([ems, serial_ms], device="cuda", dtype=torch.float64)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            ems, serial_ms = float(t[0].item()), float(t[1].item())
        e2e = {"value": world * nnz / (ems * 1e-3), "unit": UNIT, "ms_per_step": round(ems, 4),
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "mode": "double-buffered: inputs of step s+1 copy in and outputs of step s-1 copy out "
                       "while step s runs",
               "serial_ms_per_step": round(serial_ms, 4)}
        del ins, outs, run2, runs, dev_in, host_in
    jvp = None if args.no_jvp else time_jvp(cfg, run, nnz, min(args.steps, 10), torch, S)
    tot = sum(kb.get(k, 0) * v[0] for k, v in per.items()) / max(args.steps, 1)
    res = {
        "value": value, "ms_per_step": round(ms, 5),
        "config": {"workload": WORKLOAD_NAMES[cfg] + (" (overridden: %s)" % ov if ov else ""),
                   "name": cfg, "nnz": nnz, "tmode": tmode,
                   "columns": ("ranked by key count" if ranked else "as generated")
                   if cfg in ("lsq", "logreg") else None,
                   "transpose": transpose_name(blocked, split)
                   if cfg in ("lsq", "logreg") else None,
                   "l2": ("L2 flushed (256 MB write) between timed steps" if flush is not None
                          else "inputs larger than L2 (no flush)"),
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": roofline, "kernels": kernels,
        "ms_per_step_kernels_bracketed": round(bracketed_ms, 5),
        "gpu_launches": int(len(recs)), "launches_per_step": len(recs) / max(args.steps, 1),
        "hbm_gbs_step": round(tot / (ms * 1e-3) / 1e9, 1), "clocks": clocks, "e2e": e2e,
        "jvp": jvp,
    }
    del run, flush
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return p, res


SWEEP = [
    # (workload, generator overrides, what varies)
    ("lsq", dict(m=1 << 20, n=1 << 20, draws=1 << 20), "density"),
    ("lsq", dict(m=1 << 20, n=1 << 20, draws=1 << 22), "density"),
    ("lsq", dict(m=1 << 20, n=1 << 20, draws=1 << 24), "density"),
    ("lsq", dict(m=1 << 20, n=1 << 20, draws=1 << 26), "density"),
    ("lsq", dict(m=1 << 16, n=1 << 16, draws=1 << 20), "dimension"),
    ("lsq", dict(m=1 << 18, n=1 << 18, draws=1 << 22), "dimension"),
    ("lsq", dict(m=1 << 22, n=1 << 22, draws=1 << 26), "dimension"),
    ("logreg", dict(mean_row=10.0), "density"),
    ("logreg", dict(mean_row=25.0), "density"),
    ("logreg", dict(mean_row=100.0), "density"),
    ("gnn", dict(scale=16, n_edges=1 << 20), "dimension"),
    ("gnn", dict(scale=18, n_edges=1 << 22), "dimension"),
    ("gnn", dict(scale=20, n_edges=1 << 24), "dimension"),
]


def run_sweep(args):
    """Density and dimension sweep of the library's own passes (no comparison system)."""
    import torch
    from paper_2303_07030_gb300 import build as B
    from paper_2303_07030_gb300 import sdad as S
    from paper_2303_07030_gb300 import workloads as W
    B.build()
    hbm, src = peaks()
    stream = torch.cuda.current_stream()
    points = []
    for cfg, ov, what in SWEEP:
        p = W.make(cfg, "full", **ov)
        ranked, blocked, block_cols, split, transpose = layout_for(cfg, p, args, S)
        run = make_run(cfg, p, "auto", ranked, blocked, block_cols)
        for _ in range(3):
            run.step()
        torch.cuda.synchronize()
        run.check()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(10):
            run.step()
        b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / 10
        S.sdad_timing_reset()
        S.sdad_timing_enable(True)
        for _ in range(5):
            run.step()
        torch.cuda.synchronize()
        S.sdad_timing_enable(False)
        run.check()
        per = {}
        for name, kms in S.sdad_timing_records():
            per.setdefault(name, []).append(kms)
        csc = getattr(run, "csc", True)
        kb = kernel_bytes(cfg, p, p.nnz, csc, False, ranked, blocked, split)
        tot = sum(kb.get(k, 0) * len(v) for k, v in per.items()) / 5
        dom = max((k for k in per if k in kb), key=lambda k: sum(per[k]), default=None)
        pt = {"workload": cfg, "varies": what, "params": ov, "m": p.m, "n": p.n, "nnz": p.nnz,
              "density": p.nnz / (float(p.m) * p.n), "ms_per_step": round(ms, 5),
              "value": p.nnz / (ms * 1e-3), "hbm_gbs_step": round(tot / (ms * 1e-3) / 1e9, 1)}
        if dom is not None:
            dms = sum(per[dom]) / len(per[dom])
            pt["dominant"] = {"kernel": dom, "ms": round(dms, 5),
                              "frac": round(kb[dom] / (dms * 1e-3) / 1e9 / hbm, 4)}
        points.append(pt)
        print(json.dumps(pt), file=sys.stderr, flush=True)
        del run
        torch.cuda.empty_cache()
    print(json.dumps({"metric": METRIC, "unit": UNIT, "sweep": points, "peak_gbs": hbm,
                      "peak_source": src, "data": "synthetic (seeded generators)"}), flush=True)
    return 0


def main():
    args = parse()
    if args.sweep and args.impl == "ours":
        return run_sweep(args)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return 0
        return run_reference(args)

    import torch
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2303_07030_gb300 import build as B
    from paper_2303_07030_gb300 import sdad as S
    B.build()

    stream = torch.cuda.current_stream()
    fma = fp32_fma_peak(S, torch, stream)
    cfg = args.config
    ov = overrides(args)
    p, head = measure(cfg, args, ov, dist, world, local, True, fma)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, p)
    del p
    others = {}
    if args.others == "all":
        for c in ALL_CONFIGS:
            if c == cfg:
                continue
            q, r = measure(c, args, {}, dist, world, local, False, fma)
            del q
            others[c] = {k: r[k] for k in ("value", "ms_per_step", "roofline", "kernels",
                                           "gpu_launches", "hbm_gbs_step", "clocks", "jvp")}
            others[c]["workload"] = r["config"]["workload"]
            others[c]["nnz"] = r["config"]["nnz"]
            if r["config"]["transpose"]:
                others[c]["transpose"] = r["config"]["transpose"]
                others[c]["columns"] = r["config"]["columns"]

    if rank == 0:
        line = {
            "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded generators; no external dataset)",
            "config": head["config"], "roofline": head["roofline"], "kernels": head["kernels"],
            "ms_per_step_kernels_bracketed": head["ms_per_step_kernels_bracketed"],
            "gpu_launches": head["gpu_launches"],
            "gpu_launches_all_configs": head["gpu_launches"] + sum(
                o["gpu_launches"] for o in others.values()),
            "launches_per_step": head["launches_per_step"],
            "hbm_gbs_step": head["hbm_gbs_step"], "clocks": head["clocks"], "e2e": head["e2e"],
            "cpu_baseline": cpu, "fp32_fma_peak": fma, "jvp": head["jvp"], "configs": others,
        }
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def run_reference(args):
    from paper_2303_07030_gb300 import workloads as W
    import oracle  # noqa: F401
    cfg = args.config
    p = W.make(cfg, "full", **overrides(args))
    q, k, desc = oracle_sample(cfg, p, target_s=2.0)
    for _ in range(max(args.warmup, 0)):
        oracle_call(cfg, q)
    t, c = [], 0.0
    for _ in range(args.steps):
        t0, c0 = time.perf_counter(), time.process_time()
        oracle_call(cfg, q)
        t.append(time.perf_counter() - t0)
        c += time.process_time() - c0
    sec = sum(t) / len(t)
    value = k / sec
    cores = busy_cores(c, sum(t))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(sec * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded generators; no external dataset)",
        "config": {"workload": WORKLOAD_NAMES[cfg], "name": cfg, "nnz": p.nnz, "sample": desc},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": desc + ", fp64 oracle (%.1f s CPU time over %.1f s)" % (c, sum(t))},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
