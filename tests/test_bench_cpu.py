"""Host logic of bench.py, on the CPU: the algorithmic-byte formulas, the
names and overrides it reports, and the reference arm (the fp64 oracle on
the host cores) end to end on the small least-squares workload."""

import json
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_2303_07030_gb300 import workloads as W  # noqa: E402


def test_kernel_bytes_per_config():
    p = W.make("logreg", "small")
    # the default logistic layout: row pass + blocked column pass
    b = bench.kernel_bytes("logreg", p, p.nnz, True, False, ranked=True, blocked=9)
    assert set(b) >= {"logreg_row", "scalar_bcol", "bcol_combine", "rank_prep"}
    assert b["scalar_bcol"] == 8 * p.nnz + 4 * p.m
    assert b["logreg_row"] == 8 * p.nnz + 4 * (p.m + 1) + 4 * p.m + 4 * p.n + 4 * p.m
    # the plain CSC column pass and the split layout
    assert "scalar_col" in bench.kernel_bytes("logreg", p, p.nnz, True, False)
    s = bench.kernel_bytes("logreg", p, p.nnz, True, False, ranked=False, blocked=9,
                           split=(10, p.nnz // 2))
    assert s["scalar_col"] == 8 * (p.nnz - p.nnz // 2) + 4 * (p.n + 1) + 4 * p.m + 4 * p.n
    for cfg in ("smvm", "smmm", "batax"):
        q = W.make(cfg, "small", matrix="bcspwr10")
        q.params["jnnz"] = 1000
        kb = bench.kernel_bytes(cfg, q, bench.step_keys(cfg, q), True, False)
        assert kb and all(v > 0 for v in kb.values())
    q = W.make("smmm", "small", matrix="bcspwr10")
    assert bench.step_keys("smmm", q) == q.nnz + q.params["B"][0].size


def test_graph_bytes_count_rows_with_keys():
    # 4 vertices, keys (0,1), (0,2), (2,1): rows 0 and 2 and columns 1 and 2 hold keys
    row = np.array([0, 0, 2], dtype=np.int32)
    col = np.array([1, 2, 1], dtype=np.int32)
    q = W.SparseMatrixProblem("gnn", 4, 4, row, col, np.ones(3, np.float32), {}, {})
    b = bench.kernel_bytes("gnn", q, 3, True, False)
    r = 256
    assert b["gnn_fwd"] == 8 * 3 + 4 * 5 + r * 2 + 2 * r * 2
    assert b["gnn_col"] == 16 * 3 + 4 * 5 + r * 2 + 2 * r * 2
    assert b["gnn_empty"] == 4 * 5 * 2 + r * 2 + r * 2


def test_names_and_overrides():
    assert bench.transpose_name(0, None) == "CSC"
    assert "2^15" in bench.transpose_name(15, None)
    assert "12 columns" in bench.transpose_name(15, (12, 3400))

    class A:
        override = ["m=400000", "matrix=pdb1HYS", "beta=0.5"]
    assert bench.overrides(A) == {"m": 400000, "matrix": "pdb1HYS", "beta": 0.5}


def test_row_sample_keeps_whole_rows():
    p = W.make("logreg", "small")
    q, k = bench.row_sample(p, 100)
    assert q.m == 100 and k == int(np.searchsorted(p.row, 100))
    assert q.dense["y"].size == 100 and q.dense["w"].size == p.n


@pytest.mark.timeout(300)
def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--config", "lsq", "--steps", "2", "--warmup", "1"],
                       capture_output=True, text=True, timeout=280, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["steps"] == 2 and d["warmup"] == 1
    assert d["cpu_baseline"]["cores"] >= 1.0


def test_busy_cores_is_cpu_time_over_wall_time():
    assert bench.busy_cores(10.0, 10.0) == 1.0
    assert bench.busy_cores(35.0, 10.0) == 3.5
    assert bench.busy_cores(0.2, 10.0) == 1.0   # a mostly idle single thread still counts as one


def test_flops_and_traffic_tables():
    p = W.make("mf", "small")
    f = bench.kernel_flops("mf", p, p.nnz)
    assert f["mf_row"] == 256 * p.nnz and f["mf_atomic"] == 384 * p.nnz
    c = W.make("cp3", "small")
    assert bench.kernel_flops("cp3", c, c.nnz)["cp_atomic"] == 384 * c.nnz
    # a figure is given only for the layout it was captured on
    ent = bench.NCU_TRAFFIC["logreg"]
    lay = dict(ent["layout"])
    t, src = bench.measured_traffic("logreg", "logreg_row", ent["nnz"], lay)
    assert (t is None) == (src is None)
    if t is not None:   # the source file is the one captured
        assert t == ent["bytes_per_launch"]["logreg_row"][2]
    # only for the workload it was captured on
    assert bench.measured_traffic("logreg", "logreg_row", 1000, lay) == (None, None)
    lay["blocked"] = 0
    assert bench.measured_traffic("logreg", "logreg_row", ent["nnz"], lay) == (None, None)
    assert bench.measured_traffic("lsq", "lsq_row", 1000, None) == (None, None)
    g = bench.NCU_TRAFFIC["gnn"]
    assert bench.measured_traffic("gnn", "gnn_col", g["nnz"] + 1, None) == (None, None)


def test_default_headline_is_the_largest_workload():
    sizes = {"gnn": 1 << 26, "logreg": 49_997_656, "mf": 50_000_000, "cp3": 10_000_000}
    assert max(sizes, key=sizes.get) == "gnn"
    sys_argv = sys.argv
    try:
        sys.argv = ["bench.py"]
        a = bench.parse()
    finally:
        sys.argv = sys_argv
    assert a.config == "gnn" and a.others == "all"
    assert set(bench.ALL_CONFIGS) == set(bench.WORKLOAD_NAMES)


def test_sweep_covers_density_and_dimension():
    kinds = {(cfg, what) for cfg, _, what in bench.SWEEP}
    assert ("lsq", "density") in kinds and ("lsq", "dimension") in kinds
    assert ("logreg", "density") in kinds and ("gnn", "dimension") in kinds
    # every point is a valid generator call of its workload (sizes only checked here)
    for cfg, ov, _ in bench.SWEEP:
        assert cfg in bench.WORKLOAD_NAMES and isinstance(ov, dict) and ov
    d = [ov["draws"] for cfg, ov, w in bench.SWEEP if cfg == "lsq" and w == "density"]
    assert d == sorted(d) and len(set(d)) == len(d)
