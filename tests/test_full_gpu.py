"""Full-size workloads, in the launch configuration the benchmark times,
against the fp64 oracle computed in full (every output element)."""

import numpy as np
import pytest
import torch

from paper_2303_07030_gb300 import build as B
from paper_2303_07030_gb300 import runner as R
from paper_2303_07030_gb300 import sdad as S
from paper_2303_07030_gb300 import workloads as W
from tests.parity import COMPARED, assert_close, oracle_for

pytestmark = [pytest.mark.gpu, pytest.mark.full]


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    assert torch.cuda.is_available()


_cache = {}


def _problem_and_oracle(name):
    if name not in _cache:
        _cache.clear()                      # one full problem held at a time
        p = W.make(name, "full")
        _cache[name] = (p, oracle_for(name, p))
    return _cache[name]


# the logistic cases: the layout the benchmark times (ranked columns and a
# row-blocked CSC twin of every column with 2^15-row blocks: 31 blocks), the
# ranked columns with the plain CSC twin, the split column pass (blocked
# columns with >= 32 keys per 2^15-row block), the atomic transposed product,
# and the columns as generated; MF with its two passes (SDAD_T_CSC) and with
# the one-pass atomic scatter over ranked columns; CP with its one-pass atomic
# scatter (AUTO) and with the sorted per-mode passes (SDAD_T_CSC)
@pytest.mark.parametrize("name,kw", [
    ("logreg", {"ranked": True, "blocked": 15}),
    ("logreg", {"ranked": True}),
    ("logreg", {"ranked": True, "split": (15, 32.0)}),
    ("logreg", {"ranked": True, "tmode": 2}),
    ("logreg", {}),
    ("mf", {"tmode": 1}), ("mf", {"tmode": 2, "ranked": True}),
    ("cp3", {}), ("cp3", {"tmode": 1}),
    ("gnn", {}),
])
def test_full_size_parity(name, kw):
    p, ref = _problem_and_oracle(name)
    kw = dict(kw)
    if "split" in kw:
        lg, per_block = kw.pop("split")
        kw.update(blocked=lg, block_cols=S.split_columns(p.col, p.n, p.m, lg, per_block))
    r = R.RUNS[name](p, **kw)
    r.step()
    torch.cuda.synchronize()
    r.check()
    out = r.outputs()
    del r
    torch.cuda.empty_cache()
    errs = assert_close(out, ref, COMPARED[name])
    print(name, kw, "nnz", p.nnz, "errors", {k: float("%.3g" % v) for k, v in errs.items()})
