"""SMT-LIB queries from exported term lists (Sec. 3.4 "Solving"): evaluated
at concrete inputs with the uninterpreted functions given their meaning, each
query's two roots equal the oracle's fp64 value of res(y[l]) in the
reference and in the candidate."""
import math

import numpy as np
import pytest

import oracle
from paper_2609_19611_gb300 import smt
from paper_2609_19611_gb300 import workloads as W

from .smtlib_eval import evaluate

FUNCS = {
    "exp": math.exp, "tanh": math.tanh, "erf": math.erf, "log": math.log,
    "sqrt": math.sqrt, "rsqrt": lambda x: 1.0 / math.sqrt(x), "recip": lambda x: 1.0 / x,
    "gelu": lambda x: 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0))),
    "gelu_tanh": lambda x: 0.5 * x * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) *
                                                      (x + 0.044715 * x ** 3))),
}


def _case(ref, cand, values, budget):
    R, C = oracle.Program(ref), oracle.Program(cand)
    locs = np.arange(R.out_numel, dtype=np.int64)
    v, f, blob, need = oracle.compare(R, C, locs, R.keys(locs), C.keys(locs), budget=budget,
                                      capacity=1 << 28)
    assert blob is not None
    flat = np.concatenate([np.asarray(x, dtype=np.float64).ravel() for x in values])
    G = flat.size
    queries = smt.export_queries(blob, G=G)
    assert len(queries) == min(budget, int((v != 0).sum()))
    want_r = R.eval([np.asarray(x, np.float64) for x in values], locs)
    want_c = C.eval([np.asarray(x, np.float64) for x in values], locs)
    for slot, q in queries:
        assert q.count("(") == q.count(")")
        # bottom (a read outside a tensor) evaluates to NaN on both sides
        a, b = evaluate(q, lambda g: float(flat[g]), FUNCS)
        for got, want in ((a, want_r[slot]), (b, want_c[slot])):
            assert (math.isnan(got) and math.isnan(want)) or \
                math.isclose(got, want, rel_tol=1e-9, abs_tol=1e-9), (slot, got, want)
    return queries


def test_worked_example_queries():
    ref, cand = W.halfsum_gelu(N=2, C=3, H=4, W=2)
    qs = _case(ref, cand, W.random_values(ref, 3, np.float64), budget=8)
    assert all("(declare-fun gelu (Real) Real)" in q for _, q in qs)


@pytest.mark.parametrize("c,shape", [
    (2, dict(N=1, Ci=2, H=6, W=6, Co=3)),
    (4, dict(N=1, Ci=2, H=6, W=6, Co=4, bug_co=2)),
    (5, dict(B=2, M=5, K=12, N=3, tile=4, k_stop=10)),
])
def test_config_queries(c, shape):
    ref, cand = W.config(c, **shape)
    _case(ref, cand, W.make_values(c, ref), budget=6)


def test_random_pair_queries():
    """Every random program pair of the GPU parity set that has undischarged
    locations (most of them) gives correct queries."""
    tested = 0
    for seed in range(40):
        ref, cand, _ = W.random_pair(1000 + seed)
        R, C = oracle.Program(ref), oracle.Program(cand)
        locs = np.arange(R.out_numel, dtype=np.int64)
        if (R.keys(locs) == C.keys(locs)).all():
            continue
        _case(ref, cand, W.random_values(ref, seed, np.float64), budget=4)
        tested += 1
    assert tested >= 5


def test_constants_are_exact():
    assert smt._num(0.5) == "(/ 1.0 2.0)"
    assert smt._num(-3.0) == "(- 3.0)"
    assert smt._num(1e-5).startswith("(/ ")
