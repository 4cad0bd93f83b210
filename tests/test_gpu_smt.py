"""SMT-LIB queries built from the GPU's export (Sec. 3.4 "Solving"): the term
lists dirigo_compare exports, in the benchmark's launch arrangement, turned
into queries by ``smt.export_queries`` and evaluated at concrete inputs with
the uninterpreted functions given their meaning.  Each query's two roots
equal the oracle's fp64 value of res(y[l]) in the reference and the candidate.
No SMT solver is installed in this image, so the queries are checked by
evaluation rather than solved."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_19611_gb300 import dirigo as D
from paper_2609_19611_gb300 import smt
from paper_2609_19611_gb300 import workloads as W
from paper_2609_19611_gb300.pipeline import BatchChecker

from .smtlib_eval import evaluate
from .test_smt_queries import FUNCS

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("c,shape,budget", [
    (2, dict(N=1, Ci=2, H=6, W=6, Co=3), 6),
    (4, dict(N=1, Ci=2, H=6, W=6, Co=4, bug_co=2), 6),
    (5, {}, 3),                                   # the full-size bmm pair
])
def test_queries_from_the_gpu_export(c, shape, budget):
    ref, cand = W.config(c, **shape)
    R, C = oracle.Program(ref), oracle.Program(cand)
    gr, gc = D.Graph(ref), D.Graph(cand)
    q = W.make_queries(c, R.out_numel) if not shape else np.arange(R.out_numel, dtype=np.int64)
    chk = BatchChecker(gr, gc, len(q), budget=budget)
    locs = torch.as_tensor(q, device="cuda")
    chk.prepare(locs)
    st, stats = chk.step(locs)
    assert st == D.OK and stats.n_exported == budget
    blob = chk.blob(stats).cpu().numpy().tobytes()
    values = W.make_values(c, ref)
    flat = np.concatenate([np.asarray(x, dtype=np.float64).ravel() for x in values])
    queries = smt.export_queries(blob, G=flat.size)
    assert len(queries) == budget
    v = chk.verdict[:len(q)].cpu().numpy()
    slots = [s for s, _ in queries]
    assert slots == np.nonzero(v == D.EXPORTED)[0].tolist()
    sl = q[slots]
    want_r = R.eval([np.asarray(x, np.float64) for x in values], sl)
    want_c = C.eval([np.asarray(x, np.float64) for x in values], sl)
    for i, (slot, text) in enumerate(queries):
        a, b = evaluate(text, lambda g: float(flat[g]), FUNCS)
        for got, want in ((a, want_r[i]), (b, want_c[i])):
            assert (math.isnan(got) and math.isnan(want)) or \
                math.isclose(got, want, rel_tol=1e-9, abs_tol=1e-9), (slot, got, want)
