"""dirigo_cone_noalloc: the cone call for callers that cannot allocate device
memory (their device memory belongs to a memory manager, or they may not
allocate after start-up).  It must give exactly what dirigo_cone gives with a
caller workspace, call after call, although its fixed scratch array keeps the
previous call's contents.  Collected last: a failure here leaves every other
test already run."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_19611_gb300 import dirigo as D
from paper_2609_19611_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _noalloc(g, locs, cap):
    n = locs.numel()
    off = torch.empty(n + 1, dtype=torch.int64, device="cuda")
    runs = torch.empty(max(cap, 1) * 2, dtype=torch.int32, device="cuda")
    fp = torch.empty(n, dtype=torch.int64, device="cuda")
    total = ctypes.c_int64(0)
    st = D.load().dirigo_cone_noalloc(g.h, D._ptr(locs), n, D._ptr(off), D._ptr(runs), cap,
                                      D._ptr(fp), ctypes.byref(total), D._stream(None))
    return st, total.value, off, runs, fp


def test_noalloc_cone_matches_workspace_cone_twice():
    q2 = W.make_queries(2, 2048)
    cases = [
        # configuration 2's candidate: reads past a row's end (bottom past the
        # end of X) in cells without a fast plan, each location merged on its
        # own; three copies of the batch span three prefix-sum tiles
        (W.config(2)[1], np.concatenate([q2, q2, q2])),
        (W.config(4, N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)[1], np.arange(1500)),
        (W.config(1)[0], np.zeros(0, dtype=np.int64)),                           # empty batch
    ]
    g2 = D.Graph(cases[0][0])
    assert g2.n_fast_cells < g2.n_cells and (q2 % 32 == 31).any()
    assert len(cases[0][1]) > 2 * 4096
    for desc, q in cases:
        g = D.Graph(desc)
        locs = torch.as_tensor(np.asarray(q, dtype=np.int64), device="cuda")
        off_ref, runs_ref, fp_ref = D.cone(g, locs)
        total_ref = runs_ref.shape[0]
        for _ in range(2):   # two calls in a row share the fixed scratch
            st, total, off, runs, fp = _noalloc(g, locs, total_ref)
            assert st == D.OK, D.load().dirigo_last_error()
            assert total == total_ref
            assert torch.equal(off, off_ref)
            assert torch.equal(runs[:2 * total].view(total, 2), runs_ref)
            assert torch.equal(fp[:len(q)], fp_ref[:len(q)])


def test_noalloc_rejects_batches_above_its_limit():
    g = D.Graph(W.config(1)[0])
    locs = torch.zeros(8388609, dtype=torch.int64, device="cuda")
    st, total, *_ = _noalloc(g, locs, 0)
    assert st == 5   # DIRIGO_E_WORKSPACE
    assert b"8388608" in D.load().dirigo_last_error()
