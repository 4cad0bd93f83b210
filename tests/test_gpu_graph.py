"""A whole batch without host waits: dirigo_cone_async, dirigo_terms and
dirigo_compare_async captured into one CUDA graph (BatchChecker.capture) and
replayed.  Each replay must give exactly what the step with host waits gives
-- verdicts, flags, the export bytes and the statistics -- and the status and
statistics the asynchronous compare leaves on the device must equal the ones
the synchronous call returns, error cases included."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_19611_gb300 import dirigo as D
from paper_2609_19611_gb300 import workloads as W
from paper_2609_19611_gb300.pipeline import BatchChecker

pytestmark = pytest.mark.gpu

STAT_FIELDS = [k for k, _ in D.CompareStats._fields_]


@pytest.mark.parametrize("c,shape,budget", [
    (4, dict(N=3, Ci=5, H=10, W=10, Co=20, bug_co=13), 8),
    (2, dict(N=2, Ci=3, H=13, W=13, Co=5), 8),        # generic cone cells, bottom reads
    (1, {}, 4),
])
def test_graph_replay_equals_step(c, shape, budget):
    ref, cand = W.config(c, **shape)
    gr, gc = D.Graph(ref), D.Graph(cand)
    R, C = oracle.Program(ref), oracle.Program(cand)
    q = np.arange(R.out_numel, dtype=np.int64)
    locs = torch.as_tensor(q, device="cuda")
    chk = BatchChecker(gr, gc, len(q), budget=budget)
    chk.prepare(locs)
    st, stats = chk.step(locs)
    torch.cuda.synchronize()
    want = (chk.verdict[:len(q)].clone(), chk.flags[:len(q)].clone(),
            None if chk.blob(stats) is None else chk.blob(stats).clone(),
            [getattr(stats, k) for k in STAT_FIELDS], st)
    g = chk.capture(locs)
    for _ in range(2):
        chk.verdict.fill_(0xEE)
        chk.flags.fill_(0xEE)
        if chk.exp_buf is not None:
            chk.exp_buf.fill_(0)
        g.replay()
        chk.read_stats()
        torch.cuda.synchronize()
        st2, stats2 = chk.stats_host()
        assert st2 == want[4]
        assert [getattr(stats2, k) for k in STAT_FIELDS] == want[3]
        assert torch.equal(chk.verdict[:len(q)], want[0])
        assert torch.equal(chk.flags[:len(q)], want[1])
        b = chk.blob(stats2)
        assert (b is None) == (want[2] is None)
        if b is not None:
            assert torch.equal(b, want[2])
    # and the oracle agrees with what the replay left
    okr, okc = R.keys(q), C.keys(q)
    v, f, oblob, need = oracle.compare(R, C, q, okr, okc, cones=(R.cone_runs(q), C.cone_runs(q)),
                                       budget=budget)
    assert np.array_equal(chk.verdict[:len(q)].cpu().numpy(), v)
    assert np.array_equal(chk.flags[:len(q)].cpu().numpy(), f)


def test_async_compare_reports_on_the_device():
    """Short run buffer and an export buffer too small: the asynchronous
    compare's device status and statistics equal the synchronous call's."""
    ref, cand = W.config(4, N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)
    gr, gc = D.Graph(ref), D.Graph(cand)
    n = gr.out_numel
    locs = torch.arange(n, device="cuda")
    P = D._ptr
    kr, kc = D.terms(gr, locs), D.terms(gc, locs)
    tr = D.cone(gr, locs)[1].shape[0]
    tc = D.cone(gc, locs)[1].shape[0]
    for cap_r, exp_cap in ((tr - 1, 1 << 24), (tr, 64)):
        outs = []
        for asynchronous in (False, True):
            status = torch.zeros(1, dtype=torch.int32, device="cuda")
            cones = []
            for g, cap in ((gr, cap_r), (gc, tc)):
                ws = D._ws(g.workspace_size(D.CALL_CONE, n), "cuda")
                off = torch.empty(n + 1, dtype=torch.int64, device="cuda")
                runs = torch.empty(2 * cap, dtype=torch.int32, device="cuda")
                fp = torch.empty(n, dtype=torch.int64, device="cuda")
                D._check(D.dirigo_cone_async(g, P(locs), n, P(off), P(runs), cap, P(fp),
                                             P(status), P(ws), ws.numel(), D._stream(None)))
                cones.append((off, runs, fp, ws))
            ws = D._ws(D.compare_workspace_size(gr, gc, n), "cuda")
            verdict = torch.empty(n, dtype=torch.uint8, device="cuda")
            flags = torch.empty(n, dtype=torch.uint8, device="cuda")
            exp = torch.empty(exp_cap, dtype=torch.uint8, device="cuda")
            cr = (P(cones[0][0]), P(cones[0][1]), P(cones[0][2]))
            cc = (P(cones[1][0]), P(cones[1][1]), P(cones[1][2]))
            if asynchronous:
                dstats = torch.zeros(9, dtype=torch.int64, device="cuda")
                dst = torch.full((1,), -1, dtype=torch.int32, device="cuda")
                D._check(D.dirigo_compare_async(gr, gc, P(locs), n, P(kr), P(kc), cr, cc,
                                                P(verdict), P(flags), 4, P(exp), exp_cap,
                                                P(dstats), P(dst), P(ws), ws.numel(),
                                                D._stream(None), d_cone_status=P(status)))
                torch.cuda.synchronize()
                outs.append((int(dst.item()), dstats.cpu().tolist(), verdict.cpu(), flags.cpu()))
            else:
                st, stats = D.dirigo_compare(gr, gc, P(locs), n, P(kr), P(kc), cr, cc,
                                             P(verdict), P(flags), 4, P(exp), exp_cap, P(ws),
                                             ws.numel(), D._stream(None),
                                             d_cone_status=P(status))
                outs.append((st, [getattr(stats, k) for k in STAT_FIELDS], verdict.cpu(),
                             flags.cpu()))
        (s0, st0, v0, f0), (s1, st1, v1, f1) = outs
        assert s0 == s1 == D.E_CAPACITY
        assert st0 == st1
        assert torch.equal(v0, v1) and torch.equal(f0, f1)
