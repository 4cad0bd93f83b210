"""GPU parity: the CUDA path against the CPU oracle, element by element.

Bit-exact: cone offsets and runs, run-list fingerprints, key pairs, verdicts,
flags and exported bytes.  Concrete fp32 evaluation: within
|y32 - y64| <= 1e-5 |y64| + 1e-5 rms(y64) of the oracle's fp64 value of
res(y[l]) (both NaN where bottom is read).

Sizes: every configuration at reduced shapes that span several tiles of the
contraction kernel with ragged edges, then at the full benchmark shapes with
sampled locations, plus random program pairs.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_19611_gb300 import dirigo as D
from paper_2609_19611_gb300 import workloads as W

from .fingerprint import fingerprints_np as fingerprints

pytestmark = pytest.mark.gpu

def to_u32(t):
    return (t.cpu().numpy().astype(np.int64) & 0xffffffff).astype(np.uint32)


def close32(y32, y64):
    y32 = np.asarray(y32, dtype=np.float64)
    fin = np.isfinite(y64)
    rms = np.sqrt(np.mean(y64[fin] ** 2)) if fin.any() else 0.0
    both_nan = np.isnan(y32) & np.isnan(y64)
    return both_nan | (np.abs(y32 - y64) <= 1e-5 * np.abs(y64) + 1e-5 * rms)


class Case:
    def __init__(self, ref, cand, c=None, seed=0):
        self.ref, self.cand = ref, cand
        self.R, self.C = oracle.Program(ref), oracle.Program(cand)
        self.gr, self.gc = D.Graph(ref), D.Graph(cand)
        self.vals = W.make_values(c, ref) if c else W.random_values(ref, seed, np.float32)


def check_cones(case, locs, sample=None):
    d = torch.as_tensor(locs, device="cuda")
    sel = np.arange(len(locs)) if sample is None else sample
    for P, g in ((case.R, case.gr), (case.C, case.gc)):
        off, runs, fp = D.cone(g, d)
        off = off.cpu().numpy()
        runs = to_u32(runs)
        fp = fp.cpu().numpy().view(np.uint64)[:len(locs)]
        assert off[0] == 0 and np.all(np.diff(off) >= 1)
        assert np.array_equal(fingerprints(off, runs), fp)
        o_off, o_runs = P.cone_runs(np.asarray(locs)[sel])
        for j, i in enumerate(sel):
            got = runs[off[i]:off[i + 1]]
            want = o_runs[o_off[j]:o_off[j + 1]]
            assert np.array_equal(got, want), (i, got[:4], want[:4])
        # runs are maximal: sorted, pairwise non-adjacent
        for i in sel[:64]:
            r = runs[off[i]:off[i + 1]].astype(np.int64)
            assert np.all(r[1:, 0] > r[:-1, 0] + r[:-1, 1])
    torch.cuda.synchronize()


def check_keys(case, locs, sample=None):
    d = torch.as_tensor(locs, device="cuda")
    sel = np.arange(len(locs)) if sample is None else sample
    out = []
    for P, g in ((case.R, case.gr), (case.C, case.gc)):
        k = D.terms(g, d).cpu().numpy().astype(np.uint32)
        want = P.keys(np.asarray(locs)[sel])
        assert np.array_equal(k[sel], want)
        out.append(k)
    return out


def check_compare(case, locs, budget=16, capacity=1 << 26):
    d = torch.as_tensor(locs, device="cuda")
    cr, cc = D.cone(case.gr, d), D.cone(case.gc, d)
    kr, kc = D.terms(case.gr, d), D.terms(case.gc, d)
    verdict, flags, blob, stats, st = D.compare(case.gr, case.gc, d, kr, kc, cr, cc, budget=budget,
                                               export_capacity=capacity)
    okr, okc = kr.cpu().numpy().astype(np.uint32), kc.cpu().numpy().astype(np.uint32)
    ocr = (cr[0].cpu().numpy(), to_u32(cr[1]))
    occ = (cc[0].cpu().numpy(), to_u32(cc[1]))
    v, f, oblob, need = oracle.compare(case.R, case.C, np.asarray(locs), okr, okc,
                                       cones=(ocr, occ), budget=budget, capacity=capacity)
    assert np.array_equal(verdict.cpu().numpy(), v)
    assert np.array_equal(flags.cpu().numpy(), f)
    assert stats["export_required"] == (need if (v != 0).any() and budget else 0)
    if oblob is not None and budget and (v != 0).any():
        assert blob is not None and bytes(blob.cpu().numpy().tobytes()) == oblob
    assert stats["n_discharged"] == int((v == 0).sum())
    return v, f


def check_eval(case, locs, sample=None):
    d = torch.as_tensor(locs, device="cuda")
    sel = np.arange(len(locs)) if sample is None else sample
    for P, g in ((case.R, case.gr), (case.C, case.gc)):
        ins = [torch.as_tensor(x, device="cuda") for x in case.vals]
        y = D.eval_fp32(g, ins, d).cpu().numpy()
        want = P.eval([x.astype(np.float64) for x in case.vals], np.asarray(locs)[sel])
        ok = close32(y[sel], want)
        assert ok.all(), (np.nonzero(~ok)[0][:5], y[sel][~ok][:5], want[~ok][:5])


SMALL = [
    (1, {}),
    (2, dict(N=2, Ci=3, H=13, W=13, Co=5)),
    (3, dict(B=5, IN=40, OUT=24)),
    (4, dict(N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)),
    (5, dict(B=3, M=17, K=40, N=9, tile=8, k_stop=37)),
]


@pytest.mark.parametrize("c,shape", SMALL)
def test_small_configs_full_parity(c, shape):
    ref, cand = W.config(c, **shape)
    case = Case(ref, cand, c)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    rng = np.random.Generator(np.random.PCG64(c))
    locs = np.concatenate([locs, rng.integers(0, case.R.out_numel, 37)])   # duplicates
    check_cones(case, locs)
    check_keys(case, locs)
    check_compare(case, locs)
    check_eval(case, locs)


def test_worked_example_shape():
    ref, cand = W.halfsum_gelu(N=3, C=4, H=10, W=6)
    case = Case(ref, cand, seed=5)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    check_keys(case, locs)
    v, f = check_compare(case, locs)
    assert (v != 0).all()
    check_eval(case, locs)


@pytest.mark.parametrize("seed", range(40))
def test_random_pairs(seed):
    ref, cand, _ = W.random_pair(1000 + seed)
    case = Case(ref, cand, seed=seed)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    check_keys(case, locs)
    check_compare(case, locs, budget=3)
    check_eval(case, locs)


def _async_cones(g, locs, cap, status, ws=None):
    n = locs.numel()
    ws = ws if ws is not None else D._ws(g.workspace_size(D.CALL_CONE, n), locs.device)
    off = torch.empty(n + 1, dtype=torch.int64, device="cuda")
    runs = torch.full((max(cap, 1) * 2 + 64,), -7, dtype=torch.int32, device="cuda")
    fp = torch.full((max(n, 1),), -7, dtype=torch.int64, device="cuda")
    D._check(D.dirigo_cone_async(g, D._ptr(locs), n, D._ptr(off), D._ptr(runs), cap,
                                 D._ptr(fp), D._ptr(status), D._ptr(ws), ws.numel(),
                                 D._stream(None)))
    return off, runs, fp, ws


def _compare_with_status(case, d, kr, kc, cones, status, budget=4):
    (o0, r0, f0), (o1, r1, f1) = cones
    n = d.numel()
    ws = D._ws(D.compare_workspace_size(case.gr, case.gc, n), d.device)
    verdict = torch.empty(n, dtype=torch.uint8, device="cuda")
    flags = torch.empty(n, dtype=torch.uint8, device="cuda")
    exp = torch.empty(1 << 24, dtype=torch.uint8, device="cuda")
    P = D._ptr
    st, stats = D.dirigo_compare(case.gr, case.gc, P(d), n, P(kr), P(kc),
                                 (P(o0), P(r0), P(f0)), (P(o1), P(r1), P(f1)), P(verdict),
                                 P(flags), budget, P(exp), exp.numel(), P(ws), ws.numel(),
                                 D._stream(None), d_cone_status=P(status))
    return st, stats, verdict, flags, exp


def test_async_cones_match_the_oracle():
    """dirigo_cone_async (no wait) gives the oracle's cones, and a compare that
    reads its status word gives the oracle's verdicts, flags and export."""
    ref, cand = W.config(4, N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)
    case = Case(ref, cand, 4)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    d = torch.as_tensor(locs, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    cones = []
    for g, P in ((case.gr, case.R), (case.gc, case.C)):
        cap = g.max_runs_per_location * len(locs)
        assert cap > 0
        off, runs, fp, _ = _async_cones(g, d, cap, status)
        o_off, o_runs = P.cone_runs(locs)
        tot = int(off[-1].item())
        assert np.array_equal(off.cpu().numpy(), o_off)
        assert np.array_equal(to_u32(runs[:2 * tot].view(tot, 2)), o_runs)
        assert (runs[2 * tot:] == -7).all()   # nothing past the total
        cones.append((off, runs, fp))
    kr, kc = D.terms(case.gr, d), D.terms(case.gc, d)
    st, stats, verdict, flags, exp = _compare_with_status(case, d, kr, kc, cones, status)
    assert st == D.OK and stats.cone_error == 0 and int(status.item()) == 0
    okr, okc = kr.cpu().numpy().astype(np.uint32), kc.cpu().numpy().astype(np.uint32)
    v, f, oblob, need = oracle.compare(case.R, case.C, locs, okr, okc,
                                       cones=(case.R.cone_runs(locs), case.C.cone_runs(locs)),
                                       budget=4)
    assert np.array_equal(verdict.cpu().numpy(), v) and np.array_equal(flags.cpu().numpy(), f)
    assert exp[:stats.export_bytes].cpu().numpy().tobytes() == oblob


def test_async_cone_capacity_and_location_errors_reach_the_compare():
    """A run buffer one run short: the asynchronous cone writes no run and no
    fingerprint, leaves the total in offsets[n], and the compare returns
    E_CAPACITY with cone_error = DIRIGO_CONE_ERR_RUNS, NO_CONES flags and the
    verdicts of a compare without cones.  A location out of range in the cone
    batch arrives as E_INVALID (cone_error = DIRIGO_CONE_ERR_LOCATION)."""
    ref, cand = W.config(4, N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)
    case = Case(ref, cand, seed=6)
    n = case.R.out_numel
    locs = np.arange(n, dtype=np.int64)
    d = torch.as_tensor(locs, device="cuda")
    total_r = D.cone(case.gr, d)[1].shape[0]
    total_c = D.cone(case.gc, d)[1].shape[0]
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    o0, r0, f0, _ = _async_cones(case.gr, d, total_r - 1, status)
    o1, r1, f1, _ = _async_cones(case.gc, d, total_c, status)
    kr, kc = D.terms(case.gr, d), D.terms(case.gc, d)
    st, stats, verdict, flags, exp = _compare_with_status(
        case, d, kr, kc, [(o0, r0, f0), (o1, r1, f1)], status)
    assert st == D.E_CAPACITY and stats.cone_error == D.CONE_ERR_RUNS
    assert int(o0[n].item()) == total_r
    assert (r0 == -7).all() and (f0 == -7).all()   # nothing written, not even within capacity
    assert (flags.cpu().numpy() == D.FLAG_NO_CONES).all()
    okr, okc = kr.cpu().numpy().astype(np.uint32), kc.cpu().numpy().astype(np.uint32)
    ov, _, oblob, need = oracle.compare(case.R, case.C, locs, okr, okc, budget=4)
    assert np.array_equal(verdict.cpu().numpy(), ov)
    assert stats.export_required == need
    # a location past the end in the cone batch
    bad = d.clone()
    bad[n // 2] = n
    status.zero_()
    o0, r0, f0, _ = _async_cones(case.gr, bad, total_r + 64, status)
    o1, r1, f1, _ = _async_cones(case.gc, bad, total_c + 64, status)
    st, stats, verdict, flags, exp = _compare_with_status(
        case, d, kr, kc, [(o0, r0, f0), (o1, r1, f1)], status)
    assert st == D.E_INVALID and stats.cone_error & D.CONE_ERR_LOCATION
    assert (r0 == -7).all() and (r1 == -7).all()
    # the stream and the library still work: a clean batch after the errors
    status.zero_()
    cones = [_async_cones(g, d, t, status)[:3] for g, t in ((case.gr, total_r),
                                                            (case.gc, total_c))]
    st, stats, verdict, flags, exp = _compare_with_status(case, d, kr, kc, cones, status)
    assert st == D.OK and stats.cone_error == 0


def test_expired_scan_wait_is_reported(monkeypatch):
    """The prefix sum's bounded wait running out: with the test hook
    DIRIGO_TEST_SCAN_STALL=1 the first tile never publishes its sum, so the
    second tile's look-back gives up after a short bounded wait; dirigo_cone
    returns E_CUDA ("bounded wait expired").  Without the hook, the next call
    on the same stream gives the oracle's cones."""
    ref, cand = W.config(4, N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)
    case = Case(ref, cand, 4)
    locs = np.concatenate([np.arange(case.R.out_numel, dtype=np.int64)] * 6)   # three tiles
    assert len(locs) > 2 * 4096
    d = torch.as_tensor(locs, device="cuda")
    monkeypatch.setenv("DIRIGO_TEST_SCAN_STALL", "1")
    with pytest.raises(D.DirigoError) as ei:
        D.cone(case.gr, d)
    assert ei.value.status == 6 and "bounded wait expired" in str(ei.value)
    monkeypatch.delenv("DIRIGO_TEST_SCAN_STALL")
    off, runs, fp = D.cone(case.gr, d)
    o_off, o_runs = case.R.cone_runs(locs)
    assert np.array_equal(off.cpu().numpy(), o_off)
    assert np.array_equal(to_u32(runs), o_runs)


def test_errors_are_reported():
    ref, cand = W.config(1)
    g = D.Graph(ref)
    bad = torch.tensor([0, 64], dtype=torch.int64, device="cuda")
    with pytest.raises(D.DirigoError) as ei:
        D.cone(g, bad)
    assert ei.value.status == 1
    # a negative location, and one past the end in a larger batch of a
    # conv + pool + softmax graph (the counts formed inside the prefix sum)
    g4 = D.Graph(W.config(4, N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)[0])
    for locs in ([3, -1, 5], list(range(g4.out_numel)) * 40 + [g4.out_numel]):
        with pytest.raises(D.DirigoError) as ei:
            D.cone(g4, torch.tensor(locs, dtype=torch.int64, device="cuda"))
        assert ei.value.status == 1
    ws = torch.empty(8, dtype=torch.uint8, device="cuda")
    with pytest.raises(D.DirigoError) as ei:
        D.terms(g, torch.arange(4, device="cuda"), ws=ws)
    assert ei.value.status == 5
    # capacity: the C call reports the required run count
    locs = torch.arange(64, device="cuda")
    off = torch.empty(65, dtype=torch.int64, device="cuda")
    wsb = g.workspace_size(D.CALL_CONE, 64)
    w2 = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    runs = torch.empty(2, dtype=torch.int32, device="cuda")
    st, total = D.dirigo_cone(g, D._ptr(locs), 64, D._ptr(off), D._ptr(runs), 1, None,
                              D._ptr(w2), wsb, D._stream(None))
    assert st == D.E_CAPACITY and total == 64 * 18 - 1
    # mismatched programs
    other = D.Graph(W.config(2)[0])
    k = D.terms(g, locs)
    with pytest.raises(D.DirigoError) as ei:
        D.compare(g, other, locs, k, k)
    assert ei.value.status == 8


@pytest.mark.parametrize("mode", ["stationary", "mma"])
@pytest.mark.parametrize("width", [10, 32])
def test_key_contraction_variants(monkeypatch, mode, width):
    """The column-stationary tcgen05 variant and the mma.sync variant of the
    key contraction give the oracle's keys (conv pair with a split piece; at
    width 32 the tcgen05 variants read the padded limb image)."""
    if mode == "stationary":
        monkeypatch.setenv("DIRIGO_TC_STATIONARY", "1")
    else:
        monkeypatch.setenv("DIRIGO_TC", "mma")
    ref, cand = W.config(4, N=2, Ci=5, H=width, W=width, Co=20, bug_co=13)
    case = Case(ref, cand, 4)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_keys(case, locs)


@pytest.mark.parametrize("c,shape", [
    (4, dict(N=2, Ci=5, H=32, W=32, Co=20, bug_co=13)),
    (2, dict(N=2, Ci=3, H=32, W=32, Co=5)),
])
def test_convolution_limb_image_path(c, shape):
    """Convolutions with an output width of 32 read their row side from the
    padded limb image (channels padded to 64, (kh, kw, channel) reduction
    order); the keys, cones and verdicts still equal the oracle's.  Config 2's
    candidate (right padding off by one) stays on the generic path."""
    ref, cand = W.config(c, **shape)
    case = Case(ref, cand, c)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_keys(case, locs)
    check_compare(case, locs)


def test_compare_budget_capacity_and_no_cones():
    """Budget 0 (nothing exported), a budget above the undischarged count
    (every undischarged slot exported), an export buffer too small for the
    selected slots (E_CAPACITY: nothing written, the required size reported),
    and a compare without cones (every flag NO_CONES; verdicts and export as
    the oracle's, which does not read the cones for them)."""
    ref, cand = W.config(4, N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)
    case = Case(ref, cand, seed=6)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    v, _ = check_compare(case, locs, budget=0)
    assert (v != 0).any() and not (v == D.EXPORTED).any()
    v, _ = check_compare(case, locs, budget=len(locs) + 7)
    assert ((v == D.EXPORTED) == (v != 0)).all()
    v, _ = check_compare(case, locs, budget=4, capacity=64)
    assert not (v == D.EXPORTED).any()
    d = torch.as_tensor(locs, device="cuda")
    kr, kc = D.terms(case.gr, d), D.terms(case.gc, d)
    verdict, flags, blob, stats, st = D.compare(case.gr, case.gc, d, kr, kc, budget=4,
                                               export_capacity=1 << 26)
    okr, okc = kr.cpu().numpy().astype(np.uint32), kc.cpu().numpy().astype(np.uint32)
    ov, _, oblob, need = oracle.compare(case.R, case.C, locs, okr, okc, budget=4)
    assert st == D.OK and stats["export_required"] == need
    assert np.array_equal(verdict.cpu().numpy(), ov)
    assert (flags.cpu().numpy() == D.FLAG_NO_CONES).all()
    assert blob is not None and bytes(blob.cpu().numpy().tobytes()) == oblob


def test_empty_batch():
    """n = 0 through every call: offsets [0], no keys, zero counts, no export."""
    ref, cand = W.config(1)
    gr, gc = D.Graph(ref), D.Graph(cand)
    d = torch.empty(0, dtype=torch.int64, device="cuda")
    off, runs, fp = D.cone(gr, d)
    assert off.cpu().numpy().tolist() == [0]
    kr, kc = D.terms(gr, d), D.terms(gc, d)
    assert kr.numel() == 0 and kc.numel() == 0
    verdict, flags, blob, stats, st = D.compare(gr, gc, d, kr, kc, (off, runs, fp),
                                               D.cone(gc, d), budget=16,
                                               export_capacity=1 << 20)
    assert st == D.OK and blob is None
    assert stats["n_discharged"] == 0 and stats["n_exported"] == 0 and stats["export_bytes"] == 0
    vals = W.make_values(1, ref)
    y = D.eval_fp32(gr, [torch.as_tensor(x, device="cuda") for x in vals], d)
    assert y.numel() == 0


def test_two_stream_step_matches_oracle():
    """The bench's launch arrangement: both programs' term keys on a second
    stream while the cones run on the first, joined before the compare.
    Cones, keys, verdicts, flags and the export equal the oracle's."""
    ref, cand = W.config(4, N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)
    case = Case(ref, cand, 4)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    d = torch.as_tensor(locs, device="cuda")
    side.wait_stream(main)
    kr = D.terms(case.gr, d, stream=side)
    kc = D.terms(case.gc, d, stream=side)
    cr, cc = D.cone(case.gr, d, stream=main), D.cone(case.gc, d, stream=main)
    main.wait_stream(side)
    verdict, flags, blob, stats, st = D.compare(case.gr, case.gc, d, kr, kc, cr, cc, budget=8,
                                               export_capacity=1 << 26, stream=main)
    okr, okc = kr.cpu().numpy().astype(np.uint32), kc.cpu().numpy().astype(np.uint32)
    assert np.array_equal(okr, case.R.keys(locs)) and np.array_equal(okc, case.C.keys(locs))
    ocr, occ = case.R.cone_runs(locs), case.C.cone_runs(locs)
    assert np.array_equal(cr[0].cpu().numpy(), ocr[0]) and np.array_equal(to_u32(cr[1]), ocr[1])
    v, f, oblob, need = oracle.compare(case.R, case.C, locs, okr, okc, cones=(ocr, occ),
                                       budget=8, capacity=1 << 26)
    assert np.array_equal(verdict.cpu().numpy(), v) and np.array_equal(flags.cpu().numpy(), f)
    assert blob is not None and blob.cpu().numpy().tobytes() == oblob


def test_alu_peak_rates():
    """dirigo_alu_peak: positive, finite rates, the SplitMix64 finaliser (about
    20 integer instructions) slower than one 32 x 32 -> 64 multiply-add, and
    both below the integer issue bound of 152 SMs x 128 lanes x 2.1 GHz."""
    mix, mad = D.alu_peak()
    bound = 152 * 128 * 2.1e9
    assert 0 < mix < mad <= bound and np.isfinite(mix) and np.isfinite(mad)


@pytest.mark.parametrize("c,shape", [
    (4, dict(N=2, Ci=5, H=10, W=10, Co=64, bug_co=40)),     # split piece inside a 64-output tile
    (4, dict(N=2, Ci=5, H=32, W=32, Co=128, bug_co=96)),    # limb image, two column tiles
    (5, dict(B=3, M=17, K=40, N=64, tile=8, k_stop=37)),    # batched, ragged rows
    (3, dict(B=5, IN=40, OUT=64)),
])
def test_key_contraction_256_column_tiles(monkeypatch, c, shape):
    """With DIRIGO_TC_N=256, contractions with a multiple of 64 output columns
    run on the 256-limb-column tcgen05 tiles (one 128 x 256 accumulator per
    CTA, two CTAs per SM); keys, cones, verdicts and the export equal the
    oracle's."""
    monkeypatch.setenv("DIRIGO_TC_N", "256")
    ref, cand = W.config(c, **shape)
    case = Case(ref, cand, c)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_keys(case, locs)
    check_compare(case, locs)


@pytest.mark.parametrize("shape", [
    # 8,064 output rows (252 row tiles), 48 channels: tile counts and row
    # extents (7, 12, 96) that are not powers of two
    dict(N=7, Ci=5, H=12, W=96, Co=48, bug_co=30),
    # 70 input channels (two 64-channel blocks of the limb image), 72 output
    # channels (a ragged third column tile)
    dict(N=3, Ci=70, H=10, W=64, Co=72, bug_co=50),
])
def test_key_contraction_odd_sizes(shape):
    """Convolutions whose tile counts and output-row extents are not powers of
    two (the tensor-core kernel's epilogue divides by multiplies) and whose
    channel counts span several channel blocks and a ragged column tile: keys
    equal the oracle's on a sample that reaches every row tile of the
    contraction, and the verdicts on the whole batch agree with the keys."""
    ref, cand = W.conv_pool_softmax(**shape)
    case = Case(ref, cand, seed=3)
    n = case.R.out_numel
    N, Co, H, Wd = shape["N"], shape["Co"], shape["H"], shape["W"]
    Ho, Wo = H // 2, Wd // 2
    # one pooled location per 16 pooled columns of every pooled row (each covers
    # a 32-output row tile of the convolution), at a random channel, plus a
    # random sample
    rng = np.random.Generator(np.random.PCG64(11))
    picks = []
    for nn in range(N):
        for h in range(Ho):
            for w0 in range(0, Wo, 16):
                c = int(rng.integers(0, Co))
                w = w0 + int(rng.integers(0, min(16, Wo - w0)))
                picks.append(((nn * Co + c) * Ho + h) * Wo + w)
    picks = np.concatenate([np.asarray(picks, dtype=np.int64),
                            rng.integers(0, n, 64)]).astype(np.int64)
    d = torch.arange(n, dtype=torch.int64, device="cuda")
    kr_t, kc_t = D.terms(case.gr, d), D.terms(case.gc, d)
    kr = kr_t.cpu().numpy().astype(np.uint32)
    kc = kc_t.cpu().numpy().astype(np.uint32)
    assert np.array_equal(kr[picks], case.R.keys(picks))
    assert np.array_equal(kc[picks], case.C.keys(picks))
    verdict, _, _, _, _ = D.compare(case.gr, case.gc, d, kr_t, kc_t, budget=0)
    same = np.all(kr == kc, axis=1)
    assert np.array_equal(verdict.cpu().numpy() == 0, same)
    assert not same.any()   # the softmax spans every channel, so the planted stride reaches all
