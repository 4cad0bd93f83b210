"""Full-size GPU parity, in the launch arrangement the benchmark times.

Every configuration runs at its benchmark size through ``BatchChecker``:
both programs' cones on the caller's stream (``dirigo_cone_async``, one status
word), both programs' term keys on a second stream, one ``dirigo_compare``
with the export.  Results are compared with the oracle:

* configurations 1, 2, 3 and 5: every queried slot -- cones, fingerprints,
  keys, verdicts, flags and the exported bytes (budget 16), and the fp32
  evaluation; configuration 3 also on one location of every row of the
  linear layer's output;
* configuration 4 (4,194,304 locations): the whole batch is checked once;
  the oracle checks a structured sample of its slots -- every combination of
  boundary coordinates (padding edges, the candidate's channel 96), the lowest
  corner of every cone cell, one location touching every 32-pixel row tile
  of the key contraction (all 128 channels through the softmax), and every
  location of one row of the pooled output -- while properties that hold at
  any size are checked on all slots (no location discharged, every cone
  flagged as differing, runs sorted and maximal, fingerprints equal to their
  run lists).  The export of the first 64 undischarged slots is compared
  byte for byte with the oracle's, once for the flat order and once for a
  batch whose first 64 slots are 64 channels of one pooled pixel (roots that
  share every box of their equations).

Agreement is bit-exact for cones, keys, verdicts, flags and exports; the
fp32 evaluation is within |y32 - y64| <= 1e-5 |y64| + 1e-5 rms(y64) of the
oracle's fp64 value of res(y[l]).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_19611_gb300 import dirigo as D
from paper_2609_19611_gb300 import workloads as W
from paper_2609_19611_gb300.pipeline import BatchChecker

from .fingerprint import fingerprints_np, fingerprints_torch

pytestmark = pytest.mark.gpu


def close32(y32, y64):
    y32 = np.asarray(y32, dtype=np.float64)
    fin = np.isfinite(y64)
    rms = np.sqrt(np.mean(y64[fin] ** 2)) if fin.any() else 0.0
    both_nan = np.isnan(y32) & np.isnan(y64)
    err = np.abs(y32 - y64)
    ok = both_nan | (err <= 1e-5 * np.abs(y64) + 1e-5 * rms)
    rel_only = both_nan | (err <= 1e-5 * np.abs(y64))
    return ok, int((ok & ~rel_only).sum())


def gather_runs(off, runs, slots):
    """(offsets, runs uint32[R, 2]) of the given slots, gathered on the device."""
    s = torch.as_tensor(np.asarray(slots, dtype=np.int64), device=off.device)
    a, b = off[s], off[s + 1]
    lens = b - a
    o = torch.zeros(len(slots) + 1, dtype=torch.int64, device=off.device)
    o[1:] = torch.cumsum(lens, 0)
    tot = int(o[-1].item())
    pos = torch.arange(tot, device=off.device)
    idx = torch.repeat_interleave(a - o[:-1], lens) + pos
    r = runs[idx].cpu().numpy().astype(np.int64) & 0xffffffff
    return o.cpu().numpy(), r.astype(np.uint32)


def run_checks_everywhere(off, runs, fp, n):
    """Properties that hold at any size, on every slot: offsets start at 0 and
    do not decrease, runs are sorted and pairwise non-adjacent within each
    location, and each fingerprint is the one its run list defines (the
    positional sum of include/dirigo.h, 64-bit wrap-around arithmetic)."""
    dev = off.device
    assert int(off[0].item()) == 0
    assert bool((off[1:n + 1] >= off[:n]).all().item())
    total = int(off[n].item())
    first = torch.zeros(total + 1, dtype=torch.bool, device=dev)
    first[off[:n]] = True
    M32 = 0xffffffff
    chunk = 1 << 27
    for c0 in range(1, total, chunk):
        c1 = min(total, c0 + chunk)
        prev = runs[c0 - 1:c1 - 1].to(torch.int64) & M32
        cur = runs[c0:c1].to(torch.int64) & M32
        ok = cur[:, 0] > prev[:, 0] + prev[:, 1]
        assert bool((ok | first[c0:c1]).all().item()), "runs not sorted and maximal"
    got = fingerprints_torch(off, runs, n)
    assert torch.equal(got, fp[:n]), "fingerprints differ from their run lists"


class Pair:
    def __init__(self, c, **shape):
        self.c = c
        self.ref, self.cand = W.config(c, **shape)
        self.R, self.C = oracle.Program(self.ref), oracle.Program(self.cand)
        self.gr, self.gc = D.Graph(self.ref), D.Graph(self.cand)

    def checker(self, q, budget):
        chk = BatchChecker(self.gr, self.gc, len(q), budget=budget)
        locs = torch.as_tensor(np.asarray(q, dtype=np.int64), device="cuda")
        chk.prepare(locs)
        st, stats = chk.step(locs)
        torch.cuda.synchronize()
        return chk, locs, st, stats


def check_slots(P, chk, q, slots):
    """Cones, fingerprints and keys of the given slots against the oracle;
    returns the oracle's keys and cones of those slots."""
    q = np.asarray(q, dtype=np.int64)
    sl = q[slots]
    out = {}
    for i, (Prog, g) in enumerate(((P.R, P.gr), (P.C, P.gc))):
        off, runs, fp = chk.cones(i)
        g_off, g_runs = gather_runs(off, runs, slots)
        o_off, o_runs = Prog.cone_runs(sl)
        assert np.array_equal(g_off, o_off), f"program {i}: run counts differ"
        assert np.array_equal(g_runs, o_runs), f"program {i}: runs differ"
        g_fp = fp[torch.as_tensor(slots, device="cuda")].cpu().numpy().view(np.uint64)
        assert np.array_equal(g_fp, fingerprints_np(o_off, o_runs))
        k = chk.keys[i][torch.as_tensor(slots, device="cuda")].cpu().numpy().astype(np.uint32)
        ok = Prog.keys(sl)
        assert np.array_equal(k, ok), f"program {i}: keys differ"
        out[i] = (ok, (o_off, o_runs))
    return out


def check_eval(P, q, label):
    vals = W.make_values(P.c, P.ref)
    d = torch.as_tensor(np.asarray(q, dtype=np.int64), device="cuda")
    for Prog, g in ((P.R, P.gr), (P.C, P.gc)):
        y = D.eval_fp32(g, [torch.as_tensor(x, device="cuda") for x in vals], d).cpu().numpy()
        want = Prog.eval([x.astype(np.float64) for x in vals], q)
        ok, rms_only = close32(y, want)
        assert ok.all(), (np.nonzero(~ok)[0][:5], y[~ok][:5], want[~ok][:5])
        print(f"eval {label}: {len(q)} locations, {rms_only} within tolerance only by the "
              f"rms term")


@pytest.mark.parametrize("c", [1, 2, 3, 5])
def test_full_size_every_slot(c):
    P = Pair(c)
    q = W.make_queries(c, P.R.out_numel)
    n = len(q)
    chk, locs, st, stats = P.checker(q, budget=16)
    slots = np.arange(n)
    o = check_slots(P, chk, q, slots)
    (okr, ocr), (okc, occ) = o[0], o[1]
    v, f, oblob, need = oracle.compare(P.R, P.C, q, okr, okc, cones=(ocr, occ), budget=16)
    assert np.array_equal(chk.verdict[:n].cpu().numpy(), v)
    assert np.array_equal(chk.flags[:n].cpu().numpy(), f)
    assert stats.n_discharged == int((v == D.DISCHARGED).sum())
    assert stats.export_required == need
    blob = chk.blob(stats)
    if oblob is None:
        assert blob is None
    else:
        assert blob is not None and blob.cpu().numpy().tobytes() == oblob
    # the verdicts the configurations fix by construction
    und = v != D.DISCHARGED
    expect = {1: ~und.any(), 2: np.array_equal(und, q % 32 == 31), 3: ~und.any(),
              5: und.all()}[c]
    assert expect
    assert np.array_equal((f & D.FLAG_CONE_DIFFERS) != 0, und)
    check_eval(P, q, f"config {c}")


def test_full_size_linear_every_row():
    """Configuration 3: one location in every row of the 128 x 512 output
    (every row tile of the key contraction; columns spread over all column
    tiles), plus the four corners."""
    P = Pair(3)
    rows = np.arange(128)
    q = np.concatenate([rows * 512 + (rows * 37) % 512, [0, 511, 127 * 512, 128 * 512 - 1]])
    chk, locs, st, stats = P.checker(q, budget=16)
    o = check_slots(P, chk, q, np.arange(len(q)))
    assert (chk.verdict[:len(q)].cpu().numpy() == D.DISCHARGED).all()
    assert np.array_equal(o[0][0], o[1][0])
    check_eval(P, q, "config 3 rows")


def c4_sample_locations(P):
    """Slots (= locations: the batch is every location in flat order) the
    oracle checks in configuration 4's full batch."""
    N, Co, PH, PW = 128, 128, 16, 16

    def flat(n, c, ph, pw):
        return ((n * Co + c) * PH + ph) * PW + pw

    picks = []
    # every combination of boundary coordinates
    for n in (0, 1, 63, 64, 126, 127):
        for c in (0, 1, 63, 94, 95, 96, 97, 126, 127):
            for ph in (0, 1, 7, 8, 14, 15):
                for pw in (0, 1, 7, 8, 14, 15):
                    picks.append(flat(n, c, ph, pw))
    # the lowest corner of every cone cell of either program (the ranked
    # prefix of the query order lists them)
    order, pre = D.query_order(P.gr, P.gc, seed=0)
    picks.extend(order[:pre].tolist())
    # one location per pooled row: its two conv rows are two 32-pixel row
    # tiles of the key contraction, and the softmax reads all 128 channels
    for n in range(N):
        for ph in range(PH):
            picks.append(flat(n, (37 * n + 11 * ph) % Co, ph, (5 * n + 3 * ph) % PW))
    # every location of one row of the pooled output
    for c in range(Co):
        for pw in range(PW):
            picks.append(flat(77, c, 9, pw))
    return np.unique(np.asarray(picks, dtype=np.int64))


def test_full_size_conv_pool_softmax():
    P = Pair(4)
    q = W.make_queries(4, P.R.out_numel)
    n = len(q)
    assert np.array_equal(q, np.arange(n))
    chk, locs, st, stats = P.checker(q, budget=64)
    assert st == D.OK
    # properties on every slot
    for i in range(2):
        off, runs, fp = chk.cones(i)
        run_checks_everywhere(off, runs, fp, n)
    v_all = chk.verdict[:n]
    f_all = chk.flags[:n]
    assert not bool((v_all == D.DISCHARGED).any().item())
    assert bool((f_all == D.FLAG_CONE_DIFFERS).all().item())
    assert stats.n_discharged == 0 and stats.n_cone_differs == n
    assert stats.n_exported == 64 and stats.n_bot_ref == 0 and stats.n_bot_cand == 0
    assert bool((v_all[:64] == D.EXPORTED).all().item())
    assert bool((v_all[64:] == D.DIFFERS_UNEXPORTED).all().item())
    # the oracle on the structured sample
    slots = c4_sample_locations(P)
    o = check_slots(P, chk, q, slots)
    (okr, ocr), (okc, occ) = o[0], o[1]
    v, f, _, _ = oracle.compare(P.R, P.C, q[slots], okr, okc, cones=(ocr, occ), budget=0)
    assert np.array_equal(v, np.full(len(slots), D.DIFFERS_UNEXPORTED, dtype=np.uint8))
    assert np.array_equal(chk.flags[torch.as_tensor(slots, device="cuda")].cpu().numpy(), f)
    # export: slots 0..63 are the first undischarged ones (each confirmed by
    # the oracle's keys), so their export is the batch's
    first = np.arange(64)
    kr, kc = P.R.keys(q[first]), P.C.keys(q[first])
    assert not (kr == kc).all(axis=1).any()
    want = oracle.export(P.R, P.C, first, q[first])
    assert stats.export_bytes == len(want)
    assert chk.blob(stats).cpu().numpy().tobytes() == want
    check_eval(P, q[slots[::4]], "config 4 sample")


def test_full_size_shared_roots_export():
    """Configuration 4 at full size with a batch whose first 64 slots are
    channels 0..63 of one pooled pixel, then every location: the 64 exported
    roots share their pooling, exponential and convolution boxes, which the
    export's box-claim table must mark once each."""
    P = Pair(4)
    n_img, Co, PH, PW = 128, 128, 16, 16
    n0, ph0, pw0 = 5, 7, 9
    mates = np.array([((n0 * Co + c) * PH + ph0) * PW + pw0 for c in range(64)], dtype=np.int64)
    q = np.concatenate([mates, np.arange(P.R.out_numel, dtype=np.int64)])
    chk, locs, st, stats = P.checker(q, budget=64)
    assert st == D.OK and stats.n_exported == 64
    kr, kc = P.R.keys(mates), P.C.keys(mates)
    assert not (kr == kc).all(axis=1).any()
    want = oracle.export(P.R, P.C, np.arange(64), mates)
    assert chk.blob(stats).cpu().numpy().tobytes() == want
    # the duplicated slots carry the same results as their flat-order copies
    for i in range(2):
        k = chk.keys[i][:len(q)]
        assert torch.equal(k[:64], k[64 + torch.as_tensor(mates, device="cuda")])
        off, runs, fp = chk.cones(i)
        assert torch.equal(fp[:64], fp[64 + torch.as_tensor(mates, device="cuda")])
