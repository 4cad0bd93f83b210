"""Pins of the CPU oracle against facts fixed outside its own code.

Each test ties one part of the oracle to something it cannot agree with by
construction: closed-form cone sizes worked out by hand from the op
definitions, brute-force perturbation of a direct fp64 forward pass (PyTorch
library ops), exact canonical forms over Q[atoms], a direct fp64 forward pass
for concrete evaluation, primality, and the published SplitMix64 outputs.
"""
import os

import numpy as np
import pytest
import sympy

import oracle
from oracle import exact, forward64
from paper_2609_19611_gb300 import workloads as W
from tests import export_format as XF

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------------ key spec

def test_splitmix64_published_outputs():
    """The key's mixer is SplitMix64's finaliser: state k*gamma gives the
    generator's k-th output from seed 0."""
    want = [int(l, 16) for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt"))
            if l.strip() and not l.startswith("#")]
    L = oracle.lib()
    gamma = 0x9E3779B97F4A7C15
    got = [L.orc_mix64((k * gamma) % (1 << 64)) for k in range(1, len(want) + 1)]
    assert got == want


def test_primes():
    for p in (2 ** 29 - 3, 2 ** 29 - 33):
        assert sympy.isprime(p)


# ------------------------------------------------------------------ cones

def _loc(shape, coords):
    return int(np.ravel_multi_index(coords, shape))


def test_cone_c1_closed_form():
    """Y[i,j] = relu(sum_k X[i,k] W[k,j] + b[j]): K + K + 1 = 33 leaves; runs:
    X row (1) + 16 W singletons + b (1), except where the X row ends where
    W[0, j] starts (i = 7, j = 0)."""
    ref, cand = W.config(1)
    for g in (ref, cand):
        P = oracle.Program(g)
        locs = np.arange(64)
        sizes, nruns = P.cone_sizes(locs)
        assert (sizes == 33).all()
        want = np.full(64, 18)
        want[7 * 8 + 0] = 17
        assert (nruns == want).all()
        off, runs = P.cone_runs([3 * 8 + 5])
        assert runs[0].tolist() == [48, 16]                       # X[3, :]
        assert runs[1:17, 0].tolist() == [128 + 8 * k + 5 for k in range(16)]
        assert runs[17].tolist() == [256 + 5, 1]


def test_cone_c2_closed_form():
    """conv (Ci=3, 3x3, pad 1) + bias, GELU, sum over Co=16 channels.  Padded
    taps are absent, with their weight: interior 27 X + 432 W + 16 b = 475,
    border row/col 18 + 288 + 16 = 322, corner 12 + 192 + 16 = 220.  The
    candidate admits iw = W: at w = 31 its cone keeps the third tap column
    (next-row elements, or bottom past the end of X)."""
    ref, cand = W.config(2)
    R, C = oracle.Program(ref), oracle.Program(cand)
    S = [2, 32, 32]
    cases = {(0, 5, 7): (475, 475), (1, 0, 9): (322, 322), (0, 31, 0): (220, 220),
             (1, 12, 31): (322, 475), (0, 0, 31): (220, 322), (1, 31, 31): (220, 322),
             (1, 30, 31): (322, 475)}
    for co, (r, c) in cases.items():
        l = _loc(S, co)
        assert len(R.cone(l)) == r, co
        assert len(C.cone(l)) == c, co
    # bottom (global id G) is reached exactly when the image's last element's
    # right neighbour is read: n = 1, ih = 31, iw = 32
    assert C.cone(_loc(S, (1, 31, 31)))[-1] == C.G
    assert C.cone(_loc(S, (1, 30, 31)))[-1] == C.G
    assert C.cone(_loc(S, (0, 31, 31)))[-1] != C.G
    assert R.cone(_loc(S, (1, 31, 31)))[-1] != R.G


def test_cone_c3_closed_form():
    """LayerNorm of a linear layer: every output depends on its whole X row,
    all of W and b, and its own gamma and beta: 1024 + 524288 + 512 + 2."""
    ref, cand = W.config(3)
    for g in (ref, cand):
        P = oracle.Program(g)
        sizes, nruns = P.cone_sizes([0, 511, 7 * 512 + 100], nthreads=3)
        assert (sizes == 525826).all()
        # X row | W,b (+gamma[0] when j = 0) | gamma[j] | beta[j]
        assert nruns.tolist() == [3, 4, 4]


@pytest.mark.parametrize("coords,size", [((5, 3, 7, 9), 74880), ((9, 100, 0, 4), 74624),
                                         ((0, 127, 15, 0), 74432)])
def test_cone_c4_closed_form(coords, size):
    """softmax over channels of a 2x2 max-pool of conv(64ch, 3x3, pad 1) + bias:
    X is a 64 x 4 x 4 patch (clipped at the border: 3 rows or columns), all of
    W (every tap is valid for one of the pool window's conv outputs) and all
    of b.  The candidate reads W of channels >= 96 with channel stride 567, so
    its W cone is [0, 567*127 + 576) = 72585 ids: 1143 fewer."""
    ref, cand = W.config(4)
    R, C = oracle.Program(ref), oracle.Program(cand)
    l = _loc([128, 128, 16, 16], coords)
    assert R.cone_sizes([l])[0][0] == size
    c = C.cone(l)
    assert len(c) == size - 1143
    w_ids = c[(c >= 128 * 64 * 1024) & (c < 128 * 64 * 1024 + 73728)] - 128 * 64 * 1024
    assert w_ids.min() == 0 and w_ids.max() == 72584 and len(w_ids) == 72585


def test_cone_c5_closed_form():
    """tanh(sum_n (A[b] @ B[b])[m, n] + bias[m]): K + K*N + 1 = 131585; the
    candidate's K tail [480, 512) is dropped: 480 + 480*256 + 1 = 123361."""
    ref, cand = W.config(5)
    R, C = oracle.Program(ref), oracle.Program(cand)
    for l in (0, 8191, 31 * 256 + 17):
        assert R.cone_sizes([l])[0][0] == 131585
        assert C.cone_sizes([l])[0][0] == 123361


# ------------------------------------------------------------------ perturbation

TINY = [
    (1, dict(M=3, K=4, N=2), True),
    (2, dict(N=2, Ci=2, H=5, W=5, Co=3), False),
    (3, dict(B=2, IN=4, OUT=4), False),
    (4, dict(N=1, Ci=2, H=4, W=4, Co=4, bug_co=2), True),
    (5, dict(B=2, M=2, K=4, N=3, tile=2, k_stop=3), False),
]


def _changed(graph, vals, eps=0.37):
    base = forward64.flat_output(graph, vals)
    sizes = [v.size for v in vals]
    G = sum(sizes)
    changed = np.zeros((G, base.size), dtype=bool)
    g = 0
    for t, v in enumerate(vals):
        for i in range(v.size):
            pv = [x.copy() for x in vals]
            pv[t].reshape(-1)[i] += eps
            out = forward64.flat_output(graph, pv)
            changed[g] = ~np.isclose(out, base, rtol=1e-12, atol=1e-12) & ~np.isnan(base)
            g += 1
    return base, changed


@pytest.mark.parametrize("c,shape,masking", TINY)
def test_cone_membership_by_perturbation(c, shape, masking):
    """Leaves whose perturbation moves y[l] (direct fp64 forward pass) are in
    cone(l); without max/relu masking they are exactly cone(l) minus bottom."""
    for g in W.config(c, **shape):
        # the configuration's own value distributions keep GELU and tanh off
        # their flat tails, where a perturbation would vanish in fp64
        vals = W.make_values(c, g, dtype=np.float64)
        base, changed = _changed(g, vals)
        P = oracle.Program(g)
        for l in range(base.size):
            cone = set(P.cone(l).tolist()) - {P.G}
            moved = set(np.nonzero(changed[:, l])[0].tolist())
            assert moved <= cone, (c, l)
            if not masking and not np.isnan(base[l]):
                assert moved == cone, (c, l)


# ------------------------------------------------------------------ keys vs exact CFs

def _pair_check(ref, cand, atoms):
    R, C = oracle.Program(ref), oracle.Program(cand)
    n = R.out_numel
    locs = np.arange(n)
    kr, kc = R.keys(locs, nthreads=1), C.keys(locs, nthreads=1)
    er, ec = exact.ExactProgram(R, atoms), exact.ExactProgram(C, atoms)
    res = []
    vals = W.random_values(ref, seed=3)
    lv = XF.leaf_lookup(vals)
    fr, fc = forward64.flat_output(ref, vals), forward64.flat_output(cand, vals)
    for l in range(n):
        a, b = er.out_cf(l), ec.out_cf(l)
        res.append((a == b, bool((kr[l] == kc[l]).all())))
        # the CF's value is the program's value; its leaves are in the cone
        for cf, f, P in ((a, fr, R), (b, fc, C)):
            v = exact.eval_cf(cf, atoms, lv)
            # (an exp overflowing inside an unshifted softmax leaves no value
            # to compare; such locations are counted out)
            if np.isfinite(v) and np.isfinite(f[l]) and abs(f[l]) < 1e6:
                assert np.isclose(v, f[l], rtol=1e-9, atol=1e-12), (v, f[l])
                _pair_check.compared += 1
            _pair_check.total += 1
            assert exact.leaves_of(cf, atoms) <= set(P.cone(l).tolist())
    return res


_pair_check.compared = 0
_pair_check.total = 0


def test_key_equality_is_cf_equality():
    """Over random program pairs (the same expression compiled with different
    syntactic choices, half of them with one mutation), two locations have
    equal keys exactly when their canonical forms over Q[atoms] are equal."""
    atoms = exact.Atoms()
    n_eq = n_ne = 0
    for seed in range(400):
        ref, cand, _ = W.random_pair(seed)
        for cf_eq, key_eq in _pair_check(ref, cand, atoms):
            assert cf_eq == key_eq, seed
            n_eq += cf_eq
            n_ne += not cf_eq
    assert n_eq > 300 and n_ne > 300
    assert _pair_check.compared > 0.8 * _pair_check.total


def test_key_laws_on_configs_tiny():
    """Planted-bug semantics at tiny shapes, decided by exact CFs: c1, c3
    discharge everywhere; c2 differs exactly at the last column; c4 and c5
    differ everywhere; the worked example's half sum differs everywhere."""
    atoms = exact.Atoms()
    for c, shape, _ in TINY:
        ref, cand = W.config(c, **shape)
        res = _pair_check(ref, cand, atoms)
        eq = np.array([k for _, k in res])
        if c in (1, 3):
            assert eq.all()
        elif c == 2:
            S = W.out_shape(ref)
            w = np.unravel_index(np.arange(len(eq)), S)[2]
            assert (eq == (w != S[2] - 1)).all()
        else:
            assert not eq.any()
    ref, cand = W.halfsum_gelu(N=2, C=2, H=4, W=2)
    assert not any(k for _, k in _pair_check(ref, cand, atoms))


def test_axiom_gelu_merges_tags():
    ref = {"inputs": [["x", [3]]], "ops": [{"op": "gelu", "args": [0]}], "output": 1}
    cand = {"inputs": [["x", [3]]], "ops": [{"op": "gelu_tanh", "args": [0]}], "output": 1}
    R, C = oracle.Program(ref), oracle.Program(cand)
    l = np.arange(3)
    assert not (R.keys(l) == C.keys(l)).all(axis=1).any()
    assert (R.keys(l, axiom_gelu=True) == C.keys(l, axiom_gelu=True)).all()


# ------------------------------------------------------------------ verdicts

def test_verdicts_full_size_by_construction():
    """c1: 64/64 discharged; c2: discharged iff w != 31 over the 4096 seeded
    queries; c3: 1024/1024; c4, c5: none (sampled)."""
    for c in (1, 2, 3):
        ref, cand = W.config(c)
        R, C = oracle.Program(ref), oracle.Program(cand)
        q = W.make_queries(c, R.out_numel)
        eq = (R.keys(q) == C.keys(q)).all(axis=1)
        if c == 2:
            assert (eq == (q % 32 != 31)).all()
            assert (~eq).sum() > 100
        else:
            assert eq.all()
    for c in (4, 5):
        ref, cand = W.config(c)
        R, C = oracle.Program(ref), oracle.Program(cand)
        q = W.make_queries(c, R.out_numel)[::max(1, R.out_numel // 12)][:12]
        assert not (R.keys(q) == C.keys(q)).all(axis=1).any()


# ------------------------------------------------------------------ concrete eval

def _close(a, b, rel=1e-12):
    rms = np.sqrt(np.nanmean(b ** 2)) if np.isfinite(b).any() else 0.0
    both_nan = np.isnan(a) & np.isnan(b)
    return both_nan | (np.abs(a - b) <= rel * (np.abs(b) + rms))


@pytest.mark.parametrize("c,shape,_m", TINY)
def test_eval64_matches_direct_forward_tiny(c, shape, _m):
    for g in W.config(c, **shape):
        vals = W.make_values(c, g, dtype=np.float64)
        P = oracle.Program(g)
        want = forward64.flat_output(g, vals)
        got = P.eval(vals, np.arange(P.out_numel))
        assert _close(got, want).all()


@pytest.mark.parametrize("c", [1, 2, 3])
def test_eval64_matches_direct_forward_full(c):
    ref, cand = W.config(c)
    for g in (ref,) if c != 1 else (ref, cand):
        vals = W.make_values(c, g)
        P = oracle.Program(g)
        q = W.make_queries(c, P.out_numel)[:256]
        want = forward64.flat_output(g, vals)[q]
        got = P.eval(vals, q)
        assert _close(got, want).all()


# ------------------------------------------------------------------ export

@pytest.mark.parametrize("c,shape", [(2, dict(N=2, Ci=2, H=5, W=5, Co=3)),
                                     (5, dict(B=2, M=2, K=4, N=3, tile=2, k_stop=3)),
                                     (4, dict(N=1, Ci=2, H=4, W=4, Co=4, bug_co=2))])
def test_export_round_trip(c, shape):
    """Re-evaluating the exported term DAGs gives each exported location's fp64
    value (direct forward pass) in both programs; slots are the first
    undischarged ones; node lists are sorted by (tensor, elem)."""
    ref, cand = W.config(c, **shape)
    R, C = oracle.Program(ref), oracle.Program(cand)
    q = np.arange(R.out_numel)[::-1].copy()
    kr, kc = R.keys(q), C.keys(q)
    cones = (R.cone_runs(q), C.cone_runs(q))
    verdict, flags, blob, need = oracle.compare(R, C, q, kr, kc, cones=cones, budget=5)
    und = np.nonzero(~(kr == kc).all(axis=1))[0]
    assert need == len(blob)
    progs, locs = XF.parse(blob)
    assert [l[0] for l in locs] == und[:5].tolist()
    assert (verdict[und[:5]] == oracle.EXPORTED).all()
    assert (verdict[und[5:]] == oracle.DIFFERS_UNEXPORTED).all()
    assert ((flags & oracle.FLAG_CONE_DIFFERS) != 0).tolist() == (~(kr == kc).all(axis=1)).tolist()
    vals = W.make_values(c, ref, dtype=np.float64)
    lv = XF.leaf_lookup(vals)
    for p, g in enumerate((ref, cand)):
        assert progs[p]["order"] == sorted(progs[p]["order"])
        f = forward64.flat_output(g, vals)
        for slot, r0, r1 in locs:
            v = XF.evaluate(progs[p], (r0, r1)[p], lv)
            assert _close(np.array([v]), np.array([f[q[slot]]]), 1e-12).all()
    # capacity too small: nothing exported, required size reported
    v2, _, blob2, need2 = oracle.compare(R, C, q, kr, kc, budget=5, capacity=100)
    assert blob2 is None and need2 == need
    assert (v2[und] == oracle.DIFFERS_UNEXPORTED).all()


# ------------------------------------------------------------------ pin strength
# A plausible mistake planted in the oracle's lowering (on the CPU) must make
# a pin fail: the fp64 evaluation of the oracle's equations against the direct
# forward pass of the library routines.

def _planted_eval_ok(monkeypatch, graph, mutate):
    import copy
    import importlib
    L = importlib.import_module("oracle.lower")   # the module (the package re-exports lower())
    orig = L.lower_full

    def patched(g):
        inputs, prims, out, shapes = orig(g)
        prims = copy.deepcopy(prims)
        mutate(prims)
        return inputs, prims, out, shapes

    vals = W.random_values(graph, 17)
    want = forward64.flat_output(graph, vals)
    P = oracle.Program(graph)
    clean = _close(P.eval(vals, np.arange(P.out_numel)), want).all()
    monkeypatch.setattr(L, "lower_full", patched)
    Pm = oracle.Program(graph)
    planted = _close(Pm.eval(vals, np.arange(Pm.out_numel)), want).all()
    monkeypatch.setattr(L, "lower_full", orig)
    return clean, planted


def _first(prims, kind):
    return next(p for p in prims if p["kind"] == kind)


def _transpose_w(prims):           # W[k, j] read as W[j, k] (square-free: out of place)
    acc = _first(prims, "contract")["pieces"][0]["access"][1]
    acc[1], acc[2] = [0, acc[2][0]], [acc[1][1]]


def _drop_last_tap(prims):         # the channel reduction stops one short
    pc = _first(prims, "contract")["pieces"][0]
    pc["red"][0][1] -= 1


def _sub_as_add(prims):            # layernorm's centring z - mu written as z + mu
    next(p for p in prims if p["kind"] == "binary" and p["fn"] == "sub")["fn"] = "add"


def _sum_wrong_dim(prims):         # softmax's denominator sums along the last dim
    sm = [p for p in prims if p["kind"] == "contract"][-1]
    sm["pieces"][0]["access"][0][2] = [1]


@pytest.mark.parametrize("c,shape,mutate", [
    (1, {}, _transpose_w),
    (2, dict(N=1, Ci=2, H=5, W=5, Co=3), _drop_last_tap),
    (3, dict(B=3, IN=8, OUT=6), _sub_as_add),
    (4, dict(N=1, Ci=2, H=4, W=4, Co=4, bug_co=2), _sum_wrong_dim),
])
def test_pins_catch_planted_oracle_mistakes(monkeypatch, c, shape, mutate):
    ref, _ = W.config(c, **shape)
    clean, planted = _planted_eval_ok(monkeypatch, ref, mutate)
    assert clean and not planted


def test_pins_catch_a_planted_kernel_inversion_mistake(monkeypatch):
    """The oracle's kernel inversion recording each writer one location off
    fails against the thread-by-thread run of the kernel."""
    import importlib
    L = importlib.import_module("oracle.lower")
    _, cand = W.tiled_matmul_kernel(M=20, K=8, N=16, TM=8, TN=8)
    vals = W.random_values(cand, 19)
    want = forward64.flat_output(cand, vals)
    P = oracle.Program(cand)
    assert _close(P.eval(vals, np.arange(P.out_numel)), want).all()
    orig = L.kernel_writers
    n = 20 * 16
    monkeypatch.setattr(L, "kernel_writers",
                        lambda op: {(a + 1) % n: w for a, w in orig(op).items()})
    Pm = oracle.Program(cand)
    assert not _close(Pm.eval(vals, np.arange(Pm.out_numel)), want).all()
