"""Kernels given by their write sets (Sec. 3.4 "Per-element equations": a
kernel's symbolic writes are inverted -- the equation at location l is the
value of the thread whose write address is l).

CPU tests pin the oracle's inversion (it runs every thread of the launch and
records who writes each location) against a direct simulation of the kernel
in fp64 (every thread computes its value and stores it), and pin the kernel
descriptions themselves against the library routines they implement
(matmul, max_pool2d).  They also check that the library's symbolic inversion
(dirigo_graph_create, host only) rejects the write sets it cannot invert.
GPU tests compare the library's cones, keys, verdicts, exports and fp32
values with the oracle's on these kernels.
"""
import copy

import numpy as np
import pytest

import oracle
from oracle import forward64
from paper_2609_19611_gb300 import workloads as W

MATMUL_BUGS = [None, "edge", "last_tile"]


def _same64(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    both_nan = np.isnan(a) & np.isnan(b)
    scale = np.sqrt(np.nanmean(b ** 2)) if np.isfinite(b).any() else 1.0
    return np.all(both_nan | (np.abs(a - b) <= 1e-12 * (np.abs(b) + scale)))


# ------------------------------------------------------------------ oracle pins (CPU)

def test_kernel_descriptions_compute_their_ops():
    for ref, cand in (W.tiled_matmul_kernel(), W.tiled_matmul_kernel(M=48),
                      W.pool_kernel()):
        vals = W.random_values(ref, 11)
        assert _same64(forward64.flat_output(cand, vals), forward64.flat_output(ref, vals))


@pytest.mark.parametrize("bug", MATMUL_BUGS)
def test_inversion_matches_the_kernel_run(bug):
    _, cand = W.tiled_matmul_kernel(bug=bug)
    vals = W.random_values(cand, 12)
    C = oracle.Program(cand)
    got = C.eval(vals, np.arange(C.out_numel))
    assert _same64(got, forward64.flat_output(cand, vals))


def test_pool_inversion_matches_the_kernel_run():
    for bug in (None, "stride"):
        _, cand = W.pool_kernel(bug=bug)
        vals = W.random_values(cand, 13)
        C = oracle.Program(cand)
        assert _same64(C.eval(vals, np.arange(C.out_numel)), forward64.flat_output(cand, vals))


@pytest.mark.parametrize("bug", MATMUL_BUGS)
def test_verdict_pattern_of_planted_bugs(bug):
    M, N, TN = 50, 24, 8
    ref, cand = W.tiled_matmul_kernel(M=M, N=N, TN=TN, bug=bug)
    R, C = oracle.Program(ref), oracle.Program(cand)
    q = np.arange(R.out_numel)
    differs = np.any(R.keys(q) != C.keys(q), axis=1).reshape(M, N)
    want = np.zeros((M, N), dtype=bool)
    if bug == "edge":
        want[M - 1, :] = True            # never written
    elif bug == "last_tile":
        want[:, N - TN:] = True          # reads W one column to the right
    assert np.array_equal(differs, want)
    if bug == "edge":   # an unwritten location's cone holds bottom (global id G)
        off, runs = C.cone_runs(np.array([(M - 1) * N]))
        assert runs[off[1] - 1, 0] + runs[off[1] - 1, 1] == C.G + 1


def test_pool_kernel_verdicts():
    for bug, disc in ((None, True), ("stride", False)):
        ref, cand = W.pool_kernel(bug=bug)
        R, C = oracle.Program(ref), oracle.Program(cand)
        q = np.arange(R.out_numel)
        eq = np.all(R.keys(q) == C.keys(q), axis=1)
        assert eq.all() if disc else (~eq).any()


def test_oracle_rejects_races_and_stores_outside():
    _, cand = W.tiled_matmul_kernel()
    race = copy.deepcopy(cand)
    race["ops"][0]["writes"].append(race["ops"][0]["writes"][0])
    out = copy.deepcopy(cand)
    out["ops"][0]["writes"][0]["addr"][0] = 50 * 24
    for g in (race, out):
        with pytest.raises(ValueError):
            oracle.lower(g)


def test_library_rejects_what_it_cannot_invert():
    from paper_2609_19611_gb300 import dirigo as D
    _, cand = W.tiled_matmul_kernel()
    race = copy.deepcopy(cand)
    race["ops"][0]["writes"].append(race["ops"][0]["writes"][0])
    out = copy.deepcopy(cand)
    out["ops"][0]["writes"][0]["addr"][0] = 50 * 24
    # one thread column of each tile: a strided set of columns, not a box
    strided = copy.deepcopy(cand)
    w = strided["ops"][0]["writes"][0]
    w["when"][5] = [7, 8]
    for g in (race, out, strided):
        with pytest.raises(D.DirigoError) as e:
            D.Graph(g)
        assert e.value.status == 3   # DIRIGO_E_UNSUPPORTED
    # the oracle's brute-force inversion still reads the strided kernel
    oracle.lower(strided)


# ------------------------------------------------------------------ GPU parity

@pytest.mark.gpu
@pytest.mark.parametrize("bug", MATMUL_BUGS)
def test_tiled_matmul_kernel_parity(bug):
    from tests.test_gpu_parity import Case, check_cones, check_keys, check_compare, check_eval
    ref, cand = W.tiled_matmul_kernel(bug=bug)
    case = Case(ref, cand, seed=21)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    check_keys(case, locs)
    v, _ = check_compare(case, locs, budget=64)
    assert np.all(v == 0) if bug is None else np.any(v != 0)
    check_eval(case, locs)


@pytest.mark.gpu
@pytest.mark.parametrize("bug", [None, "stride"])
def test_pool_kernel_parity(bug):
    from tests.test_gpu_parity import Case, check_cones, check_keys, check_compare, check_eval
    ref, cand = W.pool_kernel(bug=bug)
    case = Case(ref, cand, seed=22)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    check_keys(case, locs)
    check_compare(case, locs)
    check_eval(case, locs)


@pytest.mark.gpu
@pytest.mark.parametrize("bug", ["edge", "last_tile"])
def test_tiled_matmul_kernel_parity_several_tiles(bug):
    """A 130 x 144 output (520 x 576 limb rows and columns: several tensor-core
    tiles with ragged edges), K = 72, tiles of 32 x 16 threads."""
    from tests.test_gpu_parity import Case, check_cones, check_keys, check_compare, check_eval
    ref, cand = W.tiled_matmul_kernel(M=130, K=72, N=144, TM=32, TN=16, bug=bug)
    case = Case(ref, cand, seed=23)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    rng = np.random.Generator(np.random.PCG64(23))
    sample = np.unique(np.concatenate([rng.integers(0, len(locs), 600),
                                       np.arange(len(locs) - 300, len(locs))]))
    check_cones(case, locs, sample)
    check_keys(case, locs, sample)
    check_compare(case, locs, budget=32)
    check_eval(case, locs, sample)


# ------------------------------------------------------------------ random pairs with variants

def test_random_pairs_with_kernel_and_shift_variants():
    """Random program pairs whose syntactic choices include kernels given by
    their write sets and max-shifted softmaxes: unmutated pairs have equal
    keys everywhere; the oracle's equations evaluate to the direct fp64
    forward pass (which runs the kernels thread by thread); the library
    accepts every graph."""
    from paper_2609_19611_gb300 import dirigo as D
    with_kernels = 0
    for seed in range(80):
        ref, cand, mutated = W.random_pair(seed, variants=True)
        with_kernels += any(op["op"].startswith("kernel") for g in (ref, cand)
                            for op in g["ops"])
        R, C = oracle.Program(ref), oracle.Program(cand)
        q = np.arange(R.out_numel)
        if not mutated:
            assert np.array_equal(R.keys(q), C.keys(q)), seed
        vals = W.random_values(ref, seed)
        for g, P in ((ref, R), (cand, C)):
            assert _same64(P.eval(vals, q), forward64.flat_output(g, vals)), seed
            D.Graph(g)
    assert with_kernels >= 15


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(24))
def test_random_pairs_with_variants_parity(seed):
    from tests.test_gpu_parity import Case, check_cones, check_keys, check_compare, check_eval
    ref, cand, _ = W.random_pair(3000 + seed, variants=True)
    case = Case(ref, cand, seed=seed)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    check_keys(case, locs)
    check_compare(case, locs)
    check_eval(case, locs)


def test_library_rejects_malformed_kernel_descriptions():
    from paper_2609_19611_gb300 import dirigo as D
    _, cand = W.tiled_matmul_kernel()
    zero_grid = copy.deepcopy(cand)
    zero_grid["ops"][0]["grid"] = [1, 0, 3]
    # X read at row by * (TM * K + 1) + ty * K: the block row's digits are not
    # combined as the output row is (by * TM + ty), so no affine map exists
    skewed = copy.deepcopy(cand)
    for w in skewed["ops"][0]["writes"]:
        w["reads"][0][1][1] += 1
    for g, status in ((zero_grid, 1), (skewed, 3)):   # E_INVALID, E_UNSUPPORTED
        with pytest.raises(D.DirigoError) as e:
            D.Graph(g)
        assert e.value.status == status


def test_merge_rejects_programs_over_different_inputs():
    from paper_2609_19611_gb300 import dirigo as D
    a, _ = W.config(4, N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)
    b, _ = W.config(4, N=2, Ci=3, H=8, W=8, Co=8, bug_co=5)
    with pytest.raises(D.DirigoError) as e:
        D.merge(a, b)
    assert e.value.status == 8   # E_MISMATCH
