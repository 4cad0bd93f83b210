"""The query order of a program pair (Sec. 4 "Search Heuristic"): a ranked
prefix (output corners and the first warp boundary, one location per cone
cell of either program, the first and last element), then a seeded random
permutation of the rest.  Host only; no GPU."""
import numpy as np
import pytest

import oracle
from paper_2609_19611_gb300 import build, dirigo as D, workloads as W


@pytest.fixture(scope="module")
def lib():
    build.build()
    return D.load()


SMALL = [
    (1, {}),
    (2, dict(N=2, Ci=3, H=13, W=13, Co=5)),
    (3, dict(B=5, IN=40, OUT=24)),
    (4, dict(N=3, Ci=5, H=10, W=10, Co=20, bug_co=13)),
    (5, dict(B=3, M=17, K=40, N=9, tile=8, k_stop=37)),
]


@pytest.mark.parametrize("c,shape", SMALL)
def test_order_is_a_permutation_with_the_ranked_prefix(lib, c, shape):
    ref, cand = W.config(c, **shape)
    gr, gc = D.Graph(ref), D.Graph(cand)
    order, pre = D.query_order(gr, gc, seed=7)
    n = gr.out_numel
    assert np.array_equal(np.sort(order), np.arange(n))
    shp = gr.out_shape
    corners = {int(np.ravel_multi_index([(m >> d) & 1 and s - 1 or 0 for d, s in enumerate(shp)],
                                        shp)) for m in range(1 << len(shp))}
    assert corners <= set(order[:len(corners)].tolist())
    assert {0, n - 1} <= set(order[:pre].tolist())
    assert pre >= len(corners)
    # deterministic per seed; another seed only changes the tail
    o2, p2 = D.query_order(gr, gc, seed=7)
    o3, p3 = D.query_order(gr, gc, seed=8)
    assert np.array_equal(order, o2) and p2 == pre
    assert p3 == pre and np.array_equal(order[:pre], o3[:pre])
    if n - pre > 8:
        assert not np.array_equal(order[pre:], o3[pre:])


def _first_bug(order, bad):
    pos = np.nonzero(bad[order])[0]
    return int(pos[0]) if len(pos) else None


def test_ranked_prefix_reaches_the_planted_padding_bug_first(lib):
    """Config 2's candidate reads one tap past the right edge: only the last
    output column differs.  The ranked prefix reaches it within the corners;
    flat order needs a whole row first."""
    ref, cand = W.config(2, N=2, Ci=3, H=13, W=13, Co=5)
    gr, gc = D.Graph(ref), D.Graph(cand)
    R, C = oracle.Program(ref), oracle.Program(cand)
    locs = np.arange(R.out_numel)
    bad = ~(R.keys(locs) == C.keys(locs)).all(axis=1)
    assert bad.any()
    order, pre = D.query_order(gr, gc, seed=3)
    heur = _first_bug(order, bad)
    seq = _first_bug(locs, bad)
    assert heur is not None and heur < 2 ** len(gr.out_shape)   # within the corners
    assert seq >= 12


def test_mismatched_outputs_are_rejected(lib):
    a = D.Graph(W.config(1)[0])
    b = D.Graph(W.config(2)[0])
    with pytest.raises(D.DirigoError) as ei:
        D.query_order(a, b)
    assert ei.value.status == 8


def test_kernel_launch_corners_lead():
    """Sec. 4 "Search Heuristic", first tier: the locations written by the
    first and last thread of the first and last block, then threads 31 and
    32 of block 0.  For the tiled kernel (grid 1 x 4 x 3, block 1 x 16 x 8 on a
    50 x 24 output) whose last column tile reads W one column off, thread 0
    of the last block (block row 3, column tile 2) writes row 48, column 16:
    the first location that differs."""
    M, N = 50, 24
    ref, cand = W.tiled_matmul_kernel(M=M, N=N, TM=16, TN=8, bug="last_tile")
    order, prefix = D.query_order(D.Graph(ref), D.Graph(cand), seed=3)
    # block 0 thread 0; block 0 thread 127 (row 15, col 7); last block thread 0
    # (row 48, col 16); the last block's last thread is outside the path
    # condition (row 63); block 0 threads 31 (row 3, col 7) and 32 (row 4, col 0)
    want = [0, 15 * N + 7, 48 * N + 16, 3 * N + 7, 4 * N + 0]
    assert list(order[:5]) == want
    assert prefix >= 5 and sorted(order) == list(range(M * N))
    R, C = oracle.Program(ref), oracle.Program(cand)
    differs = np.any(R.keys(order) != C.keys(order), axis=1)
    assert int(np.argmax(differs)) == 2


ORDER_CASES = SMALL + [("tiled", None), ("pool", None), ("halfsum", None)]


def _pair(c, shape):
    if c == "tiled":
        return W.tiled_matmul_kernel(M=50, N=24, TM=16, TN=8, bug="last_tile")
    if c == "pool":
        return W.pool_kernel()
    if c == "halfsum":
        return W.halfsum_gelu(N=2, C=3, H=6, W=4)
    return W.config(c, **shape)


@pytest.mark.parametrize("c,shape", ORDER_CASES)
def test_order_matches_the_oracle_restatement(lib, c, shape):
    """dirigo_query_order against oracle/query_order.py: the head of the
    ranked prefix (kernel launch corners, output box corners, 31 and 32) is
    exactly the restated one, the first and last element are ranked, every
    cone-shape class of either program has a
    location in the prefix, and the tail is the restated seeded shuffle."""
    from oracle import query_order as QO
    ref, cand = _pair(c, shape)
    gr, gc = D.Graph(ref), D.Graph(cand)
    seed = 11
    order, pre = D.query_order(gr, gc, seed=seed)
    n = gr.out_numel
    head = QO.ranked_head(ref, cand)
    assert order[:len(head)].tolist() == head
    prefix = order[:pre].tolist()
    assert {0, n - 1} <= set(prefix)   # the first and last element (also box corners)
    locs = np.arange(n, dtype=np.int64)
    in_prefix = np.zeros(n, dtype=bool)
    in_prefix[prefix] = True
    for desc in (ref, cand):
        classes = QO.cone_shape_classes(oracle.Program(desc), locs)
        seen = {}
        for loc, cls in enumerate(classes):
            seen.setdefault(cls, False)
            seen[cls] |= bool(in_prefix[loc])
        assert all(seen.values()), [k for k, v in seen.items() if not v][:3]
    rest = sorted(set(range(n)) - set(prefix))
    assert order[pre:].tolist() == QO.shuffled_tail(rest, seed)
