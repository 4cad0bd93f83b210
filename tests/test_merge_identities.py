"""MERGE prefix trimming (Sec. 3.2 "MERGE") and the max-shifted softmax as a
sound identity (Sec. 4.2 "Sound identities").

CPU tests pin the oracle's trimming and rewrite against the direct fp64
forward pass (torch CPU library routines, which compute the shifted softmax
literally and know nothing of trimming).  GPU tests compare the library's
trimmed graphs (dirigo_graph_create_merged) and its lowering of the shifted
softmax with the oracle's, element by element.
"""
import numpy as np
import pytest

import oracle
from oracle import forward64
from oracle.lower import merge_trim
from paper_2609_19611_gb300 import workloads as W

C3_SMALL = dict(B=5, IN=40, OUT=24)
C4_SMALL = dict(N=2, Ci=3, H=6, W=6, Co=8, bug_co=5)


def _close64(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    scale = np.sqrt(np.mean(b ** 2)) + 1e-300
    return np.all(np.abs(a - b) <= 1e-12 * (np.abs(b) + scale))


def _cut_values(graph, vals, cut):
    """The cut tensors' values: the original program's own tensors."""
    ts = forward64.tensors(graph, vals)
    return [ts[t].numpy().copy() for t in cut]


def _mul_recip(cand):
    """The shifted softmax's last step written as e * recip(s)."""
    g = {"inputs": cand["inputs"], "ops": [dict(op) for op in cand["ops"]], "output": 7}
    g["ops"][5] = {"op": "recip", "args": [5]}
    g["ops"].append({"op": "mul", "args": [4, 6]})
    return g


# ------------------------------------------------------------------ oracle pins (CPU)

def test_trim_prefix_and_cut_c3():
    ref, cand = W.config(3, **C3_SMALL)
    r2, c2, cut, n = merge_trim(ref, cand)
    # linear and scale are shared; gamma, beta and the scaled activation cross the cut
    assert n == 2 and cut == [3, 4, 6]
    assert [s for _, s in r2["inputs"]] == [[24], [24], [5, 24]]
    assert r2["inputs"] == c2["inputs"]
    assert len(r2["ops"]) == len(ref["ops"]) - 2 and len(c2["ops"]) == len(cand["ops"]) - 2


@pytest.mark.parametrize("side", [0, 1])
def test_trim_preserves_the_function_c3(side):
    ref, cand = W.config(3, **C3_SMALL)
    trimmed = merge_trim(ref, cand)
    g, g2, cut = (ref, cand)[side], trimmed[side], trimmed[2]
    vals = W.random_values(ref, 31)
    want = forward64.flat_output(g, vals)
    got = forward64.flat_output(g2, _cut_values(g, vals, cut))
    assert _close64(got, want)
    # the oracle's own evaluation of the trimmed equations agrees as well
    P = oracle.Program(g2)
    assert _close64(P.eval(_cut_values(g, vals, cut), np.arange(P.out_numel)), want)


def test_trim_keeps_discharges_c3():
    ref, cand = W.config(3, **C3_SMALL)
    r2, c2, _, _ = merge_trim(ref, cand)
    R, C = oracle.Program(r2), oracle.Program(c2)
    q = np.arange(R.out_numel)
    assert np.array_equal(R.keys(q), C.keys(q))


def test_trim_identical_programs_keeps_the_last_op():
    ref, _ = W.config(4, **C4_SMALL)
    r2, c2, cut, n = merge_trim(ref, ref)
    assert n == len(ref["ops"]) - 1
    assert cut == sorted(set(ref["ops"][-1]["args"]))
    R, C = oracle.Program(r2), oracle.Program(c2)
    q = np.arange(R.out_numel)
    assert np.array_equal(R.keys(q), C.keys(q))


def test_trim_without_common_prefix():
    ref, cand = W.config(4, **C4_SMALL)   # the convolutions already differ
    r2, c2, cut, n = merge_trim(ref, cand)
    assert n == 0 and r2 is ref and c2 is cand and cut == [0, 1, 2]


def test_trim_rejects_different_inputs():
    ref, _ = W.config(4, **C4_SMALL)
    other, _ = W.config(4, **dict(C4_SMALL, H=8))
    with pytest.raises(ValueError):
        merge_trim(ref, other)


@pytest.mark.parametrize("form", ["div", "mul_recip"])
def test_shifted_softmax_identity(form):
    ref, cand = W.softmax_shift()
    if form == "mul_recip":
        cand = _mul_recip(cand)
    vals = W.random_values(ref, 5)
    # the identity itself, computed literally by the library routines
    y_ref, y_cand = forward64.flat_output(ref, vals), forward64.flat_output(cand, vals)
    assert _close64(y_cand, y_ref)
    R, C = oracle.Program(ref), oracle.Program(cand)
    q = np.arange(R.out_numel)
    assert np.array_equal(R.keys(q), C.keys(q))
    assert _close64(C.eval(vals, q), y_cand)


def test_shift_over_another_dim_is_not_the_identity():
    ref, cand = W.softmax_shift(shift_dim=2)
    vals = W.random_values(ref, 6)
    y_ref, y_cand = forward64.flat_output(ref, vals), forward64.flat_output(cand, vals)
    assert np.all(np.abs(y_ref - y_cand) > 1e-9)
    R, C = oracle.Program(ref), oracle.Program(cand)
    q = np.arange(R.out_numel)
    assert np.all(np.any(R.keys(q) != C.keys(q), axis=1))
    # lowered literally, as written
    assert _close64(C.eval(vals, q), y_cand)


# ------------------------------------------------------------------ GPU parity

@pytest.mark.gpu
@pytest.mark.parametrize("pair", ["c3", "identical"])
def test_merged_graphs_parity(pair):
    import torch
    from paper_2609_19611_gb300 import dirigo as D
    from tests.test_gpu_parity import check_cones, check_keys, check_compare, check_eval

    if pair == "c3":
        ref, cand = W.config(3, **C3_SMALL)
    else:
        ref, _ = W.config(4, **C4_SMALL)
        cand = ref
    r2, c2, cut, n = merge_trim(ref, cand)
    gr, gc, gcut, gn = D.merge(ref, cand)
    assert (gcut, gn) == (cut, n)

    class Case:
        pass

    case = Case()
    case.ref, case.cand = r2, c2
    case.R, case.C = oracle.Program(r2), oracle.Program(c2)
    case.gr, case.gc = gr, gc
    case.vals = [x.astype(np.float32) for x in _cut_values(ref, W.random_values(ref, 7), cut)]
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    kr, kc = check_keys(case, locs)
    assert np.array_equal(kr, kc)   # both pairs are equivalent
    v, _ = check_compare(case, locs)
    assert np.all(v == 0)
    check_eval(case, locs)
    torch.cuda.synchronize()


@pytest.mark.gpu
@pytest.mark.parametrize("variant", ["div", "mul_recip", "other_dim"])
def test_shifted_softmax_parity(variant):
    from tests.test_gpu_parity import Case, check_cones, check_keys, check_compare, check_eval

    ref, cand = W.softmax_shift(shift_dim=2 if variant == "other_dim" else 1)
    if variant == "mul_recip":
        cand = _mul_recip(cand)
    case = Case(ref, cand, seed=8)
    locs = np.arange(case.R.out_numel, dtype=np.int64)
    check_cones(case, locs)
    kr, kc = check_keys(case, locs)
    v, _ = check_compare(case, locs)
    if variant == "other_dim":
        assert np.all(v != 0)
    else:
        assert np.array_equal(kr, kc) and np.all(v == 0)
    check_eval(case, locs)


@pytest.mark.gpu
def test_merged_c3_full_size():
    """Config 3 at full size (linear 128 x 1024 -> 512, scale, LayerNorm) with
    the shared linear and scale trimmed: the trimmed pair over (gamma, beta,
    z) still discharges all 1,024 queried locations, keys and cones equal to
    the oracle's on its own trimmed programs."""
    import torch
    from paper_2609_19611_gb300 import dirigo as D
    from tests.test_gpu_parity import to_u32

    ref, cand = W.config(3)
    r2, c2, cut, n = merge_trim(ref, cand)
    gr, gc, gcut, gn = D.merge(ref, cand)
    assert (gcut, gn) == (cut, n) and n == 2
    q = W.make_queries(3, gr.out_numel)
    d = torch.as_tensor(q, device="cuda")
    R, C = oracle.Program(r2), oracle.Program(c2)
    kr, kc = D.terms(gr, d).cpu().numpy().astype(np.uint32), \
        D.terms(gc, d).cpu().numpy().astype(np.uint32)
    assert np.array_equal(kr, R.keys(q)) and np.array_equal(kc, C.keys(q))
    assert np.array_equal(kr, kc)
    off, runs, _ = D.cone(gr, d)
    o_off, o_runs = R.cone_runs(q[:64])
    assert np.array_equal(off.cpu().numpy()[:65], o_off)
    assert np.array_equal(to_u32(runs)[:o_off[-1]], o_runs)


def test_kernels_with_different_write_sets_are_not_a_common_prefix():
    """Two programs that start with kernels over the same arguments but with
    different write sets (one reads W a column off in its last tile) share no
    prefix: trimming must not cut them (it would discharge a real bug)."""
    from paper_2609_19611_gb300 import dirigo as D
    good = W.tiled_matmul_kernel()[1]                 # kernel, + bias, ReLU
    bad = W.tiled_matmul_kernel(bug="last_tile")[1]
    _, _, cut, n = merge_trim(good, bad)
    assert n == 0 and cut == [0, 1, 2]
    _, _, gcut, gn = D.merge(good, bad)
    assert (gcut, gn) == (cut, n)
    # the same kernel on both sides is a common prefix (kernel and bias add)
    _, _, cut2, n2 = merge_trim(good, good)
    _, _, gcut2, gn2 = D.merge(good, good)
    assert n2 == 2 and (gcut2, gn2) == (cut2, n2)
