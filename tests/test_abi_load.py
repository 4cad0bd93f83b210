"""The C-ABI library loads without a GPU, exports every declared entry point,
and its host-side index-map compiler accepts and rejects graph descriptions
as documented (no device call is made here)."""
import os
import re

import numpy as np
import pytest

import oracle
from paper_2609_19611_gb300 import build, dirigo as D, workloads as W

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "dirigo.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return D.load()


def declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dirigo_[a-z_0-9]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    names = declared()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(D.SIGNATURES)


@pytest.mark.parametrize("c", [1, 2, 3, 4, 5])
def test_graph_create_matches_oracle_shapes(lib, c):
    for g in W.config(c):
        G = D.Graph(g)
        P = oracle.Program(g)
        assert G.G == P.G and G.out_numel == P.out_numel
        assert G.out_shape == W.out_shape(g)
        assert G.n_tensors == len(oracle.lower(g)[1]) + len(g["inputs"])


def test_primitive_tensor_count_matches_lowering_table(lib):
    for seed in range(30):
        a, b, _ = W.random_pair(seed)
        for g in (a, b):
            assert D.Graph(g).n_tensors == len(oracle.lower(g)[1]) + len(g["inputs"])


def test_rejects_bad_descriptions(lib):
    ref, _ = W.config(1)
    bad = dict(ref, ops=[{"op": "matmul", "args": [0, 2]}], output=3)    # [8,16] x [8]
    with pytest.raises(D.DirigoError) as e:
        D.Graph(bad)
    assert e.value.status == 2
    bad = dict(ref, ops=[{"op": "relu", "args": [7]}], output=3)          # not a tensor yet
    with pytest.raises(D.DirigoError) as e:
        D.Graph(bad)
    assert e.value.status == 1
    bad = dict(ref, ops=ref["ops"], output=0)                               # output is an input
    with pytest.raises(D.DirigoError) as e:
        D.Graph(bad)
    assert e.value.status == 1
    big = {"inputs": [["x", [2, 2, 2, 2, 2]]], "ops": [{"op": "relu", "args": [0]}], "output": 1}
    with pytest.raises(D.DirigoError) as e:
        D.Graph(big)
    assert e.value.status == 3


@pytest.mark.parametrize("name,graph", [
    ("broadcast", {"inputs": [["a", [3, 4]], ["b", [5]]], "ops": [{"op": "add", "args": [0, 1]}]}),
    ("conv channels", {"inputs": [["x", [1, 3, 8, 8]], ["w", [4, 2, 3, 3]]],
                       "ops": [{"op": "conv2d", "args": [0, 1], "padding": 1}]}),
    ("softmax dim", {"inputs": [["x", [2, 3]]], "ops": [{"op": "softmax", "args": [0], "dim": 2}]}),
    ("layernorm gamma", {"inputs": [["z", [2, 6]], ["g", [5]], ["b", [6]]],
                         "ops": [{"op": "layernorm", "args": [0, 1, 2]}]}),
    ("linear in", {"inputs": [["x", [2, 6]], ["w", [4, 5]], ["b", [4]]],
                   "ops": [{"op": "linear", "args": [0, 1, 2]}]}),
    ("bmm batch", {"inputs": [["a", [2, 3, 4]], ["b", [3, 4, 5]]], "ops": [{"op": "bmm", "args": [0, 1]}]}),
    ("pool window", {"inputs": [["x", [1, 1, 5, 5]]], "ops": [{"op": "maxpool2d", "args": [0], "k": 6}]}),
    ("empty extent", {"inputs": [["x", [2, 0]]], "ops": [{"op": "relu", "args": [0]}]}),
])
def test_rejects_mismatched_shapes(lib, name, graph):
    g = dict(graph, output=len(graph["inputs"]))
    with pytest.raises(D.DirigoError) as e:
        D.Graph(g)
    assert e.value.status == 2, name   # DIRIGO_E_SHAPE


def test_accepts_pytorch_shape_rules(lib):
    """Broadcasting of trailing dims, and a pooling window that does not tile
    the image (the output is floor((H - k) / s) + 1 wide, as in PyTorch)."""
    g = {"inputs": [["a", [3, 4]], ["b", [4]]], "ops": [{"op": "add", "args": [0, 1]}], "output": 2}
    assert D.Graph(g).out_shape == [3, 4]
    g = {"inputs": [["x", [1, 1, 5, 5]]], "ops": [{"op": "maxpool2d", "args": [0], "k": 2}],
         "output": 1}
    assert D.Graph(g).out_shape == [1, 1, 2, 2] == W.out_shape(g)
    with pytest.raises(ValueError):
        D.Graph({"inputs": [["x", [2, 3]]], "ops": [{"op": "frobnicate", "args": [0]}],
                 "output": 1})


def test_workspace_sizes(lib):
    ref, cand = W.config(4)
    g = D.Graph(ref)
    # terms: leaf keys (G + 1) and one key pair per element of every primitive tensor
    prims = oracle.lower(ref)[1]
    elems = sum(int(np.prod(p["shape"])) for p in prims)
    assert g.workspace_size(D.CALL_TERMS, 10) >= 8 * (g.G + 1) + 8 * elems
    assert g.workspace_size(D.CALL_EVAL, 10) >= 4 * elems


@pytest.mark.parametrize("c", [1, 2, 3, 4, 5])
def test_cone_cells_cover_the_workloads(lib, c):
    """Every benchmark program's output space splits into a handful of cone
    cells; only the candidate of the padding off-by-one keeps generic cells
    (its reads past a row end overlap the box of the next row)."""
    for i, g in enumerate(W.config(c)):
        G = D.Graph(g)
        assert 0 < G.n_cells <= 1024
        if c == 2 and i == 1:
            assert 0 < G.n_cells - G.n_fast_cells <= 8
        else:
            assert G.n_fast_cells == G.n_cells
