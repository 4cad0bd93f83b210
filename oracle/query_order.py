"""Query order of a program pair, restated for the tests (Sec. 4, "Search
Heuristic": locations likely to expose a bug first, then a random order).

TEST INFRASTRUCTURE ONLY: used by ``tests/`` to check the library's
``dirigo_query_order``; it shares no code with the library.

The order is a ranked prefix, then every other location in a seeded random
permutation.  This module restates the parts of the ranking that have a plain
definition:

* the head of the prefix (Sec. 4: launch corners and warp boundaries):
  for every kernel op whose output location is the graph output's location
  (the output is reached from it through elementwise ops whose operand has
  the op's shape), later kernels first, candidate first, the output locations
  its corner threads write -- the first and last thread of the first and the
  last block, then threads 31 and 32 of block 0, blocks and threads numbered
  with x fastest, each thread's writes in write order; then every corner of
  the output box (corner m has coordinate d at its end when bit d of m is
  set) and flat indices 31 and 32; duplicates and locations outside the
  output dropped;
* the tail: the locations not in the prefix, ascending, shuffled by
  Fisher-Yates from the last position down, the k-th draw being the
  SplitMix64 output of seed + k * gamma (Steele, Lea and Flood 2014), taken
  modulo the number of positions left;
* the purpose of the middle of the prefix (one location per region of
  output space on which a program's cone has one structure, Sec. 4's "one
  satisfying location per path condition"): ``cone_shape_classes`` groups the
  output locations by their cone's shape (run count and run lengths), so that
  a test can check that every class of either program is represented.
"""
from __future__ import annotations

import numpy as np

from .lower import lower_full

GAMMA = 0x9E3779B97F4A7C15
M64 = (1 << 64) - 1

ELEMENTWISE_UNARY = {"scale", "add_scalar", "clamp_min", "relu", "gelu", "gelu_tanh", "tanh",
                     "exp", "rsqrt", "recip", "sigmoid", "erf", "sqrt", "log"}
ELEMENTWISE_BINARY = {"add", "sub", "mul", "div"}


def splitmix64(z):
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9 & M64
    z = (z ^ (z >> 27)) * 0x94D049BB133111EB & M64
    return z ^ (z >> 31)


def _hl_shapes(graph):
    return [list(s) for s in lower_full(graph)[3]]


def _aligned_kernels(graph):
    """Indices of the kernel ops whose output locations are the graph output's."""
    I = len(graph["inputs"])
    shapes = _hl_shapes(graph)
    aligned = [False] * len(shapes)
    aligned[graph["output"]] = True
    for k in range(len(graph["ops"]) - 1, -1, -1):
        op = graph["ops"][k]
        if not aligned[I + k]:
            continue
        kind = op["op"]
        if kind in ELEMENTWISE_BINARY:
            axes = op.get("axes")
            if axes is not None and not all(list(a) == list(range(len(a))) for a in axes):
                continue
        elif kind not in ELEMENTWISE_UNARY:
            continue
        for a in op["args"]:
            if shapes[a] == shapes[I + k]:
                aligned[a] = True
    return [k for k, op in enumerate(graph["ops"])
            if op["op"] in ("kernel_contract", "kernel_maxset") and aligned[I + k]]


def kernel_corner_locations(op):
    """Output locations the corner threads of a kernel launch write."""
    gz, gy, gx = op["grid"]
    bz, by, bx = op["block"]
    nb, nt = gz * gy * gx, bz * by * bx
    out = []
    for t, b in ((0, 0), (nt - 1, 0), (0, nb - 1), (nt - 1, nb - 1), (31, 0), (32, 0)):
        if t >= nt:
            continue
        theta = (b // (gy * gx), (b // gx) % gy, b % gx, t // (by * bx), (t // bx) % by, t % bx)
        for w in op["writes"]:
            when = w.get("when", [[0, 1 << 62]] * 6)
            if all(lo <= th < hi for th, (lo, hi) in zip(theta, when)):
                a0, ac = w["addr"]
                a = a0 + sum(c * th for c, th in zip(ac, theta))
                if a not in out:
                    out.append(a)
    return out


def ranked_head(ref, cand):
    """The head of the ranked prefix (see the module docstring)."""
    shape = _hl_shapes(ref)[ref["output"]]
    n = int(np.prod(shape))
    seq = []
    for g in (cand, ref):
        for k in reversed(_aligned_kernels(g)):
            seq.extend(kernel_corner_locations(g["ops"][k]))
    for m in range(1 << len(shape)):
        c = [(s - 1) if (m >> d) & 1 else 0 for d, s in enumerate(shape)]
        seq.append(int(np.ravel_multi_index(c, shape)) if shape else 0)
    seq.extend([31, 32])
    head = []
    for loc in seq:
        if 0 <= loc < n and loc not in head:
            head.append(loc)
    return head


def shuffled_tail(rest, seed):
    """Fisher-Yates over `rest` (ascending) with the SplitMix64 draws of seed."""
    a = list(rest)
    state = seed & M64
    for i in range(len(a) - 1, 0, -1):
        state = (state + GAMMA) & M64
        j = splitmix64(state) % (i + 1)
        a[i], a[j] = a[j], a[i]
    return a


def cone_shape_classes(program, locs):
    """Class of each location: (run count, run lengths) of its cone."""
    off, runs = program.cone_runs(np.asarray(locs, dtype=np.int64))
    return [(int(off[i + 1] - off[i]), tuple(runs[off[i]:off[i + 1], 1].tolist()))
            for i in range(len(locs))]
