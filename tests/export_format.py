"""Reader for the exported term-list format (used by round-trip tests).

Layout (little-endian): a 32-byte header {u32 magic "DXP1", u32 version,
u64 total_bytes, u64 n_locations, u64 0}; then for program 0 (reference) and
program 1 (candidate) {u64 n_nodes, u64 n_entries, nodes[n_nodes] (32 bytes:
u32 tensor, u8 kind, u8 fn, u16 0, u64 elem, u64 entry_begin, u64 n_entries),
entries[n_entries] (24 bytes: f64 coef, u64 a, u64 b)}; then n_locations
records {u64 slot, u64 root_ref_program0, u64 root_ref_program1}.
A ref with bit 63 set is node (tensor = bits 40..62, elem = bits 0..39),
~0 is "none", anything else a global leaf id (the largest, G, is bottom).
"""
import math
import struct

import numpy as np

NODE_BIT = 1 << 63
NONE = (1 << 64) - 1
SUM, MAX, FUNC, DIV = 1, 2, 3, 4


def parse(blob):
    magic, version, total, nloc, _ = struct.unpack_from("<IIQQQ", blob, 0)
    assert magic == 0x31505844 and version == 1 and total == len(blob)
    pos = 32
    progs = []
    for _ in range(2):
        nn, ne = struct.unpack_from("<QQ", blob, pos)
        pos += 16
        nodes = {}
        order = []
        for i in range(nn):
            t, kind, fn, _pad, e, b, n = struct.unpack_from("<IBBHQQQ", blob, pos)
            pos += 32
            nodes[(t, e)] = (kind, fn, b, n)
            order.append((t, e))
        ents = []
        for i in range(ne):
            c, a, b = struct.unpack_from("<dQQ", blob, pos)
            pos += 24
            ents.append((c, a, b))
        progs.append({"nodes": nodes, "order": order, "entries": ents})
    locs = []
    for i in range(nloc):
        locs.append(struct.unpack_from("<QQQ", blob, pos))
        pos += 24
    assert pos == len(blob)
    return progs, locs


_UF = {1: math.exp, 2: math.tanh,
       3: lambda x: 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0))),
       4: lambda x: 0.5 * x * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) *
                                              (x + 0.044715 * x ** 3))),
       5: math.erf, 6: lambda x: 1.0 / math.sqrt(x), 7: lambda x: 1.0 / x,
       8: math.sqrt, 9: math.log}


def evaluate(prog, ref, leaf_value, memo=None):
    """fp64 value of a ref in one program's exported DAG."""
    memo = {} if memo is None else memo
    if ref == NONE:
        raise ValueError("none ref")
    if not ref & NODE_BIT:
        return leaf_value(ref)
    key = ((ref >> 40) & ((1 << 23) - 1), ref & ((1 << 40) - 1))
    if key in memo:
        return memo[key]
    kind, fn, b, n = prog["nodes"][key]
    ents = prog["entries"][b:b + n]

    def val(r):
        return evaluate(prog, r, leaf_value, memo)

    if kind == SUM:
        v = 0.0
        for c, x, y in ents:
            t = c
            if x != NONE:
                t *= val(x)
            if y != NONE:
                t *= val(y)
            v += t
    elif kind == MAX:
        v = max((c if x == NONE else val(x)) for c, x, _ in ents)
    elif kind == FUNC:
        v = _UF[fn](val(ents[0][1]))
    elif kind == DIV:
        v = val(ents[0][1]) / val(ents[0][2])
    else:
        raise ValueError(kind)
    memo[key] = v
    return v


def leaf_lookup(inputs):
    flat = np.concatenate([np.asarray(x, dtype=np.float64).ravel() for x in inputs])

    def f(g):
        return float(flat[g]) if g < flat.size else float("nan")
    return f
