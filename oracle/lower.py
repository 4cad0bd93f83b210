"""Oracle side: high-level op graph -> per-element equations (primitive ops).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package;
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
do.  It shares no code with the CUDA path.

The paper treats each Torch op as having a predefined per-element equation
T_k[l] = f_k(l) over elements of earlier tensors (Sec. 3.3 "Torch Operations",
Sec. 3.4 "Per-element equations").  This module writes those equations out,
op by op, from the textbook definition of each op.  The primitive kinds are

* ``contract``  T[o] = sum over pieces p containing o, over r in p's reduction
                box with all guards true, of coef_p * prod_i arg_i[off_{p,i}(o,r)]
* ``maxset``    T[o] = Max{ arg[off_p(o,r)] : same enumeration }
* ``unary``     T[o] = f(arg[o]) for an uninterpreted function f
* ``maxc``      T[o] = Max{ arg[o], c }
* ``affine``    T[o] = a * arg[o] + c
* ``binary``    T[o] = arg0[o|a] (+ - * /) arg1[o|b] with broadcasting

An access offset outside the operand reads the undefined value (the paper's
bottom, Sec. 3.3 "Intra-Warp Reduction", last paragraph).

The order in which a composite op emits its primitive tensors (softmax:
exp, sum, recip, mul; layernorm: mean, sub, mul, mean, +eps, rsqrt, mul,
mul gamma, add beta) fixes the node numbering of exported term lists; it is
the one interface shared by name with the CUDA path's compiler.

Also here, each written from its passage and independently of the CUDA
path's compiler:

* ``kernel_pieces``   a kernel given by its write set (Sec. 3.4 "Per-element
                      equations"): every thread of the launch is run and the
                      writer of each location recorded -- one piece per output
                      element, so only for test-sized kernels;
* ``shifted_softmax`` the max-shifted softmax written out is lowered as the
                      softmax it equals (Sec. 4.2 "Sound identities");
* ``merge_trim``      MERGE prefix trimming (Sec. 3.2 "MERGE").
"""
from __future__ import annotations

import itertools
from fractions import Fraction

UF = {"exp": 1, "tanh": 2, "gelu_erf": 3, "gelu_tanh": 4, "erf": 5,
      "rsqrt": 6, "recip": 7, "sqrt": 8, "log": 9}


def const(x):
    """Exact rational value of a constant given as float, int or [num, den]."""
    if isinstance(x, (list, tuple)):
        return Fraction(int(x[0]), int(x[1]))
    if isinstance(x, float):
        return Fraction(x)          # exact binary value of the double
    return Fraction(x)


def _numel(shape):
    n = 1
    for s in shape:
        n *= s
    return n


def _strides(shape):
    st, acc = [0] * len(shape), 1
    for i in range(len(shape) - 1, -1, -1):
        st[i] = acc
        acc *= shape[i]
    return st


def _trailing_axes(rank_op, rank_out):
    return list(range(rank_out - rank_op, rank_out))


def kernel_writers(op):
    """Who writes each output location of a kernel op: every thread of the
    launch (grid z, y, x then block z, y, x) evaluates the path condition of
    every write and records the address it stores to.  Returns a dict
    location -> (write index, thread coordinates).  Two stores to one
    location, or a store outside the output, raise ValueError."""
    total = _numel(op["shape"])
    launch = list(op["grid"]) + list(op["block"])
    writer = {}
    for wi, w in enumerate(op["writes"]):
        when = w.get("when", [[0, 1 << 62]] * 6)
        ranges = [range(max(0, lo), min(n, hi)) for (lo, hi), n in zip(when, launch)]
        a0, ac = w["addr"]
        for th in itertools.product(*ranges):
            a = a0 + sum(c * t for c, t in zip(ac, th))
            if not 0 <= a < total:
                raise ValueError("a kernel thread writes outside its output")
            if a in writer:
                raise ValueError("two kernel threads write one location")
            writer[a] = (wi, th)
    return writer


def kernel_pieces(op):
    """Per-element equations of a kernel op (Sec. 3.4 "Per-element
    equations": the equation at l is the value of the thread whose write
    address is l), one piece per output element: the writer's reduction box,
    coefficient and guards, with its thread coordinates substituted into the
    reads and guards.  A location no thread writes holds the undefined value:
    one term whose operands are all read out of range."""
    shape = list(op["shape"])
    R = len(shape)
    writer = kernel_writers(op)
    pieces = []
    for l in range(_numel(shape)):
        o, x = [0] * R, l
        for d in range(R - 1, -1, -1):
            o[d] = x % shape[d]
            x //= shape[d]
        lo, hi = list(o), [v + 1 for v in o]
        if l not in writer:
            pieces.append({"lo": lo, "hi": hi, "red": [[0, 1]], "coef": Fraction(1),
                           "guards": [],
                           "access": [[-1, [0] * R, [0]] for _ in op["args"]]})
            continue
        wi, th = writer[l]
        w = op["writes"][wi]
        dot = lambda tc: sum(a * b for a, b in zip(tc, th))   # noqa: E731
        pieces.append({
            "lo": lo, "hi": hi, "red": [list(r) for r in w["red"]],
            "coef": const(w.get("coef", 1.0)),
            "guards": [[-1, 0, rd, c + dot(tc), glo, ghi]
                       for tc, rd, c, glo, ghi in w.get("guards", [])],
            "access": [[base + dot(tc), [0] * R, list(rs)] for base, tc, rs in w["reads"]]})
    return pieces


def _plain_axes(op):
    """No operand axes given, or each operand's dims mapped to themselves."""
    axes = op.get("axes")
    return axes is None or all(list(a) == list(range(len(a))) for a in axes)


def shifted_softmax(graph, k, rank_of):
    """Sound identity (Sec. 4.2 "Sound identities"): softmax(x - max x) over a
    dim equals softmax(x) over the reals.  When op k ends a max-shifted
    softmax written out --

        m = max(x, d, keepdim)   z = sub(x, m)   e = exp(z)
        s = sum(e, d, keepdim)   y = div(e, s)  or  mul(e, recip(s))

    -- return (x, d) (d counted from 0), else None.  ``rank_of(t)`` is the
    rank of high-level tensor t."""
    n_in, ops = len(graph["inputs"]), graph["ops"]

    def op_at(t):
        return ops[t - n_in] if n_in <= t < n_in + len(ops) else None

    y = ops[k]
    if len(y["args"]) != 2 or not _plain_axes(y):
        return None
    e_id = y["args"][0]
    if y["op"] == "div":
        s_id = y["args"][1]
    elif y["op"] == "mul":
        r = op_at(y["args"][1])
        if r is None or r["op"] != "recip":
            return None
        s_id = r["args"][0]
    else:
        return None
    e, s = op_at(e_id), op_at(s_id)
    if e is None or s is None or e["op"] != "exp" or s["op"] != "sum":
        return None
    if list(s["args"]) != [e_id] or not s.get("keepdim", False):
        return None
    z = op_at(e["args"][0])
    if z is None or z["op"] != "sub" or not _plain_axes(z):
        return None
    x, m_id = z["args"]
    m = op_at(m_id)
    if m is None or m["op"] != "max" or list(m["args"]) != [x] or not m.get("keepdim", False):
        return None
    rank = rank_of(x)
    dims = []
    for d in (m["dim"], s["dim"]):
        d = d + rank if d < 0 else d
        if not 0 <= d < rank:
            return None
        dims.append(d)
    return (x, dims[0]) if dims[0] == dims[1] else None


def lower(graph):
    """Return (inputs, prims, output) with prims a list of primitive op dicts.

    inputs: list of shapes; tensor ids 0..I-1 are the inputs, I.. the prims.
    """
    inputs, prims, out, _ = lower_full(graph)
    return inputs, prims, out


def lower_full(graph):
    """lower(), plus the shape of every high-level tensor (inputs, then one
    per op)."""
    inputs = [list(s) for _, s in graph["inputs"]]
    shapes = list(inputs)
    prims = []
    hl2t = list(range(len(inputs)))        # high-level tensor id -> prim id

    def emit(p):
        prims.append(p)
        shapes.append(list(p["shape"]))
        return len(shapes) - 1

    def reduce_access(shape, dim, keepdim):
        st = _strides(shape)
        os_ = []
        for i in range(len(shape)):
            if i == dim:
                if keepdim:
                    os_.append(0)
                continue
            os_.append(st[i])
        out = [1 if i == dim else s for i, s in enumerate(shape)] if keepdim \
            else [s for i, s in enumerate(shape) if i != dim]
        return out, [0, os_, [st[dim]]]

    def reduction(kind, a, dim, keepdim, coef):
        shp = shapes[a]
        dim %= len(shp)
        out, acc = reduce_access(shp, dim, keepdim)
        piece = {"lo": [0] * len(out), "hi": list(out), "red": [[0, shp[dim]]],
                 "coef": coef, "guards": [], "access": [acc]}
        return emit({"kind": kind, "args": [a], "shape": out, "pieces": [piece]})

    def binary(fn, a, b, axes=None):
        sa, sb = shapes[a], shapes[b]
        if axes is None:
            r = max(len(sa), len(sb))
            axes = [_trailing_axes(len(sa), r), _trailing_axes(len(sb), r)]
        r = max(max(axes[0], default=-1), max(axes[1], default=-1)) + 1
        out = [1] * r
        for s, ax in ((sa, axes[0]), (sb, axes[1])):
            for d, o in enumerate(ax):
                if s[d] != 1:
                    if out[o] not in (1, s[d]):
                        raise ValueError("broadcast mismatch")
                    out[o] = s[d]
        return emit({"kind": "binary", "fn": fn, "args": [a, b],
                     "axes": [list(axes[0]), list(axes[1])], "shape": out})

    def unary(fn, a):
        return emit({"kind": "unary", "fn": fn, "args": [a], "shape": shapes[a]})

    def affine(a, mul, add):
        return emit({"kind": "affine", "a": mul, "c": add, "args": [a],
                     "shape": shapes[a]})

    for idx, op in enumerate(graph["ops"]):
        k = op["op"]
        A = [hl2t[t] for t in op["args"]]
        shift = shifted_softmax(graph, idx, lambda t: len(shapes[hl2t[t]]))
        if shift is not None:   # lowered as the softmax it equals
            k, A, op = "softmax", [hl2t[shift[0]]], {"op": "softmax", "dim": shift[1]}
        if k == "matmul":
            (M, K), (_, N) = shapes[A[0]], shapes[A[1]]
            pc = {"lo": [0, 0], "hi": [M, N], "red": [[0, K]], "coef": Fraction(1),
                  "guards": [], "access": [[0, [K, 0], [1]], [0, [0, 1], [N]]]}
            t = emit({"kind": "contract", "args": A[:2], "shape": [M, N], "pieces": [pc]})
        elif k == "bmm":
            (B, M, K), (_, _, N) = shapes[A[0]], shapes[A[1]]
            pc = {"lo": [0, 0, 0], "hi": [B, M, N], "red": [[0, K]], "coef": Fraction(1),
                  "guards": [], "access": [[0, [M * K, K, 0], [1]],
                                           [0, [K * N, 0, 1], [N]]]}
            t = emit({"kind": "contract", "args": A[:2], "shape": [B, M, N], "pieces": [pc]})
        elif k == "linear":
            (B, IN), (OUT, _) = shapes[A[0]], shapes[A[1]]
            pc = {"lo": [0, 0], "hi": [B, OUT], "red": [[0, IN]], "coef": Fraction(1),
                  "guards": [], "access": [[0, [IN, 0], [1]], [0, [0, IN], [1]]]}
            t = emit({"kind": "contract", "args": A[:2], "shape": [B, OUT], "pieces": [pc]})
            if len(A) > 2:
                t = binary("add", t, A[2], [[0, 1], [1]])
        elif k == "conv2d":
            N, Ci, H, W = shapes[A[0]]
            Co, _, kh, kw = shapes[A[1]]
            s, p = op.get("stride", 1), op.get("pad", 0)
            Ho, Wo = (H + 2 * p - kh) // s + 1, (W + 2 * p - kw) // s + 1
            # X[n, ci, s*h + i - p, s*w + j - p] * W[co, ci, i, j], taps outside the
            # image are absent (zero padding contributes no term)
            pc = {"lo": [0, 0, 0, 0], "hi": [N, Co, Ho, Wo],
                  "red": [[0, Ci], [0, kh], [0, kw]], "coef": Fraction(1),
                  "guards": [[2, s, 1, -p, 0, H], [3, s, 2, -p, 0, W]],
                  "access": [[-p * W - p, [Ci * H * W, 0, s * W, s], [H * W, W, 1]],
                             [0, [0, Ci * kh * kw, 0, 0], [kh * kw, kw, 1]]]}
            t = emit({"kind": "contract", "args": A[:2], "shape": [N, Co, Ho, Wo],
                      "pieces": [pc]})
            if len(A) > 2:
                t = binary("add", t, A[2], [[0, 1, 2, 3], [1]])
        elif k == "maxpool2d":
            N, C, H, W = shapes[A[0]]
            kk, s = op["k"], op.get("stride", op["k"])
            Ho, Wo = (H - kk) // s + 1, (W - kk) // s + 1
            pc = {"lo": [0, 0, 0, 0], "hi": [N, C, Ho, Wo], "red": [[0, kk], [0, kk]],
                  "coef": Fraction(1), "guards": [],
                  "access": [[0, [C * H * W, H * W, s * W, s], [W, 1]]]}
            t = emit({"kind": "maxset", "args": A[:1], "shape": [N, C, Ho, Wo],
                      "pieces": [pc]})
        elif k in ("add", "sub", "mul", "div"):
            t = binary(k, A[0], A[1], op.get("axes"))
        elif k == "scale":
            t = affine(A[0], const(op["c"]), Fraction(0))
        elif k == "add_scalar":
            t = affine(A[0], Fraction(1), const(op["c"]))
        elif k == "clamp_min":
            t = emit({"kind": "maxc", "c": const(op["c"]), "args": A[:1],
                      "shape": shapes[A[0]]})
        elif k == "relu":
            t = emit({"kind": "maxc", "c": Fraction(0), "args": A[:1],
                      "shape": shapes[A[0]]})
        elif k == "gelu":
            t = unary("gelu_erf", A[0])
        elif k in ("gelu_tanh", "tanh", "exp", "rsqrt", "recip", "erf", "sqrt", "log"):
            t = unary(k, A[0])
        elif k == "sigmoid":   # sound identity: sigmoid(x) = recip(1 + exp(-x))
            t = affine(A[0], Fraction(-1), Fraction(0))
            t = unary("exp", t)
            t = affine(t, Fraction(1), Fraction(1))
            t = unary("recip", t)
        elif k == "sum":
            t = reduction("contract", A[0], op["dim"], op.get("keepdim", False), Fraction(1))
        elif k == "mean":
            D = shapes[A[0]][op["dim"] % len(shapes[A[0]])]
            t = reduction("contract", A[0], op["dim"], op.get("keepdim", False),
                          Fraction(1, D))
        elif k == "max":
            t = reduction("maxset", A[0], op["dim"], op.get("keepdim", False), Fraction(1))
        elif k == "softmax":
            # s_c = exp(x_c) * recip(sum_c' exp(x_c')) (no max shift: equal over R)
            e = unary("exp", A[0])
            sm = reduction("contract", e, op["dim"], True, Fraction(1))
            rc = unary("recip", sm)
            t = binary("mul", e, rc)
        elif k == "layernorm":
            z = A[0]
            D = shapes[z][-1]
            mu = reduction("contract", z, -1, True, Fraction(1, D))
            d = binary("sub", z, mu)
            q = binary("mul", d, d)
            v = reduction("contract", q, -1, True, Fraction(1, D))
            ve = affine(v, Fraction(1), const(op.get("eps", 1e-5)))
            rs = unary("rsqrt", ve)
            t = binary("mul", d, rs)
            if len(A) > 1:
                t = binary("mul", t, A[1])
            if len(A) > 2:
                t = binary("add", t, A[2])
        elif k in ("kernel_contract", "kernel_maxset"):
            t = emit({"kind": k[len("kernel_"):], "args": A, "shape": list(op["shape"]),
                      "pieces": kernel_pieces(op)})
        elif k in ("contract", "maxset"):
            pieces = []
            for pc in op["pieces"]:
                pieces.append({"lo": list(pc.get("lo", [0] * len(op["shape"]))),
                               "hi": list(pc.get("hi", op["shape"])),
                               "red": [list(x) for x in pc["red"]],
                               "coef": const(pc.get("coef", 1.0)),
                               "guards": [list(g) for g in pc.get("guards", [])],
                               "access": [[a[0], list(a[1]), list(a[2])]
                                          for a in pc["access"]]})
            t = emit({"kind": k, "args": A, "shape": list(op["shape"]), "pieces": pieces})
        else:
            raise ValueError(f"unknown op {k}")
        hl2t.append(t)
    return inputs, prims, hl2t[graph["output"]], [list(shapes[t]) for t in hl2t]


# ----------------------------------------------------------------------------
# MERGE prefix trimming (Sec. 3.2 "MERGE")
# ----------------------------------------------------------------------------

def _op_meaning(op):
    """What an op computes: kind, arguments and the attributes its lowering
    reads, with the lowering's defaults filled in."""
    k = op["op"]
    key = [k, tuple(op["args"])]
    if k == "conv2d":
        key += [op.get("stride", 1) or 1, op.get("pad", 0)]
    elif k == "maxpool2d":
        key += [op["k"], op.get("stride", op["k"]) or op["k"]]
    elif k in ("add", "sub", "mul", "div"):
        ax = op.get("axes")
        key.append(None if ax is None else tuple(tuple(a) for a in ax))
    elif k in ("scale", "add_scalar", "clamp_min"):
        key.append(const(op["c"]))
    elif k == "layernorm":
        key.append(const(op.get("eps", 1e-5)))
    elif k in ("sum", "mean", "max"):
        key += [op["dim"], bool(op.get("keepdim", False))]
    elif k == "softmax":
        key.append(op["dim"])
    elif k in ("kernel_contract", "kernel_maxset"):
        key += [tuple(op["shape"]), tuple(op["grid"]), tuple(op["block"])]
        for w in op["writes"]:
            key.append((tuple(tuple(x) for x in w.get("when", [[0, 1 << 62]] * 6)),
                        w["addr"][0], tuple(w["addr"][1]),
                        tuple(tuple(x) for x in w["red"]), const(w.get("coef", 1.0)),
                        tuple((tuple(g[0]),) + tuple(g[1:]) for g in w.get("guards", [])),
                        tuple((r[0], tuple(r[1]), tuple(r[2])) for r in w["reads"])))
    elif k in ("contract", "maxset"):
        key.append(tuple(op["shape"]))
        for pc in op["pieces"]:
            key.append((tuple(pc.get("lo", [0] * len(op["shape"]))),
                        tuple(pc.get("hi", op["shape"])),
                        tuple(tuple(x) for x in pc["red"]), const(pc.get("coef", 1.0)),
                        tuple(tuple(g) for g in pc.get("guards", [])),
                        tuple((a[0], tuple(a[1]), tuple(a[2])) for a in pc["access"])))
    return tuple(key)


def merge_trim(ref, cand):
    """Cut the longest common op prefix of two programs over the same inputs.

    Returns (ref', cand', cut, n_shared): both programs rewritten so that
    their inputs are the tensors ``cut`` (ids in the given numbering,
    ascending) that the rest of either program reads from the prefix; each
    program keeps the op that computes its output.  With no common prefix the
    programs are returned as given and ``cut`` lists their inputs."""
    if [list(s) for _, s in ref["inputs"]] != [list(s) for _, s in cand["inputs"]]:
        raise ValueError("the programs declare different inputs")
    n_in = len(ref["inputs"])
    last = min(ref["output"], cand["output"]) - n_in
    n = 0
    while (n < len(ref["ops"]) and n < len(cand["ops"]) and n < last and
           _op_meaning(ref["ops"][n]) == _op_meaning(cand["ops"][n])):
        n += 1
    if n == 0:
        return ref, cand, list(range(n_in)), 0
    used = set()
    for g in (ref, cand):
        for op in g["ops"][n:]:
            used.update(t for t in op["args"] if t < n_in + n)
    cut = sorted(used)
    shapes = lower_full(ref)[3]

    def rewrite(g):
        new = {t: i for i, t in enumerate(cut)}
        for j in range(n, len(g["ops"])):
            new[n_in + j] = len(cut) + (j - n)
        ops = []
        for op in g["ops"][n:]:
            o = dict(op)
            o["args"] = [new[t] for t in op["args"]]
            ops.append(o)
        return {"inputs": [[f"t{t}", list(shapes[t])] for t in cut], "ops": ops,
                "output": new[g["output"]]}

    return rewrite(ref), rewrite(cand), cut, n


# ----------------------------------------------------------------------------
# flat encoding for the C++ interpreter (oracle-private format)
# ----------------------------------------------------------------------------

KIND = {"contract": 1, "maxset": 2, "unary": 3, "maxc": 4, "affine": 5, "binary": 6}
BIN = {"add": 1, "sub": 2, "mul": 3, "div": 4}


def _enc_const(f):
    """Fraction -> (m, e, d) with value m * 2**e / d, m and d odd (or m = 0)."""
    f = Fraction(f)
    if f == 0:
        return [0, 0, 1]
    n, d = f.numerator, f.denominator
    e = 0
    while n % 2 == 0:
        n //= 2
        e += 1
    while d % 2 == 0:
        d //= 2
        e -= 1
    if abs(n) >= 2 ** 62 or d >= 2 ** 62:
        raise ValueError("constant too large for the oracle encoding")
    return [n, e, d]


def encode(graph):
    inputs, prims, out = lower(graph)
    w = [len(inputs), len(prims), out]
    for s in inputs:
        w += [len(s)] + list(s)
    for p in prims:
        kind = KIND[p["kind"]]
        fn = UF.get(p.get("fn"), 0) if kind == 3 else BIN.get(p.get("fn"), 0)
        w += [kind, fn, len(p["args"])] + list(p["args"])
        w += [len(p["shape"])] + list(p["shape"])
        if kind in (1, 2):
            w += [len(p["pieces"])]
            for pc in p["pieces"]:
                w += list(pc["lo"]) + list(pc["hi"])
                w += [len(pc["red"])]
                for lo, hi in pc["red"]:
                    w += [lo, hi]
                w += _enc_const(pc["coef"])
                w += [len(pc["guards"])]
                for g in pc["guards"]:
                    w += list(g)
                for a in pc["access"]:
                    w += [a[0]] + list(a[1]) + list(a[2])
        elif kind == 4:
            w += _enc_const(p["c"])
        elif kind == 5:
            w += _enc_const(p["a"]) + _enc_const(p["c"])
        elif kind == 6:
            w += [len(p["axes"][0])] + list(p["axes"][0])
            w += [len(p["axes"][1])] + list(p["axes"][1])
    return w
