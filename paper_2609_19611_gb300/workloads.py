"""Seeded synthetic workloads: graph descriptions, query batches and input values.

This module only *describes* the two programs of each equivalence query (the
reference and the candidate, as op graphs) and draws seeded inputs for them.
It holds none of the checking method's arithmetic (no cones, no terms, no
keys, no evaluation), and it imports nothing else from this package, so the
CPU oracle under ``oracle/`` and the CUDA path can both be fed from it.

Graph description (plain dict, JSON-serialisable)
-------------------------------------------------
``{"inputs": [[name, shape], ...], "ops": [op, ...], "output": tid}``

Tensor ids: inputs are ``0 .. I-1`` in declared order, then one id per op in
SSA order.  An op is ``{"op": kind, "args": [tid, ...], **attrs}`` with kind one
of

* ``matmul`` [M,K]x[K,N]; ``bmm`` [B,M,K]x[B,K,N]; ``linear`` (x[B,in], W[out,in], b[out]?)
* ``conv2d`` (X NCHW, W [Co,Ci,kh,kw], b[Co]?) with ``stride``, ``pad``
* ``maxpool2d`` with ``k``, ``stride``
* ``add`` ``sub`` ``mul`` ``div`` (broadcast; optional ``axes`` = per operand the
  output dim of each operand dim; default numpy trailing alignment)
* ``scale`` / ``add_scalar`` / ``clamp_min`` with constant ``c``
* ``relu`` ``gelu`` ``gelu_tanh`` ``tanh`` ``exp`` ``rsqrt`` ``recip`` ``sigmoid``
* ``sum`` ``mean`` ``max`` with ``dim``, ``keepdim``; ``softmax`` with ``dim``
* ``layernorm`` (z, gamma?, beta?) over the last dim with ``eps``
* ``kernel_contract`` / ``kernel_maxset``: a kernel given by its write set
  (Sec. 3.4: under a path condition on the thread coordinates a thread writes
  a value to an address), with ``shape`` (output), ``grid`` and ``block``
  (z, y, x) and ``writes``: each ``{"when": [[lo, hi]] * 6, "addr": [a0, a],
  "red": [[lo, hi], ...], "coef": c, "guards": [[tc, rd, c, lo, hi], ...],
  "reads": [[base, tc, rs], ...]}`` over thread coordinates
  theta = (bz, by, bx, tz, ty, tx): threads in the ``when`` box store
  ``sum_r coef * prod_i arg_i[base_i + tc_i.theta + rs_i.r]`` (or the max) at
  ``a0 + a.theta``, the terms kept where ``lo <= tc.theta + r[rd] + c < hi``.
  Locations no thread writes hold the undefined value.
* ``contract`` / ``maxset``: an explicit per-element equation (the form a
  hand-written kernel's write set takes once inverted, Sec. 3.4 "Per-element
  equations"), given as ``shape`` and a list of ``pieces``.  A piece is
  ``{"lo": [...], "hi": [...], "red": [[lo, hi], ...], "coef": c,
  "guards": [[od, oa, rd, c, lo, hi], ...], "access": [[base, os, rs], ...]}``:
  for output coordinates ``o`` inside ``[lo, hi)`` and reduction coordinates
  ``r`` inside the ``red`` box, the term is present when every guard
  ``lo <= oa*o[od] + r[rd] + c < hi`` holds (``od``/``rd`` = -1: absent), and
  operand ``i`` is read at flat offset ``base + sum(os*o) + sum(rs*r)``.
  ``contract`` sums ``coef * prod(operands)``, ``maxset`` takes the max.

Constants (``c``, ``coef``, ``eps``) are floats or ``[num, den]`` rationals.
"""
from __future__ import annotations

import math
import numpy as np

__all__ = [
    "CONFIGS", "config", "make_values", "make_queries", "numel",
    "tiny_matmul", "conv_gelu_sum", "linear_layernorm", "conv_pool_softmax",
    "bmm_sum_tanh", "halfsum_gelu", "softmax_shift", "tiled_matmul_kernel", "pool_kernel",
]


def numel(shape):
    n = 1
    for s in shape:
        n *= int(s)
    return n


# ----------------------------------------------------------------------------
# piece helpers (descriptions of hand-written kernels' per-element equations)
# ----------------------------------------------------------------------------

def _conv_pieces(N, Ci, H, W, Co, k, pad, w_co_stride=None, w_split=None,
                 iw_hi=None):
    """Per-element equation of a stride-1 conv kernel as contract pieces.

    Output coords (n, co, h, w); reduction coords (ci, kh, kw).  ``iw_hi`` lets a
    kernel's right-edge padding test differ from the image width (an
    off-by-one), ``w_split``/``w_co_stride`` let output channels ``co >= w_split``
    read the weight with a different channel stride.
    """
    Ho, Wo = H + 2 * pad - k + 1, W + 2 * pad - k + 1
    if iw_hi is None:
        iw_hi = W
    x_acc = [-pad * W - pad, [Ci * H * W, 0, W, 1], [H * W, W, 1]]
    guards = [[2, 1, 1, -pad, 0, H], [3, 1, 2, -pad, 0, iw_hi]]

    def piece(co_lo, co_hi, co_stride):
        return {
            "lo": [0, co_lo, 0, 0], "hi": [N, co_hi, Ho, Wo],
            "red": [[0, Ci], [0, k], [0, k]], "coef": 1.0,
            "guards": [list(g) for g in guards],
            "access": [list(x_acc), [0, [0, co_stride, 0, 0], [k * k, k, 1]]],
        }

    full = Ci * k * k
    if w_split is None:
        return [piece(0, Co, full)]
    return [piece(0, w_split, full), piece(w_split, Co, w_co_stride)]


def _matmul_piece(M, K, N, k_lo, k_hi):
    return {"lo": [0, 0], "hi": [M, N], "red": [[k_lo, k_hi]], "coef": 1.0,
            "guards": [], "access": [[0, [K, 0], [1]], [0, [0, 1], [N]]]}


# ----------------------------------------------------------------------------
# the workloads
# ----------------------------------------------------------------------------

def tiny_matmul(M=8, K=16, N=8):
    """X[M,K] @ W[K,N] + b[N] then ReLU; the candidate splits K in two halves,
    adds the bias between them and writes ReLU as max(x, 0)."""
    inputs = [["X", [M, K]], ["W", [K, N]], ["b", [N]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "matmul", "args": [0, 1]},
        {"op": "add", "args": [3, 2]},
        {"op": "relu", "args": [4]},
    ], "output": 5}
    h = K // 2
    cand = {"inputs": inputs, "ops": [
        {"op": "contract", "args": [0, 1], "shape": [M, N],
         "pieces": [_matmul_piece(M, K, N, 0, h)]},
        {"op": "add", "args": [3, 2]},
        {"op": "contract", "args": [0, 1], "shape": [M, N],
         "pieces": [_matmul_piece(M, K, N, h, K)]},
        {"op": "add", "args": [4, 5]},
        {"op": "clamp_min", "args": [6], "c": 0.0},
    ], "output": 7}
    return ref, cand


def conv_gelu_sum(N=2, Ci=3, H=32, W=32, Co=16, k=3, pad=1):
    """conv2d + bias, GELU, sum over channels; the candidate's kernel lets the
    input column index reach W (one past the right edge)."""
    inputs = [["X", [N, Ci, H, W]], ["W", [Co, Ci, k, k]], ["b", [Co]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "conv2d", "args": [0, 1, 2], "stride": 1, "pad": pad},
        {"op": "gelu", "args": [3]},
        {"op": "sum", "args": [4], "dim": 1, "keepdim": False},
    ], "output": 5}
    Ho, Wo = H + 2 * pad - k + 1, W + 2 * pad - k + 1
    cand = {"inputs": inputs, "ops": [
        {"op": "contract", "args": [0, 1], "shape": [N, Co, Ho, Wo],
         "pieces": _conv_pieces(N, Ci, H, W, Co, k, pad, iw_hi=W + 1)},
        {"op": "add", "args": [3, 2], "axes": [[0, 1, 2, 3], [1]]},
        {"op": "gelu", "args": [4]},
        {"op": "sum", "args": [5], "dim": 1, "keepdim": False},
    ], "output": 6}
    return ref, cand


def linear_layernorm(B=128, IN=1024, OUT=512, eps=1e-5):
    """Linear, scale 0.5, LayerNorm over the last dim; the candidate takes the
    variance from the second moment (E[z^2] - mu^2, reduced before centring)
    and sums the mean as two half reductions."""
    inputs = [["X", [B, IN]], ["W", [OUT, IN]], ["b", [OUT]],
              ["gamma", [OUT]], ["beta", [OUT]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "linear", "args": [0, 1, 2]},
        {"op": "scale", "args": [5], "c": 0.5},
        {"op": "layernorm", "args": [6, 3, 4], "eps": eps},
    ], "output": 7}
    h = OUT // 2
    half = lambda lo, hi: {"lo": [0, 0], "hi": [B, 1], "red": [[lo, hi]],
                           "coef": [1, OUT], "guards": [],
                           "access": [[0, [OUT, 0], [1]]]}
    cand = {"inputs": inputs, "ops": [
        {"op": "linear", "args": [0, 1, 2]},                        # 5
        {"op": "scale", "args": [5], "c": 0.5},                     # 6  z
        {"op": "mul", "args": [6, 6]},                              # 7  z*z
        {"op": "mean", "args": [7], "dim": 1, "keepdim": True},     # 8  E[z^2]
        {"op": "contract", "args": [6], "shape": [B, 1],
         "pieces": [half(h, OUT)]},                                 # 9  upper half / OUT
        {"op": "contract", "args": [6], "shape": [B, 1],
         "pieces": [half(0, h)]},                                   # 10 lower half / OUT
        {"op": "add", "args": [10, 9]},                             # 11 mu
        {"op": "mul", "args": [11, 11]},                            # 12 mu^2
        {"op": "sub", "args": [8, 12]},                             # 13 var
        {"op": "add_scalar", "args": [13], "c": eps},               # 14
        {"op": "rsqrt", "args": [14]},                              # 15
        {"op": "sub", "args": [6, 11]},                             # 16 z - mu
        {"op": "mul", "args": [16, 15]},                            # 17
        {"op": "mul", "args": [17, 3]},                             # 18 * gamma
        {"op": "add", "args": [18, 4]},                             # 19 + beta
    ], "output": 19}
    return ref, cand


def conv_pool_softmax(N=128, Ci=64, H=32, W=32, Co=128, k=3, pad=1, bug_co=96):
    """conv2d + bias, 2x2 max-pool, softmax over channels; the candidate's
    kernel reads the weight of output channels >= bug_co with channel stride
    (Ci-1)*k*k instead of Ci*k*k."""
    inputs = [["X", [N, Ci, H, W]], ["W", [Co, Ci, k, k]], ["b", [Co]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "conv2d", "args": [0, 1, 2], "stride": 1, "pad": pad},
        {"op": "maxpool2d", "args": [3], "k": 2, "stride": 2},
        {"op": "softmax", "args": [4], "dim": 1},
    ], "output": 5}
    Ho, Wo = H + 2 * pad - k + 1, W + 2 * pad - k + 1
    cand = {"inputs": inputs, "ops": [
        {"op": "contract", "args": [0, 1], "shape": [N, Co, Ho, Wo],
         "pieces": _conv_pieces(N, Ci, H, W, Co, k, pad, w_split=bug_co,
                                w_co_stride=(Ci - 1) * k * k)},
        {"op": "add", "args": [3, 2], "axes": [[0, 1, 2, 3], [1]]},
        {"op": "maxpool2d", "args": [4], "k": 2, "stride": 2},
        {"op": "softmax", "args": [5], "dim": 1},
    ], "output": 6}
    return ref, cand


def bmm_sum_tanh(B=32, M=256, K=512, N=256, tile=64, k_stop=480):
    """Batched matmul, sum over the last dim, bias, tanh; the candidate tiles K
    by ``tile`` and its last tile stops at ``k_stop`` (the K tail is dropped)."""
    inputs = [["A", [B, M, K]], ["B", [B, K, N]], ["bias", [M]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "bmm", "args": [0, 1]},
        {"op": "sum", "args": [3], "dim": 2, "keepdim": False},
        {"op": "add", "args": [4, 2]},
        {"op": "tanh", "args": [5]},
    ], "output": 6}
    nt = K // tile
    acc = [[0, [M * K, K, 0], [tile, 1]], [0, [K * N, 0, 1], [tile * N, N]]]
    full_t = k_stop // tile
    pieces = [{"lo": [0, 0, 0], "hi": [B, M, N], "red": [[0, full_t], [0, tile]],
               "coef": 1.0, "guards": [], "access": [list(a) for a in acc]}]
    if k_stop % tile:
        pieces.append({"lo": [0, 0, 0], "hi": [B, M, N],
                       "red": [[full_t, full_t + 1], [0, k_stop % tile]],
                       "coef": 1.0, "guards": [], "access": [list(a) for a in acc]})
    assert nt * tile == K
    cand = {"inputs": inputs, "ops": [
        {"op": "contract", "args": [0, 1], "shape": [B, M, N], "pieces": pieces},
        {"op": "sum", "args": [3], "dim": 2, "keepdim": False},
        {"op": "add", "args": [4, 2]},
        {"op": "tanh", "args": [5]},
    ], "output": 6}
    return ref, cand


def halfsum_gelu(N=4, C=4, H=16, W=8):
    """The shape of the paper's worked example (Sec. 2, Fig. "checker"): min over
    channels, a sum over H, GELU and a per-channel bias.  Written with max in
    place of min (max(-x) = -min(x) would add two scales); the candidate sums
    only the first half of H."""
    inputs = [["M", [N, C, H, W]], ["b", [C]]]
    red = lambda hh: {"lo": [0, 0], "hi": [N, W], "red": [[0, hh]], "coef": 1.0,
                      "guards": [], "access": [[0, [H * W, 1], [W]]]}

    def prog(hh):
        return {"inputs": inputs, "ops": [
            {"op": "max", "args": [0], "dim": 1, "keepdim": False},       # 2 R[n,h,w]
            {"op": "contract", "args": [2], "shape": [N, W],
             "pieces": [red(hh)]},                                          # 3 S[n,w]
            {"op": "gelu", "args": [3]},                                    # 4 G[n,w]
            {"op": "add", "args": [4, 1], "axes": [[0, 2], [1]]},          # 5 Y[n,c,w]
        ], "output": 5}

    ref = prog(H)
    cand = prog(H // 2)
    # Y[n, c, w] = G[n, w] + b[c]: the add's output rank is 3 with these axes
    for g in (ref, cand):
        g["ops"][3]["shape"] = [N, C, W]
    return ref, cand


_ALL = 1 << 62   # "no bound" in a path condition


def _when(**iv):
    """Path-condition box over (bz, by, bx, tz, ty, tx); unnamed coords free."""
    names = ["bz", "by", "bx", "tz", "ty", "tx"]
    return [list(iv.get(n, (0, _ALL))) for n in names]


def tiled_matmul_kernel(M=50, K=40, N=24, TM=16, TN=8, bug=None):
    """X[M,K] @ W[K,N] + b[N], ReLU.  The reference calls matmul; the candidate
    runs a tiled kernel given by its write set (the form symbolic execution
    gives a hand-written kernel, Sec. 3.4): grid (1, ceil(M/TM), N/TN),
    block (1, TM, TN); thread (by, bx, ty, tx) computes row by*TM + ty and
    column bx*TN + tx, the path condition row < M splitting the threads into
    the full block rows and the last, partial one.  Planted bugs: ``"edge"``
    -- the last block row's bound drops its last row (never written: the
    undefined value); ``"last_tile"`` -- the last column tile reads W one
    column to the right."""
    assert N % TN == 0
    GY, GX = -(-M // TM), N // TN
    rows_last = M - (GY - 1) * TM
    inputs = [["X", [M, K]], ["W", [K, N]], ["b", [N]]]
    addr = [0, [0, TM * N, TN, 0, N, 1]]                       # row * N + col

    def write(by, ty, bx, dcol=0):
        return {"when": _when(by=by, ty=ty, bx=bx), "addr": addr, "red": [[0, K]],
                "coef": 1.0, "guards": [],
                "reads": [[0, [0, TM * K, 0, 0, K, 0], [1]],       # X[row, k]
                          [dcol, [0, 0, TN, 0, 0, 1], [N]]]}       # W[k, col + dcol]

    row_parts = [((0, GY - 1), (0, TM))] if rows_last < TM else []
    last_rows = rows_last - 1 if bug == "edge" else rows_last
    row_parts.append(((GY - 1, GY), (0, last_rows)) if rows_last < TM else ((0, GY), (0, TM)))
    if bug == "edge" and rows_last == TM:
        row_parts = [((0, GY - 1), (0, TM)), ((GY - 1, GY), (0, TM - 1))]
    writes = []
    for by, ty in row_parts:
        if bug == "last_tile":
            writes.append(write(by, ty, (0, GX - 1)))
            writes.append(write(by, ty, (GX - 1, GX), dcol=1))
        else:
            writes.append(write(by, ty, (0, GX)))
    kernel = {"op": "kernel_contract", "args": [0, 1], "shape": [M, N],
              "grid": [1, GY, GX], "block": [1, TM, TN], "writes": writes}
    ref = {"inputs": inputs, "ops": [
        {"op": "matmul", "args": [0, 1]},
        {"op": "add", "args": [3, 2]},
        {"op": "relu", "args": [4]},
    ], "output": 5}
    cand = {"inputs": inputs, "ops": [
        kernel,
        {"op": "add", "args": [3, 2]},
        {"op": "relu", "args": [4]},
    ], "output": 5}
    return ref, cand


def pool_kernel(N=2, C=3, H=8, W=8, bug=None):
    """2x2 max pooling.  The reference calls maxpool2d; the candidate is a
    kernel (grid (N, C, 1), block (1, H/2, W/2), thread (n, c, h, w) writes
    out[n, c, h, w] = max over its window).  Bug ``"stride"``: the window's
    columns step by 1 instead of 2 (overlapping windows)."""
    Ho, Wo = H // 2, W // 2
    sw = 1 if bug == "stride" else 2
    kernel = {"op": "kernel_maxset", "args": [0], "shape": [N, C, Ho, Wo],
              "grid": [N, C, 1], "block": [1, Ho, Wo],
              "writes": [{"addr": [0, [C * Ho * Wo, Ho * Wo, 0, 0, Wo, 1]],
                          "red": [[0, 2], [0, 2]], "guards": [],
                          "reads": [[0, [C * H * W, H * W, 0, 0, 2 * W, sw], [W, 1]]]}]}
    inputs = [["X", [N, C, H, W]]]
    ref = {"inputs": inputs, "ops": [{"op": "maxpool2d", "args": [0], "k": 2}], "output": 1}
    cand = {"inputs": inputs, "ops": [kernel], "output": 1}
    return ref, cand


def softmax_shift(N=4, C=16, L=8, shift_dim=1):
    """softmax over channels of 0.5 * X: the reference calls softmax, the
    candidate writes it out with the usual max shift,
    exp(x - max_c x) / sum_c exp(x - max_c x) -- equal over the reals (the
    sound identity of Sec. 4.2).  ``shift_dim`` != 1 takes the max over
    another dim instead: that shift is not constant along the channels, so
    the candidate then differs from the reference."""
    inputs = [["X", [N, C, L]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "scale", "args": [0], "c": 0.5},                            # 1 x
        {"op": "softmax", "args": [1], "dim": 1},                          # 2
    ], "output": 2}
    cand = {"inputs": inputs, "ops": [
        {"op": "scale", "args": [0], "c": 0.5},                            # 1 x
        {"op": "max", "args": [1], "dim": shift_dim, "keepdim": True},     # 2 m
        {"op": "sub", "args": [1, 2]},                                     # 3 x - m
        {"op": "exp", "args": [3]},                                        # 4 e
        {"op": "sum", "args": [4], "dim": 1, "keepdim": True},             # 5 s
        {"op": "div", "args": [4, 5]},                                     # 6 e / s
    ], "output": 6}
    return ref, cand


def channel_max(N=2, Ci=3, H=8, W=8, Co=128, k=3, pad=1, bug_co=96, bug_stride=None):
    """conv2d + bias, max over all Co output channels, tanh (a long max-set:
    Co members per element); the candidate reads the weight of channels
    >= bug_co with channel stride ``bug_stride`` (default (Ci+1)*k*k, which
    reads past the weight's end for the last channels)."""
    inputs = [["X", [N, Ci, H, W]], ["W", [Co, Ci, k, k]], ["b", [Co]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "conv2d", "args": [0, 1, 2], "stride": 1, "pad": pad},
        {"op": "max", "args": [3], "dim": 1, "keepdim": False},
        {"op": "tanh", "args": [4]},
    ], "output": 5}
    Ho, Wo = H + 2 * pad - k + 1, W + 2 * pad - k + 1
    cand = {"inputs": inputs, "ops": [
        {"op": "contract", "args": [0, 1], "shape": [N, Co, Ho, Wo],
         "pieces": _conv_pieces(N, Ci, H, W, Co, k, pad, w_split=bug_co,
                                w_co_stride=bug_stride or (Ci + 1) * k * k)},
        {"op": "add", "args": [3, 2], "axes": [[0, 1, 2, 3], [1]]},
        {"op": "max", "args": [4], "dim": 1, "keepdim": False},
        {"op": "tanh", "args": [5]},
    ], "output": 6}
    return ref, cand


def row_max(B=4, L=1024, split=None):
    """relu of the max over a row of L elements of 0.5 X (L members per
    element); the candidate takes the max of the row's two halves' maxima
    when ``split`` is given (equal as sets), else the row without its last
    element."""
    inputs = [["X", [B, L]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "scale", "args": [0], "c": 0.5},
        {"op": "max", "args": [1], "dim": 1, "keepdim": False},
        {"op": "relu", "args": [2]},
    ], "output": 3}
    if split:
        cand = {"inputs": inputs, "ops": [
            {"op": "scale", "args": [0], "c": 0.5},
            {"op": "maxset", "args": [1], "shape": [B], "pieces": [
                {"lo": [0], "hi": [B], "red": [[0, split]], "guards": [],
                 "access": [[0, [L], [1]]]},
                {"lo": [0], "hi": [B], "red": [[split, L]], "guards": [],
                 "access": [[0, [L], [1]]]}]},
            {"op": "relu", "args": [2]},
        ], "output": 3}
    else:
        cand = {"inputs": inputs, "ops": [
            {"op": "scale", "args": [0], "c": 0.5},
            {"op": "maxset", "args": [1], "shape": [B], "pieces": [
                {"lo": [0], "hi": [B], "red": [[0, L - 1]], "guards": [],
                 "access": [[0, [L], [1]]]}]},
            {"op": "relu", "args": [2]},
        ], "output": 3}
    return ref, cand


def softmax_shift_broadcast(N=3, C=64, L=5):
    """softmax over C channels of 0.5 X against the max-shifted form whose
    shift is taken without keepdim and broadcast back with explicit axes: the
    rewrite to softmax does not apply, so the candidate keeps a max over C
    members and its exponentials' arguments differ from the reference's."""
    inputs = [["X", [N, C, L]]]
    ref = {"inputs": inputs, "ops": [
        {"op": "scale", "args": [0], "c": 0.5},
        {"op": "softmax", "args": [1], "dim": 1},
    ], "output": 2}
    cand = {"inputs": inputs, "ops": [
        {"op": "scale", "args": [0], "c": 0.5},                                   # 1 x
        {"op": "max", "args": [1], "dim": 1, "keepdim": False},                   # 2 m [N, L]
        {"op": "sub", "args": [1, 2], "axes": [[0, 1, 2], [0, 2]]},               # 3 x - m
        {"op": "exp", "args": [3]},                                               # 4
        {"op": "sum", "args": [4], "dim": 1, "keepdim": True},                    # 5
        {"op": "div", "args": [4, 5]},                                            # 6
    ], "output": 6}
    return ref, cand


# ----------------------------------------------------------------------------
# the five benchmark configurations and their seeded inputs
# ----------------------------------------------------------------------------

CONFIGS = {
    1: dict(name="tiny_matmul_relu", build=tiny_matmul, n_queries=None,
            order="all"),
    2: dict(name="conv_gelu_sum", build=conv_gelu_sum, n_queries=4096,
            order="random"),
    3: dict(name="linear_scale_layernorm", build=linear_layernorm,
            n_queries=1024, order="random"),
    4: dict(name="conv_maxpool_softmax", build=conv_pool_softmax,
            n_queries=None, order="all"),
    5: dict(name="bmm_sum_bias_tanh", build=bmm_sum_tanh, n_queries=None,
            order="all"),
}


def config(c, **shape_overrides):
    """(ref, cand) graph descriptions of configuration ``c`` (1..5), optionally
    at reduced shapes (same structure, same planted bug)."""
    return CONFIGS[c]["build"](**shape_overrides)


def out_shape(graph):
    """Output shape of a graph description, by shape bookkeeping only."""
    shapes = [list(s) for _, s in graph["inputs"]]
    for op in graph["ops"]:
        shapes.append(_shape_of(op, shapes))
    return shapes[graph["output"]]


def _bcast(sa, sb, axes=None):
    if axes is not None:
        ra = max(max(axes[0], default=-1), max(axes[1], default=-1)) + 1
        out = [1] * ra
        for s, ax in ((sa, axes[0]), (sb, axes[1])):
            for d, a in enumerate(ax):
                out[a] = max(out[a], s[d])
        return out
    r = max(len(sa), len(sb))
    pa = [1] * (r - len(sa)) + list(sa)
    pb = [1] * (r - len(sb)) + list(sb)
    return [max(x, y) for x, y in zip(pa, pb)]


def _shape_of(op, shapes):
    k, a = op["op"], op["args"]
    if "shape" in op:
        return list(op["shape"])
    s0 = shapes[a[0]]
    if k == "matmul":
        return [s0[0], shapes[a[1]][1]]
    if k == "bmm":
        return [s0[0], s0[1], shapes[a[1]][2]]
    if k == "linear":
        return [s0[0], shapes[a[1]][0]]
    if k == "conv2d":
        w = shapes[a[1]]
        st, p = op.get("stride", 1), op.get("pad", 0)
        return [s0[0], w[0], (s0[2] + 2 * p - w[2]) // st + 1,
                (s0[3] + 2 * p - w[3]) // st + 1]
    if k == "maxpool2d":
        kk, st = op["k"], op.get("stride", op["k"])
        return [s0[0], s0[1], (s0[2] - kk) // st + 1, (s0[3] - kk) // st + 1]
    if k in ("add", "sub", "mul", "div"):
        return _bcast(s0, shapes[a[1]], op.get("axes"))
    if k in ("sum", "mean", "max"):
        d = op["dim"] % len(s0)
        if op.get("keepdim", False):
            return [1 if i == d else s for i, s in enumerate(s0)]
        return [s for i, s in enumerate(s0) if i != d]
    return list(s0)


def make_values(c, graph, seed=None, dtype=np.float32):
    """Seeded input tensors for configuration ``c`` (distributions of the
    configuration's table), in declared input order."""
    seed = 1000 * c + 1 if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    vals = []
    shapes = {n: s for n, s in graph["inputs"]}
    for name, shape in graph["inputs"]:
        if c == 1:
            v = rng.standard_normal(shape)
        elif c in (2, 4):
            if name == "X":
                v = rng.standard_normal(shape)
            else:
                w = shapes["W"]
                bound = 1.0 / math.sqrt(w[1] * w[2] * w[3])
                v = rng.uniform(-bound, bound, shape)
        elif c == 3:
            fan_in = shapes["W"][1]
            if name == "X":
                v = rng.standard_normal(shape)
            elif name in ("W", "b"):
                b = 1.0 / math.sqrt(fan_in)
                v = rng.uniform(-b, b, shape)
            elif name == "gamma":
                v = 1.0 + 0.1 * rng.standard_normal(shape)
            else:
                v = 0.1 * rng.standard_normal(shape)
        elif c == 5:
            v = rng.standard_normal(shape)
            if name == "B":
                v = v / math.sqrt(shape[1])
        else:
            v = rng.standard_normal(shape)
        vals.append(np.ascontiguousarray(v, dtype=dtype))
    return vals


def make_queries(c, n_out, n=None, seed=None):
    """Queried output locations (flat row-major indices, int64)."""
    spec = CONFIGS[c]
    n = spec["n_queries"] if n is None else n
    if spec["order"] == "all" and n is None:
        return np.arange(n_out, dtype=np.int64)
    seed = 1000 * c + 2 if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.integers(0, n_out, int(n), dtype=np.int64)


def random_values(graph, seed, dtype=np.float64):
    """Generic N(0,1) inputs for any graph description."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return [np.ascontiguousarray(rng.standard_normal(s), dtype=dtype)
            for _, s in graph["inputs"]]


# ----------------------------------------------------------------------------
# random small program pairs (equivalent rewrites and planted mutations)
# ----------------------------------------------------------------------------

_UFS = ("exp", "tanh", "gelu", "sigmoid", "gelu_tanh")


def _rand_tree(rng, depth, shape_kind):
    """A random expression tree over X[B,D], Y[B,D], w[D] and Wm[D,D]: a 'full'
    [B,D] value, a 'row' [B,1] reduction result or the 'w' [D] leaf."""
    if shape_kind == "w":
        return ("in", 2)
    if shape_kind == "row":
        op = rng.choice(["sum", "mean", "max"])
        return (op, _rand_tree(rng, depth - 1, "full"))
    if depth <= 0:
        return ("in", int(rng.choice([0, 1, 3])))
    r = rng.random()
    if r < 0.12:
        return ("in", int(rng.choice([0, 1, 3])))
    if r < 0.45:
        op = rng.choice(["add", "sub", "mul"])
        u = rng.random()
        second = "row" if u < 0.2 else ("w" if u < 0.35 else "full")
        return (op, _rand_tree(rng, depth - 1, "full"), _rand_tree(rng, depth - 1, second))
    if r < 0.58:
        return ("scale", float(rng.choice([0.5, -1.0, 0.25, 2.0, 3.0])),
                _rand_tree(rng, depth - 1, "full"))
    if r < 0.7:
        return ("uf", str(rng.choice(_UFS)), _rand_tree(rng, depth - 1, "full"))
    if r < 0.78:
        return ("relu", _rand_tree(rng, depth - 1, "full"))
    if r < 0.86:
        return ("softmax", _rand_tree(rng, depth - 1, "full"))
    return ("matmul", _rand_tree(rng, depth - 1, "full"))


def _mutate(rng, t):
    """Apply one small change somewhere in the tree (usually not equivalent)."""
    kids = [i for i, x in enumerate(t) if isinstance(x, tuple)]
    if kids and rng.random() < 0.6:
        i = int(rng.choice(kids))
        return t[:i] + (_mutate(rng, t[i]),) + t[i + 1:]
    k = t[0]
    if k == "in":
        return ("in", {0: 1, 1: 0, 2: 2, 3: 0}[t[1]]) if t[1] != 2 else ("scale", 2.0, t)
    if k == "scale":
        return ("scale", t[1] * 0.5, t[2])
    if k == "sub":
        return ("sub", t[2], t[1]) if _shape_of_tree(t[2]) == "full" else ("add",) + t[1:]
    if k in ("add", "mul"):
        return (("mul" if k == "add" else "add"),) + t[1:]
    if k == "uf":
        alt = [u for u in _UFS if u != t[1]]
        return ("uf", str(rng.choice(alt)), t[2])
    if k in ("sum", "mean", "max"):
        return ("dropone", k, t[1])
    return ("scale", 2.0, t)


def _shape_of_tree(t):
    if t == ("in", 2):
        return "w"
    return "row" if t[0] in ("sum", "mean", "max", "dropone") else "full"


class _GraphBuilder:
    def __init__(self, B, D, rng, variants=False):
        self.B, self.D, self.rng = B, D, rng
        # variants: also write matmuls and row maxima as kernels given by their
        # write sets, and softmaxes with the max shift
        self.variants = variants
        self.inputs = [["X", [B, D]], ["Y", [B, D]], ["w", [D]], ["Wm", [D, D]]]
        self.ops = []

    def op(self, **kw):
        self.ops.append(kw)
        return len(self.inputs) + len(self.ops) - 1

    def reduce_pieces(self, kind, a, drop=False):
        B, D = self.B, self.D
        acc = [[0, [D, 0], [1]]]
        h = int(self.rng.integers(1, D)) if D > 1 else 1
        if self.rng.random() < 0.5 or D == 1:
            ranges = [[0, D]]
        else:   # split (and reverse) the reduction order
            ranges = [[h, D], [0, h]]
        if drop:
            ranges = [[0, D - 1]] if D > 1 else [[0, 0]]
        coef = [1, D] if kind == "mean" else 1.0
        return self.op(op="maxset" if kind == "max" else "contract", args=[a],
                       shape=[B, 1],
                       pieces=[{"lo": [0, 0], "hi": [B, 1], "red": [r], "coef": coef,
                                "guards": [], "access": [list(x) for x in acc]}
                               for r in ranges])

    def build(self, t):
        rng = self.rng
        k = t[0]
        if k == "in":
            if t[1] == 3:       # the [B, D] value X @ Wm
                return self.op(op="matmul", args=[0, 3])
            return t[1]
        if k in ("add", "mul"):
            a, b = self.build(t[1]), self.build(t[2])
            if rng.random() < 0.5 and _shape_of_tree(t[2]) == "full":
                a, b = b, a
            return self.op(op=k, args=[a, b])
        if k == "sub":
            a, b = self.build(t[1]), self.build(t[2])
            if rng.random() < 0.5:
                nb = self.op(op="scale", args=[b], c=-1.0)
                return self.op(op="add", args=[a, nb])
            return self.op(op="sub", args=[a, b])
        if k == "scale":
            c, sub = t[1], t[2]
            if sub[0] == "add" and rng.random() < 0.5:     # distribute
                return self.build(("add", ("scale", c, sub[1]), ("scale", c, sub[2])))
            a = self.build(sub)
            if rng.random() < 0.3 and c != 0:
                a = self.op(op="scale", args=[a], c=c * 2.0)
                return self.op(op="scale", args=[a], c=0.5)
            return self.op(op="scale", args=[a], c=c)
        if k == "uf":
            a = self.build(t[2])
            return self.op(op=t[1], args=[a])
        if k == "relu":
            a = self.build(t[1])
            return self.op(op="relu", args=[a]) if rng.random() < 0.5 else \
                self.op(op="clamp_min", args=[a], c=0.0)
        if k == "softmax":
            a = self.build(t[1])
            r = rng.random()
            if self.variants and rng.random() < 0.3:   # with the max shift
                m = self.op(op="max", args=[a], dim=1, keepdim=True)
                z = self.op(op="sub", args=[a, m])
                e = self.op(op="exp", args=[z])
                s = self.op(op="sum", args=[e], dim=1, keepdim=True)
                return self.op(op="div", args=[e, s])
            if r < 0.4:
                return self.op(op="softmax", args=[a], dim=1)
            e = self.op(op="exp", args=[a])
            s = self.op(op="sum", args=[e], dim=1, keepdim=True)
            if r < 0.7:
                return self.op(op="div", args=[e, s])
            rc = self.op(op="recip", args=[s])
            return self.op(op="mul", args=[rc, e]) if rng.random() < 0.5 else \
                self.op(op="mul", args=[e, rc])
        if k in ("sum", "mean", "max"):
            a = self.build(t[1])
            if k == "max" and self.variants and rng.random() < 0.3:
                # a kernel: one thread per row (blockIdx.y) takes the row's max
                B, D = self.B, self.D
                return self.op(op="kernel_maxset", args=[a], shape=[B, 1],
                               grid=[1, B, 1], block=[1, 1, 1],
                               writes=[{"addr": [0, [0, 1, 0, 0, 0, 0]], "red": [[0, D]],
                                        "guards": [],
                                        "reads": [[0, [0, D, 0, 0, 0, 0], [1]]]}])
            if rng.random() < 0.5:
                return self.op(op=k, args=[a], dim=1, keepdim=True)
            if k == "mean" and rng.random() < 0.5:
                s = self.reduce_pieces("sum", a)
                return self.op(op="scale", args=[s], c=[1, self.D])
            return self.reduce_pieces(k, a)
        if k == "dropone":
            a = self.build(t[2])
            return self.reduce_pieces(t[1], a, drop=True)
        if k == "matmul":
            a = self.build(t[1])
            if self.variants and rng.random() < 0.4:
                # a kernel: block row by = output row, columns split into
                # (blockIdx.x, threadIdx.x) tiles of TX
                B, D = self.B, self.D
                TX = int(rng.choice([x for x in (1, 2, D) if D % x == 0]))
                return self.op(op="kernel_contract", args=[a, 3], shape=[B, D],
                               grid=[1, B, D // TX], block=[1, 1, TX],
                               writes=[{"addr": [0, [0, D, TX, 0, 0, 1]], "red": [[0, D]],
                                        "coef": 1.0, "guards": [],
                                        "reads": [[0, [0, D, 0, 0, 0, 0], [1]],
                                                  [0, [0, 0, TX, 0, 0, 1], [D]]]}])
            if rng.random() < 0.5 or self.D < 2:
                return self.op(op="matmul", args=[a, 3])
            h = int(rng.integers(1, self.D))
            D, B = self.D, self.B
            pcs = [{"lo": [0, 0], "hi": [B, D], "red": [[h, D]], "coef": 1.0, "guards": [],
                    "access": [[0, [D, 0], [1]], [0, [0, 1], [D]]]},
                   {"lo": [0, 0], "hi": [B, D], "red": [[0, h]], "coef": 1.0, "guards": [],
                    "access": [[0, [D, 0], [1]], [0, [0, 1], [D]]]}]
            return self.op(op="contract", args=[a, 3], shape=[B, D], pieces=pcs)
        raise ValueError(k)


def random_pair(seed, depth=3, variants=False):
    """Two programs over the same inputs: the same random expression compiled
    with independent syntactic choices; with probability 1/2 the candidate's
    expression carries one mutation.  Returns (ref, cand, mutated).  With
    ``variants`` the choices also include kernels given by their write sets
    (matmuls, row maxima) and max-shifted softmaxes."""
    rng = np.random.Generator(np.random.PCG64(seed))
    B = int(rng.integers(1, 3))
    D = int(rng.choice([2, 4]))
    tree = _rand_tree(rng, depth, "full")
    mutated = bool(rng.random() < 0.5)
    t2 = _mutate(rng, tree) if mutated else tree
    graphs = []
    for t in (tree, t2):
        gb = _GraphBuilder(B, D, rng, variants)
        out = gb.build(t)
        if out < len(gb.inputs):           # make the output an op
            out = gb.op(op="scale", args=[out], c=1.0)
        graphs.append({"inputs": gb.inputs, "ops": gb.ops, "output": out})
    return graphs[0], graphs[1], mutated
