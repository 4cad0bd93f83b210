"""Direct fp64 forward pass of a high-level op graph (oracle pin machinery).

TEST INFRASTRUCTURE ONLY.

Independent of the oracle's per-element equations: standard ops run as
PyTorch CPU library routines in float64 (conv2d, max_pool2d, softmax,
layer_norm, ...); the explicit ``contract``/``maxset`` equations are evaluated
straight from their definition with numpy, one output element at a time
(tiny shapes only).  Reading outside an operand yields NaN (the undefined
value).
"""
from __future__ import annotations

import itertools
import math
from fractions import Fraction

import numpy as np
import torch
import torch.nn.functional as F


def _c(x):
    if isinstance(x, (list, tuple)):
        return float(Fraction(int(x[0]), int(x[1])))
    return float(x)


def _explicit(op, args, maximum):
    shape = op["shape"]
    out = np.full(shape, np.nan if maximum else 0.0)
    flat = [a.reshape(-1).numpy() for a in args]
    for o in itertools.product(*[range(s) for s in shape]):
        vals = []
        for pc in op["pieces"]:
            lo = pc.get("lo", [0] * len(shape))
            hi = pc.get("hi", shape)
            if any(not (l <= x < h) for x, l, h in zip(o, lo, hi)):
                continue
            coef = _c(pc.get("coef", 1.0))
            for r in itertools.product(*[range(a, b) for a, b in pc["red"]]):
                ok = True
                for od, oa, rd, c, glo, ghi in pc.get("guards", []):
                    v = c + (oa * o[od] if od >= 0 else 0) + (r[rd] if rd >= 0 else 0)
                    if not (glo <= v < ghi):
                        ok = False
                if not ok:
                    continue
                prod = coef if not maximum else 1.0
                for i, (base, os_, rs) in enumerate(pc["access"]):
                    off = base + sum(a * b for a, b in zip(os_, o)) + \
                        sum(a * b for a, b in zip(rs, r))
                    x = flat[i][off] if 0 <= off < flat[i].size else np.nan
                    prod = x if maximum else prod * x
                vals.append(prod)
        if maximum:
            out[o] = max(vals) if vals and not any(np.isnan(vals)) else np.nan
        else:
            out[o] = sum(vals)
    return torch.from_numpy(out)


def _kernel(op, args, maximum):
    """Run the kernel: every thread of the launch evaluates each write whose
    path condition it satisfies and stores the value at the write's address
    (unwritten locations stay NaN, the undefined value)."""
    shape = op["shape"]
    total = int(np.prod(shape))
    out = np.full(total, np.nan)
    written = np.zeros(total, dtype=bool)
    flat = [a.reshape(-1).numpy() for a in args]
    launch = list(op["grid"]) + list(op["block"])
    for w in op["writes"]:
        when = w.get("when", [[0, 1 << 62]] * 6)
        ranges = [range(max(0, lo), min(n, hi)) for (lo, hi), n in zip(when, launch)]
        a0, ac = w["addr"]
        coef = _c(w.get("coef", 1.0))
        for th in itertools.product(*ranges):
            vals = []
            for r in itertools.product(*[range(a, b) for a, b in w["red"]]):
                ok = True
                for tc, rd, c, glo, ghi in w.get("guards", []):
                    v = c + sum(x * y for x, y in zip(tc, th)) + (r[rd] if rd >= 0 else 0)
                    ok = ok and glo <= v < ghi
                if not ok:
                    continue
                prod = 1.0 if maximum else coef
                for i, (base, tc, rs) in enumerate(w["reads"]):
                    off = base + sum(x * y for x, y in zip(tc, th)) + \
                        sum(x * y for x, y in zip(rs, r))
                    x = flat[i][off] if 0 <= off < flat[i].size else np.nan
                    prod = x if maximum else prod * x
                vals.append(prod)
            a = a0 + sum(x * y for x, y in zip(ac, th))
            if not 0 <= a < total or written[a]:
                raise ValueError("kernel store outside the output or twice to one location")
            written[a] = True
            if maximum:
                out[a] = max(vals) if vals and not any(np.isnan(vals)) else np.nan
            else:
                out[a] = sum(vals)
    return torch.from_numpy(out.reshape(shape))


def _bcast(a, b, axes):
    if axes is None:
        return a, b
    r = max(max(axes[0], default=-1), max(axes[1], default=-1)) + 1

    def lift(x, ax):
        shp = [1] * r
        for d, o in enumerate(ax):
            shp[o] = x.shape[d]
        # operand dims must appear in increasing output order for a plain view
        perm = sorted(range(len(ax)), key=lambda d: ax[d])
        return x.permute(*perm).reshape(shp) if perm != list(range(len(ax))) \
            else x.reshape(shp)

    return lift(a, axes[0]), lift(b, axes[1])


def forward(graph, inputs):
    """Output tensor (torch float64) of the graph on concrete inputs."""
    return tensors(graph, inputs)[graph["output"]]


def tensors(graph, inputs):
    """Every tensor of the graph (inputs, then one per op) on concrete inputs."""
    ts = [torch.as_tensor(np.asarray(x, dtype=np.float64)) for x in inputs]
    for op in graph["ops"]:
        k = op["op"]
        a = [ts[i] for i in op["args"]]
        if k == "matmul":
            y = a[0] @ a[1]
        elif k == "bmm":
            y = torch.bmm(a[0], a[1])
        elif k == "linear":
            y = F.linear(a[0], a[1], a[2] if len(a) > 2 else None)
        elif k == "conv2d":
            y = F.conv2d(a[0], a[1], a[2] if len(a) > 2 else None,
                         stride=op.get("stride", 1), padding=op.get("pad", 0))
        elif k == "maxpool2d":
            y = F.max_pool2d(a[0], op["k"], op.get("stride", op["k"]))
        elif k in ("add", "sub", "mul", "div"):
            x0, x1 = _bcast(a[0], a[1], op.get("axes"))
            y = {"add": torch.add, "sub": torch.sub, "mul": torch.mul,
                 "div": torch.div}[k](x0, x1)
        elif k == "scale":
            y = a[0] * _c(op["c"])
        elif k == "add_scalar":
            y = a[0] + _c(op["c"])
        elif k == "clamp_min":
            y = torch.clamp_min(a[0], _c(op["c"]))
        elif k == "relu":
            y = torch.relu(a[0])
        elif k == "gelu":
            y = F.gelu(a[0])
        elif k == "gelu_tanh":
            y = F.gelu(a[0], approximate="tanh")
        elif k == "tanh":
            y = torch.tanh(a[0])
        elif k == "exp":
            y = torch.exp(a[0])
        elif k == "rsqrt":
            y = torch.rsqrt(a[0])
        elif k == "recip":
            y = torch.reciprocal(a[0])
        elif k == "sigmoid":
            y = torch.sigmoid(a[0])
        elif k == "erf":
            y = torch.erf(a[0])
        elif k == "sqrt":
            y = torch.sqrt(a[0])
        elif k == "log":
            y = torch.log(a[0])
        elif k == "sum":
            y = a[0].sum(dim=op["dim"], keepdim=op.get("keepdim", False))
        elif k == "mean":
            y = a[0].mean(dim=op["dim"], keepdim=op.get("keepdim", False))
        elif k == "max":
            y = a[0].amax(dim=op["dim"], keepdim=op.get("keepdim", False))
        elif k == "softmax":
            y = torch.softmax(a[0], dim=op["dim"])
        elif k == "layernorm":
            D = a[0].shape[-1]
            y = F.layer_norm(a[0], (D,), a[1] if len(a) > 1 else None,
                             a[2] if len(a) > 2 else None, eps=_c(op.get("eps", 1e-5)))
        elif k in ("kernel_contract", "kernel_maxset"):
            y = _kernel(op, a, maximum=k == "kernel_maxset")
        elif k == "contract":
            y = _explicit(op, a, maximum=False)
        elif k == "maxset":
            y = _explicit(op, a, maximum=True)
        else:
            raise ValueError(k)
        if "shape" in op and k not in ("contract", "maxset", "kernel_contract", "kernel_maxset"):
            y = y.reshape(op["shape"])
        ts.append(y)
    return ts


def flat_output(graph, inputs):
    return forward(graph, inputs).reshape(-1).numpy()


__all__ = ["forward", "tensors", "flat_output", "math"]
