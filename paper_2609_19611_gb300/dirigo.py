"""Python binding of the C ABI in include/dirigo.h (argument marshalling only).

Every step of the check runs in the CUDA library; this module converts graph
descriptions (the dict format of ``workloads``) to the C structs, passes
device pointers of torch tensors, and raises on any non-OK status.  There is
no CPU fallback: without the compiled library (or without a GPU) the calls
fail.
"""
from __future__ import annotations

import ctypes
import os
from fractions import Fraction

import numpy as np

import torch

from . import build as _build

MAX_RANK, MAX_RED, MAX_GUARDS = 4, 4, 4

STATUS = {0: "OK", 1: "E_INVALID", 2: "E_SHAPE", 3: "E_UNSUPPORTED", 4: "E_CAPACITY",
          5: "E_WORKSPACE", 6: "E_CUDA", 7: "E_NOMEM", 8: "E_MISMATCH"}
(OK, E_INVALID, E_SHAPE, E_UNSUPPORTED, E_CAPACITY, E_WORKSPACE, E_CUDA, E_NOMEM,
 E_MISMATCH) = range(9)
# error bits a cone call latches (dirigo_cone_async's status word)
CONE_ERR_UNSUPPORTED, CONE_ERR_BOXES, CONE_ERR_LOCATION, CONE_ERR_NONMONOTONE, CONE_ERR_WAIT, \
    CONE_ERR_RUNS = 1, 2, 4, 8, 16, 32

OPS = {name: i + 1 for i, name in enumerate([
    "matmul", "bmm", "linear", "conv2d", "maxpool2d", "add", "sub", "mul", "div", "scale",
    "add_scalar", "clamp_min", "relu", "gelu", "gelu_tanh", "tanh", "exp", "rsqrt", "recip",
    "sigmoid", "erf", "sqrt", "log", "sum", "mean", "max", "softmax", "layernorm",
    "contract", "maxset", "kernel_contract", "kernel_maxset"])}
THREAD_DIMS = 6

CALL_CONE, CALL_TERMS, CALL_EVAL = 1, 2, 3
DISCHARGED, EXPORTED, DIFFERS_UNEXPORTED = 0, 1, 2
FLAG_CONE_DIFFERS, FLAG_BOT_REF, FLAG_BOT_CAND, FLAG_NO_CONES = 1, 2, 4, 8
AXIOM_GELU = 1
KERNEL_CLASSES = ["cone_count", "cone_write", "key_leaf", "key_gemm", "key_elem", "compare",
                  "export", "eval", "scan", "key_limbs"]


class Const(ctypes.Structure):
    _fields_ = [("value", ctypes.c_double), ("num", ctypes.c_int64), ("den", ctypes.c_int64)]


class Guard(ctypes.Structure):
    _fields_ = [("od", ctypes.c_int32), ("rd", ctypes.c_int32), ("oa", ctypes.c_int64),
                ("c", ctypes.c_int64), ("lo", ctypes.c_int64), ("hi", ctypes.c_int64)]


class Access(ctypes.Structure):
    _fields_ = [("base", ctypes.c_int64), ("os", ctypes.c_int64 * MAX_RANK),
                ("rs", ctypes.c_int64 * MAX_RED)]


class Piece(ctypes.Structure):
    _fields_ = [("lo", ctypes.c_int64 * MAX_RANK), ("hi", ctypes.c_int64 * MAX_RANK),
                ("n_red", ctypes.c_int32), ("n_guards", ctypes.c_int32),
                ("red_lo", ctypes.c_int64 * MAX_RED), ("red_hi", ctypes.c_int64 * MAX_RED),
                ("coef", Const), ("guards", Guard * MAX_GUARDS), ("access", Access * 2)]


class KGuard(ctypes.Structure):
    _fields_ = [("tc", ctypes.c_int64 * 6), ("rd", ctypes.c_int32), ("c", ctypes.c_int64),
                ("lo", ctypes.c_int64), ("hi", ctypes.c_int64)]


class KAccess(ctypes.Structure):
    _fields_ = [("base", ctypes.c_int64), ("tc", ctypes.c_int64 * 6),
                ("rs", ctypes.c_int64 * MAX_RED)]


class KernelWrite(ctypes.Structure):
    _fields_ = [("when_lo", ctypes.c_int64 * 6), ("when_hi", ctypes.c_int64 * 6),
                ("addr_base", ctypes.c_int64), ("addr", ctypes.c_int64 * 6),
                ("n_red", ctypes.c_int32), ("n_guards", ctypes.c_int32),
                ("red_lo", ctypes.c_int64 * MAX_RED), ("red_hi", ctypes.c_int64 * MAX_RED),
                ("coef", Const), ("guards", KGuard * MAX_GUARDS), ("reads", KAccess * 2)]


class OpDesc(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("n_args", ctypes.c_int32),
                ("args", ctypes.c_int32 * 3), ("rank", ctypes.c_int32),
                ("shape", ctypes.c_int64 * MAX_RANK), ("stride", ctypes.c_int32),
                ("pad", ctypes.c_int32), ("k", ctypes.c_int32), ("dim", ctypes.c_int32),
                ("keepdim", ctypes.c_int32), ("axes_rank", ctypes.c_int32 * 2),
                ("axes", (ctypes.c_int32 * MAX_RANK) * 2), ("c", Const),
                ("n_pieces", ctypes.c_int32), ("pieces", ctypes.POINTER(Piece)),
                ("grid", ctypes.c_int64 * 3), ("block", ctypes.c_int64 * 3),
                ("n_writes", ctypes.c_int32), ("writes", ctypes.POINTER(KernelWrite))]


class TensorDesc(ctypes.Structure):
    _fields_ = [("rank", ctypes.c_int32), ("shape", ctypes.c_int64 * MAX_RANK)]


class GraphDesc(ctypes.Structure):
    _fields_ = [("n_inputs", ctypes.c_int32), ("inputs", ctypes.POINTER(TensorDesc)),
                ("n_ops", ctypes.c_int32), ("ops", ctypes.POINTER(OpDesc)),
                ("output", ctypes.c_int32)]


class Options(ctypes.Structure):
    _fields_ = [("flags", ctypes.c_uint32)]


class MergeInfo(ctypes.Structure):
    _fields_ = [("n_shared_ops", ctypes.c_int32), ("n_inputs", ctypes.c_int32)]


class GraphInfo(ctypes.Structure):
    _fields_ = [("n_leaves", ctypes.c_int64), ("out_numel", ctypes.c_int64),
                ("out_rank", ctypes.c_int32), ("out_shape", ctypes.c_int64 * MAX_RANK),
                ("n_tensors", ctypes.c_int32), ("n_inputs", ctypes.c_int32),
                ("n_cells", ctypes.c_int64), ("n_fast_cells", ctypes.c_int64),
                ("key_tc_flops", ctypes.c_double), ("key_limb_bytes", ctypes.c_double),
                ("n_tc_contractions", ctypes.c_int64), ("max_runs_per_location", ctypes.c_int64),
                ("key_mix_ops", ctypes.c_double)]


class CompareStats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "n_discharged", "n_exported", "n_unexported", "n_cone_differs", "n_bot_ref",
        "n_bot_cand", "export_bytes", "export_required", "cone_error")]


class DirigoError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


_lib = None

VP, I64, I32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32

# exported entry points and their argument types (every symbol the header declares)
SIGNATURES = {
    "dirigo_graph_create": ([ctypes.POINTER(GraphDesc), ctypes.POINTER(Options), ctypes.POINTER(VP)], I32),
    "dirigo_graph_destroy": ([VP], None),
    "dirigo_graph_create_merged": ([ctypes.POINTER(GraphDesc), ctypes.POINTER(GraphDesc),
                                    ctypes.POINTER(Options), ctypes.POINTER(VP),
                                    ctypes.POINTER(VP), ctypes.POINTER(ctypes.c_int32), I32,
                                    ctypes.POINTER(MergeInfo)], I32),
    "dirigo_graph_info_get": ([VP, ctypes.POINTER(GraphInfo)], I32),
    "dirigo_workspace_size": ([VP, I32, I64, ctypes.POINTER(ctypes.c_size_t)], I32),
    "dirigo_compare_workspace_size": ([VP, VP, I64, ctypes.POINTER(ctypes.c_size_t)], I32),
    "dirigo_cone": ([VP, VP, I64, VP, VP, I64, VP, ctypes.POINTER(I64), VP, ctypes.c_size_t, VP], I32),
    "dirigo_cone_async": ([VP, VP, I64, VP, VP, I64, VP, VP, VP, ctypes.c_size_t, VP], I32),
    "dirigo_cone_noalloc": ([VP, VP, I64, VP, VP, I64, VP, ctypes.POINTER(I64), VP], I32),
    "dirigo_terms": ([VP, VP, I64, VP, VP, ctypes.c_size_t, VP], I32),
    "dirigo_compare": ([VP, VP, VP, I64, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, I64, VP, I64,
                        ctypes.POINTER(CompareStats), VP, ctypes.c_size_t, VP], I32),
    "dirigo_compare_async": ([VP, VP, VP, I64, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP, I64,
                              VP, I64, VP, VP, VP, ctypes.c_size_t, VP], I32),
    "dirigo_eval": ([VP, ctypes.POINTER(VP), VP, I64, VP, VP, ctypes.c_size_t, VP], I32),
    "dirigo_profile_enable": ([I32], I32),
    "dirigo_profile_read": ([ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I64), I32, I32], I32),
    "dirigo_query_order": ([VP, VP, ctypes.c_uint64, VP, ctypes.POINTER(I64)], I32),
    "dirigo_alu_peak": ([ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double), VP], I32),
    "dirigo_launch_count": ([], I64),
    "dirigo_last_error": ([], ctypes.c_char_p),
}


def lib_path():
    return _build.LIB


def load(path=None):
    """Load the compiled library (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or lib_path()
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library not built: {path} (run build())")
    L = ctypes.CDLL(path)
    for name, (args, res) in SIGNATURES.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _lib = L
    return L


def _check(st):
    if st != OK:
        raise DirigoError(st, load().dirigo_last_error().decode())


def _const(x):
    if isinstance(x, (list, tuple)):
        f = Fraction(int(x[0]), int(x[1]))
        return Const(float(f), f.numerator, f.denominator)
    return Const(float(x), 0, 0)


def _trail(n, r):
    return list(range(r - n, r))


def _marshal(desc):
    """ctypes dirigo_graph_desc of a graph description (and the buffers it points into)."""
    shapes = [s for _, s in desc["inputs"]] + [op["shape"] for op in desc["ops"] if "shape" in op]
    if any(len(s) > MAX_RANK for s in shapes):
        raise DirigoError(3, "rank above 4 cannot be described")
    ins = (TensorDesc * len(desc["inputs"]))()
    for i, (_, shape) in enumerate(desc["inputs"]):
        ins[i].rank = len(shape)
        for d, s in enumerate(shape):
            ins[i].shape[d] = s
    ops = (OpDesc * max(1, len(desc["ops"])))()
    keep = [ins, ops]
    for k, op in enumerate(desc["ops"]):
        o = ops[k]
        if op["op"] not in OPS:
            raise ValueError(f"op {k}: unknown op {op['op']!r}")
        o.kind = OPS[op["op"]]
        o.n_args = len(op["args"])
        for i, a in enumerate(op["args"]):
            o.args[i] = a
        o.stride = op.get("stride", 0)
        o.pad = op.get("pad", 0)
        o.k = op.get("k", 0)
        o.dim = op.get("dim", 0)
        o.keepdim = int(bool(op.get("keepdim", False)))
        o.axes_rank[0] = o.axes_rank[1] = -1
        if "axes" in op:
            for s in range(2):
                o.axes_rank[s] = len(op["axes"][s])
                for d, ax in enumerate(op["axes"][s]):
                    o.axes[s][d] = ax
        if "c" in op:
            o.c = _const(op["c"])
        elif "eps" in op:
            o.c = _const(op["eps"])
        if "shape" in op and op["op"] in ("contract", "maxset", "kernel_contract",
                                          "kernel_maxset"):
            o.rank = len(op["shape"])
            for d, s in enumerate(op["shape"]):
                o.shape[d] = s
        if op["op"] in ("contract", "maxset"):
            pcs = (Piece * len(op["pieces"]))()
            for q, pc in enumerate(op["pieces"]):
                p = pcs[q]
                lo = pc.get("lo", [0] * len(op["shape"]))
                hi = pc.get("hi", op["shape"])
                for d in range(len(op["shape"])):
                    p.lo[d], p.hi[d] = lo[d], hi[d]
                p.n_red = len(pc["red"])
                for e, (a, b) in enumerate(pc["red"]):
                    p.red_lo[e], p.red_hi[e] = a, b
                p.coef = _const(pc.get("coef", 1.0))
                gs = pc.get("guards", [])
                p.n_guards = len(gs)
                for j, (od, oa, rd, c, glo, ghi) in enumerate(gs):
                    p.guards[j] = Guard(od, rd, oa, c, glo, ghi)
                for i, (base, os_, rs) in enumerate(pc["access"]):
                    p.access[i].base = base
                    for d, v in enumerate(os_):
                        p.access[i].os[d] = v
                    for e, v in enumerate(rs):
                        p.access[i].rs[e] = v
            keep.append(pcs)
            o.n_pieces = len(op["pieces"])
            o.pieces = ctypes.cast(pcs, ctypes.POINTER(Piece))
        if op["op"] in ("kernel_contract", "kernel_maxset"):
            for d in range(3):
                o.grid[d], o.block[d] = op["grid"][d], op["block"][d]
            ws = (KernelWrite * max(1, len(op["writes"])))()
            for q, w in enumerate(op["writes"]):
                kw = ws[q]
                when = w.get("when", [[0, 1 << 62]] * THREAD_DIMS)
                for j in range(THREAD_DIMS):
                    kw.when_lo[j], kw.when_hi[j] = when[j]
                kw.addr_base = w["addr"][0]
                for j in range(THREAD_DIMS):
                    kw.addr[j] = w["addr"][1][j]
                kw.n_red = len(w["red"])
                for e, (a, b) in enumerate(w["red"]):
                    kw.red_lo[e], kw.red_hi[e] = a, b
                kw.coef = _const(w.get("coef", 1.0))
                gs = w.get("guards", [])
                kw.n_guards = len(gs)
                for j, (tc, rd, c, glo, ghi) in enumerate(gs):
                    g = kw.guards[j]
                    for i in range(THREAD_DIMS):
                        g.tc[i] = tc[i]
                    g.rd, g.c, g.lo, g.hi = rd, c, glo, ghi
                for i, (base, tc, rs) in enumerate(w["reads"]):
                    kw.reads[i].base = base
                    for j in range(THREAD_DIMS):
                        kw.reads[i].tc[j] = tc[j]
                    for e, v in enumerate(rs):
                        kw.reads[i].rs[e] = v
            keep.append(ws)
            o.n_writes = len(op["writes"])
            o.writes = ctypes.cast(ws, ctypes.POINTER(KernelWrite))
    gd = GraphDesc(len(desc["inputs"]), ctypes.cast(ins, ctypes.POINTER(TensorDesc)),
                   len(desc["ops"]), ctypes.cast(ops, ctypes.POINTER(OpDesc)),
                   desc["output"])
    return gd, keep


class Graph:
    """One program compiled by dirigo_graph_create (or one side of
    dirigo_graph_create_merged: ``Graph(None, handle=h)``)."""

    def __init__(self, desc, axiom_gelu=False, handle=None):
        L = load()
        if handle is None:
            gd, _keep = _marshal(desc)
            opt = Options(AXIOM_GELU if axiom_gelu else 0)
            h = VP()
            _check(L.dirigo_graph_create(ctypes.byref(gd), ctypes.byref(opt), ctypes.byref(h)))
        else:
            h = handle
        self.h = h
        self.desc = desc
        info = GraphInfo()
        _check(L.dirigo_graph_info_get(h, ctypes.byref(info)))
        self.G = info.n_leaves
        self.out_numel = info.out_numel
        self.out_shape = list(info.out_shape)[:info.out_rank]
        self.n_tensors = info.n_tensors
        self.n_cells = info.n_cells
        self.n_fast_cells = info.n_fast_cells
        self.key_tc_flops = info.key_tc_flops
        self.key_limb_bytes = info.key_limb_bytes
        self.n_gemm = info.n_tc_contractions
        self.max_runs_per_location = info.max_runs_per_location
        self.key_mix_ops = info.key_mix_ops

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.dirigo_graph_destroy(self.h)
            self.h = None

    def workspace_size(self, call, n):
        b = ctypes.c_size_t()
        _check(load().dirigo_workspace_size(self.h, call, n, ctypes.byref(b)))
        return b.value


def merge(ref_desc, cand_desc, axiom_gelu=False):
    """dirigo_graph_create_merged: both programs with their common op prefix
    trimmed (Sec. 3.2 "MERGE").  Returns (ref Graph, cand Graph, cut_ids,
    n_shared_ops): input i of the trimmed programs is tensor cut_ids[i] of the
    given descriptions."""
    L = load()
    gr, keep_r = _marshal(ref_desc)
    gc, keep_c = _marshal(cand_desc)
    opt = Options(AXIOM_GELU if axiom_gelu else 0)
    cap = len(ref_desc["inputs"]) + len(ref_desc["ops"])
    cut = (ctypes.c_int32 * max(cap, 1))()
    info = MergeInfo()
    hr, hc = VP(), VP()
    _check(L.dirigo_graph_create_merged(ctypes.byref(gr), ctypes.byref(gc), ctypes.byref(opt),
                                        ctypes.byref(hr), ctypes.byref(hc), cut, cap,
                                        ctypes.byref(info)))
    ids = [int(cut[i]) for i in range(info.n_inputs)]
    return Graph(None, handle=hr), Graph(None, handle=hc), ids, int(info.n_shared_ops)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ws(nbytes, device):
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


# --------------------------------------------------------------- raw C-ABI calls

def dirigo_cone(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, d_ws, ws_bytes, stream):
    total = ctypes.c_int64(0)
    st = load().dirigo_cone(g.h, d_locs, n, d_offsets, d_runs, run_capacity, d_fp,
                            ctypes.byref(total), d_ws, ws_bytes, stream)
    return st, total.value


def dirigo_cone_async(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, d_status, d_ws,
                      ws_bytes, stream):
    return load().dirigo_cone_async(g.h, d_locs, n, d_offsets, d_runs, run_capacity, d_fp,
                                    d_status, d_ws, ws_bytes, stream)


def dirigo_terms(g, d_locs, n, d_keys, d_ws, ws_bytes, stream):
    return load().dirigo_terms(g.h, d_locs, n, d_keys, d_ws, ws_bytes, stream)


def dirigo_compare(ref, cand, d_locs, n, d_kref, d_kcand, cone_ref, cone_cand, d_verdict,
                   d_flags, budget, d_export, export_capacity, d_ws, ws_bytes, stream,
                   d_cone_status=None, cones_ready=None):
    stats = CompareStats()
    (orr, rr, fr), (oc, rc, fc) = cone_ref, cone_cand
    st = load().dirigo_compare(ref.h, cand.h, d_locs, n, d_kref, d_kcand, orr, rr, fr, oc, rc, fc,
                               d_cone_status, cones_ready, d_verdict, d_flags, budget, d_export,
                               export_capacity, ctypes.byref(stats), d_ws, ws_bytes, stream)
    return st, stats


def dirigo_compare_async(ref, cand, d_locs, n, d_kref, d_kcand, cone_ref, cone_cand, d_verdict,
                         d_flags, budget, d_export, export_capacity, d_stats, d_status, d_ws,
                         ws_bytes, stream, d_cone_status=None, cones_ready=None):
    (orr, rr, fr), (oc, rc, fc) = cone_ref, cone_cand
    return load().dirigo_compare_async(ref.h, cand.h, d_locs, n, d_kref, d_kcand, orr, rr, fr, oc,
                                       rc, fc, d_cone_status, cones_ready, d_verdict, d_flags,
                                       budget, d_export, export_capacity, d_stats, d_status, d_ws,
                                       ws_bytes, stream)


def dirigo_eval(g, d_inputs, d_locs, n, d_out, d_ws, ws_bytes, stream):
    arr = (VP * len(d_inputs))(*[p.value if isinstance(p, ctypes.c_void_p) else p for p in d_inputs])
    return load().dirigo_eval(g.h, arr, d_locs, n, d_out, d_ws, ws_bytes, stream)


def compare_workspace_size(ref, cand, n):
    b = ctypes.c_size_t()
    _check(load().dirigo_compare_workspace_size(ref.h, cand.h, n, ctypes.byref(b)))
    return b.value


# --------------------------------------------------------------- torch-level helpers

def _used_on(stream, *tensors):
    """Tensors allocated here but used by kernels on another stream: tell the
    caching allocator, so their memory is not reused before that stream's
    work on them is done."""
    if stream is None or stream == torch.cuda.current_stream(stream.device):
        return
    for t in tensors:
        if t is not None:
            t.record_stream(stream)


def cone(g, locs, with_fp=True, stream=None, run_capacity=None, ws=None):
    """(offsets int64[n+1], runs int32 view [R, 2] of uint32 data, fingerprints)."""
    dev = locs.device
    n = locs.numel()
    ws = ws if ws is not None else _ws(g.workspace_size(CALL_CONE, n), dev)
    off = torch.empty(n + 1, dtype=torch.int64, device=dev)
    fp = torch.empty(max(n, 1), dtype=torch.int64, device=dev) if with_fp else None
    s = _stream(stream)
    cap = run_capacity if run_capacity is not None else 0
    runs = torch.empty(max(cap, 1) * 2, dtype=torch.int32, device=dev)
    st, total = dirigo_cone(g, _ptr(locs), n, _ptr(off), _ptr(runs), cap, _ptr(fp), _ptr(ws),
                            ws.numel(), s)
    if st == E_CAPACITY:
        runs = torch.empty(max(total, 1) * 2, dtype=torch.int32, device=dev)
        st, total = dirigo_cone(g, _ptr(locs), n, _ptr(off), _ptr(runs), total, _ptr(fp),
                                _ptr(ws), ws.numel(), s)
    _check(st)
    _used_on(stream, ws, off, fp, runs)
    return off, runs[:2 * total].view(total, 2), fp


def terms(g, locs, stream=None, ws=None):
    dev = locs.device
    n = locs.numel()
    ws = ws if ws is not None else _ws(g.workspace_size(CALL_TERMS, n), dev)
    keys = torch.empty((max(n, 1), 2), dtype=torch.int32, device=dev)
    _check(dirigo_terms(g, _ptr(locs), n, _ptr(keys), _ptr(ws), ws.numel(), _stream(stream)))
    _used_on(stream, ws, keys)
    return keys[:n]


def compare(ref, cand, locs, kref, kcand, cone_ref=None, cone_cand=None, budget=4096,
            export_capacity=0, stream=None, ws=None):
    """(verdict uint8[n], flags uint8[n], export bytes tensor or None, stats dict, status)."""
    dev = locs.device
    n = locs.numel()
    ws = ws if ws is not None else _ws(compare_workspace_size(ref, cand, n), dev)
    verdict = torch.empty(max(n, 1), dtype=torch.uint8, device=dev)
    flags = torch.empty(max(n, 1), dtype=torch.uint8, device=dev)
    exp = torch.empty(max(export_capacity, 1), dtype=torch.uint8, device=dev) \
        if export_capacity > 0 else None
    cr = tuple(_ptr(x) for x in cone_ref) if cone_ref else (None, None, None)
    cc = tuple(_ptr(x) for x in cone_cand) if cone_cand else (None, None, None)
    st, stats = dirigo_compare(ref, cand, _ptr(locs), n, _ptr(kref), _ptr(kcand), cr, cc,
                               _ptr(verdict), _ptr(flags), budget, _ptr(exp), export_capacity,
                               _ptr(ws), ws.numel(), _stream(stream))
    if st not in (OK, E_CAPACITY):
        _check(st)
    _used_on(stream, ws, verdict, flags, exp)
    sd = {k: getattr(stats, k) for k, _ in CompareStats._fields_}
    blob = exp[:stats.export_bytes] if (exp is not None and stats.export_bytes) else None
    return verdict[:n], flags[:n], blob, sd, st


def eval_fp32(g, inputs, locs, stream=None, ws=None):
    dev = locs.device
    n = locs.numel()
    ws = ws if ws is not None else _ws(g.workspace_size(CALL_EVAL, n), dev)
    out = torch.empty(max(n, 1), dtype=torch.float32, device=dev)
    ptrs = [ctypes.c_void_p(x.data_ptr()) for x in inputs]
    _check(dirigo_eval(g, ptrs, _ptr(locs), n, _ptr(out), _ptr(ws), ws.numel(), _stream(stream)))
    _used_on(stream, ws, out)
    return out[:n]


def profile_enable(on=True):
    _check(load().dirigo_profile_enable(int(on)))


def profile_read(reset=True):
    n = len(KERNEL_CLASSES)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int64 * n)()
    _check(load().dirigo_profile_read(ms, cnt, n, int(reset)))
    return {k: (ms[i], cnt[i]) for i, k in enumerate(KERNEL_CLASSES)}


def query_order(ref, cand, seed=0):
    """Output locations of a program pair in the heuristic query order:
    (order int64[out_numel], length of the ranked prefix)."""
    order = np.empty(ref.out_numel, dtype=np.int64)
    pre = I64()
    _check(load().dirigo_query_order(ref.h, cand.h, seed, order.ctypes.data, ctypes.byref(pre)))
    return order, int(pre.value)


def alu_peak(stream=None):
    """(SplitMix64 finalisers / s, 32x32->64 multiply-adds / s) on this GPU."""
    a, b = ctypes.c_double(), ctypes.c_double()
    _check(load().dirigo_alu_peak(ctypes.byref(a), ctypes.byref(b), _stream(stream)))
    return a.value, b.value


def launch_count():
    return load().dirigo_launch_count()
