"""CPU oracle for the per-output-location equivalence check (Dirigo, Sec. 3.4).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline leg, never by the product path.  It shares no
code with the CUDA library and does not import it.

* ``lower.py``  -- per-element equations of every op (the oracle's own lowering)
* ``core.cpp``  -- back-projection res(), cones, keys, fp64 evaluation, export
* ``exact.py``  -- exact canonical forms over Q[atoms] for tiny graphs (pins)
* ``forward64.py`` -- an independent fp64 direct forward pass (torch CPU ops)

Parity unpinned: the key's constants (the two primes, the two seeds, the
function tags) are arbitrary choices; they are fixed only by the key laws the
pins check and by agreement with the CUDA path.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .lower import encode, lower  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

I64P = ctypes.POINTER(ctypes.c_int64)
U32P = ctypes.POINTER(ctypes.c_uint32)
F64P = ctypes.POINTER(ctypes.c_double)
U64P = ctypes.POINTER(ctypes.c_uint64)


def build(force=False):
    """Compile the oracle core with the host C++ compiler."""
    src = os.path.join(_HERE, "core.cpp")
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(src):
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    subprocess.check_call(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread",
                           "-o", tmp, src])
    os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            L.orc_create.restype = ctypes.c_void_p
            L.orc_create.argtypes = [I64P, ctypes.c_int64]
            L.orc_destroy.argtypes = [ctypes.c_void_p]
            for f in ("orc_num_leaves", "orc_out_numel", "orc_num_tensors"):
                getattr(L, f).restype = ctypes.c_int64
                getattr(L, f).argtypes = [ctypes.c_void_p]
            L.orc_tensor_numel.restype = ctypes.c_int64
            L.orc_tensor_numel.argtypes = [ctypes.c_void_p, ctypes.c_int64]
            L.orc_cone.restype = ctypes.c_int64
            L.orc_cone.argtypes = [ctypes.c_void_p, ctypes.c_int64, U32P, ctypes.c_int64]
            L.orc_cone_stats.argtypes = [ctypes.c_void_p, I64P, ctypes.c_int64, I64P, I64P,
                                         ctypes.c_int]
            L.orc_cone_runs.argtypes = [ctypes.c_void_p, I64P, ctypes.c_int64, I64P, U32P,
                                        ctypes.c_int]
            L.orc_keys.argtypes = [ctypes.c_void_p, I64P, ctypes.c_int64, U32P, ctypes.c_int,
                                   ctypes.c_int]
            L.orc_keys_of.argtypes = [ctypes.c_void_p, ctypes.c_int64, I64P, ctypes.c_int64,
                                      U32P, ctypes.c_int]
            L.orc_eval.argtypes = [ctypes.c_void_p, ctypes.POINTER(F64P), I64P, ctypes.c_int64,
                                   F64P, ctypes.c_int]
            L.orc_export.restype = ctypes.c_int64
            L.orc_export.argtypes = [ctypes.c_void_p, ctypes.c_void_p, I64P, I64P,
                                     ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64]
            L.orc_terms.restype = ctypes.c_int64
            L.orc_terms.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, F64P,
                                    U64P, U64P, ctypes.c_int64]
            L.orc_mix64.restype = ctypes.c_uint64
            L.orc_mix64.argtypes = [ctypes.c_uint64]
            L.orc_last_error.restype = ctypes.c_char_p
            _lib = L
    return _lib


def _p(a, t):
    return a.ctypes.data_as(t)


def default_threads():
    return max(1, os.cpu_count() or 1)


class Program:
    """One program (reference or candidate) under the oracle."""

    def __init__(self, graph):
        self.graph = graph
        words = np.asarray(encode(graph), dtype=np.int64)
        L = lib()
        self.h = L.orc_create(_p(words, I64P), len(words))
        if not self.h:
            raise ValueError(L.orc_last_error().decode())
        self.G = L.orc_num_leaves(self.h)
        self.out_numel = L.orc_out_numel(self.h)

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_destroy(self.h)
            self.h = None

    def cone(self, loc):
        """Sorted unique global leaf ids of res(y[loc]) (bottom = G)."""
        n = lib().orc_cone(self.h, int(loc), None, 0)
        out = np.empty(n, dtype=np.uint32)
        lib().orc_cone(self.h, int(loc), _p(out, U32P), n)
        return out

    def cone_runs(self, locs, nthreads=None):
        """(offsets int64[n+1], runs uint32[R, 2]) with maximal runs."""
        locs = np.ascontiguousarray(locs, dtype=np.int64)
        n = len(locs)
        nt = nthreads or default_threads()
        sizes = np.empty(n, dtype=np.int64)
        nruns = np.empty(n, dtype=np.int64)
        lib().orc_cone_stats(self.h, _p(locs, I64P), n, _p(sizes, I64P), _p(nruns, I64P), nt)
        off = np.zeros(n + 1, dtype=np.int64)
        np.cumsum(nruns, out=off[1:])
        runs = np.empty((int(off[-1]), 2), dtype=np.uint32)
        lib().orc_cone_runs(self.h, _p(locs, I64P), n, _p(off, I64P), _p(runs, U32P), nt)
        return off, runs

    def cone_sizes(self, locs, nthreads=None):
        locs = np.ascontiguousarray(locs, dtype=np.int64)
        n = len(locs)
        sizes = np.empty(n, dtype=np.int64)
        nruns = np.empty(n, dtype=np.int64)
        lib().orc_cone_stats(self.h, _p(locs, I64P), n, _p(sizes, I64P), _p(nruns, I64P),
                             nthreads or default_threads())
        return sizes, nruns

    def keys(self, locs, axiom_gelu=False, nthreads=None):
        """Root keys, uint32[n, 2] (lane 0, lane 1)."""
        locs = np.ascontiguousarray(locs, dtype=np.int64)
        out = np.empty((len(locs), 2), dtype=np.uint32)
        lib().orc_keys(self.h, _p(locs, I64P), len(locs), _p(out, U32P), int(axiom_gelu),
                       nthreads or default_threads())
        return out

    def keys_of(self, tensor, elems, axiom_gelu=False):
        elems = np.ascontiguousarray(elems, dtype=np.int64)
        out = np.empty((len(elems), 2), dtype=np.uint32)
        lib().orc_keys_of(self.h, int(tensor), _p(elems, I64P), len(elems), _p(out, U32P),
                          int(axiom_gelu))
        return out

    def eval(self, inputs, locs, nthreads=None):
        """fp64 value of res(y[l]) on concrete inputs (NaN where bottom is read)."""
        ins = [np.ascontiguousarray(x, dtype=np.float64).ravel() for x in inputs]
        arr = (F64P * len(ins))(*[_p(x, F64P) for x in ins])
        locs = np.ascontiguousarray(locs, dtype=np.int64)
        out = np.empty(len(locs), dtype=np.float64)
        lib().orc_eval(self.h, arr, _p(locs, I64P), len(locs), _p(out, F64P),
                       nthreads or default_threads())
        return out

    def terms(self, tensor, elem, cap=1 << 20):
        coef = np.empty(cap, dtype=np.float64)
        ra = np.empty(cap, dtype=np.uint64)
        rb = np.empty(cap, dtype=np.uint64)
        k = lib().orc_terms(self.h, int(tensor), int(elem), _p(coef, F64P), _p(ra, U64P),
                            _p(rb, U64P), cap)
        k = min(k, cap)
        return coef[:k], ra[:k], rb[:k]


# verdict codes and flag bits (Sec. 3.4 "Solving": an identical canonical term
# discharges the location; the rest is handed to a solver as term lists)
DISCHARGED, EXPORTED, DIFFERS_UNEXPORTED = 0, 1, 2
FLAG_CONE_DIFFERS, FLAG_BOT_REF, FLAG_BOT_CAND = 1, 2, 4


def compare(ref, cand, locs, kref, kcand, cones=None, budget=4096, capacity=1 << 62):
    """Verdicts, flags and the export bytes of one batch.

    cones: optional ((off_r, runs_r), (off_c, runs_c)) from Program.cone_runs.
    The first ``budget`` undischarged query slots are exported when the whole
    export fits in ``capacity`` bytes; otherwise none is and the required size
    is returned.
    """
    locs = np.ascontiguousarray(locs, dtype=np.int64)
    n = len(locs)
    eq = np.all(kref == kcand, axis=1)
    verdict = np.where(eq, DISCHARGED, DIFFERS_UNEXPORTED).astype(np.uint8)
    flags = np.zeros(n, dtype=np.uint8)
    if cones is not None:
        (orr, rr), (oc, rc) = cones
        for i in range(n):
            a = rr[orr[i]:orr[i + 1]]
            b = rc[oc[i]:oc[i + 1]]
            if a.shape != b.shape or not np.array_equal(a, b):
                flags[i] |= FLAG_CONE_DIFFERS
            if len(a) and int(a[-1, 0]) + int(a[-1, 1]) == ref.G + 1:
                flags[i] |= FLAG_BOT_REF
            if len(b) and int(b[-1, 0]) + int(b[-1, 1]) == cand.G + 1:
                flags[i] |= FLAG_BOT_CAND
    und = np.nonzero(~eq)[0]
    sel = und[:budget]
    if len(sel) == 0:   # nothing selected: no export at all (not even a header)
        return verdict, flags, None, 0
    need = export_size(ref, cand, sel, locs[sel])
    blob = None
    if need <= capacity:
        blob = export(ref, cand, sel, locs[sel])
        verdict[sel] = EXPORTED
    return verdict, flags, blob, need


def export_size(ref, cand, slots, locs):
    """Bytes of the DXP1 export of the given query slots (at their locations)."""
    slots = np.ascontiguousarray(slots, dtype=np.int64)
    sl = np.ascontiguousarray(locs, dtype=np.int64)
    return lib().orc_export(ref.h, cand.h, _p(slots, I64P), _p(sl, I64P), len(slots), None, 0)


def export(ref, cand, slots, locs):
    """The DXP1 export (bytes) of the given query slots, in the given order:
    both programs' equation nodes reachable from the slots' roots, then one
    record per slot (Sec. 3.4 "Solving": the term lists a solver receives)."""
    slots = np.ascontiguousarray(slots, dtype=np.int64)
    sl = np.ascontiguousarray(locs, dtype=np.int64)
    need = export_size(ref, cand, slots, sl)
    buf = np.empty(need, dtype=np.uint8)
    lib().orc_export(ref.h, cand.h, _p(slots, I64P), _p(sl, I64P), len(slots),
                     buf.ctypes.data_as(ctypes.c_void_p), need)
    return buf.tobytes()
