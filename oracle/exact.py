"""Exact canonical forms for tiny programs (oracle pin machinery).

TEST INFRASTRUCTURE ONLY.

The canonical form CF(e) of a resolved expression is its normal form in the
polynomial ring Q[atoms] (Sec. 3.3 "Setup": floats are reals, so ring laws
hold exactly).  Atoms are input leaves, uninterpreted-function applications
f(CF(arg)) (one UF per transcendental, Sec. 3.4 "Flipping the quantifiers"),
and max-sets Max{CF(a_i)} (the data-dependent conditional of max, kept as an
unordered set of argument forms).  Two expressions are "identical canonical
terms" exactly when their CFs are equal.  This module builds CFs with Python
Fractions and hash-consed atoms, so tests can check that the oracle's key
equality coincides with CF equality.
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np

from .lower import lower, UF

NODE_BIT = 1 << 63
NONE = (1 << 64) - 1


class Atoms:
    """Hash-consing table: structural atom -> small integer id."""

    def __init__(self):
        self.ids = {}
        self.items = []

    def intern(self, key):
        i = self.ids.get(key)
        if i is None:
            i = len(self.items)
            self.ids[key] = i
            self.items.append(key)
        return i


def p_const(c):
    c = Fraction(c)
    return () if c == 0 else (((), c),)


def p_atom(a):
    return ((((a, 1),), Fraction(1)),)


def p_add(*ps):
    acc = {}
    for p in ps:
        for m, c in p:
            acc[m] = acc.get(m, 0) + c
    return tuple(sorted((m, c) for m, c in acc.items() if c != 0))


def p_scale(p, c):
    c = Fraction(c)
    if c == 0:
        return ()
    return tuple((m, v * c) for m, v in p)


def _m_mul(m1, m2):
    d = dict(m1)
    for a, k in m2:
        d[a] = d.get(a, 0) + k
    return tuple(sorted(d.items()))


def p_mul(p, q):
    acc = {}
    for m1, c1 in p:
        for m2, c2 in q:
            m = _m_mul(m1, m2)
            acc[m] = acc.get(m, 0) + c1 * c2
    return tuple(sorted((m, c) for m, c in acc.items() if c != 0))


def decode_ref(w):
    if w == NONE:
        return None
    if w & NODE_BIT:
        return ("n", (w >> 40) & ((1 << 23) - 1), w & ((1 << 40) - 1))
    return ("l", w)


class ExactProgram:
    """CFs of a program's output locations (uses the oracle's term enumeration)."""

    def __init__(self, prog, atoms, axiom_gelu=False):
        self.prog = prog
        self.atoms = atoms
        self.axiom_gelu = axiom_gelu
        inputs, prims, out = lower(prog.graph)
        self.n_inputs = len(inputs)
        self.prims = prims
        self.memo = {}

    def ref_cf(self, r):
        if r[0] == "l":
            return p_atom(self.atoms.intern(("L", r[1])))
        return self.node_cf(r[1], r[2])

    def node_cf(self, t, e):
        key = (t, e)
        if key in self.memo:
            return self.memo[key]
        p = self.prims[t - self.n_inputs]
        coef, ra, rb = self.prog.terms(t, e)
        ents = [(Fraction(float(c)), decode_ref(int(a)), decode_ref(int(b)))
                for c, a, b in zip(coef, ra, rb)]
        kind = p["kind"]
        if kind in ("maxset", "maxc"):
            members = set()
            for c, a, _ in ents:
                members.add(p_const(c) if a is None else self.ref_cf(a))
            if len(members) == 1:
                cf = next(iter(members))
            else:
                cf = p_atom(self.atoms.intern(("M", frozenset(members))))
        elif kind == "unary":
            fid = UF[p["fn"]]
            if self.axiom_gelu and fid == UF["gelu_tanh"]:
                fid = UF["gelu_erf"]
            cf = p_atom(self.atoms.intern(("F", fid, self.ref_cf(ents[0][1]))))
        elif kind == "binary" and p["fn"] == "div":
            _, a, b = ents[0]
            rc = p_atom(self.atoms.intern(("F", UF["recip"], self.ref_cf(b))))
            cf = p_mul(self.ref_cf(a), rc)
        else:
            parts = []
            for c, a, b in ents:
                term = p_const(c)
                for r in (a, b):
                    if r is not None:
                        term = p_mul(term, self.ref_cf(r))
                parts.append(term)
            cf = p_add(*parts)
        self.memo[key] = cf
        return cf

    def out_cf(self, loc):
        out_t = lower(self.prog.graph)[2]
        if out_t < self.n_inputs:
            base = sum(math.prod(s) for _, s in self.prog.graph["inputs"][:out_t])
            return p_atom(self.atoms.intern(("L", base + loc)))
        return self.node_cf(out_t, int(loc))


def eval_cf(cf, atoms, leaf_value, memo=None):
    """Numerical value of a CF (UFs evaluated as the real functions)."""
    memo = {} if memo is None else memo

    def atom_val(i):
        if i in memo:
            return memo[i]
        a = atoms.items[i]
        if a[0] == "L":
            v = leaf_value(a[1])
        elif a[0] == "F":
            x = eval_cf(a[2], atoms, leaf_value, memo)
            v = _uf(a[1], x)
        else:
            v = max(eval_cf(m, atoms, leaf_value, memo) for m in a[1])
        memo[i] = v
        return v

    s = 0.0
    with np.errstate(all="ignore"):
        for m, c in cf:
            t = np.float64(c)
            for a, k in m:
                t = t * np.float64(atom_val(a)) ** k
            s = s + t
    return float(s)


def _uf(fid, x):
    if not math.isfinite(x):
        return float("nan")
    if fid == UF["exp"]:
        return math.exp(x) if x < 700 else float("inf")
    if fid == UF["tanh"]:
        return math.tanh(x)
    if fid == UF["gelu_erf"]:
        return 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))
    if fid == UF["gelu_tanh"]:
        k = math.sqrt(2.0 / math.pi)
        return 0.5 * x * (1.0 + math.tanh(k * (x + 0.044715 * x ** 3)))
    if fid == UF["erf"]:
        return math.erf(x)
    if fid == UF["rsqrt"]:
        return 1.0 / math.sqrt(x) if x > 0 else float("nan")
    if fid == UF["recip"]:
        return 1.0 / x if x != 0 else float("nan")
    if fid == UF["sqrt"]:
        return math.sqrt(x) if x >= 0 else float("nan")
    if fid == UF["log"]:
        return math.log(x) if x > 0 else float("nan")
    raise ValueError(fid)


def leaves_of(cf, atoms, acc=None):
    """Leaf ids occurring in a CF (after simplification)."""
    acc = set() if acc is None else acc
    for m, _ in cf:
        for a, _ in m:
            it = atoms.items[a]
            if it[0] == "L":
                acc.add(it[1])
            elif it[0] == "F":
                leaves_of(it[2], atoms, acc)
            else:
                for mm in it[1]:
                    leaves_of(mm, atoms, acc)
    return acc
