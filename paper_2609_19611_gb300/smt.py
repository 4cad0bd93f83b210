"""SMT-LIB 2 queries from exported term lists (Sec. 3.4 "Solving").

For one exported location the solver decides e_A != e_B, where e_A and e_B
are res(y[l]) in the reference and the candidate: a quantifier-free formula
over the reals with one uninterpreted function per transcendental (Sec. 3.4:
floats are modelled as reals).  ``unsat`` means the location is equivalent
under that model; ``sat`` yields a witness input.

The export ("DXP1", read by ``shard.parse_export``) holds each program's
equation DAG: a node is (tensor, element) with a kind and a list of entries
{coef, a, b}; a ref is a node, a global leaf id (the largest, G, is bottom,
the value read outside a tensor) or none.  The query declares one real per
leaf reached (``x<g>``; bottom is ``bot``), defines one term per node
(``r_<t>_<e>`` / ``c_<t>_<e>``, shared subterms once), and asserts that the
two roots differ:

  kind 1 (sum)   sum of coef * a * b over the entries (absent a/b omitted)
  kind 2 (max)   the maximum of the members (a constant member when a is none)
  kind 3 (func)  f(a) for the node's function f (uninterpreted)
  kind 4 (div)   a / b

This module only formats text; it needs no solver (none is installed here).
"""
from __future__ import annotations

from fractions import Fraction

from .shard import parse_export

__all__ = ["FUNCTIONS", "location_query", "export_queries"]

NODE_BIT = 1 << 63
NONE = (1 << 64) - 1

# function ids of the export's kind-3 nodes and their uninterpreted names
FUNCTIONS = {1: "exp", 2: "tanh", 3: "gelu", 4: "gelu_tanh", 5: "erf", 6: "rsqrt",
             7: "recip", 8: "sqrt", 9: "log"}


def _num(x):
    """Exact SMT-LIB real literal of a float."""
    f = Fraction(x)
    n, d = f.numerator, f.denominator
    lit = f"{abs(n)}.0" if d == 1 else f"(/ {abs(n)}.0 {d}.0)"
    return f"(- {lit})" if n < 0 else lit


class _Emitter:
    def __init__(self, progs, G):
        self.progs = progs
        self.G = G
        self.lines = []
        self.leaves = set()
        self.bottom = False
        self.funcs = set()
        self.done = set()

    def ref(self, p, r):
        if r == NONE:
            raise ValueError("none ref")
        if r & NODE_BIT:
            key = ((r >> 40) & ((1 << 23) - 1), r & ((1 << 40) - 1))
            self.node(p, key)
            return f"{'rc'[p]}_{key[0]}_{key[1]}"
        return self.leaf(r)

    def leaf(self, g):
        if self.G is not None and g >= self.G:
            self.bottom = True
            return "bot"
        self.leaves.add(g)
        return f"x{g}"

    def node(self, p, key):
        if (p, key) in self.done:
            return
        self.done.add((p, key))
        kind, fn, ents = self.progs[p][key]
        if kind == 1:
            terms = []
            for c, a, b in ents:
                fac = [self.ref(p, x) for x in (a, b) if x != NONE]
                if not fac:
                    terms.append(_num(c))
                elif c == 1.0:
                    terms.append(fac[0] if len(fac) == 1 else f"(* {' '.join(fac)})")
                else:
                    terms.append(f"(* {_num(c)} {' '.join(fac)})")
            body = terms[0] if len(terms) == 1 else (f"(+ {' '.join(terms)})" if terms else "0.0")
        elif kind == 2:
            members = [_num(c) if a == NONE else self.ref(p, a) for c, a, _ in ents]
            body = members[0]
            for m in members[1:]:
                body = f"(ite (>= {body} {m}) {body} {m})"
        elif kind == 3:
            name = FUNCTIONS[fn]
            self.funcs.add(name)
            body = f"({name} {self.ref(p, ents[0][1])})"
        elif kind == 4:
            body = f"(/ {self.ref(p, ents[0][1])} {self.ref(p, ents[0][2])})"
        else:
            raise ValueError(f"node kind {kind}")
        self.lines.append(f"(define-fun {'rc'[p]}_{key[0]}_{key[1]} () Real {body})")


def location_query(blob, i, G=None):
    """SMT-LIB 2 script deciding e_A != e_B for the i-th exported location.

    G: the programs' bottom leaf id (the largest global id); leaf ids >= G
    read the shared undefined value ``bot``.  Without G every leaf is a
    variable.
    """
    progs, locs = parse_export(blob)
    slot, r0, r1 = locs[i]
    em = _Emitter(progs, G)
    a = em.ref(0, r0)
    b = em.ref(1, r1)
    head = ["; dirigo: exported location slot %d" % slot, "(set-logic QF_UFNRA)"]
    head += [f"(declare-fun x{g} () Real)" for g in sorted(em.leaves)]
    if em.bottom:
        head.append("(declare-fun bot () Real)")
    head += [f"(declare-fun {f} (Real) Real)" for f in sorted(em.funcs)]
    tail = [f"(assert (not (= {a} {b})))", "(check-sat)"]
    return "\n".join(head + em.lines + tail) + "\n"


def export_queries(blob, G=None):
    """One query per exported location: list of (slot, script)."""
    _, locs = parse_export(blob)
    return [(locs[i][0], location_query(blob, i, G)) for i in range(len(locs))]
