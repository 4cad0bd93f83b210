"""A small evaluator for the SMT-LIB 2 subset the query emitter writes (test
infrastructure): declare-fun / define-fun over Real, +, -, *, /, ite, >=,
numerals, and unary functions given by the caller."""
import math
from fractions import Fraction


def tokens(text):
    out = []
    for line in text.splitlines():
        line = line.split(";", 1)[0]
        out += line.replace("(", " ( ").replace(")", " ) ").split()
    return out


def parse(text):
    toks = tokens(text)
    pos = 0

    def expr():
        nonlocal pos
        t = toks[pos]
        pos += 1
        if t != "(":
            return t
        lst = []
        while toks[pos] != ")":
            lst.append(expr())
        pos += 1
        return lst

    forms = []
    while pos < len(toks):
        forms.append(expr())
    return forms


def evaluate(text, leaf, funcs, bot=float("nan")):
    """Values of the two roots compared by the script's assertion."""
    defs = {}
    roots = None
    for f in parse(text):
        if f[0] == "define-fun":
            defs[f[1]] = f[4]
        elif f[0] == "assert":
            _, eq = f[1]
            roots = eq[1], eq[2]
    memo = {}

    def ev(e):
        if isinstance(e, str):
            if e in memo:
                return memo[e]
            if e in defs:
                v = ev(defs[e])
            elif e == "bot":
                v = bot
            elif e.startswith("x") and e[1:].isdigit():
                v = leaf(int(e[1:]))
            else:
                v = float(Fraction(e))
            memo[e] = v
            return v
        op, args = e[0], [ev(a) for a in e[1:]]
        if op == "+":
            return sum(args)
        if op == "*":
            return math.prod(args)
        if op == "-":
            return -args[0] if len(args) == 1 else args[0] - sum(args[1:])
        if op == "/":
            return args[0] / args[1]
        if op == ">=":
            return args[0] >= args[1]
        if op == "ite":
            return args[1] if args[0] else args[2]
        return funcs[op](*args)

    return ev(roots[0]), ev(roots[1])
