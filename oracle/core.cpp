// Dirigo oracle: a plain, slow, obviously-correct CPU interpreter of the
// per-output-location equivalence check.
//
// TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
// CPU-baseline leg load this library.  It shares no code, header, table or
// constant generator with the CUDA path.
//
// What it computes, per queried output location l of a program (Sec. 3.4):
//   * res(y[l]) by back-projection through the per-element equations
//     (Sec. 3.4 "Back-projection"), memoised per (tensor, element) within one
//     location;
//   * cone(l): the sorted unique global leaf ids occurring in res(y[l]) before
//     any simplification, bottom (id G) included when an out-of-range read is
//     reached (Sec. 3.3, undefined values);
//   * key(l): the value of res(y[l]) under a ring homomorphism from Q[atoms]
//     into F_p0 x F_p1 (leaves and uninterpreted-function applications are
//     atoms, Sec. 3.3 "Setup": floats as reals, transcendentals as UFs; max as
//     an unordered set).  Equal canonical forms give equal keys;
//   * eval(l): res(y[l]) evaluated in double precision on concrete inputs
//     (the semantics [[R_y(i)]]_x of Sec. 3.3 "Setup");
//   * the exported term lists of undischarged locations.
//
// Key definition (both sides implement it from this text, nothing is shared):
//   mix64       = the SplitMix64 output finaliser (Steele, Lea, Flood 2014)
//   p0 = 2^29-3, p1 = 2^29-33; sigma0 = 0x243F6A8885A308D3, sigma1 = 0x13198A2E03707344
//   leaf g      : mix64(sigma_s + (g+1)*0x9E3779B97F4A7C15) mod p_s
//   constant    : m*2^e/d  ->  m * 2^e * d^-1 mod p_s
//   sum/product : ring operations mod p_s
//   f(a)        : mix64(mix64(K0(a) | K1(a)<<32) ^ (fid*0x9E3779B97F4A7C15) ^ sigma_s) mod p_s
//   a / b       : K(a) * K(recip(b))
//   Max{a_i}    : u_i = K0(a_i) | K1(a_i)<<32, sorted ascending, duplicates dropped;
//                 one member -> that member; else h = 0x4D41585345545F31,
//                 h = mix64(h ^ u) over the sorted u, key_s = mix64(h ^ sigma_s) mod p_s
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <string>
#include <thread>
#include <unordered_map>
#include <unordered_set>
#include <vector>

namespace {

const uint64_t kP[2] = {536870909ull, 536870879ull};
const uint64_t kSigma[2] = {0x243F6A8885A308D3ull, 0x13198A2E03707344ull};
const uint64_t kGamma = 0x9E3779B97F4A7C15ull;
const uint64_t kMaxTag = 0x4D41585345545F31ull;
const uint64_t kNone = ~0ull;

enum Kind { CONTRACT = 1, MAXSET = 2, UNARY = 3, MAXC = 4, AFFINE = 5, BINARY = 6 };
enum Fn { EXP = 1, TANH = 2, GELU_ERF = 3, GELU_TANH = 4, ERF = 5, RSQRT = 6,
          RECIP = 7, SQRT = 8, LOG = 9 };
enum Bin { ADD = 1, SUB = 2, MUL = 3, DIV = 4 };
enum NodeKind { N_SUM = 1, N_MAX = 2, N_FUNC = 3, N_DIV = 4 };

uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  return z ^ (z >> 31);
}

uint64_t mulmod(uint64_t a, uint64_t b, uint64_t p) { return (a % p) * (b % p) % p; }
uint64_t addmod(uint64_t a, uint64_t b, uint64_t p) { return (a + b) % p; }
uint64_t powmod(uint64_t b, uint64_t e, uint64_t p) {
  uint64_t r = 1;
  b %= p;
  while (e) {
    if (e & 1) r = r * b % p;
    b = b * b % p;
    e >>= 1;
  }
  return r;
}
uint64_t invmod(uint64_t a, uint64_t p) { return powmod(a, p - 2, p); }

struct Const {
  int64_t m = 0;
  int64_t e = 0;
  int64_t d = 1;
  double val() const { return std::ldexp((double)m, (int)e) / (double)d; }
  bool zero() const { return m == 0; }
  uint64_t enc(int s) const {
    uint64_t p = kP[s];
    uint64_t mm = (uint64_t)(m < 0 ? -m : m) % p;
    if (m < 0) mm = (p - mm) % p;
    uint64_t two = e >= 0 ? powmod(2, (uint64_t)e, p) : powmod(invmod(2, p), (uint64_t)(-e), p);
    return mulmod(mulmod(mm, two, p), invmod((uint64_t)d % p, p), p);
  }
};

struct Guard { int64_t od, oa, rd, c, lo, hi; };
struct Access { int64_t base; std::vector<int64_t> os, rs; };
struct Piece {
  std::vector<int64_t> lo, hi, rlo, rhi;
  Const coef;
  std::vector<Guard> guards;
  std::vector<Access> acc;
};
struct Op {
  int kind = 0, fn = 0;
  std::vector<int> args;
  std::vector<int64_t> shape;
  std::vector<Piece> pieces;
  Const a, c;
  std::vector<int64_t> axes[2];
};

struct Prog {
  int n_inputs = 0;
  int output = 0;
  std::vector<std::vector<int64_t>> shapes;   // every tensor
  std::vector<int64_t> numel, base;           // base: global id base of inputs
  int64_t G = 0;
  std::vector<Op> ops;                        // ops[t - n_inputs]
  std::string err;
};

// A reference to a value: a leaf (global id, bottom = G) or an element of an
// intermediate tensor.
struct Ref {
  int64_t t;   // -1: leaf; otherwise tensor id >= n_inputs
  int64_t e;   // leaf: global id; node: flat element index
};

bool parse(const int64_t* w, int64_t len, Prog& P) {
  int64_t i = 0;
  auto rd = [&](int64_t& x) {
    if (i >= len) return false;
    x = w[i++];
    return true;
  };
  int64_t ni, nops, out;
  if (!rd(ni) || !rd(nops) || !rd(out)) return false;
  P.n_inputs = (int)ni;
  P.output = (int)out;
  int64_t gbase = 0;
  for (int64_t t = 0; t < ni; ++t) {
    int64_t r;
    if (!rd(r)) return false;
    std::vector<int64_t> s(r);
    int64_t n = 1;
    for (auto& x : s) {
      if (!rd(x)) return false;
      n *= x;
    }
    P.shapes.push_back(s);
    P.numel.push_back(n);
    P.base.push_back(gbase);
    gbase += n;
  }
  P.G = gbase;
  auto rdc = [&](Const& c) { return rd(c.m) && rd(c.e) && rd(c.d); };
  for (int64_t k = 0; k < nops; ++k) {
    Op op;
    int64_t kind, fn, na;
    if (!rd(kind) || !rd(fn) || !rd(na)) return false;
    op.kind = (int)kind;
    op.fn = (int)fn;
    for (int64_t j = 0; j < na; ++j) {
      int64_t a;
      if (!rd(a)) return false;
      op.args.push_back((int)a);
    }
    int64_t r;
    if (!rd(r)) return false;
    op.shape.resize(r);
    int64_t n = 1;
    for (auto& x : op.shape) {
      if (!rd(x)) return false;
      n *= x;
    }
    if (kind == CONTRACT || kind == MAXSET) {
      int64_t np;
      if (!rd(np)) return false;
      for (int64_t q = 0; q < np; ++q) {
        Piece pc;
        pc.lo.resize(r);
        pc.hi.resize(r);
        for (auto& x : pc.lo) if (!rd(x)) return false;
        for (auto& x : pc.hi) if (!rd(x)) return false;
        int64_t nr;
        if (!rd(nr)) return false;
        pc.rlo.resize(nr);
        pc.rhi.resize(nr);
        for (int64_t j = 0; j < nr; ++j)
          if (!rd(pc.rlo[j]) || !rd(pc.rhi[j])) return false;
        if (!rdc(pc.coef)) return false;
        int64_t ng;
        if (!rd(ng)) return false;
        for (int64_t j = 0; j < ng; ++j) {
          Guard g;
          if (!rd(g.od) || !rd(g.oa) || !rd(g.rd) || !rd(g.c) || !rd(g.lo) || !rd(g.hi))
            return false;
          pc.guards.push_back(g);
        }
        for (int64_t j = 0; j < na; ++j) {
          Access a;
          if (!rd(a.base)) return false;
          a.os.resize(r);
          a.rs.resize(nr);
          for (auto& x : a.os) if (!rd(x)) return false;
          for (auto& x : a.rs) if (!rd(x)) return false;
          pc.acc.push_back(a);
        }
        op.pieces.push_back(pc);
      }
    } else if (kind == MAXC) {
      if (!rdc(op.c)) return false;
    } else if (kind == AFFINE) {
      if (!rdc(op.a) || !rdc(op.c)) return false;
    } else if (kind == BINARY) {
      for (int s = 0; s < 2; ++s) {
        int64_t ra;
        if (!rd(ra)) return false;
        op.axes[s].resize(ra);
        for (auto& x : op.axes[s]) if (!rd(x)) return false;
      }
    }
    P.shapes.push_back(op.shape);
    P.numel.push_back(n);
    P.ops.push_back(op);
  }
  return i == len;
}

// flat index -> coordinates (row-major)
void unflatten(int64_t e, const std::vector<int64_t>& shape, std::vector<int64_t>& o) {
  o.assign(shape.size(), 0);
  for (int64_t d = (int64_t)shape.size() - 1; d >= 0; --d) {
    o[d] = e % shape[d];
    e /= shape[d];
  }
}

int64_t flatten(const std::vector<int64_t>& o, const std::vector<int64_t>& shape) {
  int64_t e = 0;
  for (size_t d = 0; d < shape.size(); ++d) e = e * shape[d] + o[d];
  return e;
}

// Reference to element `off` of tensor t, or bottom when off is out of range.
Ref ref_of(const Prog& P, int t, int64_t off) {
  if (off < 0 || off >= P.numel[t]) return Ref{-1, P.G};
  if (t < P.n_inputs) return Ref{-1, P.base[t] + off};
  return Ref{t, off};
}

// One term of a per-element equation: coef * ref0 * ref1 (absent refs have
// t = -2).
struct Term {
  Const coef;
  Ref r[2];
  int nref;
};

const Ref kAbsent{-2, 0};

// Enumerate the terms of T_t[e] in equation order (pieces in declared order,
// reduction coordinates row-major).  Calls f(Term).
template <class F>
void for_each_term(const Prog& P, int t, int64_t e, F&& f) {
  const Op& op = P.ops[t - P.n_inputs];
  std::vector<int64_t> o;
  unflatten(e, op.shape, o);
  switch (op.kind) {
    case CONTRACT:
    case MAXSET: {
      for (const Piece& pc : op.pieces) {
        bool in = true;
        for (size_t d = 0; d < o.size(); ++d)
          if (o[d] < pc.lo[d] || o[d] >= pc.hi[d]) in = false;
        if (!in) continue;
        size_t nr = pc.rlo.size();
        bool empty = false;
        for (size_t j = 0; j < nr; ++j)
          if (pc.rlo[j] >= pc.rhi[j]) empty = true;
        if (empty) continue;
        std::vector<int64_t> r(pc.rlo);
        while (true) {
          bool ok = true;
          for (const Guard& g : pc.guards) {
            int64_t v = g.c;
            if (g.od >= 0) v += g.oa * o[g.od];
            if (g.rd >= 0) v += r[g.rd];
            if (v < g.lo || v >= g.hi) ok = false;
          }
          if (ok) {
            Term tm;
            tm.coef = op.kind == CONTRACT ? pc.coef : Const{1, 0, 1};
            tm.nref = (int)op.args.size();
            tm.r[0] = tm.r[1] = kAbsent;
            for (size_t i = 0; i < op.args.size(); ++i) {
              const Access& a = pc.acc[i];
              int64_t off = a.base;
              for (size_t d = 0; d < o.size(); ++d) off += a.os[d] * o[d];
              for (size_t j = 0; j < nr; ++j) off += a.rs[j] * r[j];
              tm.r[i] = ref_of(P, op.args[i], off);
            }
            f(tm);
          }
          // next reduction coordinate, row-major
          int64_t j = (int64_t)nr - 1;
          while (j >= 0) {
            if (++r[j] < pc.rhi[j]) break;
            r[j] = pc.rlo[j];
            --j;
          }
          if (j < 0) break;
        }
      }
      break;
    }
    case UNARY:
    case MAXC:
    case AFFINE: {
      Term tm;
      tm.coef = op.kind == AFFINE ? op.a : Const{1, 0, 1};
      tm.nref = 1;
      tm.r[0] = ref_of(P, op.args[0], e);
      tm.r[1] = kAbsent;
      f(tm);
      if (op.kind == MAXC || (op.kind == AFFINE && !op.c.zero())) {
        Term c;
        c.coef = op.c;
        c.nref = 0;
        c.r[0] = c.r[1] = kAbsent;
        f(c);
      }
      break;
    }
    case BINARY: {
      int64_t idx[2];
      for (int s = 0; s < 2; ++s) {
        const auto& sh = P.shapes[op.args[s]];
        std::vector<int64_t> oi(sh.size());
        for (size_t d = 0; d < sh.size(); ++d)
          oi[d] = sh[d] == 1 ? 0 : o[op.axes[s][d]];
        idx[s] = flatten(oi, sh);
      }
      Ref ra = ref_of(P, op.args[0], idx[0]);
      Ref rb = ref_of(P, op.args[1], idx[1]);
      if (op.fn == ADD || op.fn == SUB) {
        f(Term{Const{1, 0, 1}, {ra, kAbsent}, 1});
        f(Term{Const{op.fn == ADD ? 1 : -1, 0, 1}, {rb, kAbsent}, 1});
      } else {  // MUL, DIV: one term with both operands
        f(Term{Const{1, 0, 1}, {ra, rb}, 2});
      }
      break;
    }
  }
}

int node_kind(const Op& op) {
  switch (op.kind) {
    case CONTRACT: case AFFINE: return N_SUM;
    case MAXSET: case MAXC: return N_MAX;
    case UNARY: return N_FUNC;
    case BINARY: return op.fn == DIV ? N_DIV : N_SUM;
  }
  return 0;
}

uint64_t nkey(int64_t t, int64_t e) { return ((uint64_t)t << 40) | (uint64_t)e; }

// ---------------------------------------------------------------- keys
struct Key {
  uint64_t k[2];
};

Key leaf_key(int64_t g) {
  Key r;
  for (int s = 0; s < 2; ++s) r.k[s] = mix64(kSigma[s] + (uint64_t)(g + 1) * kGamma) % kP[s];
  return r;
}

Key uf_key(int fid, const Key& a) {
  uint64_t inner = mix64(a.k[0] | (a.k[1] << 32));
  Key r;
  for (int s = 0; s < 2; ++s)
    r.k[s] = mix64(inner ^ ((uint64_t)fid * kGamma) ^ kSigma[s]) % kP[s];
  return r;
}

Key maxset_key(std::vector<uint64_t> u) {
  std::sort(u.begin(), u.end());
  u.erase(std::unique(u.begin(), u.end()), u.end());
  Key r;
  if (u.size() == 1) {
    r.k[0] = u[0] & 0xffffffffull;
    r.k[1] = u[0] >> 32;
    return r;
  }
  uint64_t h = kMaxTag;
  for (uint64_t x : u) h = mix64(h ^ x);
  for (int s = 0; s < 2; ++s) r.k[s] = mix64(h ^ kSigma[s]) % kP[s];
  return r;
}

struct KeyEval {
  const Prog& P;
  bool axiom_gelu;
  std::unordered_map<uint64_t, Key> memo;
  KeyEval(const Prog& p, bool ax) : P(p), axiom_gelu(ax) {}

  Key of(const Ref& r) {
    if (r.t < 0) return leaf_key(r.e);
    uint64_t nk = nkey(r.t, r.e);
    auto it = memo.find(nk);
    if (it != memo.end()) return it->second;
    Key v = compute((int)r.t, r.e);
    memo.emplace(nk, v);
    return v;
  }

  Key compute(int t, int64_t e) {
    const Op& op = P.ops[t - P.n_inputs];
    Key out{{0, 0}};
    if (op.kind == MAXSET || op.kind == MAXC) {
      std::vector<uint64_t> u;
      for_each_term(P, t, e, [&](const Term& tm) {
        Key k;
        if (tm.nref == 0) {
          k.k[0] = tm.coef.enc(0);
          k.k[1] = tm.coef.enc(1);
        } else {
          k = of(tm.r[0]);
        }
        u.push_back(k.k[0] | (k.k[1] << 32));
      });
      return maxset_key(u);
    }
    if (op.kind == UNARY) {
      Key a = of(ref_of(P, op.args[0], e));
      int fid = op.fn;
      if (axiom_gelu && fid == GELU_TANH) fid = GELU_ERF;
      return uf_key(fid, a);
    }
    if (op.kind == BINARY && op.fn == DIV) {
      Key a{{0, 0}}, b{{0, 0}};
      for_each_term(P, t, e, [&](const Term& tm) {
        a = of(tm.r[0]);
        b = of(tm.r[1]);
      });
      Key rb = uf_key(RECIP, b);
      for (int s = 0; s < 2; ++s) out.k[s] = mulmod(a.k[s], rb.k[s], kP[s]);
      return out;
    }
    // sums of products: contract, affine, add/sub/mul
    for_each_term(P, t, e, [&](const Term& tm) {
      uint64_t prod[2] = {tm.coef.enc(0), tm.coef.enc(1)};
      for (int i = 0; i < tm.nref; ++i) {
        Key k = of(tm.r[i]);
        for (int s = 0; s < 2; ++s) prod[s] = mulmod(prod[s], k.k[s], kP[s]);
      }
      for (int s = 0; s < 2; ++s) out.k[s] = addmod(out.k[s], prod[s], kP[s]);
    });
    return out;
  }
};

// ---------------------------------------------------------------- fp64 eval
double uf_eval(int fid, double x) {
  switch (fid) {
    case EXP: return std::exp(x);
    case TANH: return std::tanh(x);
    case GELU_ERF: return 0.5 * x * (1.0 + std::erf(x / std::sqrt(2.0)));
    case GELU_TANH: {
      const double k = std::sqrt(2.0 / M_PI);
      return 0.5 * x * (1.0 + std::tanh(k * (x + 0.044715 * x * x * x)));
    }
    case ERF: return std::erf(x);
    case RSQRT: return 1.0 / std::sqrt(x);
    case RECIP: return 1.0 / x;
    case SQRT: return std::sqrt(x);
    case LOG: return std::log(x);
  }
  return NAN;
}

struct ValEval {
  const Prog& P;
  const double* const* inputs;
  std::unordered_map<uint64_t, double> memo;
  ValEval(const Prog& p, const double* const* in) : P(p), inputs(in) {}

  double leaf(int64_t g) {
    if (g >= P.G) return NAN;  // bottom
    for (int t = P.n_inputs - 1; t >= 0; --t)
      if (g >= P.base[t]) return inputs[t][g - P.base[t]];
    return NAN;
  }
  double of(const Ref& r) {
    if (r.t < 0) return leaf(r.e);
    uint64_t nk = nkey(r.t, r.e);
    auto it = memo.find(nk);
    if (it != memo.end()) return it->second;
    double v = compute((int)r.t, r.e);
    memo.emplace(nk, v);
    return v;
  }
  double compute(int t, int64_t e) {
    const Op& op = P.ops[t - P.n_inputs];
    if (op.kind == MAXSET || op.kind == MAXC) {
      double m = -INFINITY;
      bool any = false, bot = false;
      for_each_term(P, t, e, [&](const Term& tm) {
        double v = tm.nref == 0 ? tm.coef.val() : of(tm.r[0]);
        if (std::isnan(v)) bot = true;
        m = any ? std::max(m, v) : v;
        any = true;
      });
      return bot ? NAN : m;
    }
    if (op.kind == UNARY) return uf_eval(op.fn, of(ref_of(P, op.args[0], e)));
    if (op.kind == BINARY && op.fn == DIV) {
      double r = NAN;
      for_each_term(P, t, e, [&](const Term& tm) { r = of(tm.r[0]) / of(tm.r[1]); });
      return r;
    }
    double s = 0.0;
    for_each_term(P, t, e, [&](const Term& tm) {
      double p = tm.coef.val();
      for (int i = 0; i < tm.nref; ++i) p *= of(tm.r[i]);
      s += p;
    });
    return s;
  }
};

// ---------------------------------------------------------------- cones
void cone_ids(const Prog& P, int64_t loc, std::vector<uint32_t>& ids) {
  ids.clear();
  std::unordered_set<uint64_t> seen;
  std::vector<Ref> stack;
  Ref root = ref_of(P, P.output, loc);
  stack.push_back(root);
  while (!stack.empty()) {
    Ref r = stack.back();
    stack.pop_back();
    if (r.t < 0) {
      ids.push_back((uint32_t)r.e);
      continue;
    }
    if (!seen.insert(nkey(r.t, r.e)).second) continue;
    for_each_term(P, (int)r.t, r.e, [&](const Term& tm) {
      for (int i = 0; i < tm.nref; ++i) stack.push_back(tm.r[i]);
    });
  }
  std::sort(ids.begin(), ids.end());
  ids.erase(std::unique(ids.begin(), ids.end()), ids.end());
}

template <class F>
void parallel_for(int64_t n, int nthreads, F&& f) {
  if (nthreads <= 1 || n < 2) {
    for (int64_t i = 0; i < n; ++i) f(i);
    return;
  }
  std::atomic<int64_t> next{0};
  std::vector<std::thread> th;
  for (int w = 0; w < nthreads; ++w)
    th.emplace_back([&]() {
      while (true) {
        int64_t i = next.fetch_add(1);
        if (i >= n) break;
        f(i);
      }
    });
  for (auto& x : th) x.join();
}

uint64_t ref_word(const Ref& r) {
  if (r.t == -2) return kNone;
  if (r.t < 0) return (uint64_t)r.e;
  return (1ull << 63) | ((uint64_t)r.t << 40) | (uint64_t)r.e;
}

void put64(std::vector<uint8_t>& b, uint64_t x) {
  for (int i = 0; i < 8; ++i) b.push_back((uint8_t)(x >> (8 * i)));
}
void put32(std::vector<uint8_t>& b, uint32_t x) {
  for (int i = 0; i < 4; ++i) b.push_back((uint8_t)(x >> (8 * i)));
}
void putf64(std::vector<uint8_t>& b, double v) {
  uint64_t x;
  std::memcpy(&x, &v, 8);
  put64(b, x);
}

// Program section of the export format.
void export_program(const Prog& P, const std::vector<int64_t>& locs, std::vector<uint8_t>& b) {
  std::unordered_set<uint64_t> seen;
  std::vector<std::pair<int64_t, int64_t>> nodes;
  std::vector<Ref> stack;
  for (int64_t l : locs) stack.push_back(ref_of(P, P.output, l));
  while (!stack.empty()) {
    Ref r = stack.back();
    stack.pop_back();
    if (r.t < 0) continue;
    if (!seen.insert(nkey(r.t, r.e)).second) continue;
    nodes.push_back({r.t, r.e});
    for_each_term(P, (int)r.t, r.e, [&](const Term& tm) {
      for (int i = 0; i < tm.nref; ++i) stack.push_back(tm.r[i]);
    });
  }
  std::sort(nodes.begin(), nodes.end());
  std::vector<uint8_t> recs, ents;
  uint64_t n_ent = 0;
  for (auto& nd : nodes) {
    const Op& op = P.ops[nd.first - P.n_inputs];
    uint64_t begin = n_ent;
    for_each_term(P, (int)nd.first, nd.second, [&](const Term& tm) {
      putf64(ents, tm.coef.val());
      put64(ents, tm.nref > 0 ? ref_word(tm.r[0]) : kNone);
      put64(ents, tm.nref > 1 ? ref_word(tm.r[1]) : kNone);
      ++n_ent;
    });
    put32(recs, (uint32_t)nd.first);
    recs.push_back((uint8_t)node_kind(op));
    recs.push_back((uint8_t)(op.kind == UNARY ? op.fn : 0));
    recs.push_back(0);
    recs.push_back(0);
    put64(recs, (uint64_t)nd.second);
    put64(recs, begin);
    put64(recs, n_ent - begin);
  }
  put64(b, nodes.size());
  put64(b, n_ent);
  b.insert(b.end(), recs.begin(), recs.end());
  b.insert(b.end(), ents.begin(), ents.end());
}

thread_local std::string g_err;

}  // namespace

extern "C" {

const char* orc_last_error() { return g_err.c_str(); }

void* orc_create(const int64_t* words, int64_t len) {
  Prog* P = new Prog();
  if (!parse(words, len, *P)) {
    g_err = "malformed program encoding";
    delete P;
    return nullptr;
  }
  return P;
}

void orc_destroy(void* h) { delete (Prog*)h; }

int64_t orc_num_leaves(void* h) { return ((Prog*)h)->G; }
int64_t orc_out_numel(void* h) {
  Prog* P = (Prog*)h;
  return P->numel[P->output];
}
int64_t orc_num_tensors(void* h) { return (int64_t)((Prog*)h)->numel.size(); }
int64_t orc_tensor_numel(void* h, int64_t t) { return ((Prog*)h)->numel[t]; }

// Sorted unique cone of one location.  Returns its size; writes at most cap ids.
int64_t orc_cone(void* h, int64_t loc, uint32_t* ids, int64_t cap) {
  std::vector<uint32_t> v;
  cone_ids(*(Prog*)h, loc, v);
  for (int64_t i = 0; i < (int64_t)v.size() && i < cap; ++i) ids[i] = v[i];
  return (int64_t)v.size();
}

// Cone sizes and run counts of a batch (sizes[n], nruns[n]).
void orc_cone_stats(void* h, const int64_t* locs, int64_t n, int64_t* sizes, int64_t* nruns,
                    int nthreads) {
  const Prog& P = *(Prog*)h;
  parallel_for(n, nthreads, [&](int64_t i) {
    std::vector<uint32_t> v;
    cone_ids(P, locs[i], v);
    sizes[i] = (int64_t)v.size();
    int64_t r = 0;
    for (size_t j = 0; j < v.size(); ++j)
      if (j == 0 || v[j] != v[j - 1] + 1) ++r;
    nruns[i] = r;
  });
}

// Maximal runs of each location's cone, CSR: offsets[n+1] must be the exclusive
// prefix sum of nruns (from orc_cone_stats); runs[2*total] = (start, len).
void orc_cone_runs(void* h, const int64_t* locs, int64_t n, const int64_t* offsets,
                   uint32_t* runs, int nthreads) {
  const Prog& P = *(Prog*)h;
  parallel_for(n, nthreads, [&](int64_t i) {
    std::vector<uint32_t> v;
    cone_ids(P, locs[i], v);
    int64_t w = offsets[i];
    for (size_t j = 0; j < v.size(); ++j) {
      if (j == 0 || v[j] != v[j - 1] + 1) {
        runs[2 * w] = v[j];
        runs[2 * w + 1] = 1;
        ++w;
      } else {
        runs[2 * (w - 1) + 1] += 1;
      }
    }
  });
}

void orc_keys(void* h, const int64_t* locs, int64_t n, uint32_t* keys, int axiom_gelu,
              int nthreads) {
  const Prog& P = *(Prog*)h;
  parallel_for(n, nthreads, [&](int64_t i) {
    KeyEval ke(P, axiom_gelu != 0);
    Key k = ke.of(ref_of(P, P.output, locs[i]));
    keys[2 * i] = (uint32_t)k.k[0];
    keys[2 * i + 1] = (uint32_t)k.k[1];
  });
}

// Keys of arbitrary elements of arbitrary tensors (leaves: global ids).
void orc_keys_of(void* h, int64_t t, const int64_t* elems, int64_t n, uint32_t* keys,
                 int axiom_gelu) {
  const Prog& P = *(Prog*)h;
  KeyEval ke(P, axiom_gelu != 0);
  for (int64_t i = 0; i < n; ++i) {
    Key k = ke.of(ref_of(P, (int)t, elems[i]));
    keys[2 * i] = (uint32_t)k.k[0];
    keys[2 * i + 1] = (uint32_t)k.k[1];
  }
}

void orc_eval(void* h, const double* const* inputs, const int64_t* locs, int64_t n,
              double* out, int nthreads) {
  const Prog& P = *(Prog*)h;
  parallel_for(n, nthreads, [&](int64_t i) {
    ValEval ve(P, inputs);
    out[i] = ve.of(ref_of(P, P.output, locs[i]));
  });
}

// Export of the term lists of the given (already selected) locations.
// Returns the byte size; writes only when it fits in cap.
int64_t orc_export(void* href, void* hcand, const int64_t* slots, const int64_t* locs,
                   int64_t n, uint8_t* buf, int64_t cap) {
  const Prog& R = *(Prog*)href;
  const Prog& C = *(Prog*)hcand;
  std::vector<int64_t> L(locs, locs + n);
  std::vector<uint8_t> b;
  put32(b, 0x31505844u);   // "DXP1"
  put32(b, 1u);
  put64(b, 0);             // total bytes, patched below
  put64(b, (uint64_t)n);
  put64(b, 0);
  export_program(R, L, b);
  export_program(C, L, b);
  for (int64_t i = 0; i < n; ++i) {
    put64(b, (uint64_t)slots[i]);
    put64(b, ref_word(ref_of(R, R.output, locs[i])));
    put64(b, ref_word(ref_of(C, C.output, locs[i])));
  }
  uint64_t total = b.size();
  for (int i = 0; i < 8; ++i) b[8 + i] = (uint8_t)(total >> (8 * i));
  if ((int64_t)total <= cap && buf) std::memcpy(buf, b.data(), total);
  return (int64_t)total;
}

// Debug/pin helper: the raw terms of one element (coef as double, refs).
int64_t orc_terms(void* h, int64_t t, int64_t e, double* coef, uint64_t* ra, uint64_t* rb,
                  int64_t cap) {
  const Prog& P = *(Prog*)h;
  int64_t k = 0;
  for_each_term(P, (int)t, e, [&](const Term& tm) {
    if (k < cap) {
      coef[k] = tm.coef.val();
      ra[k] = tm.nref > 0 ? ref_word(tm.r[0]) : kNone;
      rb[k] = tm.nref > 1 ? ref_word(tm.r[1]) : kNone;
    }
    ++k;
  });
  return k;
}

uint64_t orc_mix64(uint64_t x) { return mix64(x); }

}  // extern "C"
