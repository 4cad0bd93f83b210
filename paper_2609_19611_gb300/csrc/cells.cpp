// Cone cells: the cone kernels' box propagation and run plan, run once per
// box of output coordinates with every quantity an affine function of the
// coordinates (see cells.h).
//
// Each step below restates the per-location step of the cone kernels
// (cone_prop.cuh, cone.cu) over a box C of output coordinates.  Every
// comparison must have one outcome on all of C; when it does not, the
// evaluation stops and asks for C to be cut at the coordinate where the
// outcome changes (or, for comparisons in several coordinates, in half).
// Quantities that the run plan stores as plain numbers (run lengths, counts)
// must be constant on C, and divisions are only taken of constants.  When a
// cell's plan leaves the fast form (a read past a tensor's end, overlapping
// streams), the cell is generic.
#include "cells.h"

#include <algorithm>
#include <array>
#include <map>
#include <cstring>

namespace dirigo {
namespace {

// c + sum_d a[d] * o[d]
struct Aff {
  int64_t c = 0;
  int64_t a[MR] = {0, 0, 0, 0};
  Aff() = default;
  Aff(int64_t v) : c(v) {}
};

Aff operator+(Aff x, const Aff& y) {
  x.c += y.c;
  for (int d = 0; d < MR; ++d) x.a[d] += y.a[d];
  return x;
}
Aff operator-(Aff x, const Aff& y) {
  x.c -= y.c;
  for (int d = 0; d < MR; ++d) x.a[d] -= y.a[d];
  return x;
}
Aff operator*(Aff x, int64_t k) {
  x.c *= k;
  for (int d = 0; d < MR; ++d) x.a[d] *= k;
  return x;
}
Aff coord(int d) {
  Aff x;
  x.a[d] = 1;
  return x;
}

struct Split {   // cut the cell at o[d] = t
  int d;
  int64_t t;
};
struct Generic {};

int64_t fdiv(int64_t a, int64_t b) {
  int64_t q = a / b;
  if ((a % b != 0) && ((a < 0) != (b < 0))) --q;
  return q;
}
int64_t cdiv(int64_t a, int64_t b) { return -fdiv(-a, b); }

// Decisions over the box lo <= o < hi of output coordinates.
struct Box {
  int64_t lo[MR], hi[MR];

  // constant part on the box's singleton dims, and the dims along which x varies
  int64_t fold(const Aff& x, int* dims, int& nd) const {
    int64_t c = x.c;
    nd = 0;
    for (int d = 0; d < MR; ++d) {
      if (x.a[d] == 0) continue;
      if (hi[d] - lo[d] == 1)
        c += x.a[d] * lo[d];
      else
        dims[nd++] = d;
    }
    return c;
  }
  int64_t vmin(const Aff& x) const {
    int64_t v = x.c;
    for (int d = 0; d < MR; ++d) v += x.a[d] * (x.a[d] > 0 ? lo[d] : hi[d] - 1);
    return v;
  }
  int64_t vmax(const Aff& x) const {
    int64_t v = x.c;
    for (int d = 0; d < MR; ++d) v += x.a[d] * (x.a[d] > 0 ? hi[d] - 1 : lo[d]);
    return v;
  }
  [[noreturn]] void halve(const int* dims, int nd) const {
    int k = dims[0];
    for (int i = 1; i < nd; ++i)
      if (hi[dims[i]] - lo[dims[i]] > hi[k] - lo[k]) k = dims[i];
    throw Split{k, lo[k] + (hi[k] - lo[k]) / 2};
  }
  bool pos(const Aff& x) const {   // x > 0
    if (vmin(x) > 0) return true;
    if (vmax(x) <= 0) return false;
    int dims[MR], nd;
    int64_t c = fold(x, dims, nd);
    if (nd != 1) halve(dims, nd);
    int k = dims[0];
    int64_t a = x.a[k];
    throw Split{k, a > 0 ? fdiv(-c, a) + 1 : cdiv(c, -a)};
  }
  bool zero(const Aff& x) const {   // x == 0
    int64_t mn = vmin(x), mx = vmax(x);
    if (mn == 0 && mx == 0) return true;
    if (mn > 0 || mx < 0) return false;
    int dims[MR], nd;
    int64_t c = fold(x, dims, nd);
    if (nd != 1) halve(dims, nd);
    int k = dims[0];
    int64_t a = x.a[k];
    if ((-c) % a != 0) return false;
    int64_t z = -c / a;
    throw Split{k, z > lo[k] ? z : z + 1};
  }
  int64_t K(const Aff& x) const {   // x, which must be constant on the box
    int dims[MR], nd;
    int64_t c = fold(x, dims, nd);
    if (nd) halve(dims, nd);
    return c;
  }
  bool lt(const Aff& x, const Aff& y) const { return pos(y - x); }
  bool le(const Aff& x, const Aff& y) const { return pos(y - x + 1); }
  bool ge(const Aff& x, const Aff& y) const { return !lt(x, y); }
  bool gt(const Aff& x, const Aff& y) const { return lt(y, x); }
  Aff mx(const Aff& x, const Aff& y) const { return lt(x, y) ? y : x; }
  Aff mn(const Aff& x, const Aff& y) const { return lt(y, x) ? y : x; }
};

struct SBox {
  int t;
  Aff lo[MR], hi[MR];
};

struct SStream {
  int t;
  Aff start;
  int64_t L;
  int nd;
  int64_t step[4], cnt[4];
};

struct Contrib {
  int64_t step, cnt;
};

struct SegOut {
  Aff gs;
  int64_t L, step[3], cnt[2], j0, j1, pos;
};
struct BwOut {
  Aff start;
  int64_t len, pos;
};
struct CellPlan {
  int64_t count = 0;
  std::vector<SegOut> seg;
  std::vector<BwOut> bw;
};

// Work budget of the fingerprint constants (one step per run of a plan).
constexpr int64_t kFpCellRuns = 1 << 20, kFpTotalRuns = 1 << 26;

// Affine fingerprint of a fast cell: the run list's fingerprint (cells.h) is
// fp[0] + sum_d fp[1 + d] * o[d] mod 2^64, since every start is affine in the
// location's coordinates o and every length and position is fixed.
void cell_fingerprint(const CellPlan& pl, uint64_t* fp) {
  for (int d = 0; d <= MR; ++d) fp[d] = 0;
  for (const SegOut& g : pl.seg) {
    // runs j in [j0, j1) at positions pos + j - j0
    uint64_t rk = fp_pow((uint64_t)g.pos), sum_r = 0, sum_roff = 0;
    const int64_t c0 = g.cnt[0], c1 = g.cnt[1];
    for (int64_t j = g.j0; j < g.j1; ++j) {
      const int64_t i0 = j % c0, r1 = j / c0, i1 = r1 % c1, i2 = r1 / c1;
      const int64_t off = g.step[0] * i0 + g.step[1] * i1 + g.step[2] * i2;
      sum_r += rk;
      sum_roff += rk * (uint64_t)off;
      rk *= kFpR;
    }
    fp[0] += kFpA * ((uint64_t)g.gs.c * sum_r + sum_roff) + (kFpB * (uint64_t)g.L + kFpC) * sum_r;
    for (int d = 0; d < MR; ++d) fp[1 + d] += kFpA * (uint64_t)g.gs.a[d] * sum_r;
  }
  for (const BwOut& b : pl.bw) {
    const uint64_t rk = fp_pow((uint64_t)b.pos);
    fp[0] += rk * fp_term((uint64_t)b.start.c, (uint64_t)b.len);
    for (int d = 0; d < MR; ++d) fp[1 + d] += rk * kFpA * (uint64_t)b.start.a[d];
  }
}

int64_t last_off(const SStream& s) {
  int64_t x = 0;
  for (int k = 0; k < s.nd; ++k) x += s.step[k] * (s.cnt[k] - 1);
  return x;
}

int64_t runs_of(const SStream& s) {
  int64_t r = 1;
  for (int k = 0; k < s.nd; ++k) r *= s.cnt[k];
  return r;
}

struct Sym {
  const Prog& P;
  const Box& C;
  std::vector<SBox> pool;
  std::vector<SStream> st;

  Sym(const Prog& p, const Box& c) : P(p), C(c) {}

  void push(int t, const Aff* lo, const Aff* hi) {
    SBox b;
    b.t = t;
    for (int d = 0; d < MR; ++d) {
      b.lo[d] = lo[d];
      b.hi[d] = hi[d];
    }
    pool.push_back(b);
  }

  std::vector<SBox> take(int t) {
    std::vector<SBox> cur, rest;
    for (const SBox& b : pool) (b.t == t ? cur : rest).push_back(b);
    pool.swap(rest);
    return cur;
  }

  // contained boxes dropped, boxes differing in one touching dim merged
  void simplify(std::vector<SBox>& b, int rank) {
    bool changed = true;
    while (changed) {
      changed = false;
      for (size_t i = 0; i < b.size() && !changed; ++i) {
        for (size_t j = 0; j < b.size() && !changed; ++j) {
          if (j == i) continue;
          bool contains = true;
          int ndiff = 0, dd = 0;
          for (int d = 0; d < rank; ++d) {
            if (contains) contains = C.le(b[i].lo[d], b[j].lo[d]) && C.le(b[j].hi[d], b[i].hi[d]);
            if (!C.zero(b[i].lo[d] - b[j].lo[d]) || !C.zero(b[i].hi[d] - b[j].hi[d])) {
              ++ndiff;
              dd = d;
            }
          }
          bool merge = !contains && ndiff == 1 && C.le(b[i].lo[dd], b[j].hi[dd]) &&
                       C.le(b[j].lo[dd], b[i].hi[dd]);
          if (contains || merge) {
            if (merge) {
              b[i].lo[dd] = C.mn(b[i].lo[dd], b[j].lo[dd]);
              b[i].hi[dd] = C.mx(b[i].hi[dd], b[j].hi[dd]);
            }
            b[j] = b.back();
            b.pop_back();
            changed = true;
          }
        }
      }
    }
  }

  // steps ascending; innermost contiguous block folded into the run length;
  // outer dims that tile exactly merged
  bool canonical(int t, const Aff& start, Contrib* c, int nc, SStream& s) {
    std::stable_sort(c, c + nc, [](const Contrib& x, const Contrib& y) { return x.step < y.step; });
    int64_t L = 1;
    int k = 0;
    while (k < nc && c[k].step <= L) {
      L = c[k].step * (c[k].cnt - 1) + L;
      ++k;
    }
    s.t = t;
    s.start = start;
    s.nd = 0;
    if (L >= ((int64_t)1 << 32)) return false;
    s.L = L;
    for (; k < nc; ++k) {
      if (c[k].step >= ((int64_t)1 << 32) || c[k].cnt >= ((int64_t)1 << 32)) return false;
      if (s.nd > 0 && s.step[s.nd - 1] * s.cnt[s.nd - 1] == c[k].step &&
          s.cnt[s.nd - 1] * c[k].cnt < ((int64_t)1 << 32)) {
        s.cnt[s.nd - 1] *= c[k].cnt;
        continue;
      }
      if (s.nd >= 4) return false;
      s.step[s.nd] = c[k].step;
      s.cnt[s.nd] = c[k].cnt;
      ++s.nd;
    }
    // a dim whose step is a multiple q <= cnt of the previous one's adds no
    // start beyond a longer lattice (the device planner folds it the same way)
    for (int i = 0; i + 1 < s.nd;) {
      const int64_t q = s.step[i + 1] / s.step[i];
      const int64_t merged = s.cnt[i] + q * (s.cnt[i + 1] - 1);
      if (s.step[i + 1] % s.step[i] == 0 && q <= s.cnt[i] && merged < ((int64_t)1 << 32)) {
        s.cnt[i] = merged;
        for (int j = i + 1; j + 1 < s.nd; ++j) {
          s.step[j] = s.step[j + 1];
          s.cnt[j] = s.cnt[j + 1];
        }
        --s.nd;
      } else {
        ++i;
      }
    }
    return true;
  }

  // a strided set of A that is a box of A
  bool to_natural(const Tensor& A, const Aff& start, const Contrib* c, int nc, int64_t* lo,
                  int64_t* hi) {
    if (C.lt(start, 0) || C.ge(start, A.numel)) return false;
    int64_t x = C.K(start);
    int64_t reach[MR], crd[MR];
    for (int d = MR - 1; d >= 0; --d) {
      reach[d] = 1;
      if (d < A.rank) {
        crd[d] = x % A.shape[d];
        x /= A.shape[d];
      } else {
        crd[d] = 0;
      }
    }
    for (int i = 0; i < nc; ++i) {
      int dd = -1;
      int64_t q = 0;
      for (int d = 0; d < A.rank; ++d) {
        if (A.stride[d] <= c[i].step) {
          if (c[i].step % A.stride[d] == 0 && c[i].step / A.stride[d] < A.shape[d]) {
            dd = d;
            q = c[i].step / A.stride[d];
          }
          break;
        }
      }
      if (dd < 0 || q > reach[dd]) return false;
      reach[dd] = q * (c[i].cnt - 1) + reach[dd];
    }
    for (int d = 0; d < MR; ++d) {
      if (d < A.rank) {
        if (crd[d] + reach[d] > A.shape[d]) return false;
        lo[d] = crd[d];
        hi[d] = crd[d] + reach[d];
      } else {
        lo[d] = 0;
        hi[d] = 1;
      }
    }
    return true;
  }

  void image(int arg, const Aff& start, Contrib* c, int nc) {
    const Tensor& A = P.t[arg];
    std::stable_sort(c, c + nc, [](const Contrib& x, const Contrib& y) { return x.step < y.step; });
    int64_t lo[MR], hi[MR];
    if (to_natural(A, start, c, nc, lo, hi)) {
      Aff l[MR], h[MR];
      for (int d = 0; d < MR; ++d) {
        l[d] = lo[d];
        h[d] = hi[d];
      }
      push(arg, l, h);
      return;
    }
    if (A.kind != K_INPUT) throw Generic{};
    SStream s;
    if (!canonical(arg, start, c, nc, s)) throw Generic{};
    st.push_back(s);
  }

  void pieces(const Tensor& T, const SBox& B) {
    for (int q = 0; q < T.npieces; ++q) {
      const Piece& pc = P.p[T.piece0 + q];
      Aff Olo[MR], Ohi[MR], Rlo[MRED], Rhi[MRED];
      bool empty = false;
      for (int d = 0; d < MR && !empty; ++d) {
        Olo[d] = C.mx(B.lo[d], d < T.rank ? pc.lo[d] : 0);
        Ohi[d] = C.mn(B.hi[d], d < T.rank ? pc.hi[d] : 1);
        empty = C.ge(Olo[d], Ohi[d]);
      }
      for (int e = 0; e < MRED && !empty; ++e) {
        Rlo[e] = e < pc.nred ? pc.rlo[e] : 0;
        Rhi[e] = e < pc.nred ? pc.rhi[e] : 1;
        empty = C.ge(Rlo[e], Rhi[e]);
      }
      if (empty) continue;
      int gdo[MR] = {-1, -1, -1, -1}, gdr[MRED] = {-1, -1, -1, -1};
      for (int j = 0; j < pc.nguard; ++j) {
        const Guard& g = pc.g[j];
        if (g.od >= 0) {
          if (gdo[g.od] >= 0) throw Generic{};
          gdo[g.od] = j;
        }
        if (g.rd >= 0) {
          if (gdr[g.rd] >= 0) throw Generic{};
          gdr[g.rd] = j;
        }
      }
      Aff Vlo[MG], Vhi[MG];
      bool vcontig[MG], rcontig[MG];
      for (int j = 0; j < pc.nguard && !empty; ++j) {
        const Guard& g = pc.g[j];
        int64_t lo = g.lo - (int64_t)g.c, hi = g.hi - (int64_t)g.c, a = g.oa;
        vcontig[j] = rcontig[j] = true;
        if (g.od < 0 && g.rd < 0) {
          empty = !(0 >= lo && 0 < hi);
        } else if (g.rd < 0) {   // lo <= a*o < hi
          Aff& o0 = Olo[g.od];
          Aff& o1 = Ohi[g.od];
          if (a > 0) {
            o0 = C.mx(o0, cdiv(lo, a));
            o1 = C.mn(o1, cdiv(hi, a));
          } else if (a < 0) {
            o0 = C.mx(o0, fdiv(hi, a) + 1);
            o1 = C.mn(o1, fdiv(lo, a) + 1);
          } else if (!(0 >= lo && 0 < hi)) {
            empty = true;
          }
          if (!empty) empty = C.ge(o0, o1);
        } else if (g.od < 0) {   // lo <= r < hi
          Rlo[g.rd] = C.mx(Rlo[g.rd], lo);
          Rhi[g.rd] = C.mn(Rhi[g.rd], hi);
          empty = C.ge(Rlo[g.rd], Rhi[g.rd]);
        } else {   // lo <= a*o + r < hi
          int64_t R0 = C.K(Rlo[g.rd]), R1 = C.K(Rhi[g.rd]);
          Aff& o0 = Olo[g.od];
          Aff& o1 = Ohi[g.od];
          if (a > 0) {
            o0 = C.mx(o0, cdiv(lo - R1 + 1, a));
            o1 = C.mn(o1, cdiv(hi - R0, a));
          } else if (a < 0) {
            o0 = C.mx(o0, fdiv(hi - R0, a) + 1);
            o1 = C.mn(o1, fdiv(lo - R1 + 1, a) + 1);
          } else if (!(R0 < hi && R1 - 1 >= lo)) {
            empty = true;
          }
          if (empty || C.ge(o0, o1)) {
            empty = true;
            break;
          }
          Aff amin = a >= 0 ? o0 * a : (o1 - 1) * a;
          Aff amax = a >= 0 ? (o1 - 1) * a : o0 * a;
          int64_t aa = a < 0 ? -a : a;
          rcontig[j] = aa <= hi - lo || C.zero(o1 - o0 - 1);
          vcontig[j] = aa <= R1 - R0 || C.zero(o1 - o0 - 1);
          Aff r0 = C.mx(R0, Aff(lo) - amax), r1 = C.mn(R1, Aff(hi) - amin);
          Vlo[j] = C.mx(lo, amin + R0);
          Vhi[j] = C.mn(hi, amax + R1);
          Rlo[g.rd] = r0;
          Rhi[g.rd] = r1;
          empty = C.ge(r0, r1) || C.ge(Vlo[j], Vhi[j]);
        }
      }
      if (empty) continue;
      for (int i = 0; i < T.nargs; ++i) {
        const Access& ac = pc.acc[i];
        const AccTpl& tp = pc.tpl[i];
        if (tp.unsupported) throw Generic{};
        const Tensor& A = P.t[T.args[i]];
        Aff start = ac.base;
        bool nat = tp.natural;
        Aff crd[MR];
        int64_t reach[MR];
        for (int d = 0; d < MR; ++d) {
          crd[d] = tp.cbase[d];
          reach[d] = 1;
        }
        Contrib c[MSLOT];
        int nc = 0;
        for (int k = 0; k < tp.nslot; ++k) {
          const Slot& sl = tp.s[k];
          Aff lo, hi;
          if (sl.kind == SL_O) {
            lo = Olo[sl.ref];
            hi = Ohi[sl.ref];
          } else if (sl.kind == SL_R) {
            lo = Rlo[sl.ref];
            hi = Rhi[sl.ref];
          } else if (sl.kind == SL_V) {
            if (!vcontig[sl.ref]) throw Generic{};
            lo = Vlo[sl.ref];
            hi = Vhi[sl.ref];
          } else if (sl.kind == SL_GR) {
            if (!rcontig[sl.ref]) throw Generic{};
            lo = Rlo[pc.g[sl.ref].rd];
            hi = Rhi[pc.g[sl.ref].rd];
          } else {
            lo = Olo[pc.g[sl.ref].od];
            hi = Ohi[pc.g[sl.ref].od];
          }
          start = start + lo * sl.step;
          crd[sl.nd] = crd[sl.nd] + lo * sl.q;
          if (C.gt(hi - lo, 1)) {
            int64_t cnt = C.K(hi - lo);
            int64_t stp = sl.step;
            if (stp < 0) {
              start = start + Aff(stp * (cnt - 1));
              stp = -stp;
              nat = false;
            }
            if ((int64_t)sl.q > reach[sl.nd]) nat = false;
            reach[sl.nd] += (int64_t)sl.q * (cnt - 1);
            c[nc++] = Contrib{stp, cnt};
          }
        }
        if (nat) {
          bool ok = true;
          Aff lo2[MR], hi2[MR];
          for (int d = 0; d < MR; ++d) {
            if (d < A.rank) {
              if (ok) ok = C.ge(crd[d], 0) && C.le(crd[d] + reach[d], A.shape[d]);
              lo2[d] = crd[d];
              hi2[d] = crd[d] + reach[d];
            } else {
              lo2[d] = 0;
              hi2[d] = 1;
            }
          }
          if (ok) {
            push(T.args[i], lo2, hi2);
            continue;
          }
        }
        image(T.args[i], start, c, nc);
      }
    }
  }

  void propagate() {
    const Tensor& Y = P.t[P.output];
    Aff lo[MR], hi[MR];
    for (int d = 0; d < MR; ++d) {
      if (d < Y.rank) {
        lo[d] = coord(d);
        hi[d] = coord(d) + 1;
      } else {
        lo[d] = 0;
        hi[d] = 1;
      }
    }
    push(P.output, lo, hi);
    for (int t = P.output; t >= P.n_inputs; --t) {
      const Tensor& T = P.t[t];
      std::vector<SBox> cur = take(t);
      if (cur.empty()) continue;
      simplify(cur, T.rank);
      for (const SBox& B : cur) {
        if (T.kind == K_CONTRACT || T.kind == K_MAXSET) {
          pieces(T, B);
        } else if (T.kind == K_BINARY) {
          for (int s = 0; s < 2; ++s) {
            const Tensor& A = P.t[T.args[s]];
            Aff lo2[MR], hi2[MR];
            for (int d = 0; d < MR; ++d) {
              if (d < T.arg_rank[s] && A.shape[d] != 1) {
                lo2[d] = B.lo[T.axes[s][d]];
                hi2[d] = B.hi[T.axes[s][d]];
              } else {
                lo2[d] = 0;
                hi2[d] = 1;
              }
            }
            push(T.args[s], lo2, hi2);
          }
        } else {
          push(T.args[0], B.lo, B.hi);
        }
      }
    }
    for (int u = 0; u < P.n_inputs; ++u) {
      const Tensor& A = P.t[u];
      std::vector<SBox> cur = take(u);
      simplify(cur, A.rank);
      for (const SBox& b : cur) {
        Contrib c[MR];
        int nc = 0;
        Aff start = 0;
        for (int d = 0; d < A.rank; ++d) {
          start = start + b.lo[d] * A.stride[d];
          if (C.gt(b.hi[d] - b.lo[d], 1)) c[nc++] = Contrib{A.stride[d], C.K(b.hi[d] - b.lo[d])};
        }
        SStream s;
        if (!canonical(u, start, c, nc, s)) throw Generic{};
        st.push_back(s);
      }
    }
  }

  // the fast run plan: in-range, regular, disjoint streams; junction runs
  // where one stream's last run touches the next stream's first
  void plan(CellPlan& out) {
    for (const SStream& S : st) {
      const Tensor& A = P.t[S.t];
      if (C.lt(S.start, 0) || C.gt(S.start + last_off(S) + S.L, A.numel)) throw Generic{};
      if (S.nd > 3) throw Generic{};
      int64_t span = S.L;
      for (int k = 0; k < S.nd; ++k) {
        if (S.step[k] <= span) throw Generic{};
        span += S.step[k] * (S.cnt[k] - 1);
      }
    }
    const int ns = (int)st.size();
    std::vector<Aff> gs(ns);
    for (int s = 0; s < ns; ++s) gs[s] = st[s].start + P.t[st[s].t].gbase;
    for (int i = 1; i < ns; ++i) {
      SStream x = st[i];
      Aff gx = gs[i];
      int j = i;
      while (j > 0 && C.gt(gs[j - 1], gx)) {
        st[j] = st[j - 1];
        gs[j] = gs[j - 1];
        --j;
      }
      st[j] = x;
      gs[j] = gx;
    }
    int m = 0;
    for (int s = 0; s < ns; ++s) {
      if (m > 0 && st[m - 1].nd == 0 && st[s].nd == 0 && C.le(gs[s], gs[m - 1] + st[m - 1].L)) {
        Aff e = C.mx(gs[m - 1] + st[m - 1].L, gs[s] + st[s].L);
        st[m - 1].L = C.K(e - gs[m - 1]);
        continue;
      }
      st[m] = st[s];
      gs[m] = gs[s];
      ++m;
    }
    st.resize(m);
    gs.resize(m);
    for (int s = 1; s < m; ++s)
      if (C.lt(gs[s], gs[s - 1] + last_off(st[s - 1]) + st[s - 1].L)) throw Generic{};
    int64_t pos = 0;
    bool pend = false;
    Aff pst, pen;
    for (int s = 0; s < m; ++s) {
      const SStream& S = st[s];
      int64_t R = runs_of(S);
      Aff first = gs[s], last = gs[s] + last_off(S);
      int64_t j0 = 0;
      if (pend && C.zero(pen - first)) {
        pen = first + S.L;
        if (R == 1) continue;
        out.bw.push_back(BwOut{pst, C.K(pen - pst), pos});
        ++pos;
        j0 = 1;
      } else if (pend) {
        out.bw.push_back(BwOut{pst, C.K(pen - pst), pos});
        ++pos;
      }
      int64_t j1 = R - 1 > j0 ? R - 1 : j0;
      if (j1 > j0) {
        SegOut g;
        g.gs = gs[s];
        g.L = S.L;
        for (int d = 0; d < 3; ++d) g.step[d] = d < S.nd ? S.step[d] : 0;
        for (int d = 0; d < 2; ++d) g.cnt[d] = d < S.nd ? S.cnt[d] : 1;
        g.j0 = j0;
        g.j1 = j1;
        g.pos = pos;
        out.seg.push_back(g);
      }
      pos += j1 - j0;
      pst = last;
      pen = last + S.L;
      pend = true;
    }
    if (pend) {
      out.bw.push_back(BwOut{pst, C.K(pen - pst), pos});
      ++pos;
    }
    out.count = pos;
  }
};

uint32_t magic_of(uint32_t d) {
  return (d > 1 && d < (1u << 27)) ? (uint32_t)(((1ull << 32) + d - 1) / d) : 0u;
}

bool fits_u32(int64_t x) { return x >= 0 && x < ((int64_t)1 << 32); }

// 0: plan; 1: generic; 2: split requested (in *sp)
int eval_cell(const Prog& P, const Box& C, CellPlan& out, Split* sp) {
  try {
    Sym s(P, C);
    s.propagate();
    s.plan(out);
  } catch (const Split& x) {
    *sp = x;
    return 2;
  } catch (const Generic&) {
    return 1;
  }
  if (!fits_u32(out.count)) return 1;
  for (const SegOut& g : out.seg) {
    if (!fits_u32(g.L) || !fits_u32(g.j1) || !fits_u32(g.pos)) return 1;
    for (int d = 0; d < 3; ++d)
      if (!fits_u32(g.step[d])) return 1;
    for (int d = 0; d < 2; ++d)
      if (!fits_u32(g.cnt[d])) return 1;
  }
  for (const BwOut& b : out.bw)
    if (!fits_u32(b.len) || !fits_u32(b.pos)) return 1;
  return 0;
}

template <class T>
void put(std::vector<uint8_t>& blob, size_t off, const T& v) {
  std::memcpy(blob.data() + off, &v, sizeof(T));
}

}  // namespace

bool build_cells(Prog& P, std::vector<uint8_t>& blob) {
  P.cell_on = 0;
  blob.clear();
  const Tensor& Y = P.t[P.output];
  const int rank = Y.rank;
  int64_t tab = 0;
  for (int d = 0; d < rank; ++d) tab += Y.shape[d];
  if (tab > (1 << 20)) return false;
  constexpr int64_t kMaxCells = 1 << 14;
  constexpr int64_t kMaxEvals = 1 << 17;
  std::vector<std::vector<int64_t>> thr(MR);
  for (int d = 0; d < MR; ++d) thr[d] = {0, d < rank ? (int64_t)Y.shape[d] : 1};
  auto ncells = [&]() {
    int64_t n = 1;
    for (int d = 0; d < MR; ++d) n *= (int64_t)thr[d].size() - 1;
    return n;
  };
  std::vector<CellPlan> plans;
  std::vector<int> kind;
  int64_t evals = 0;
  while (true) {
    const int64_t n = ncells();
    plans.assign(n, CellPlan());
    kind.assign(n, 1);
    std::vector<Split> req;
    for (int64_t id = 0; id < n; ++id) {
      Box C;
      int64_t x = id;
      for (int d = MR - 1; d >= 0; --d) {
        int64_t k = (int64_t)thr[d].size() - 1, i = x % k;
        x /= k;
        C.lo[d] = thr[d][i];
        C.hi[d] = thr[d][i + 1];
      }
      Split sp{0, 0};
      kind[id] = eval_cell(P, C, plans[id], &sp);
      if (kind[id] == 2) req.push_back(sp);
      if (++evals > kMaxEvals) return false;
    }
    bool changed = false;
    for (const Split& sp : req) {
      std::vector<int64_t>& v = thr[sp.d];
      if (std::binary_search(v.begin(), v.end(), sp.t)) continue;
      if (ncells() / ((int64_t)v.size() - 1) * (int64_t)v.size() > kMaxCells) continue;
      v.insert(std::upper_bound(v.begin(), v.end(), sp.t), sp.t);
      changed = true;
    }
    if (!changed) break;
  }
  const int64_t n = ncells();
  int64_t nfast = 0, nseg = 0, nbw = 0, fp_work = 0;
  for (int64_t id = 0; id < n; ++id) {
    if (kind[id] != 0) continue;
    // the fingerprint constants take one step per run of the cell's plan: a
    // cell beyond the budget is planned per location instead
    fp_work += plans[id].count;
    if (plans[id].count > kFpCellRuns || fp_work > kFpTotalRuns) {
      kind[id] = 1;
      continue;
    }
    ++nfast;
    nseg += (int64_t)plans[id].seg.size();
    nbw += (int64_t)plans[id].bw.size();
  }
  if (nfast == 0) return false;
  // layout
  int64_t off = (tab * 2 + 15) / 16 * 16;
  P.cell_rec_off = off;
  off += n * (int64_t)sizeof(CellRec);
  off = (off + 15) / 16 * 16;
  P.cell_seg_off = off;
  off += nseg * (int64_t)sizeof(CellSeg);
  P.cell_bw_off = off;
  off += nbw * (int64_t)sizeof(CellBw);
  off = (off + 255) / 256 * 256;
  if (off > (64 << 20)) return false;
  blob.assign((size_t)off, 0);
  int64_t e = 0;
  for (int d = 0; d < MR; ++d) {
    P.cell_tab[d] = (int32_t)e;
    if (d >= rank) continue;
    const std::vector<int64_t>& v = thr[d];
    for (int64_t xcrd = 0, i = 0; xcrd < Y.shape[d]; ++xcrd) {
      while (xcrd >= v[i + 1]) ++i;
      put(blob, (size_t)(2 * (e + xcrd)), (uint16_t)i);
    }
    e += Y.shape[d];
  }
  int64_t r = 1;
  for (int d = MR - 1; d >= 0; --d) {
    P.cell_radix[d] = (int32_t)r;
    r *= (int64_t)thr[d].size() - 1;
  }
  int64_t si = 0, bi = 0;
  std::map<std::array<uint32_t, 7>, uint32_t> tabs;   // offset tables, by steps, counts and range
  for (int64_t id = 0; id < n; ++id) {
    CellRec rec{};
    if (kind[id] != 0) {
      rec.nseg = kCellGeneric;
    } else {
      const CellPlan& pl = plans[id];
      cell_fingerprint(pl, rec.fp);
      rec.count = (uint32_t)pl.count;
      rec.nseg = (uint16_t)pl.seg.size();
      rec.nbw = (uint16_t)pl.bw.size();
      rec.seg0 = (uint32_t)si;
      rec.bw0 = (uint32_t)bi;
      for (const SegOut& g : pl.seg) {
        CellSeg cs{};
        cs.gc = g.gs.c;
        for (int d = 0; d < MR; ++d) cs.ga[d] = g.gs.a[d];
        cs.L = (uint32_t)g.L;
        cs.st0 = (uint32_t)g.step[0];
        cs.st1 = (uint32_t)g.step[1];
        cs.st2 = (uint32_t)g.step[2];
        cs.ct0 = (uint32_t)g.cnt[0];
        cs.ct1 = (uint32_t)g.cnt[1];
        cs.mg0 = magic_of(cs.ct0);
        cs.mg1 = magic_of(cs.ct1);
        cs.j0 = (uint32_t)g.j0;
        cs.j1 = (uint32_t)g.j1;
        cs.pos = (uint32_t)g.pos;
        cs.tab = tabs.emplace(std::array<uint32_t, 7>{cs.st0, cs.st1, cs.st2, cs.ct0, cs.ct1,
                                                      cs.j0, cs.j1},
                              (uint32_t)si).first->second;
        put(blob, (size_t)(P.cell_seg_off + si * (int64_t)sizeof(CellSeg)), cs);
        ++si;
      }
      for (const BwOut& b : pl.bw) {
        CellBw cb{};
        cb.sc = b.start.c;
        for (int d = 0; d < MR; ++d) cb.sa[d] = b.start.a[d];
        cb.len = (uint32_t)b.len;
        cb.pos = (uint32_t)b.pos;
        put(blob, (size_t)(P.cell_bw_off + bi * (int64_t)sizeof(CellBw)), cb);
        ++bi;
      }
    }
    put(blob, (size_t)(P.cell_rec_off + id * (int64_t)sizeof(CellRec)), rec);
  }
  P.n_cells = (int32_t)n;
  P.cell_bytes = off;
  P.cell_on = 1;
  return true;
}

}  // namespace dirigo
