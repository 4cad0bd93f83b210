// Backward box propagation: the cone of one output location without
// enumerating its elements.
//
// res(y[l]) visits, for every tensor, the set of its elements that some
// per-element equation on the way from y[l] reads (Sec. 3.4,
// "Back-projection").  For index maps of the supported form that set is a
// union of boxes: starting from the point box {l} of y, each tensor's boxes
// (in reverse SSA order, merged where they touch) are pushed through its
// equation to boxes of its operands:
//   UNARY/AFFINE/MAXC  same box;  BINARY  the box through the broadcast axes;
//   CONTRACT/MAXSET    per piece: the output box clipped to the piece, the
//                      reduction box clipped by the guards, and the image of
//                      the access map (an arithmetic progression per
//                      independent index component) as a box of the operand.
// Guards couple at most one output dim with one reduction dim (the padding
// tests of a convolution); the projections and images of such a pair are
// intervals whenever consecutive windows touch, which every stride-s kernel
// with s <= k satisfies.  Accesses that are not boxes of the operand (a
// kernel reading with a wrong stride, or past a row end) become raw strided
// sets on input tensors.  Input boxes end as strided "streams" of runs over
// global ids.
#pragma once
#include <cstdint>

#include "../../include/dirigo.h"
#include "dev.cuh"

namespace dirigo {

constexpr int NB = 12;    // natural boxes per location (all tensors)
constexpr int NS = 6;     // run streams per location
constexpr int MSD = 4;    // outer dims of a stream

enum ConeErr : int32_t { CE_OK = 0, CE_UNSUPPORTED = 1, CE_CAPACITY = 2, CE_LOCATION = 4,
                         CE_NONMONOTONE = 8, CE_WAIT = 16 /* a bounded wait expired */,
                         CE_RUNCAP = 32 /* the runs do not fit the caller's run buffer */ };

// Status of a cone's latched error bits (the first that applies, in this
// order), host and device.
__host__ __device__ inline int cone_bits_status(int32_t st) {
  if (st & CE_LOCATION) return DIRIGO_E_INVALID;
  if (st & (CE_UNSUPPORTED | CE_NONMONOTONE | CE_CAPACITY)) return DIRIGO_E_UNSUPPORTED;
  if (st & CE_WAIT) return DIRIGO_E_CUDA;
  if (st & CE_RUNCAP) return DIRIGO_E_CAPACITY;
  return DIRIGO_OK;
}

struct NBox {
  int32_t lo[MR], hi[MR];
  int32_t t;
};

// Runs start + sum_k step[k] * i_k + [0, L), i_k < cnt[k], steps ascending,
// in the flat offsets of input tensor t (possibly out of its range).
struct Stream {
  int64_t start;
  uint32_t L;
  int32_t t;
  int32_t nd;
  uint32_t step[MSD];
  uint32_t cnt[MSD];
};

struct Contrib {
  int64_t step, lo, cnt;
};

struct LocState {
  NBox pool[NB];
  int npool;
  uint64_t pending;   // bit t: the pool holds a box of tensor t
  Stream st[NS];
  int nst;
  int err;
};

__device__ __forceinline__ int64_t floordiv(int64_t a, int64_t b) {
  if (b == 1) return a;
  int64_t q = a / b;
  if ((a % b != 0) && ((a < 0) != (b < 0))) --q;
  return q;
}
__device__ __forceinline__ int64_t ceildiv(int64_t a, int64_t b) { return -floordiv(-a, b); }

__device__ __forceinline__ void push_box(LocState& L, int t, const int32_t* lo, const int32_t* hi) {
  if (L.npool >= NB) {
    L.err |= CE_CAPACITY;
    return;
  }
  NBox& b = L.pool[L.npool++];
  L.pending |= 1ull << t;
  b.t = t;
  for (int d = 0; d < MR; ++d) {
    b.lo[d] = lo[d];
    b.hi[d] = hi[d];
  }
}

// Sort contributions by step ascending, fold the innermost contiguous (or
// overlapping) block into the run length, merge exact tilings of outer dims.
__device__ inline bool canonical_stream(int t, int64_t start, Contrib* c, int nc, Stream& s) {
  for (int i = 1; i < nc; ++i) {
    Contrib x = c[i];
    int j = i;
    while (j > 0 && c[j - 1].step > x.step) {
      c[j] = c[j - 1];
      --j;
    }
    c[j] = x;
  }
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
  s.L = (uint32_t)L;
  for (; k < nc; ++k) {
    if (c[k].step >= ((int64_t)1 << 32) || c[k].cnt >= ((int64_t)1 << 32)) return false;
    if (s.nd > 0 && (int64_t)s.step[s.nd - 1] * s.cnt[s.nd - 1] == c[k].step &&
        (int64_t)s.cnt[s.nd - 1] * c[k].cnt < ((int64_t)1 << 32)) {
      s.cnt[s.nd - 1] *= (uint32_t)c[k].cnt;
      continue;
    }
    if (s.nd >= MSD) return false;
    s.step[s.nd] = (uint32_t)c[k].step;
    s.cnt[s.nd] = (uint32_t)c[k].cnt;
    ++s.nd;
  }
  // A dim whose step is a multiple q <= cnt of the previous dim's step adds
  // no new run starts beyond a longer lattice: the starts of the two dims are
  // {step0 * (a + q b)}, a < cnt0, b < cnt1, which is the lattice of step0
  // with cnt0 + q (cnt1 - 1) points (the cone is a set; repeats do not
  // matter).  Merging keeps the stream's starts increasing where the
  // overlapping form would not be (a read whose outer stride is smaller than
  // its inner extent, as a weight read with the wrong channel stride).
  for (int i = 0; i + 1 < s.nd;) {
    const uint64_t st0 = s.step[i], st1 = s.step[i + 1];
    const uint64_t q = st1 / st0;
    const uint64_t merged = (uint64_t)s.cnt[i] + q * (uint64_t)(s.cnt[i + 1] - 1);
    if (st1 % st0 == 0 && q <= s.cnt[i] && merged < ((uint64_t)1 << 32)) {
      s.cnt[i] = (uint32_t)merged;
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

__device__ __forceinline__ void push_stream(LocState& L, const Stream& s) {
  if (L.nst >= NS) {
    L.err |= CE_CAPACITY;
    return;
  }
  L.st[L.nst++] = s;
}

// A strided set of tensor A as a natural box, when it is one.
__device__ inline bool to_natural(const Tensor& A, int64_t start, const Contrib* c, int nc, int32_t* lo,
                           int32_t* hi) {
  if (start < 0 || start >= A.numel) return false;
  int64_t reach[MR];
  int64_t coord[MR];
  int64_t x = start;
  for (int d = MR - 1; d >= 0; --d) {
    reach[d] = 1;
    if (d < A.rank) {
      int64_t q, r;
      divmod64(x, A.shape[d], q, r);
      coord[d] = r;
      x = q;
    } else {
      coord[d] = 0;
    }
  }
  // contributions sorted by step ascending: within one dim, multipliers come
  // in ascending order, so the contiguity test applies incrementally
  for (int i = 0; i < nc; ++i) {
    // the step is a multiple q < shape[d] of exactly one stride: that of the
    // outermost dim whose stride does not exceed it
    int dd = -1;
    int64_t q = 0;
    for (int d = 0; d < A.rank; ++d) {
      if (A.stride[d] <= c[i].step) {
        int64_t qq, rr;
        divmod64(c[i].step, A.stride[d], qq, rr);
        if (rr == 0 && qq < A.shape[d]) {
          dd = d;
          q = qq;
        }
        break;
      }
    }
    if (dd < 0) return false;
    if (q > reach[dd]) return false;
    reach[dd] = q * (c[i].cnt - 1) + reach[dd];
  }
  for (int d = 0; d < MR; ++d) {
    if (d < A.rank) {
      if (coord[d] + reach[d] > A.shape[d]) return false;
      lo[d] = (int32_t)coord[d];
      hi[d] = (int32_t)(coord[d] + reach[d]);
    } else {
      lo[d] = 0;
      hi[d] = 1;
    }
  }
  return true;
}

__device__ __forceinline__ void sort_contribs(Contrib* c, int nc) {
  for (int i = 1; i < nc; ++i) {
    Contrib x = c[i];
    int j = i;
    while (j > 0 && c[j - 1].step > x.step) {
      c[j] = c[j - 1];
      --j;
    }
    c[j] = x;
  }
}

// Push the image of operand `arg` read through `acc` over the given
// contributions.
__device__ inline void push_image(const Prog& P, int arg, int64_t start, Contrib* c, int nc,
                           LocState& L) {
  const Tensor& A = P.t[arg];
  sort_contribs(c, nc);
  int32_t lo[MR], hi[MR];
  if (to_natural(A, start, c, nc, lo, hi)) {
    push_box(L, arg, lo, hi);
    return;
  }
  if (A.kind != K_INPUT) {   // intermediate tensors are only read as boxes
    L.err |= CE_UNSUPPORTED;
    return;
  }
  Stream s;
  if (!canonical_stream(arg, start, c, nc, s)) {
    L.err |= CE_UNSUPPORTED;
    return;
  }
  push_stream(L, s);
}

// Operand boxes of one box of a CONTRACT/MAXSET tensor.
__device__ inline void propagate_pieces(const Prog& P, const Tensor& T, const NBox& B, LocState& L) {
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    int64_t Olo[MR], Ohi[MR], Rlo[MRED], Rhi[MRED];
    bool empty = false;
    for (int d = 0; d < MR; ++d) {
      Olo[d] = max(B.lo[d], d < T.rank ? pc.lo[d] : 0);
      Ohi[d] = min(B.hi[d], d < T.rank ? pc.hi[d] : 1);
      empty |= Olo[d] >= Ohi[d];
    }
    for (int e = 0; e < MRED; ++e) {
      Rlo[e] = e < pc.nred ? pc.rlo[e] : 0;
      Rhi[e] = e < pc.nred ? pc.rhi[e] : 1;
      empty |= Rlo[e] >= Rhi[e];
    }
    if (empty) continue;
    int gdo[MR] = {-1, -1, -1, -1}, gdr[MRED] = {-1, -1, -1, -1};
    int64_t Vlo[MG], Vhi[MG];
    bool vcontig[MG], rcontig[MG];
    for (int j = 0; j < pc.nguard; ++j) {
      const Guard& g = pc.g[j];
      if (g.od >= 0) {
        if (gdo[g.od] >= 0) L.err |= CE_UNSUPPORTED;
        gdo[g.od] = j;
      }
      if (g.rd >= 0) {
        if (gdr[g.rd] >= 0) L.err |= CE_UNSUPPORTED;
        gdr[g.rd] = j;
      }
    }
    if (L.err) return;
    for (int j = 0; j < pc.nguard && !empty; ++j) {
      const Guard& g = pc.g[j];
      int64_t lo = g.lo - (int64_t)g.c, hi = g.hi - (int64_t)g.c, a = g.oa;
      vcontig[j] = rcontig[j] = true;
      if (g.od < 0 && g.rd < 0) {
        empty |= !(0 >= lo && 0 < hi);
      } else if (g.rd < 0) {   // lo <= a*o < hi
        int64_t& o0 = Olo[g.od];
        int64_t& o1 = Ohi[g.od];
        if (a > 0) {
          o0 = max(o0, ceildiv(lo, a));
          o1 = min(o1, ceildiv(hi, a));
        } else if (a < 0) {
          o0 = max(o0, floordiv(hi, a) + 1);
          o1 = min(o1, floordiv(lo, a) + 1);
        } else if (!(0 >= lo && 0 < hi)) {
          empty = true;
        }
        empty |= o0 >= o1;
      } else if (g.od < 0) {   // lo <= r < hi
        Rlo[g.rd] = max(Rlo[g.rd], lo);
        Rhi[g.rd] = min(Rhi[g.rd], hi);
        empty |= Rlo[g.rd] >= Rhi[g.rd];
      } else {   // lo <= a*o + r < hi
        int64_t R0 = Rlo[g.rd], R1 = Rhi[g.rd];
        int64_t& o0 = Olo[g.od];
        int64_t& o1 = Ohi[g.od];
        // o admits some r: a*o < hi - R0 and a*o >= lo - R1 + 1
        if (a > 0) {
          o0 = max(o0, ceildiv(lo - R1 + 1, a));
          o1 = min(o1, ceildiv(hi - R0, a));
        } else if (a < 0) {
          o0 = max(o0, floordiv(hi - R0, a) + 1);
          o1 = min(o1, floordiv(lo - R1 + 1, a) + 1);
        } else if (!(R0 < hi && R1 - 1 >= lo)) {
          empty = true;
        }
        if (o0 >= o1) {
          empty = true;
          break;
        }
        int64_t amin = a >= 0 ? a * o0 : a * (o1 - 1);   // min of a*o over the o range
        int64_t amax = a >= 0 ? a * (o1 - 1) : a * o0;
        bool single = o1 - o0 == 1;
        int64_t aa = a < 0 ? -a : a;
        // r-projection: union over o of [lo - a*o, hi - a*o)
        rcontig[j] = single || aa <= hi - lo;
        int64_t r0 = max(R0, lo - amax), r1 = min(R1, hi - amin);
        // image of v = a*o + r: union over o of [a*o + R0, a*o + R1) within [lo, hi)
        vcontig[j] = single || aa <= R1 - R0;
        Vlo[j] = max(lo, amin + R0);
        Vhi[j] = min(hi, amax + R1);
        Rlo[g.rd] = r0;
        Rhi[g.rd] = r1;
        empty |= r0 >= r1 || Vlo[j] >= Vhi[j];
      }
    }
    if (empty) continue;
    for (int i = 0; i < T.nargs; ++i) {
      const Access& ac = pc.acc[i];
      const AccTpl& tp = pc.tpl[i];
      if (tp.unsupported) {
        L.err |= CE_UNSUPPORTED;
        return;
      }
      const Tensor& A = P.t[T.args[i]];
      int64_t start = ac.base;
      bool nat = tp.natural;
      int64_t coord[MR], reach[MR];
      for (int d = 0; d < MR; ++d) {
        coord[d] = tp.cbase[d];
        reach[d] = 1;
      }
      Contrib c[MSLOT];
      int nc = 0;
      for (int k = 0; k < tp.nslot; ++k) {
        const Slot& sl = tp.s[k];
        int64_t lo, cnt;
        if (sl.kind == SL_O) {
          lo = Olo[sl.ref];
          cnt = Ohi[sl.ref] - lo;
        } else if (sl.kind == SL_R) {
          lo = Rlo[sl.ref];
          cnt = Rhi[sl.ref] - lo;
        } else if (sl.kind == SL_V) {
          if (!vcontig[sl.ref]) L.err |= CE_UNSUPPORTED;
          lo = Vlo[sl.ref];
          cnt = Vhi[sl.ref] - lo;
        } else if (sl.kind == SL_GR) {
          if (!rcontig[sl.ref]) L.err |= CE_UNSUPPORTED;
          lo = Rlo[pc.g[sl.ref].rd];
          cnt = Rhi[pc.g[sl.ref].rd] - lo;
        } else {
          lo = Olo[pc.g[sl.ref].od];
          cnt = Ohi[pc.g[sl.ref].od] - lo;
        }
        start += sl.step * lo;
        coord[sl.nd] += (int64_t)sl.q * lo;
        if (cnt > 1) {
          int64_t st = sl.step;
          if (st < 0) {
            start += st * (cnt - 1);
            st = -st;
            nat = false;
          }
          if ((int64_t)sl.q > reach[sl.nd]) nat = false;
          reach[sl.nd] += (int64_t)sl.q * (cnt - 1);
          c[nc++] = Contrib{st, 0, cnt};
        }
      }
      if (L.err) return;
      if (nat) {
        bool ok = true;
        int32_t lo2[MR], hi2[MR];
        for (int d = 0; d < MR; ++d) {
          if (d < A.rank) {
            ok &= coord[d] >= 0 && coord[d] + reach[d] <= A.shape[d];
            lo2[d] = (int32_t)coord[d];
            hi2[d] = (int32_t)(coord[d] + reach[d]);
          } else {
            lo2[d] = 0;
            hi2[d] = 1;
          }
        }
        if (ok) {
          push_box(L, T.args[i], lo2, hi2);
          continue;
        }
      }
      push_image(P, T.args[i], start, c, nc, L);
    }
  }
}

// Box simplification within one tensor's list: drop contained boxes and
// merge boxes that differ in one dim where their ranges touch or overlap.
constexpr int NCUR = 8;   // boxes of one tensor at a time

__device__ inline void simplify_list(NBox* b, int& k, int rank) {
  bool changed = true;
  while (changed) {
    changed = false;
    for (int i = 0; i < k && !changed; ++i) {
      for (int j = 0; j < k && !changed; ++j) {
        if (j == i) continue;
        bool contains = true;
        int ndiff = 0, dd = 0;
        for (int d = 0; d < rank; ++d) {
          contains &= b[i].lo[d] <= b[j].lo[d] && b[j].hi[d] <= b[i].hi[d];
          if (b[i].lo[d] != b[j].lo[d] || b[i].hi[d] != b[j].hi[d]) {
            ++ndiff;
            dd = d;
          }
        }
        bool merge = !contains && ndiff == 1 && b[i].lo[dd] <= b[j].hi[dd] &&
                     b[j].lo[dd] <= b[i].hi[dd];
        if (contains || merge) {
          if (merge) {
            b[i].lo[dd] = min(b[i].lo[dd], b[j].lo[dd]);
            b[i].hi[dd] = max(b[i].hi[dd], b[j].hi[dd]);
          }
          b[j] = b[--k];
          changed = true;
        }
      }
    }
  }
}

// Move the boxes of tensor t out of the pool into cur[] (at most NCUR).
__device__ inline int take_boxes(LocState& L, int t, NBox* cur) {
  int k = 0;
  for (int i = 0; i < L.npool;) {
    if (L.pool[i].t == t) {
      if (k < NCUR) {
        cur[k++] = L.pool[i];
      } else {
        L.err |= CE_CAPACITY;
      }
      L.pool[i] = L.pool[--L.npool];
    } else {
      ++i;
    }
  }
  return k;
}

// Propagate from location `loc` of the output down to the inputs.  visit(t,
// box) sees every (merged) box of every primitive tensor before it is
// expanded.  Afterwards the pool holds input boxes and the streams raw reads.
template <class Visit>
__device__ void propagate(const Prog& P, int64_t loc, LocState& L, Visit& visit) {
  L.npool = 0;
  L.nst = 0;
  L.err = 0;
  L.pending = 0;
  const Tensor& Y = P.t[P.output];
  if (loc < 0 || loc >= Y.numel) {
    L.err |= CE_LOCATION;
    return;
  }
  int32_t o[MR], hi[MR];
  unflatten(loc, Y, o);
  for (int d = 0; d < MR; ++d) hi[d] = o[d] + 1;
  push_box(L, P.output, o, hi);
  NBox cur[NCUR];
  for (int t = P.output; t >= P.n_inputs && !L.err; --t) {
    if (!((L.pending >> t) & 1)) continue;
    const Tensor& T = P.t[t];
    int k = take_boxes(L, t, cur);
    if (k == 0) continue;
    simplify_list(cur, k, T.rank);
    for (int i = 0; i < k && !L.err; ++i) {
      const NBox& B = cur[i];
      visit(t, B);
      if (T.kind == K_CONTRACT || T.kind == K_MAXSET) {
        propagate_pieces(P, T, B, L);
      } else if (T.kind == K_BINARY) {
        for (int s = 0; s < 2; ++s) {
          const Tensor& A = P.t[T.args[s]];
          int32_t lo2[MR], hi2[MR];
          for (int d = 0; d < MR; ++d) {
            if (d < T.arg_rank[s] && A.shape[d] != 1) {
              lo2[d] = B.lo[T.axes[s][d]];
              hi2[d] = B.hi[T.axes[s][d]];
            } else {
              lo2[d] = 0;
              hi2[d] = 1;
            }
          }
          push_box(L, T.args[s], lo2, hi2);
        }
      } else {
        push_box(L, T.args[0], B.lo, B.hi);
      }
    }
  }
}

struct NoVisit {
  __device__ void operator()(int, const NBox&) {}
};

// Input boxes (merged per tensor) -> streams of runs (tensor-local offsets).
__device__ inline void boxes_to_streams(const Prog& P, LocState& L) {
  NBox cur[NCUR];
  for (int u = 0; u < P.n_inputs && !L.err; ++u) {
    if (!((L.pending >> u) & 1)) continue;
    const Tensor& A = P.t[u];
    int k = take_boxes(L, u, cur);
    simplify_list(cur, k, A.rank);
    for (int i = 0; i < k && !L.err; ++i) {
      const NBox& b = cur[i];
      Contrib c[MR];
      int nc = 0;
      int64_t start = 0;
      for (int d = 0; d < A.rank; ++d) {
        start += A.stride[d] * b.lo[d];
        if (b.hi[d] - b.lo[d] > 1) c[nc++] = Contrib{A.stride[d], 0, b.hi[d] - b.lo[d]};
      }
      Stream s;
      if (!canonical_stream(u, start, c, nc, s)) {
        L.err |= CE_UNSUPPORTED;
        return;
      }
      push_stream(L, s);
    }
  }
  L.npool = 0;
}

}  // namespace dirigo
