// Index-map compiler: validates an op-graph description and lowers every op to
// primitive per-element equations (Sec. 3.3 "Torch Operations": each op has a
// predefined mapping to symbolic expressions; Sec. 3.4 "Per-element
// equations").
//
// Lowering table (the order of the primitive tensors a composite op emits is
// part of the exported term-list format):
//   matmul, bmm, linear, conv2d -> CONTRACT [-> BINARY add bias]
//       conv2d: X[n, ci, s*h + i - p, s*w + j - p] * W[co, ci, i, j]; taps outside
//       the image are absent (guards), so neither factor of a padded tap is read
//   maxpool2d, max             -> MAXSET
//   sum, mean                  -> CONTRACT with one operand (coef 1 or 1/D)
//   add, sub, mul, div         -> BINARY
//   scale, add_scalar          -> AFFINE;  relu, clamp_min -> MAXC
//   gelu, tanh, exp, ...       -> UNARY (uninterpreted function)
//   sigmoid                    -> AFFINE(-1, 0), UNARY exp, AFFINE(1, 1), UNARY recip
//                                 (a sound identity, Sec. 4.2)
//   softmax(dim)               -> UNARY exp, CONTRACT sum (keepdim), UNARY recip, BINARY mul
//   layernorm(z, g, b, eps)    -> CONTRACT mean, BINARY sub, BINARY mul (square),
//                                 CONTRACT mean, AFFINE(1, eps), UNARY rsqrt,
//                                 BINARY mul, [BINARY mul gamma], [BINARY add beta]
//   contract, maxset           -> as given (explicit pieces)
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "cells.h"
#include "internal.h"
#include "keyspec.cuh"

namespace dirigo {

namespace {

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

// m * 2^e / d mod p, with d odd and p prime not dividing d
uint32_t enc_lane(int64_t m, int64_t e, int64_t d, uint64_t p) {
  uint64_t mag = m < 0 ? (uint64_t)0 - (uint64_t)m : (uint64_t)m;
  uint64_t am = mag % p;
  if (m < 0) am = (p - am) % p;
  uint64_t two = e >= 0 ? powmod(2, (uint64_t)e, p) : powmod(powmod(2, p - 2, p), (uint64_t)(-e), p);
  uint64_t dinv = powmod((uint64_t)d % p, p - 2, p);
  return (uint32_t)(am * two % p * dinv % p);
}

}  // namespace

KConst encode_const(const dirigo_const& c, bool* ok) {
  KConst k{0, 0, 0.0f, 1, 0.0};
  *ok = true;
  int64_t m, e = 0, d = 1;
  if (c.den != 0) {
    m = c.num;
    d = c.den;
    if (d < 0) {
      d = -d;
      m = -m;
    }
    if (m == 0) return k;
    while ((m & 1) == 0) {
      m /= 2;
      ++e;
    }
    while ((d & 1) == 0) {
      d /= 2;
      --e;
    }
    k.f = (float)((double)c.num / (double)c.den);
  } else {
    double v = c.value;
    if (!std::isfinite(v)) {
      *ok = false;
      return k;
    }
    if (v == 0.0) return k;
    int ex;
    double mant = std::frexp(v, &ex);          // v = mant * 2^ex, |mant| in [0.5, 1)
    m = (int64_t)std::ldexp(mant, 53);         // exact
    e = ex - 53;
    while ((m & 1) == 0) {
      m /= 2;
      ++e;
    }
    k.f = (float)v;
  }
  if (d % kP0 == 0 || d % kP1 == 0) {
    *ok = false;
    return k;
  }
  k.k0 = enc_lane(m, e, d, kP0);
  k.k1 = enc_lane(m, e, d, kP1);
  k.is_zero = 0;
  k.d = std::ldexp((double)m, (int)e) / (double)d;
  return k;
}

namespace {

struct Builder {
  dirigo_graph* g;
  Prog& P;
  std::string err;
  dirigo_status st = DIRIGO_OK;

  explicit Builder(dirigo_graph* gg) : g(gg), P(gg->prog) {}

  bool fail(dirigo_status s, const std::string& m) {
    if (st == DIRIGO_OK) {
      st = s;
      err = m;
    }
    return false;
  }

  static int64_t numel(const int32_t* s, int r) {
    int64_t n = 1;
    for (int i = 0; i < r; ++i) n *= s[i];
    return n;
  }

  int new_tensor(int kind, int fn, int nargs, const int* args, int rank, const int32_t* shape) {
    if (P.n_tensors >= MT) {
      fail(DIRIGO_E_UNSUPPORTED, "too many primitive tensors (max 40)");
      return -1;
    }
    if (rank < 0 || rank > MR) {
      fail(DIRIGO_E_UNSUPPORTED, "rank above 4");
      return -1;
    }
    Tensor& t = P.t[P.n_tensors];
    std::memset(&t, 0, sizeof(t));
    t.kind = (int8_t)kind;
    t.fn = (int8_t)fn;
    t.nargs = (int8_t)nargs;
    t.rank = (int8_t)rank;
    for (int i = 0; i < nargs; ++i) t.args[i] = args[i];
    int64_t acc = 1;
    for (int d = rank - 1; d >= 0; --d) {
      t.shape[d] = shape[d];
      t.stride[d] = acc;
      acc *= shape[d];
    }
    for (int d = rank; d < MR; ++d) t.shape[d] = 1;
    t.numel = acc;
    t.piece0 = -1;
    return P.n_tensors++;
  }

  int add_piece(const Piece& pc) {
    if (P.n_pieces >= MP) {
      fail(DIRIGO_E_UNSUPPORTED, "too many pieces (max 24)");
      return -1;
    }
    P.p[P.n_pieces] = pc;
    return P.n_pieces++;
  }

  const Tensor& T(int id) const { return P.t[id]; }

  static Piece blank_piece(const Tensor& out) {
    Piece pc;
    std::memset(&pc, 0, sizeof(pc));
    for (int d = 0; d < MR; ++d) {
      pc.lo[d] = 0;
      pc.hi[d] = d < out.rank ? out.shape[d] : 1;
    }
    pc.coef = KConst{1, 1, 1.0f, 0, 1.0};
    return pc;
  }

  int contract_like(int kind, int nargs, const int* args, int rank, const int32_t* shape,
                    std::vector<Piece> pieces) {
    int id = new_tensor(kind, 0, nargs, args, rank, shape);
    if (id < 0) return -1;
    Tensor& t = P.t[id];
    t.piece0 = (int16_t)P.n_pieces;
    int64_t terms = 0;
    for (auto& pc : pieces) {
      int64_t vol = 1;
      for (int e = 0; e < pc.nred; ++e) vol *= std::max(0, pc.rhi[e] - pc.rlo[e]);
      terms += vol;
      if (add_piece(pc) < 0) return -1;
    }
    t.npieces = (int16_t)pieces.size();
    t.max_terms = (int32_t)std::min<int64_t>(terms, 1 << 30);
    if (kind == K_CONTRACT && nargs == 2) t.flags |= TF_GEMM;
    return id;
  }

  // sum / mean / max over one dim of tensor a
  int reduction(int kind, int a, int dim, bool keepdim, KConst coef) {
    const Tensor ta = T(a);
    if (ta.rank == 0) {
      fail(DIRIGO_E_SHAPE, "reduction of a rank-0 tensor");
      return -1;
    }
    if (dim < 0) dim += ta.rank;
    if (dim < 0 || dim >= ta.rank) {
      fail(DIRIGO_E_SHAPE, "reduction dim out of range");
      return -1;
    }
    int32_t shape[MR];
    int rank = 0;
    Piece pc;
    std::memset(&pc, 0, sizeof(pc));
    for (int d = 0; d < ta.rank; ++d) {
      if (d == dim) {
        if (keepdim) {
          shape[rank] = 1;
          pc.acc[0].os[rank] = 0;
          ++rank;
        }
        continue;
      }
      shape[rank] = ta.shape[d];
      pc.acc[0].os[rank] = ta.stride[d];
      ++rank;
    }
    for (int d = 0; d < MR; ++d) {
      pc.lo[d] = 0;
      pc.hi[d] = d < rank ? shape[d] : 1;
    }
    pc.nred = 1;
    pc.rlo[0] = 0;
    pc.rhi[0] = ta.shape[dim];
    pc.acc[0].rs[0] = ta.stride[dim];
    pc.coef = coef;
    int args[1] = {a};
    return contract_like(kind, 1, args, rank, shape, {pc});
  }

  int unary(int fn, int a) {
    const Tensor ta = T(a);
    int args[1] = {a};
    return new_tensor(K_UNARY, fn, 1, args, ta.rank, ta.shape);
  }

  int affine(int a, KConst mul, KConst add) {
    const Tensor ta = T(a);
    int args[1] = {a};
    int id = new_tensor(K_AFFINE, 0, 1, args, ta.rank, ta.shape);
    if (id >= 0) {
      P.t[id].a = mul;
      P.t[id].c = add;
    }
    return id;
  }

  int maxc(int a, KConst c) {
    const Tensor ta = T(a);
    int args[1] = {a};
    int id = new_tensor(K_MAXC, 0, 1, args, ta.rank, ta.shape);
    if (id >= 0) P.t[id].c = c;
    return id;
  }

  // broadcasting binary op; axes_rank < 0: trailing alignment
  int binary(int fn, int a, int b, const int32_t* axes_rank, const int32_t (*axes)[MR]) {
    const Tensor ta = T(a), tb = T(b);
    int ax[2][MR];
    int rk[2] = {ta.rank, tb.rank};
    int out_rank = 0;
    for (int s = 0; s < 2; ++s) {
      if (axes_rank && axes_rank[s] >= 0) {
        if (axes_rank[s] != rk[s]) {
          fail(DIRIGO_E_SHAPE, "axes rank differs from operand rank");
          return -1;
        }
        for (int d = 0; d < rk[s]; ++d) {
          ax[s][d] = axes[s][d];
          if (ax[s][d] < 0 || ax[s][d] >= MR) {
            fail(DIRIGO_E_SHAPE, "axis out of range");
            return -1;
          }
          out_rank = std::max(out_rank, ax[s][d] + 1);
        }
      }
    }
    bool dflt = !(axes_rank && axes_rank[0] >= 0 && axes_rank[1] >= 0);
    if (dflt) {
      out_rank = std::max(ta.rank, tb.rank);
      for (int s = 0; s < 2; ++s)
        for (int d = 0; d < rk[s]; ++d) ax[s][d] = out_rank - rk[s] + d;
    }
    int32_t shape[MR];
    for (int d = 0; d < MR; ++d) shape[d] = 1;
    const Tensor* ts[2] = {&ta, &tb};
    for (int s = 0; s < 2; ++s)
      for (int d = 0; d < rk[s]; ++d) {
        int32_t v = ts[s]->shape[d];
        int o = ax[s][d];
        if (v != 1) {
          if (shape[o] != 1 && shape[o] != v) {
            fail(DIRIGO_E_SHAPE, "broadcast shapes do not match");
            return -1;
          }
          shape[o] = v;
        }
      }
    int args[2] = {a, b};
    int id = new_tensor(K_BINARY, fn, 2, args, out_rank, shape);
    if (id < 0) return -1;
    Tensor& t = P.t[id];
    for (int s = 0; s < 2; ++s) {
      t.arg_rank[s] = (int8_t)rk[s];
      for (int d = 0; d < MR; ++d) t.axes[s][d] = d < rk[s] ? (int8_t)ax[s][d] : (int8_t)-1;
    }
    return id;
  }

  bool konst(const dirigo_const& c, KConst* out) {
    bool ok;
    *out = encode_const(c, &ok);
    if (!ok) return fail(DIRIGO_E_INVALID, "constant not representable");
    return true;
  }

  int lower(const dirigo_op_desc& op, const std::vector<int>& hl2t) {
    int A[3];
    if (op.n_args < 0 || op.n_args > 3) {
      fail(DIRIGO_E_INVALID, "bad argument count");
      return -1;
    }
    for (int i = 0; i < op.n_args; ++i) {
      if (op.args[i] < 0 || op.args[i] >= (int)hl2t.size()) {
        fail(DIRIGO_E_INVALID, "argument is not an earlier tensor");
        return -1;
      }
      A[i] = hl2t[op.args[i]];
    }
    auto need = [&](int lo, int hi) {
      if (op.n_args < lo || op.n_args > hi) return fail(DIRIGO_E_INVALID, "wrong number of arguments");
      return true;
    };
    KConst one{1, 1, 1.0f, 0, 1.0}, zero{0, 0, 0.0f, 1, 0.0};
    switch (op.kind) {
      case DIRIGO_OP_MATMUL: {
        if (!need(2, 2)) return -1;
        const Tensor x = T(A[0]), w = T(A[1]);
        if (x.rank != 2 || w.rank != 2 || x.shape[1] != w.shape[0])
          return fail(DIRIGO_E_SHAPE, "matmul shapes"), -1;
        int32_t shape[2] = {x.shape[0], w.shape[1]};
        Piece pc = blank_piece(x);
        pc.hi[0] = shape[0];
        pc.hi[1] = shape[1];
        pc.nred = 1;
        pc.rhi[0] = x.shape[1];
        pc.acc[0].os[0] = x.shape[1];
        pc.acc[0].rs[0] = 1;
        pc.acc[1].os[1] = 1;
        pc.acc[1].rs[0] = w.shape[1];
        return contract_like(K_CONTRACT, 2, A, 2, shape, {pc});
      }
      case DIRIGO_OP_BMM: {
        if (!need(2, 2)) return -1;
        const Tensor x = T(A[0]), w = T(A[1]);
        if (x.rank != 3 || w.rank != 3 || x.shape[0] != w.shape[0] || x.shape[2] != w.shape[1])
          return fail(DIRIGO_E_SHAPE, "bmm shapes"), -1;
        int32_t B = x.shape[0], M = x.shape[1], K = x.shape[2], N = w.shape[2];
        int32_t shape[3] = {B, M, N};
        Piece pc = blank_piece(x);
        pc.hi[0] = B;
        pc.hi[1] = M;
        pc.hi[2] = N;
        pc.nred = 1;
        pc.rhi[0] = K;
        pc.acc[0].os[0] = (int64_t)M * K;
        pc.acc[0].os[1] = K;
        pc.acc[0].rs[0] = 1;
        pc.acc[1].os[0] = (int64_t)K * N;
        pc.acc[1].os[2] = 1;
        pc.acc[1].rs[0] = N;
        return contract_like(K_CONTRACT, 2, A, 3, shape, {pc});
      }
      case DIRIGO_OP_LINEAR: {
        if (!need(2, 3)) return -1;
        const Tensor x = T(A[0]), w = T(A[1]);
        if (x.rank != 2 || w.rank != 2 || x.shape[1] != w.shape[1])
          return fail(DIRIGO_E_SHAPE, "linear shapes"), -1;
        int32_t shape[2] = {x.shape[0], w.shape[0]};
        Piece pc = blank_piece(x);
        pc.hi[0] = shape[0];
        pc.hi[1] = shape[1];
        pc.nred = 1;
        pc.rhi[0] = x.shape[1];
        pc.acc[0].os[0] = x.shape[1];
        pc.acc[0].rs[0] = 1;
        pc.acc[1].os[1] = w.shape[1];
        pc.acc[1].rs[0] = 1;
        int t = contract_like(K_CONTRACT, 2, A, 2, shape, {pc});
        if (t < 0 || op.n_args < 3) return t;
        const Tensor b = T(A[2]);
        if (b.rank != 1 || b.shape[0] != shape[1]) return fail(DIRIGO_E_SHAPE, "linear bias"), -1;
        int32_t ar[2] = {2, 1};
        int32_t ax[2][MR] = {{0, 1, 0, 0}, {1, 0, 0, 0}};
        return binary(B_ADD, t, A[2], ar, ax);
      }
      case DIRIGO_OP_CONV2D: {
        if (!need(2, 3)) return -1;
        const Tensor x = T(A[0]), w = T(A[1]);
        int32_t s = op.stride > 0 ? op.stride : 1, p = op.pad;
        if (x.rank != 4 || w.rank != 4 || x.shape[1] != w.shape[1] || p < 0)
          return fail(DIRIGO_E_SHAPE, "conv2d shapes"), -1;
        int32_t N = x.shape[0], Ci = x.shape[1], H = x.shape[2], W = x.shape[3];
        int32_t Co = w.shape[0], kh = w.shape[2], kw = w.shape[3];
        int32_t Ho = (H + 2 * p - kh) / s + 1, Wo = (W + 2 * p - kw) / s + 1;
        if (Ho <= 0 || Wo <= 0) return fail(DIRIGO_E_SHAPE, "conv2d output is empty"), -1;
        int32_t shape[4] = {N, Co, Ho, Wo};
        Piece pc = blank_piece(x);
        for (int d = 0; d < 4; ++d) pc.hi[d] = shape[d];
        pc.nred = 3;
        pc.rhi[0] = Ci;
        pc.rhi[1] = kh;
        pc.rhi[2] = kw;
        pc.nguard = 2;
        pc.g[0] = Guard{2, 1, s, -p, 0, H};
        pc.g[1] = Guard{3, 2, s, -p, 0, W};
        pc.acc[0].base = -(int64_t)p * W - p;
        pc.acc[0].os[0] = (int64_t)Ci * H * W;
        pc.acc[0].os[2] = (int64_t)s * W;
        pc.acc[0].os[3] = s;
        pc.acc[0].rs[0] = (int64_t)H * W;
        pc.acc[0].rs[1] = W;
        pc.acc[0].rs[2] = 1;
        pc.acc[1].os[1] = (int64_t)Ci * kh * kw;
        pc.acc[1].rs[0] = (int64_t)kh * kw;
        pc.acc[1].rs[1] = kw;
        pc.acc[1].rs[2] = 1;
        int t = contract_like(K_CONTRACT, 2, A, 4, shape, {pc});
        if (t < 0 || op.n_args < 3) return t;
        const Tensor b = T(A[2]);
        if (b.rank != 1 || b.shape[0] != Co) return fail(DIRIGO_E_SHAPE, "conv2d bias"), -1;
        int32_t ar[2] = {4, 1};
        int32_t ax[2][MR] = {{0, 1, 2, 3}, {1, 0, 0, 0}};
        return binary(B_ADD, t, A[2], ar, ax);
      }
      case DIRIGO_OP_MAXPOOL2D: {
        if (!need(1, 1)) return -1;
        const Tensor x = T(A[0]);
        int32_t k = op.k, s = op.stride > 0 ? op.stride : op.k;
        if (x.rank != 4 || k <= 0 || x.shape[2] < k || x.shape[3] < k)
          return fail(DIRIGO_E_SHAPE, "maxpool2d shapes"), -1;
        int32_t N = x.shape[0], C = x.shape[1], H = x.shape[2], W = x.shape[3];
        int32_t shape[4] = {N, C, (H - k) / s + 1, (W - k) / s + 1};
        Piece pc = blank_piece(x);
        for (int d = 0; d < 4; ++d) pc.hi[d] = shape[d];
        pc.nred = 2;
        pc.rhi[0] = k;
        pc.rhi[1] = k;
        pc.acc[0].os[0] = (int64_t)C * H * W;
        pc.acc[0].os[1] = (int64_t)H * W;
        pc.acc[0].os[2] = (int64_t)s * W;
        pc.acc[0].os[3] = s;
        pc.acc[0].rs[0] = W;
        pc.acc[0].rs[1] = 1;
        return contract_like(K_MAXSET, 1, A, 4, shape, {pc});
      }
      case DIRIGO_OP_ADD: case DIRIGO_OP_SUB: case DIRIGO_OP_MUL: case DIRIGO_OP_DIV: {
        if (!need(2, 2)) return -1;
        int fn = op.kind == DIRIGO_OP_ADD ? B_ADD : op.kind == DIRIGO_OP_SUB ? B_SUB
                 : op.kind == DIRIGO_OP_MUL ? B_MUL : B_DIV;
        return binary(fn, A[0], A[1], op.axes_rank, op.axes);
      }
      case DIRIGO_OP_SCALE: {
        if (!need(1, 1)) return -1;
        KConst c;
        if (!konst(op.c, &c)) return -1;
        return affine(A[0], c, zero);
      }
      case DIRIGO_OP_ADD_SCALAR: {
        if (!need(1, 1)) return -1;
        KConst c;
        if (!konst(op.c, &c)) return -1;
        return affine(A[0], one, c);
      }
      case DIRIGO_OP_CLAMP_MIN: {
        if (!need(1, 1)) return -1;
        KConst c;
        if (!konst(op.c, &c)) return -1;
        return maxc(A[0], c);
      }
      case DIRIGO_OP_RELU:
        if (!need(1, 1)) return -1;
        return maxc(A[0], zero);
      case DIRIGO_OP_GELU: if (!need(1, 1)) return -1; return unary(F_GELU_ERF, A[0]);
      case DIRIGO_OP_GELU_TANH: if (!need(1, 1)) return -1; return unary(F_GELU_TANH, A[0]);
      case DIRIGO_OP_TANH: if (!need(1, 1)) return -1; return unary(F_TANH, A[0]);
      case DIRIGO_OP_EXP: if (!need(1, 1)) return -1; return unary(F_EXP, A[0]);
      case DIRIGO_OP_RSQRT: if (!need(1, 1)) return -1; return unary(F_RSQRT, A[0]);
      case DIRIGO_OP_RECIP: if (!need(1, 1)) return -1; return unary(F_RECIP, A[0]);
      case DIRIGO_OP_ERF: if (!need(1, 1)) return -1; return unary(F_ERF, A[0]);
      case DIRIGO_OP_SQRT: if (!need(1, 1)) return -1; return unary(F_SQRT, A[0]);
      case DIRIGO_OP_LOG: if (!need(1, 1)) return -1; return unary(F_LOG, A[0]);
      case DIRIGO_OP_SIGMOID: {
        if (!need(1, 1)) return -1;
        dirigo_const m1{-1.0, 0, 0};
        KConst neg;
        konst(m1, &neg);
        int t = affine(A[0], neg, zero);
        if (t < 0) return -1;
        t = unary(F_EXP, t);
        if (t < 0) return -1;
        t = affine(t, one, one);
        if (t < 0) return -1;
        return unary(F_RECIP, t);
      }
      case DIRIGO_OP_SUM: case DIRIGO_OP_MEAN: case DIRIGO_OP_MAX: {
        if (!need(1, 1)) return -1;
        const Tensor x = T(A[0]);
        int dim = op.dim < 0 ? op.dim + x.rank : op.dim;
        if (dim < 0 || dim >= x.rank) return fail(DIRIGO_E_SHAPE, "reduction dim"), -1;
        KConst c = one;
        if (op.kind == DIRIGO_OP_MEAN) {
          dirigo_const q{0.0, 1, x.shape[dim]};
          if (!konst(q, &c)) return -1;
        }
        return reduction(op.kind == DIRIGO_OP_MAX ? K_MAXSET : K_CONTRACT, A[0], dim,
                         op.keepdim != 0, c);
      }
      case DIRIGO_OP_SOFTMAX: {
        if (!need(1, 1)) return -1;
        int e = unary(F_EXP, A[0]);
        if (e < 0) return -1;
        int s = reduction(K_CONTRACT, e, op.dim, true, one);
        if (s < 0) return -1;
        int r = unary(F_RECIP, s);
        if (r < 0) return -1;
        return binary(B_MUL, e, r, nullptr, nullptr);
      }
      case DIRIGO_OP_LAYERNORM: {
        if (!need(1, 3)) return -1;
        int z = A[0];
        const Tensor tz = T(z);
        if (tz.rank < 1) return fail(DIRIGO_E_SHAPE, "layernorm rank"), -1;
        int32_t D = tz.shape[tz.rank - 1];
        dirigo_const q{0.0, 1, D};
        KConst invD;
        if (!konst(q, &invD)) return -1;
        KConst eps;
        dirigo_const ec = op.c;
        if (ec.den == 0 && ec.value == 0.0) ec.value = 1e-5;
        if (!konst(ec, &eps)) return -1;
        int mu = reduction(K_CONTRACT, z, tz.rank - 1, true, invD);
        if (mu < 0) return -1;
        int d = binary(B_SUB, z, mu, nullptr, nullptr);
        if (d < 0) return -1;
        int sq = binary(B_MUL, d, d, nullptr, nullptr);
        if (sq < 0) return -1;
        int v = reduction(K_CONTRACT, sq, tz.rank - 1, true, invD);
        if (v < 0) return -1;
        int ve = affine(v, one, eps);
        if (ve < 0) return -1;
        int rs = unary(F_RSQRT, ve);
        if (rs < 0) return -1;
        int t = binary(B_MUL, d, rs, nullptr, nullptr);
        if (t < 0) return -1;
        if (op.n_args > 1) {
          if (T(A[1]).rank != 1 || T(A[1]).shape[0] != D) return fail(DIRIGO_E_SHAPE, "gamma"), -1;
          t = binary(B_MUL, t, A[1], nullptr, nullptr);
          if (t < 0) return -1;
        }
        if (op.n_args > 2) {
          if (T(A[2]).rank != 1 || T(A[2]).shape[0] != D) return fail(DIRIGO_E_SHAPE, "beta"), -1;
          t = binary(B_ADD, t, A[2], nullptr, nullptr);
        }
        return t;
      }
      case DIRIGO_OP_CONTRACT: case DIRIGO_OP_MAXSET: {
        bool mx = op.kind == DIRIGO_OP_MAXSET;
        if (!need(1, mx ? 1 : 2)) return -1;
        if (op.rank < 0 || op.rank > MR) return fail(DIRIGO_E_UNSUPPORTED, "rank above 4"), -1;
        if (op.n_pieces < 1 || !op.pieces) return fail(DIRIGO_E_INVALID, "no pieces"), -1;
        int32_t shape[MR];
        for (int d = 0; d < op.rank; ++d) {
          if (op.shape[d] <= 0 || op.shape[d] > INT32_MAX)
            return fail(DIRIGO_E_SHAPE, "bad output shape"), -1;
          shape[d] = (int32_t)op.shape[d];
        }
        std::vector<Piece> pcs;
        for (int q = 0; q < op.n_pieces; ++q) {
          const dirigo_piece& s = op.pieces[q];
          Piece pc;
          std::memset(&pc, 0, sizeof(pc));
          for (int d = 0; d < MR; ++d) {
            if (d < op.rank) {
              int64_t lo = std::max<int64_t>(0, s.lo[d]);
              int64_t hi = std::min<int64_t>(shape[d], s.hi[d]);
              pc.lo[d] = (int32_t)lo;
              pc.hi[d] = (int32_t)std::max(lo, hi);
            } else {
              pc.lo[d] = 0;
              pc.hi[d] = 1;
            }
          }
          if (s.n_red < 0 || s.n_red > MRED) return fail(DIRIGO_E_UNSUPPORTED, "too many reduction dims"), -1;
          if (s.n_guards < 0 || s.n_guards > MG) return fail(DIRIGO_E_UNSUPPORTED, "too many guards"), -1;
          pc.nred = s.n_red;
          for (int e = 0; e < s.n_red; ++e) {
            if (s.red_lo[e] < INT32_MIN / 2 || s.red_hi[e] > INT32_MAX / 2)
              return fail(DIRIGO_E_UNSUPPORTED, "reduction box too large"), -1;
            pc.rlo[e] = (int32_t)s.red_lo[e];
            pc.rhi[e] = (int32_t)std::max(s.red_lo[e], s.red_hi[e]);
          }
          pc.nguard = s.n_guards;
          for (int j = 0; j < s.n_guards; ++j) {
            const dirigo_guard& gd = s.guards[j];
            if (gd.od < -1 || gd.od >= op.rank || gd.rd < -1 || gd.rd >= s.n_red)
              return fail(DIRIGO_E_INVALID, "guard dims out of range"), -1;
            auto fits = [](int64_t v) { return v > INT32_MIN / 2 && v < INT32_MAX / 2; };
            if (!fits(gd.oa) || !fits(gd.c) || !fits(gd.lo) || !fits(gd.hi))
              return fail(DIRIGO_E_UNSUPPORTED, "guard constants too large"), -1;
            pc.g[j] = Guard{gd.od, gd.rd, (int32_t)gd.oa, (int32_t)gd.c, (int32_t)gd.lo, (int32_t)gd.hi};
          }
          if (mx) {
            pc.coef = one;
          } else if (!konst(s.coef, &pc.coef)) {
            return -1;
          }
          for (int i = 0; i < op.n_args; ++i) {
            pc.acc[i].base = s.access[i].base;
            for (int d = 0; d < MR; ++d) pc.acc[i].os[d] = d < op.rank ? s.access[i].os[d] : 0;
            for (int e = 0; e < MRED; ++e) pc.acc[i].rs[e] = e < s.n_red ? s.access[i].rs[e] : 0;
          }
          pcs.push_back(pc);
        }
        return contract_like(mx ? K_MAXSET : K_CONTRACT, op.n_args, A, op.rank, shape, pcs);
      }
      case DIRIGO_OP_KERNEL_CONTRACT: case DIRIGO_OP_KERNEL_MAXSET: {
        // a kernel's write set, inverted into pieces over output coordinates
        std::vector<dirigo_piece> pcs;
        std::string why;
        dirigo_status s = invert_kernel_writes(op, &pcs, &why);
        if (s != DIRIGO_OK) return fail(s, why.c_str()), -1;
        dirigo_op_desc eq = op;
        eq.kind = op.kind == DIRIGO_OP_KERNEL_MAXSET ? DIRIGO_OP_MAXSET : DIRIGO_OP_CONTRACT;
        eq.n_pieces = (int32_t)pcs.size();
        eq.pieces = pcs.data();
        return lower(eq, hl2t);
      }
      default:
        fail(DIRIGO_E_INVALID, "unknown op kind");
        return -1;
    }
  }
};

}  // namespace

namespace {

// Location-independent image template of operand i of a piece (see AccTpl).
void build_template(const Prog& P, const Tensor& T, Piece& pc, int i) {
  AccTpl& tp = pc.tpl[i];
  std::memset(&tp, 0, sizeof(tp));
  const Access& a = pc.acc[i];
  const Tensor& A = P.t[T.args[i]];
  Slot sl[MSLOT];
  int n = 0;
  bool used_o[MR] = {false, false, false, false}, used_r[MRED] = {false, false, false, false};
  for (int j = 0; j < pc.nguard; ++j) {
    const Guard& g = pc.g[j];
    if (g.od < 0 || g.rd < 0) continue;
    used_o[g.od] = used_r[g.rd] = true;
    int64_t sa = a.os[g.od], sr = a.rs[g.rd];
    if (sa == 0 && sr == 0) continue;
    Slot x{0, (int8_t)j, 0, 0, 0, 0};
    if (sr != 0 && sa == (int64_t)g.oa * sr) {
      x.kind = SL_V;
      x.step = sr;
    } else if (sa == 0) {
      x.kind = SL_GR;
      x.step = sr;
    } else if (sr == 0) {
      x.kind = SL_GO;
      x.step = sa;
    } else {
      tp.unsupported = 1;
      continue;
    }
    sl[n++] = x;
  }
  for (int d = 0; d < T.rank; ++d)
    if (!used_o[d] && a.os[d] != 0) sl[n++] = Slot{SL_O, (int8_t)d, 0, 0, 0, a.os[d]};
  for (int e = 0; e < pc.nred; ++e)
    if (!used_r[e] && a.rs[e] != 0) sl[n++] = Slot{SL_R, (int8_t)e, 0, 0, 0, a.rs[e]};
  // ascending |step|
  for (int x = 1; x < n; ++x)
    for (int y = x; y > 0 && std::llabs(sl[y - 1].step) > std::llabs(sl[y].step); --y) {
      Slot t = sl[y];
      sl[y] = sl[y - 1];
      sl[y - 1] = t;
    }
  tp.natural = 1;
  for (int k = 0; k < n; ++k) {
    int64_t st = sl[k].step;
    int nd = -1;
    int64_t q = 0;
    if (st > 0) {
      for (int d = 0; d < A.rank; ++d)
        if (A.stride[d] <= st) {
          if (st % A.stride[d] == 0 && st / A.stride[d] < A.shape[d]) {
            nd = d;
            q = st / A.stride[d];
          }
          break;
        }
    }
    if (nd < 0) {
      tp.natural = 0;
      nd = 0;
    }
    sl[k].nd = (int8_t)nd;
    sl[k].q = (int32_t)q;
    tp.s[k] = sl[k];
  }
  tp.nslot = (int8_t)n;
  // base offset over the natural dims, remainders truncated toward zero
  int64_t x = a.base;
  for (int d = A.rank - 1; d >= 1; --d) {
    tp.cbase[d] = (int32_t)(x % A.shape[d]);
    x /= A.shape[d];
  }
  if (A.rank > 0) {
    if (x < INT32_MIN || x > INT32_MAX) tp.natural = 0;
    tp.cbase[0] = (int32_t)x;
  }
}

}  // namespace

// Sound identity (Sec. 4.2 "Sound identities"): a softmax written out with the
// max shift,
//   m = max(x, d, keepdim); z = x - m; e = exp(z); s = sum(e, d, keepdim);
//   y = e / s   (or e * recip(s)),
// equals softmax(x) over d over the reals, so y is lowered as that softmax and
// its canonical term does not depend on the shift (m, z, e, s are still
// lowered as written, for any other reader).
namespace {

const dirigo_op_desc* hl_op(const dirigo_graph_desc* g, int id) {
  const int k = id - g->n_inputs;
  return k >= 0 && k < g->n_ops ? &g->ops[k] : nullptr;
}

bool default_axes(const dirigo_op_desc& op) {
  for (int s = 0; s < 2; ++s) {
    if (op.axes_rank[s] < 0) continue;
    for (int d = 0; d < op.axes_rank[s] && d < DIRIGO_MAX_RANK; ++d)
      if (op.axes[s][d] != d) return false;
  }
  return true;
}

// x and d of a matched pattern ending at op k, or x = -1; shapes[id] is the
// shape of high-level tensor id (known for every tensor before op k)
int match_softmax_shift(const dirigo_graph_desc* g, int k,
                        const std::vector<std::vector<int64_t>>& shapes, int* dim_out) {
  const dirigo_op_desc& y = g->ops[k];
  if (y.n_args != 2 || !default_axes(y)) return -1;
  int e_id = y.args[0], s_id = -1;
  if (y.kind == DIRIGO_OP_DIV) {
    s_id = y.args[1];
  } else if (y.kind == DIRIGO_OP_MUL) {
    const dirigo_op_desc* r = hl_op(g, y.args[1]);
    if (!r || r->kind != DIRIGO_OP_RECIP || r->n_args != 1) return -1;
    s_id = r->args[0];
  } else {
    return -1;
  }
  const dirigo_op_desc* e = hl_op(g, e_id);
  const dirigo_op_desc* s = hl_op(g, s_id);
  if (!e || !s || e->kind != DIRIGO_OP_EXP || e->n_args != 1) return -1;
  if (s->kind != DIRIGO_OP_SUM || s->n_args != 1 || s->args[0] != e_id || !s->keepdim) return -1;
  const dirigo_op_desc* z = hl_op(g, e->args[0]);
  if (!z || z->kind != DIRIGO_OP_SUB || z->n_args != 2 || !default_axes(*z)) return -1;
  const int x = z->args[0];
  const dirigo_op_desc* m = hl_op(g, z->args[1]);
  if (!m || m->kind != DIRIGO_OP_MAX || m->n_args != 1 || m->args[0] != x || !m->keepdim)
    return -1;
  if (x < 0 || x >= (int)shapes.size()) return -1;
  // the same reduction dim (negative dims counted from the end of x's rank)
  const int rank = (int)shapes[x].size();
  const int dm = m->dim < 0 ? m->dim + rank : m->dim, ds = s->dim < 0 ? s->dim + rank : s->dim;
  if (dm != ds || dm < 0 || dm >= rank) return -1;
  *dim_out = dm;
  return x;
}

}  // namespace

dirigo_status compile_graph(const dirigo_graph_desc* desc, const dirigo_options* opt,
                            dirigo_graph* g) {
  Builder b(g);
  Prog& P = g->prog;
  std::memset(&P, 0, sizeof(P));
  if (!desc || desc->n_inputs <= 0 || !desc->inputs || desc->n_ops < 0 ||
      (desc->n_ops > 0 && !desc->ops))
    return set_error(DIRIGO_E_INVALID, "graph description is incomplete");
  P.axiom_gelu = (opt && (opt->flags & DIRIGO_AXIOM_GELU)) ? 1 : 0;
  std::vector<int> hl2t;
  int64_t gbase = 0;
  for (int i = 0; i < desc->n_inputs; ++i) {
    const dirigo_tensor_desc& td = desc->inputs[i];
    if (td.rank < 0 || td.rank > MR) return set_error(DIRIGO_E_UNSUPPORTED, "input rank above 4");
    int32_t shape[MR];
    std::vector<int64_t> sh;
    for (int d = 0; d < td.rank; ++d) {
      if (td.shape[d] <= 0 || td.shape[d] > INT32_MAX)
        return set_error(DIRIGO_E_SHAPE, "bad input shape");
      shape[d] = (int32_t)td.shape[d];
      sh.push_back(td.shape[d]);
    }
    g->in_shapes.push_back(sh);
    g->hl_shapes.push_back(sh);
    int id = b.new_tensor(K_INPUT, 0, 0, nullptr, td.rank, shape);
    if (id < 0) return set_error(b.st, b.err);
    P.t[id].gbase = gbase;
    gbase += P.t[id].numel;
    hl2t.push_back(id);
  }
  P.n_inputs = desc->n_inputs;
  P.G = gbase;
  if (gbase + 1 >= (int64_t)UINT32_MAX) return set_error(DIRIGO_E_UNSUPPORTED, "more than 2^32-2 input elements");
  for (int k = 0; k < desc->n_ops; ++k) {
    int t, sdim = 0;
    const int sx = match_softmax_shift(desc, k, g->hl_shapes, &sdim);
    if (sx >= 0) {
      // sound identity: a max-shifted softmax written out is the softmax
      dirigo_op_desc sm;
      std::memset(&sm, 0, sizeof(sm));
      sm.kind = DIRIGO_OP_SOFTMAX;
      sm.n_args = 1;
      sm.args[0] = sx;
      sm.dim = sdim;
      t = b.lower(sm, hl2t);
    } else {
      t = b.lower(desc->ops[k], hl2t);
    }
    if (t < 0) return set_error(b.st == DIRIGO_OK ? DIRIGO_E_INVALID : b.st, b.err + " (op " + std::to_string(k) + ")");
    hl2t.push_back(t);
    const Tensor& ht = P.t[t];
    g->hl_shapes.emplace_back(ht.shape, ht.shape + ht.rank);
  }
  if (desc->output < 0 || desc->output >= (int)hl2t.size())
    return set_error(DIRIGO_E_INVALID, "output is not a tensor of the graph");
  P.output = hl2t[desc->output];
  if (P.output < P.n_inputs) return set_error(DIRIGO_E_INVALID, "output must be computed by an op");
  // kernels whose output locations are the graph output's: walk back from the
  // output through elementwise ops whose operand has the op's own shape
  {
    const int I = desc->n_inputs;
    std::vector<char> aligned(hl2t.size(), 0);
    aligned[desc->output] = 1;
    for (int k = desc->n_ops - 1; k >= 0; --k) {
      const dirigo_op_desc& op = desc->ops[k];
      if (!aligned[I + k]) continue;
      bool elementwise = false;
      switch (op.kind) {
        case DIRIGO_OP_ADD: case DIRIGO_OP_SUB: case DIRIGO_OP_MUL: case DIRIGO_OP_DIV:
          elementwise = default_axes(op);
          break;
        case DIRIGO_OP_SCALE: case DIRIGO_OP_ADD_SCALAR: case DIRIGO_OP_CLAMP_MIN:
        case DIRIGO_OP_RELU: case DIRIGO_OP_GELU: case DIRIGO_OP_GELU_TANH: case DIRIGO_OP_TANH:
        case DIRIGO_OP_EXP: case DIRIGO_OP_RSQRT: case DIRIGO_OP_RECIP: case DIRIGO_OP_SIGMOID:
        case DIRIGO_OP_ERF: case DIRIGO_OP_SQRT: case DIRIGO_OP_LOG:
          elementwise = true;
          break;
        default:
          break;
      }
      if (!elementwise) continue;
      for (int i = 0; i < op.n_args; ++i)
        if (g->hl_shapes[op.args[i]] == g->hl_shapes[I + k]) aligned[op.args[i]] = 1;
    }
    for (int k = 0; k < desc->n_ops; ++k) {
      const dirigo_op_desc& op = desc->ops[k];
      if ((op.kind == DIRIGO_OP_KERNEL_CONTRACT || op.kind == DIRIGO_OP_KERNEL_MAXSET) &&
          aligned[I + k])
        g->kernel_corners.push_back(kernel_corner_locations(op));
    }
  }
  // value layout of the primitive tensors (one array per tensor)
  int64_t off = 0;
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    P.t[t].ws_off = off;
    off += (P.t[t].numel + 63) / 64 * 64;
    if (P.t[t].kind == K_MAXSET && P.t[t].max_terms > 4096)
      return set_error(DIRIGO_E_UNSUPPORTED, "max over more than 4096 terms per element");
    if (P.t[t].numel >= ((int64_t)1 << 40)) return set_error(DIRIGO_E_UNSUPPORTED, "tensor too large");
  }
  g->value_elems = off;
  const Tensor& out = P.t[P.output];
  g->out_numel = out.numel;
  g->out_rank = out.rank;
  for (int d = 0; d < DIRIGO_MAX_RANK; ++d) g->out_shape[d] = d < out.rank ? out.shape[d] : 0;
  // image templates of every contraction/max access
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    const Tensor& T = P.t[t];
    if (T.kind != K_CONTRACT && T.kind != K_MAXSET) continue;
    for (int q = 0; q < T.npieces; ++q)
      for (int i = 0; i < T.nargs; ++i) build_template(P, T, P.p[T.piece0 + q], i);
  }
  // GEMM view of two-operand contractions: a dim read by operand 0 only is a
  // row dim, by operand 1 only a column dim, by both a batch dim
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    Tensor& T = P.t[t];
    if (!(T.flags & TF_GEMM)) continue;
    for (int d = 0; d < T.rank; ++d) {
      bool ua = false, ub = false;
      for (int q = 0; q < T.npieces; ++q) {
        const Piece& pc = P.p[T.piece0 + q];
        ua |= pc.acc[0].os[d] != 0;
        ub |= pc.acc[1].os[d] != 0;
        for (int j = 0; j < pc.nguard; ++j)
          if (pc.g[j].od == d) ua = true;   // guards are tested on the row side
      }
      if (ua && ub) T.batch_mask |= 1 << d;
      else if (ub) T.col_mask |= 1 << d;
      else T.row_mask |= 1 << d;
    }
  }
  // a contraction whose only reader adds a broadcast operand to it (a bias):
  // the contraction's epilogue writes the sum's keys (its own are not needed)
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    Tensor& T = P.t[t];
    if (!(T.flags & TF_GEMM) || t == P.output) continue;
    int consumer = -1, uses = 0;
    for (int u = t + 1; u < P.n_tensors; ++u)
      for (int a = 0; a < P.t[u].nargs; ++a)
        if (P.t[u].args[a] == t) {
          consumer = u;
          ++uses;
        }
    if (uses != 1) continue;
    Tensor& U = P.t[consumer];
    // the added operand must be ready when the contraction runs
    if (U.kind != K_BINARY || U.fn != B_ADD || U.args[0] != t || U.args[1] >= t ||
        U.rank != T.rank || U.arg_rank[0] != T.rank)
      continue;
    bool same = true;
    for (int d = 0; d < T.rank; ++d) same &= U.shape[d] == T.shape[d] && U.axes[0][d] == d;
    if (!same) continue;
    T.fused = consumer;
    U.flags |= TF_BY_GEMM;
  }
  // a max-set or a (non-tiled) sum whose only reader is a UNARY: its kernel
  // writes the UNARY's keys (the UF key of each element) directly
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    Tensor& T = P.t[t];
    if (t == P.output || (T.kind != K_MAXSET && !(T.kind == K_CONTRACT && !(T.flags & TF_GEMM))))
      continue;
    int consumer = -1, uses = 0;
    for (int u = t + 1; u < P.n_tensors; ++u)
      for (int a = 0; a < P.t[u].nargs; ++a)
        if (P.t[u].args[a] == t) {
          consumer = u;
          ++uses;
        }
    if (uses != 1 || P.t[consumer].kind != K_UNARY || P.t[consumer].numel != T.numel) continue;
    T.unary_next = consumer;
    P.t[consumer].flags |= TF_BY_PRODUCER;
  }
  // cone cells of the output (cells off when the partition is too fine)
  if (build_cells(P, g->cells)) {
    const CellRec* rec = reinterpret_cast<const CellRec*>(g->cells.data() + P.cell_rec_off);
    for (int i = 0; i < P.n_cells; ++i) g->n_generic_cells += rec[i].nseg == kCellGeneric;
  }
  return DIRIGO_OK;
}

}  // namespace dirigo
