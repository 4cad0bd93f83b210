// Compiled program: the per-element equations of every primitive tensor of
// one op graph, in the form the kernels read (library-internal).
//
// Every op is lowered to primitive tensors of six kinds (Sec. 3.4, "Per-element
// equations": T_k[l] = f_k(l) over elements of earlier tensors):
//   CONTRACT  T[o] = sum_{pieces p containing o} sum_{r in R_p, guards} coef_p * prod_i arg_i[acc_{p,i}(o, r)]
//   MAXSET    T[o] = Max{ arg[acc_p(o, r)] }   (same enumeration; an unordered set)
//   UNARY     T[o] = f(arg[o])                  (f an uninterpreted function)
//   MAXC      T[o] = Max{ arg[o], c }
//   AFFINE    T[o] = a * arg[o] + c
//   BINARY    T[o] = arg0[.] op arg1[.]         (broadcast through axes)
// An access offset outside its operand reads the undefined value bottom.
//
// The whole program is passed to kernels by value as a __grid_constant__
// parameter (it lives in the constant bank, and every thread of a warp reads
// the same fields, so the reads are broadcasts).
#pragma once
#include <cstdint>

namespace dirigo {

constexpr int MR = 4;     // max tensor rank
constexpr int MRED = 4;   // max reduction dims of a piece
constexpr int MG = 4;     // max guards of a piece
constexpr int MT = 40;    // max tensors (inputs + primitive)
constexpr int MP = 24;    // max pieces of a program

// Key field: two primes just below 2^29 (p = 2^29 - c).
constexpr uint32_t kP0 = 536870909u;   // 2^29 - 3
constexpr uint32_t kP1 = 536870879u;   // 2^29 - 33

enum PKind : int8_t { K_INPUT = 0, K_CONTRACT = 1, K_MAXSET = 2, K_UNARY = 3, K_MAXC = 4,
                      K_AFFINE = 5, K_BINARY = 6 };
enum Fn : int8_t { F_EXP = 1, F_TANH = 2, F_GELU_ERF = 3, F_GELU_TANH = 4, F_ERF = 5,
                   F_RSQRT = 6, F_RECIP = 7, F_SQRT = 8, F_LOG = 9 };
enum Bin : int8_t { B_ADD = 1, B_SUB = 2, B_MUL = 3, B_DIV = 4 };

// A constant: its key in both lanes and its fp32 value.
struct KConst {
  uint32_t k0, k1;
  float f;
  int32_t is_zero;
  double d;     // exact double when the constant is dyadic (exported coefficients)
};

// lo <= oa * o[od] + r[rd] + c < hi   (od / rd = -1: absent)
struct Guard {
  int32_t od, rd, oa, c, lo, hi;
};

// flat offset = base + sum_d os[d] * o[d] + sum_e rs[e] * r[e]
struct Access {
  int64_t base;
  int64_t os[MR];
  int64_t rs[MRED];
};

// Image template of one operand access of a piece (location-independent,
// built by the compiler): the offset is base + sum over slots of step * v,
// where v ranges over an interval the cone kernel computes per location.
// Slots are sorted by step; each is tied to one natural dim of the operand
// (dim `nd`, multiplier `q`) when the access reads a box of the operand.
enum SlotKind : int8_t {
  SL_O = 1,     // v = o[ref]                  (output dim in no two-sided guard)
  SL_R = 2,     // v = r[ref]                  (reduction dim in no two-sided guard)
  SL_V = 3,     // v = oa * o + r of guard ref (the offset reads the guarded sum)
  SL_GR = 4,    // v = r of guard ref          (projection onto the reduction dim)
  SL_GO = 5,    // v = o of guard ref          (projection onto the output dim)
};
struct Slot {
  int8_t kind, ref, nd, pad;
  int32_t q;
  int64_t step;
};
constexpr int MSLOT = MR + MRED;
struct AccTpl {
  int8_t nslot;
  int8_t natural;       // every slot maps to a natural dim with q > 0
  int8_t unsupported;   // the access couples an output and a reduction dim otherwise
  int8_t pad;
  int32_t cbase[MR];    // base offset split over the natural dims (truncating)
  Slot s[MSLOT];
};

struct Piece {
  int32_t lo[MR], hi[MR];       // output box the piece applies to
  int32_t rlo[MRED], rhi[MRED]; // reduction box
  int32_t nred, nguard;
  KConst coef;
  Guard g[MG];
  Access acc[2];
  AccTpl tpl[2];
};

enum TFlags : int32_t {
  TF_GEMM = 1,      // CONTRACT with two operands that the tiled kernel handles
  TF_BY_GEMM = 2,   // BINARY add whose keys the epilogue of its operand 0's contraction writes
  TF_BY_PRODUCER = 4,   // UNARY whose keys its operand's (max-set / sum) kernel writes
};

struct Tensor {
  int8_t kind, fn, nargs, rank;
  int16_t piece0, npieces;
  int32_t args[2];
  int32_t shape[MR];
  int64_t stride[MR];   // row-major strides
  int64_t numel;
  int64_t gbase;        // inputs: global id of element 0
  int64_t ws_off;       // element offset of the value array in a call's value area
  KConst a, c;          // AFFINE: a, c; MAXC: c
  int8_t axes[2][MR];   // BINARY: output dim of each operand dim
  int8_t arg_rank[2];
  int32_t flags;
  int32_t max_terms;    // bound on terms of one element (CONTRACT/MAXSET)
  // GEMM view (TF_GEMM): output dims split into row (arg0 only), col (arg1
  // only) and batch (both) dims; bit d of *_mask set when dim d is in that set
  int32_t row_mask, col_mask, batch_mask;
  // TF_GEMM: the BINARY add (t + broadcast operand) that is this tensor's only
  // reader; its keys are written by this contraction's epilogue (0: none)
  int32_t fused;
  // MAXSET / non-tiled CONTRACT: the UNARY that is this tensor's only reader;
  // the kernel writes that UNARY's keys (its own are not needed; 0: none)
  int32_t unary_next;
};

struct Prog {
  int32_t n_tensors, n_inputs, output, n_pieces;
  int64_t G;            // number of global input ids; G is bottom
  int32_t axiom_gelu;
  int32_t pad_;
  // cone cells of the output (see cells.h): cell id = sum_d idx_d[o_d] *
  // cell_radix[d], idx_d read at entry cell_tab[d] of the blob's uint16 table
  int32_t cell_on, n_cells;
  int32_t cell_tab[MR], cell_radix[MR];
  int64_t cell_rec_off, cell_seg_off, cell_bw_off, cell_bytes;
  Tensor t[MT];
  Piece p[MP];
};

}  // namespace dirigo
