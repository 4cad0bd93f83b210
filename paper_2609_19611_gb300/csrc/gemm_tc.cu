// Two-operand CONTRACT keys on the tensor cores.
//
// The key of an output element is sum_k a_k * b_k mod p (a, b < 2^29: the
// keys of the operands).  Each key is split into four signed 8-bit limbs,
// a = sum_i a_i 256^i with a_i in [-128, 128), which bf16 holds exactly.  Then
//   sum_k a_k b_k = sum_{i,j} 256^(i+j) * (sum_k a_{k,i} b_{k,j}),
// and every inner sum is an integer of magnitude <= K * 2^14, exact in fp32
// for K <= 1024 (longer reductions are flushed every 1024 steps).
//
// Per contraction and key lane S:
//   tc_limb_image   (convolution pieces) writes the row side once as a padded
//                   channel-last limb image [N][H+kh-1][W+kw-1][4][Cpad], read
//                   at each window offset by TMA (no im2col);
//   tc_materialize  (other pieces, and every column side) gathers the
//                   operands through the piece's access map (guards and piece
//                   boxes masked to zero, out-of-range reads to the key of
//                   bottom) into dense limb matrices A'[(r, i), k] and
//                   B'[(c, j), k] in bf16, four limb rows per operand row;
//   tc5_gemm        C'[(r,i), (c,j)] = A' B'^T on the tcgen05 tensor cores:
//                   TMA loads into an mbarrier ring, one thread issues the
//                   MMAs into TMEM accumulators, epilogue warps read them back,
//                   round each C' value and combine sum_{i,j} 256^(i+j) C'
//                   mod p, times the piece coefficient (a fused bias add
//                   included).
// tc_gemm is the same product with cp.async-staged tiles, ldmatrix and
// mma.sync m16n8k16 (selected with DIRIGO_TC=mma; it reads materialised
// matrices only).
// Rows are the output dims read by operand 0 only, columns those read by
// operand 1 only, batch the dims read by both (grid z).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <string>
#include <type_traits>

#include "dev.cuh"
#include "fastdiv.h"
#include "internal.h"
#include "launch.h"

namespace dirigo {

namespace {

constexpr int TO = 32;          // outputs per CTA along rows and along columns
constexpr int TK = 32;          // reduction steps per pipeline stage (mma.sync path)
constexpr int KPAD = 64;        // reduction padding of the limb matrices (one TMA box)
constexpr int LDR = 40;         // padded smem row (bf16): conflict-free ldmatrix
constexpr int LR = TO * 4;      // limb rows of a tile (128)
constexpr int KBLK = 1024;      // reduction steps between exact flushes
constexpr int NTHR = 256;
constexpr int NSTAGE = 3;

struct GemmSmem {
  union {
    struct {
      uint16_t A[NSTAGE][LR][LDR];
      uint16_t B[NSTAGE][LR][LDR];
    } ab;
    float C[LR][LR + 4];
  } u;
  int32_t orow[TO][MR], ocol[TO][MR];
};

struct Split {
  int nd;
  int dims[MR];
  int64_t count;
};

__host__ __device__ __forceinline__ Split split_of(const Tensor& T, int mask) {
  Split s;
  s.nd = 0;
  s.count = 1;
  for (int d = 0; d < T.rank; ++d)
    if (mask & (1 << d)) {
      s.dims[s.nd++] = d;
      s.count *= T.shape[d];
    }
  return s;
}

__device__ __forceinline__ void split_coords(const Tensor& T, const Split& s, int64_t x,
                                             int32_t* o) {
#pragma unroll
  for (int i = MR - 1; i >= 0; --i) {
    if (i < s.nd) {
      const int d = s.dims[i];
      int64_t q, r;
      divmod64(x, T.shape[d], q, r);
      set4(o, d, (int32_t)r);
      x = q;
    }
  }
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Geometry of one contraction's limb matrices (host and device agree).
struct TcGeom {
  int64_t rows, cols, batch;       // outputs
  int64_t rpad, cpad;              // padded to TO
  int64_t kp[MP];                  // padded reduction length of each piece
  int64_t offA[MP], offB[MP];      // element offsets (bf16) of each piece's matrices, lane 0
  int64_t lane_stride;             // bf16 elements per lane
  // rows [r0, r1) and columns [c0, c1) that hold every output of the piece
  // (flattened over the row / column dims); tiles outside add nothing
  int64_t r0[MP], r1[MP], c0[MP], c1[MP];
  int32_t a_src[MP];               // piece whose row-side matrix this piece reads
  Split rsp, csp, bsp;             // row, column and batch dims of the output
  // Convolution pieces (stride 1, padding by the image bounds, output width a
  // multiple of TO): the row side is a padded channel-last limb image
  // [N][Hp][Wp][4 limbs][Cpad] read by TMA at the window offset, and the
  // reduction runs in (kh, kw, channel) order with channels padded to Cpad.
  // fused bias add (Tensor::fused): the sum's value offset, the added
  // operand's key array and stride per output dim; brow: the operand depends
  // on a row or batch dim (filled at launch)
  int64_t out_ws_off;
  const uint2* bsrc;
  int64_t bos[MR];
  int32_t brow;
  int32_t conv[MP];
  int32_t cv_C[MP], cv_Cpad[MP], cv_KH[MP], cv_KW[MP], cv_H[MP], cv_W[MP];
  int32_t cv_Hp[MP], cv_Wp[MP], cv_ph[MP], cv_pw[MP], cv_Ho[MP], cv_Wo[MP], cv_N[MP];
  // division by a multiply: q = umulhi(x, fd_m) >> fd_s for x < 2^31 (fd_m = 0:
  // the divisor is 1), for the column-tile count [0], the row-tile count [1]
  // and the extents of the row split's dims [2 + i]; fd_ok when every
  // dividend stays below 2^31 (filled at launch)
  uint32_t fd_m[2 + MR], fd_s[2 + MR];
  int32_t fd_ok;
};

// Whether piece pc of T reads its row side as a stride-1 convolution window
// whose taps outside the image are exactly the ones its guards drop.
__host__ __device__ inline bool conv_piece(const Prog& P, const Tensor& T, const Piece& pc) {
  const Tensor& X = P.t[T.args[0]];
  if (T.rank != 4 || X.rank != 4 || pc.nred != 3 || pc.nguard != 2) return false;
  if (T.row_mask != 0b1101 || T.col_mask != 0b0010 || T.batch_mask != 0) return false;
  const int64_t C = X.shape[1], H = X.shape[2], W = X.shape[3];
  if (pc.rlo[0] != 0 || pc.rlo[1] != 0 || pc.rlo[2] != 0 || pc.rhi[0] != C) return false;
  const Access& a = pc.acc[0];
  if (a.os[0] != C * H * W || a.os[1] != 0 || a.os[2] != W || a.os[3] != 1) return false;
  if (a.rs[0] != H * W || a.rs[1] != W || a.rs[2] != 1) return false;
  int gh = pc.g[0].od == 2 ? 0 : 1, gw = 1 - gh;
  const Guard &h = pc.g[gh], &w = pc.g[gw];
  if (h.od != 2 || h.rd != 1 || h.oa != 1 || h.lo != 0 || h.hi != H) return false;
  if (w.od != 3 || w.rd != 2 || w.oa != 1 || w.lo != 0 || w.hi != W) return false;
  if (a.base != (int64_t)h.c * W + w.c) return false;
  for (int d = 0; d < 4; ++d)
    if (d != 1 && (pc.lo[d] != 0 || pc.hi[d] != T.shape[d])) return false;
  return T.shape[0] == X.shape[0] && T.shape[3] % TO == 0;
}

// sum over the dims of s of w[d] * coordinate, for flat index x over them
__device__ __forceinline__ int64_t split_offset_w(const Tensor& T, const Split& s, int64_t x,
                                                  const int64_t* w) {
  if (s.nd == 1) {   // x is the coordinate itself
    int64_t v = 0;
#pragma unroll
    for (int y = 0; y < MR; ++y)
      if (y == s.dims[0]) v = w[y] * x;
    return v;
  }
  int64_t off = 0;
#pragma unroll
  for (int i = MR - 1; i >= 0; --i) {
    if (i < s.nd) {
      const int d = s.dims[i];
      int64_t q, r;
      divmod64(x, (int64_t)T.shape[d], q, r);
#pragma unroll
      for (int y = 0; y < MR; ++y)
        if (y == d) off += w[y] * r;
      x = q;
    }
  }
  return off;
}

// sum over the dims of s of stride * coordinate, for flat index x over them
__device__ __forceinline__ int64_t split_offset(const Tensor& T, const Split& s, int64_t x) {
  if (s.nd == 1) return T.stride[s.dims[0]] * x;   // x is the coordinate itself
  int64_t off = 0;
#pragma unroll
  for (int i = MR - 1; i >= 0; --i) {
    if (i < s.nd) {
      const int d = s.dims[i];
      int64_t q, r;
      divmod64(x, (int64_t)T.shape[d], q, r);
      off += T.stride[d] * r;
      x = q;
    }
  }
  return off;
}

// Range of flattened indices over the dims of `s` that cover the piece's box.
__host__ __device__ inline void split_range(const Tensor& T, const Split& s, const Piece& pc,
                                            int64_t& lo, int64_t& hi) {
  int64_t a = 0, b = 0;
  for (int i = 0; i < s.nd; ++i) {
    const int d = s.dims[i];
    const int64_t l = pc.lo[d] > 0 ? pc.lo[d] : 0, h = pc.hi[d] < T.shape[d] ? pc.hi[d] : T.shape[d];
    if (l >= h) {
      lo = hi = 0;
      return;
    }
    a = a * T.shape[d] + l;
    b = b * T.shape[d] + (h - 1);
  }
  lo = a;
  hi = b + 1;
}

// Whether piece q can have outputs in row tile tr, column tile tc (tiles of
// TO rows and wc columns of outputs).
__host__ __device__ inline bool piece_hits(const TcGeom& g, int q, int64_t tr, int64_t tc,
                                           int64_t wc = TO) {
  return g.r0[q] < (tr + 1) * TO && tr * TO < g.r1[q] && g.c0[q] < (tc + 1) * wc &&
         tc * wc < g.c1[q];
}

// Two pieces read the same row-side matrix when their row-side access,
// reduction box, guards and row/batch ranges agree.
__host__ __device__ inline bool same_row_side(const Tensor& T, const Piece& a, const Piece& b) {
  if (a.nred != b.nred || a.nguard != b.nguard) return false;
  if (a.acc[0].base != b.acc[0].base) return false;
  for (int d = 0; d < MR; ++d)
    if (a.acc[0].os[d] != b.acc[0].os[d]) return false;
  for (int e = 0; e < MRED; ++e)
    if (a.acc[0].rs[e] != b.acc[0].rs[e] || a.rlo[e] != b.rlo[e] || a.rhi[e] != b.rhi[e])
      return false;
  for (int j = 0; j < a.nguard; ++j) {
    const Guard &x = a.g[j], &y = b.g[j];
    if (x.od != y.od || x.rd != y.rd || x.oa != y.oa || x.c != y.c || x.lo != y.lo || x.hi != y.hi)
      return false;
  }
  const int m = T.row_mask | T.batch_mask;
  for (int d = 0; d < T.rank; ++d)
    if (((m >> d) & 1) && (a.lo[d] != b.lo[d] || a.hi[d] != b.hi[d])) return false;
  return true;
}

// tc5: the tcgen05 path (convolution pieces read padded limb images)
__host__ __device__ inline TcGeom tc_geom(const Prog& P, const Tensor& T, bool tc5) {
  TcGeom g;
  g.fd_ok = 0;
  Split rs = split_of(T, T.row_mask), cs = split_of(T, T.col_mask), bs = split_of(T, T.batch_mask);
  g.rows = rs.count;
  g.cols = cs.count;
  g.batch = bs.count;
  g.rsp = rs;
  g.csp = cs;
  g.bsp = bs;
  g.rpad = (g.rows + TO - 1) / TO * TO;
  g.cpad = (g.cols + TO - 1) / TO * TO;
  int64_t off = 0;
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    int64_t kv = 1;
    for (int e = 0; e < pc.nred; ++e) kv *= (pc.rhi[e] > pc.rlo[e] ? pc.rhi[e] - pc.rlo[e] : 0);
    g.conv[q] = tc5 && conv_piece(P, T, pc);
    if (g.conv[q]) {
      const Tensor& X = P.t[T.args[0]];
      g.cv_C[q] = X.shape[1];
      g.cv_Cpad[q] = (X.shape[1] + KPAD - 1) / KPAD * KPAD;
      g.cv_KH[q] = pc.rhi[1];
      g.cv_KW[q] = pc.rhi[2];
      g.cv_H[q] = X.shape[2];
      g.cv_W[q] = X.shape[3];
      g.cv_N[q] = T.shape[0];
      g.cv_Ho[q] = T.shape[2];
      g.cv_Wo[q] = T.shape[3];
      g.cv_ph[q] = -pc.g[pc.g[0].od == 2 ? 0 : 1].c;
      g.cv_pw[q] = -pc.g[pc.g[0].od == 2 ? 1 : 0].c;
      g.cv_Hp[q] = g.cv_Ho[q] + g.cv_KH[q] - 1;
      g.cv_Wp[q] = g.cv_Wo[q] + g.cv_KW[q] - 1;
      g.kp[q] = (int64_t)g.cv_KH[q] * g.cv_KW[q] * g.cv_Cpad[q];
    } else {
      g.kp[q] = (kv + KPAD - 1) / KPAD * KPAD;
    }
    split_range(T, rs, pc, g.r0[q], g.r1[q]);
    split_range(T, cs, pc, g.c0[q], g.c1[q]);
    g.a_src[q] = q;
    for (int u = 0; u < q; ++u)
      if (g.a_src[u] == u && g.kp[u] == g.kp[q] && g.conv[u] == g.conv[q] &&
          same_row_side(T, P.p[T.piece0 + u], pc)) {
        g.a_src[q] = u;
        break;
      }
    if (g.a_src[q] == q) {
      g.offA[q] = off;
      off += g.conv[q] ? (int64_t)g.cv_N[q] * g.cv_Hp[q] * g.cv_Wp[q] * 4 * g.cv_Cpad[q]
                       : g.batch * 4 * g.rpad * g.kp[q];
    } else {
      g.offA[q] = g.offA[g.a_src[q]];
    }
    g.offB[q] = off;
    off += g.batch * 4 * g.cpad * g.kp[q];
  }
  g.lane_stride = (off + 127) / 128 * 128;
  return g;
}

}  // namespace

void tc_work(const Prog& P, double* flops_per_lane, double* limb_bytes) {
  double f = 0, b = 0;
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    const Tensor& T = P.t[t];
    if (!(T.flags & TF_GEMM)) continue;
    TcGeom g = tc_geom(P, T, T.npieces <= 4);
    for (int q = 0; q < T.npieces; ++q) {
      const Piece& pc = P.p[T.piece0 + q];
      double kv = 1;
      for (int e = 0; e < pc.nred; ++e) kv *= (pc.rhi[e] > pc.rlo[e] ? pc.rhi[e] - pc.rlo[e] : 0);
      f += 2.0 * 4.0 * (double)(g.r1[q] - g.r0[q]) * 4.0 * (double)(g.c1[q] - g.c0[q]) * kv *
           (double)g.batch;
      // both lanes: row-side matrix (or limb image) unless shared, column-side matrix
      const double arow = g.a_src[q] != q ? 0.0
                          : g.conv[q] ? (double)g.cv_N[q] * g.cv_Hp[q] * g.cv_Wp[q] * 4.0 * g.cv_Cpad[q]
                                      : 4.0 * (double)g.batch * (double)g.rpad * (double)g.kp[q];
      b += 2.0 * 2.0 * (arow + 4.0 * (double)g.batch * (double)g.cpad * (double)g.kp[q]);
    }
  }
  *flops_per_lane = f;
  *limb_bytes = b;
}

size_t tc_ws_bytes(const Prog& P) {
  size_t m = 0;
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    const Tensor& T = P.t[t];
    if (!(T.flags & TF_GEMM)) continue;
    for (int mode = 0; mode < 2; ++mode) {
      TcGeom g = tc_geom(P, T, mode == 1);
      m = std::max(m, (size_t)g.lane_stride * 2 * 2);
    }
  }
  return m;
}

// bf16 limbs of a key (< 2^29): with y = x + 0x808080 the balanced base-256
// digits are byte_i(y) - 128 (i < 3) and y >> 24; each digit becomes a float
// exactly as (2^23 + byte) - bias, whose upper half is its bf16 pattern.
__device__ __forceinline__ void limb_floats(uint32_t x, float* f) {
  const uint32_t y = x + 0x808080u;
  f[0] = __uint_as_float(__byte_perm(y, 0x4B000000u, 0x7550)) - 8388736.0f;
  f[1] = __uint_as_float(__byte_perm(y, 0x4B000000u, 0x7551)) - 8388736.0f;
  f[2] = __uint_as_float(__byte_perm(y, 0x4B000000u, 0x7552)) - 8388736.0f;
  f[3] = __uint_as_float(__byte_perm(y, 0x4B000000u, 0x7553)) - 8388608.0f;
}

// bf16 patterns of a (low half) and b (high half)
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  return __byte_perm(__float_as_uint(a), __float_as_uint(b), 0x7632);
}

constexpr int kMatK = 256;   // reduction steps per materialisation block (large matrices)

// Limb matrices of one piece.  A block covers 32 rows (or columns) x KM
// reduction steps of one batch index: it first tabulates the offset and guard
// parts of its steps and of its lines in shared memory, then each thread
// gathers the keys of one line at 8 steps at a time (offset = line part +
// step part; guards tested on the sums) and writes their limbs, 16 bytes per
// limb row and key lane.  KM = 64 for small matrices (a weight's few hundred
// lines): four times the blocks, each thread one pass of 8 steps, so that the
// gathers' latency is paid once.
template <int KM>
__global__ void __launch_bounds__(256) tc_materialize_kernel(const __grid_constant__ Prog P, int t,
                                                             int q, int b_only,
                                                             const uint2* leafk,
                                                             const uint2* vals, uint16_t* buf,
                                                             TcGeom g) {
  // step tables, index k + k / 8 (the 8 threads of a line read steps 8 apart)
  __shared__ int64_t koff[KM + KM / 8];
  __shared__ int32_t kg[MG][KM + KM / 8];
  __shared__ uint8_t kok[KM + KM / 8];
  __shared__ int64_t loff[32];
  __shared__ int32_t lg[MG][32];
  __shared__ uint8_t lok[32];
  const Tensor& T = P.t[t];
  const Piece& pc = P.p[T.piece0 + q];
  const int tid = threadIdx.x;
  const int64_t nkb = (g.kp[q] + KM - 1) / KM;
  const int64_t lblocks = ((b_only ? 0 : g.rpad) + g.cpad) / 32;
  int64_t bid = blockIdx.x, kbi, lb, b;
  divmod64(bid, nkb, lb, kbi);
  divmod64(lb, lblocks, b, lb);
  if (b_only) lb += g.rpad / 32;
  const bool side_b = lb * 32 >= g.rpad;
  const int64_t line0 = side_b ? lb * 32 - g.rpad : lb * 32;
  const int si = side_b ? 1 : 0;
  const Access& ac = pc.acc[si];
  int64_t kv = 1;
  for (int e = 0; e < pc.nred; ++e) kv *= pc.rhi[e] - pc.rlo[e];
  if (tid < KM) {  // step tables: one step per thread
    int64_t k = kbi * KM + tid;
    bool ok = k < kv;
    int32_t r[MRED] = {0, 0, 0, 0};
    if (g.conv[q]) {   // (kh, kw, channel) order, channels padded to Cpad
      int64_t t2, c, kw, kh;
      divmod64(k, (int64_t)g.cv_Cpad[q], t2, c);
      divmod64(t2, (int64_t)g.cv_KW[q], kh, kw);
      ok = k < g.kp[q] && c < g.cv_C[q];
      if (ok) {
        r[0] = (int32_t)c;
        r[1] = (int32_t)kh;
        r[2] = (int32_t)kw;
      }
    } else {
      int64_t x = ok ? k : 0;
#pragma unroll
      for (int e = MRED - 1; e >= 0; --e) {
        if (e < pc.nred) {
          int64_t qq, rr;
          divmod64(x, (int64_t)(pc.rhi[e] - pc.rlo[e]), qq, rr);
          r[e] = pc.rlo[e] + (int32_t)rr;
          x = qq;
        }
      }
    }
    int64_t o = 0;
#pragma unroll
    for (int e = 0; e < MRED; ++e)
      if (e < pc.nred) o += ac.rs[e] * r[e];
    const int kx = tid + (tid >> 3);
    koff[kx] = o;
    kok[kx] = ok;
#pragma unroll
    for (int j = 0; j < MG; ++j)
      kg[j][kx] = (!side_b && j < pc.nguard && pc.g[j].rd >= 0) ? sel4(r, pc.g[j].rd) : 0;
  }
  if (tid < 32) {  // line tables
    const int li = tid;
    int64_t rc = line0 + li;
    const Split bs = split_of(T, T.batch_mask);
    const Split ss = split_of(T, side_b ? T.col_mask : T.row_mask);
    int32_t o[MR] = {0, 0, 0, 0};
    split_coords(T, bs, b, o);
    bool ok = rc < ss.count;
    if (ok) split_coords(T, ss, rc, o);
    const int mine = T.batch_mask | (side_b ? T.col_mask : T.row_mask);
#pragma unroll
    for (int d = 0; d < MR; ++d)
      if (d < T.rank && ((mine >> d) & 1)) ok &= o[d] >= pc.lo[d] && o[d] < pc.hi[d];
    int64_t off = ac.base;
#pragma unroll
    for (int d = 0; d < MR; ++d)
      if (d < T.rank) off += ac.os[d] * o[d];
    loff[li] = off;
    lok[li] = ok;
#pragma unroll
    for (int j = 0; j < MG; ++j) {
      int32_t v = 0;
      if (!side_b && j < pc.nguard) {
        v = pc.g[j].c;
        if (pc.g[j].od >= 0) v += pc.g[j].oa * sel4(o, pc.g[j].od);
      }
      lg[j][li] = v;
    }
  }
  __syncthreads();
  // 8 threads per line: a warp's stores fill 128-byte segments of 4 lines'
  // limb rows
  const int li = tid >> 3;
  const int arg = T.args[si];
  const int ng = side_b ? 0 : pc.nguard;
  // operand keys: every load is issued (in-range index or element 0), bottom
  // and absent terms are selected afterwards, so the 8 gathers overlap
  const Tensor& A = P.t[arg];
  const uint2* src = A.kind == K_INPUT ? leafk + A.gbase : vals + A.ws_off;
  const int64_t numel = A.numel;
  const uint2 bot = leafk[P.G];
  const bool lin = lok[li];
  const int64_t lo_off = loff[li];
  int32_t lgv[MG];
#pragma unroll
  for (int j = 0; j < MG; ++j) lgv[j] = lg[j][li];
  const int64_t nlines = side_b ? g.cpad : g.rpad;
  const int64_t rowbase = (side_b ? g.offB[q] : g.offA[q]) + b * 4 * nlines * g.kp[q] +
                          4 * (line0 + li) * g.kp[q];
  const int nk = (int)min((int64_t)KM, g.kp[q] - kbi * KM);
  for (int k0 = (tid & 7) * 8; k0 < nk; k0 += 64) {
    uint32_t w0[4][4], w1[4][4];   // [limb][pair of steps], per key lane
#pragma unroll
    for (int u = 0; u < 8; u += 2) {
      float fa[2][4], fb[2][4];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int k = k0 + u + h, kx = k + (k >> 3);
        bool ok = lin && kok[kx];
#pragma unroll
        for (int j = 0; j < MG; ++j) {
          if (j >= ng) continue;
          int32_t v = lgv[j] + kg[j][kx];
          ok &= v >= pc.g[j].lo && v < pc.g[j].hi;
        }
        const int64_t idx = lo_off + koff[kx];
        const bool inr = idx >= 0 && idx < numel;
        const uint2 v = __ldg(src + (inr ? idx : 0));
        const uint2 key = ok ? (inr ? v : bot) : make_uint2(0, 0);
        limb_floats(key.x, fa[h]);
        limb_floats(key.y, fb[h]);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        w0[i][u >> 1] = pack_bf16(fa[0][i], fa[1][i]);
        w1[i][u >> 1] = pack_bf16(fb[0][i], fb[1][i]);
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t e0 = rowbase + i * g.kp[q] + kbi * KM + k0;
      *reinterpret_cast<uint4*>(buf + e0) = make_uint4(w0[i][0], w0[i][1], w0[i][2], w0[i][3]);
      *reinterpret_cast<uint4*>(buf + g.lane_stride + e0) =
          make_uint4(w1[i][0], w1[i][1], w1[i][2], w1[i][3]);
    }
  }
}

// Padded channel-last limb image of a convolution piece's row-side operand
// X[N, C, H, W]: image[n][hp][wp][i][c] = limb i of the key of
// X[n, c, hp - ph, wp - pw] inside the image, 0 outside it and for c >= C.
// One thread per (pixel, 8 channels), the channel group fastest: the threads
// of a pixel write each limb row's 128 bytes side by side (whole lines), and
// for each channel a warp reads the keys of consecutive pixels (32-byte
// segments).  An input's keys are formed from its global ids, not loaded.
__global__ void __launch_bounds__(256) tc_limb_image_kernel(const __grid_constant__ Prog P, int t,
                                                            int q, const uint2* leafk,
                                                            const uint2* vals, uint16_t* buf,
                                                            TcGeom g) {
  const Tensor& T = P.t[t];
  const Tensor& X = P.t[T.args[0]];
  const int64_t Cp = g.cv_Cpad[q], C = g.cv_C[q], H = g.cv_H[q], W = g.cv_W[q];
  const int64_t Hp = g.cv_Hp[q], Wp = g.cv_Wp[q], nch = Cp / 8;
  const int64_t id = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (id >= (int64_t)g.cv_N[q] * Hp * Wp * nch) return;
  int64_t wp, hp, cc, n, rest;
  divmod64(id, nch, rest, cc);
  divmod64(rest, Wp, rest, wp);
  divmod64(rest, Hp, n, hp);
  const int64_t h = hp - g.cv_ph[q], w = wp - g.cv_pw[q];
  const bool in = h >= 0 && h < H && w >= 0 && w < W;
  const uint2* src = X.kind == K_INPUT ? leafk + X.gbase : vals + X.ws_off;
  uint32_t w0[4][4], w1[4][4];
#pragma unroll
  for (int j = 0; j < 8; j += 2) {
    float fa[2][4], fb[2][4];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int64_t c = cc * 8 + j + u;
      const bool ok = in && c < C;
      const int64_t off = ((n * C + c) * H + h) * W + w;
      uint2 key = make_uint2(0, 0);
      if (ok) {
        if (X.kind == K_INPUT)
          key = make_uint2(leaf_key0((uint64_t)(X.gbase + off)), leaf_key1((uint64_t)(X.gbase + off)));
        else
          key = __ldg(src + off);
      }
      limb_floats(key.x, fa[u]);
      limb_floats(key.y, fb[u]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      w0[i][j >> 1] = pack_bf16(fa[0][i], fa[1][i]);
      w1[i][j >> 1] = pack_bf16(fb[0][i], fb[1][i]);
    }
  }
  const int64_t base = g.offA[q] + ((n * Hp + hp) * Wp + wp) * 4 * Cp + cc * 8;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    *reinterpret_cast<uint4*>(buf + base + i * Cp) =
        make_uint4(w0[i][0], w0[i][1], w0[i][2], w0[i][3]);
    *reinterpret_cast<uint4*>(buf + g.lane_stride + base + i * Cp) =
        make_uint4(w1[i][0], w1[i][1], w1[i][2], w1[i][3]);
  }
}

template <int S>
__global__ void __launch_bounds__(NTHR, 2) tc_gemm_kernel(const __grid_constant__ Prog P, int t,
                                                          const uint16_t* buf, TcGeom g,
                                                          const uint2* leafk, uint2* vals) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GemmSmem& sm = *reinterpret_cast<GemmSmem*>(smem_raw);
  const Tensor& T = P.t[t];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wm = warp & 3, wn = warp >> 2;   // warp tile: 32 limb rows x 64 limb columns
  const int64_t col0 = (int64_t)blockIdx.x * TO, row0 = (int64_t)blockIdx.y * TO;
  const int64_t bz = blockIdx.z;
  const Split rs = split_of(T, T.row_mask), cs = split_of(T, T.col_mask),
              bs = split_of(T, T.batch_mask);
  int32_t ob[MR] = {0, 0, 0, 0};
  split_coords(T, bs, bz, ob);
  if (tid < TO) {
    int32_t o[MR];
    for (int d = 0; d < MR; ++d) o[d] = ob[d];
    if (row0 + tid < rs.count) split_coords(T, rs, row0 + tid, o);
    for (int d = 0; d < MR; ++d) sm.orow[tid][d] = o[d];
  } else if (tid >= 64 && tid < 64 + TO) {
    int c = tid - 64;
    int32_t o[MR];
    for (int d = 0; d < MR; ++d) o[d] = ob[d];
    if (col0 + c < cs.count) split_coords(T, cs, col0 + c, o);
    for (int d = 0; d < MR; ++d) sm.ocol[c][d] = o[d];
  }
  uint32_t w256[7];
  w256[0] = 1;
#pragma unroll
  for (int k = 1; k < 7; ++k) w256[k] = mulmod<S>(w256[k - 1], 256u);
  uint32_t tot[4] = {0, 0, 0, 0};
  const uint16_t* lanebuf = buf + (S ? g.lane_stride : 0);

  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    const int64_t kp = g.kp[q];
    if (kp == 0) continue;
    const uint16_t* Ag = lanebuf + g.offA[q] + (bz * 4 * g.rpad + 4 * row0) * kp;
    const uint16_t* Bg = lanebuf + g.offB[q] + (bz * 4 * g.cpad + 4 * col0) * kp;
    for (int64_t kb0 = 0; kb0 < kp; kb0 += KBLK) {
      const int nchunk = (int)(((kb0 + KBLK < kp ? kb0 + KBLK : kp) - kb0) / TK);
      float acc[2][8][4];
#pragma unroll
      for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int b = 0; b < 8; ++b)
#pragma unroll
          for (int r = 0; r < 4; ++r) acc[a][b][r] = 0.0f;
      // each stage: 128 rows x 64 bytes of A and of B = 512 + 512 chunks of 16 B
      auto load = [&](int c, int st) {
        const int64_t k = kb0 + (int64_t)c * TK;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          int ch = tid + NTHR * h;
          int row = ch >> 2, part = ch & 3;
          cp_async16(smem_u32(&sm.u.ab.A[st][row][part * 8]), Ag + row * kp + k + part * 8);
          cp_async16(smem_u32(&sm.u.ab.B[st][row][part * 8]), Bg + row * kp + k + part * 8);
        }
      };
      __syncthreads();
#pragma unroll
      for (int st = 0; st < NSTAGE - 1; ++st) {
        if (st < nchunk) load(st, st);
        cp_async_commit();
      }
      for (int c = 0; c < nchunk; ++c) {
        cp_async_wait<NSTAGE - 2>();
        __syncthreads();
        if (c + NSTAGE - 1 < nchunk) load(c + NSTAGE - 1, (c + NSTAGE - 1) % NSTAGE);
        cp_async_commit();
        const int st = c % NSTAGE;
#pragma unroll
        for (int ks = 0; ks < TK; ks += 16) {
          uint32_t af[2][4], bfr[8][2];
#pragma unroll
          for (int a = 0; a < 2; ++a) {
            int row = wm * 32 + a * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
            int col = ks + 8 * (lane >> 4);
            ldsm_x4(smem_u32(&sm.u.ab.A[st][row][col]), af[a][0], af[a][1], af[a][2], af[a][3]);
          }
#pragma unroll
          for (int b = 0; b < 4; ++b) {
            int row = wn * 64 + b * 16 + (lane & 7) + 8 * (lane >> 4);
            int col = ks + 8 * ((lane >> 3) & 1);
            ldsm_x4(smem_u32(&sm.u.ab.B[st][row][col]), bfr[2 * b][0], bfr[2 * b][1],
                    bfr[2 * b + 1][0], bfr[2 * b + 1][1]);
          }
#pragma unroll
          for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int b = 0; b < 8; ++b) mma_bf16(acc[a][b], af[a], bfr[b][0], bfr[b][1]);
        }
      }
      cp_async_wait<0>();
      // exact flush: C' to shared memory, then recombination of the limbs
      __syncthreads();
#pragma unroll
      for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int b = 0; b < 8; ++b) {
          int row = wm * 32 + a * 16 + (lane >> 2);
          int col = wn * 64 + b * 8 + 2 * (lane & 3);
          sm.u.C[row][col] = acc[a][b][0];
          sm.u.C[row][col + 1] = acc[a][b][1];
          sm.u.C[row + 8][col] = acc[a][b][2];
          sm.u.C[row + 8][col + 1] = acc[a][b][3];
        }
      __syncthreads();
      constexpr uint32_t PS = S ? kP1 : kP0;
      const uint32_t cf = S ? pc.coef.k1 : pc.coef.k0;
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        int idx = tid + NTHR * v;
        int m = idx >> 5, n = idx & 31;
        uint64_t sum = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            int32_t d = __float2int_rn(sm.u.C[4 * m + i][4 * n + j]);
            uint32_t rr = d < 0 ? (uint32_t)(d + (int32_t)PS) : (uint32_t)d;
            sum += (uint64_t)rr * w256[i + j];
          }
        tot[v] = addmod<S>(tot[v], mulmod<S>(reduce<S>(sum), cf));
      }
    }
  }
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    int idx = tid + NTHR * v;
    int m = idx >> 5, n = idx & 31;
    if (row0 + m >= rs.count || col0 + n >= cs.count) continue;
    int64_t flat = 0, bflat = 0;
    for (int d = 0; d < T.rank; ++d) {
      int32_t x = ((T.col_mask >> d) & 1) ? sm.ocol[n][d] : sm.orow[m][d];
      flat += T.stride[d] * x;
      bflat += g.bos[d] * x;
    }
    uint32_t key = tot[v];
    if (g.bsrc) {
      const uint2 b = g.bsrc[bflat];
      key = addmod<S>(key, S ? b.y : b.x);
    }
    reinterpret_cast<uint32_t*>(&vals[g.out_ws_off + flat])[S] = key;
  }
}

// ---------------------------------------------------------------- tcgen05 path
//
// Same product on the 5th-generation tensor cores: per CTA a 128 x 128 tile
// of C' (32 x 32 outputs), K in blocks of 64.  Warp 0 lane 0 streams the A'
// and B' tiles with TMA (128-byte swizzle) into a 3-stage ring guarded by
// mbarriers; warp 1 lane 0 issues tcgen05.mma (M 128, N 128, K 16, bf16 in,
// fp32 accumulator in tensor memory) and commits each stage back to the
// producer; after each exact block all four warps read their 32 lanes of
// the accumulator with tcgen05.ld and recombine the limbs.  Every wait is
// bounded: on a timeout the kernel records an error and stops issuing work.
namespace {

constexpr int T5_STAGES = 3;
constexpr int T5_BK = 64;                       // K per stage (one 128-byte swizzle row)
constexpr int T5_TILE_BYTES = 128 * T5_BK * 2;  // 16 KB per operand tile
constexpr int T5_MAXP = 4;                      // pieces per contraction on this path
constexpr uint32_t T5_TMEM_COLS = 128;
constexpr uint32_t T5_WAIT_LIMIT = 1u << 23;

struct TmaMaps {
  CUtensorMap a[T5_MAXP];
  CUtensorMap b[T5_MAXP];
};


__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(a), "r"(n));
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(a), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(a), "r"(parity)
      : "memory");
  return ok != 0;
}
// a * b + c with a 32 x 32 -> 64-bit product (one wide multiply-add)
__device__ __forceinline__ int64_t mad_wide_s32(int32_t a, int32_t b, int64_t c) {
  int64_t d;
  asm("mad.wide.s32 %0, %1, %2, %3;\n" : "=l"(d) : "r"(a), "r"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t mad_wide_u32(uint32_t a, uint32_t b, uint64_t c) {
  uint64_t d;
  asm("mad.wide.u32 %0, %1, %2, %3;\n" : "=l"(d) : "r"(a), "r"(b), "l"(c));
  return d;
}
// bounded wait; false on timeout
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity) {
  for (uint32_t i = 0; i < T5_WAIT_LIMIT; ++i)
    if (mbar_try(a, parity)) return true;
  return false;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t x,
                                            int32_t y, uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, "
      "{%2, %3}], [%4];\n" ::"r"(dst),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(mbar)
      : "memory");
}
// K-major operand in the 128-byte swizzled canonical layout: 8-row groups of
// 1024 bytes (stride byte offset), start address advanced 32 bytes per K = 16
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1 << 16;             // leading byte offset (unused with this swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;   // stride byte offset
  d |= (uint64_t)1 << 46;             // descriptor version
  d |= (uint64_t)2 << 61;             // 128-byte swizzle
  return d;
}
// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both
// K-major, N = 128, M = 128
constexpr uint32_t T5_IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 3) << 17) |
                              ((128u >> 4) << 24);
// the same with N = 256 (256-column tiles)
constexpr uint32_t T5_IDESC_N256 = (1u << 4) | (1u << 7) | (1u << 10) | ((256u >> 3) << 17) |
                                   ((128u >> 4) << 24);

__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                     uint32_t accumulate, uint32_t idesc = T5_IDESC) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t mbar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(mbar)
      : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, "
      "%30, %31}, [%32];\n"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

}  // namespace

// Persistent, warp-specialised kernel: warp 0 produces (TMA), warp 1 issues
// the MMAs, warps 2..9 drain the accumulators.  Two TMEM accumulators of 128
// columns let the epilogue of one exact block overlap the MMAs of the next.
// A unit is one (piece, block of <= 1024 reduction steps) of one tile; all
// roles walk the same sequence of tiles and units.
constexpr int T5_THREADS = 320;   // producer, MMA, 8 epilogue warps

struct T5Smem2 {
  uint8_t tiles[T5_STAGES][2][T5_TILE_BYTES];   // [stage][A|B], 1024-byte aligned
  uint64_t full[T5_STAGES], empty[T5_STAGES];
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int32_t abort_flag;
};

// 256-column variant: two CTAs per SM, each with one 256-column accumulator
// (the two fill the SM's tensor memory) and two stages of a 128-row A tile
// and a 256-row B tile; an MMA instruction covers 128 x 256 x 16, twice the
// work per instruction of the 128-column tiles.
constexpr int T5N_STAGES = 2;
constexpr int T5N_B_BYTES = 2 * T5_TILE_BYTES;   // 256 rows x 64 K
struct T5SmemN {
  uint8_t a[T5N_STAGES][T5_TILE_BYTES];
  uint8_t b[T5N_STAGES][T5N_B_BYTES];
  uint64_t full[T5N_STAGES], empty[T5N_STAGES];
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int32_t abort_flag;
};

// Column-stationary variant: the column-side tiles of one column tile (all
// pieces that reach it, all reduction blocks) stay in shared memory while
// the CTA walks its row tiles; only row-side tiles stream through the ring.
constexpr int T5W_MAXKB = 9;    // stationary 16 KB tiles (144 KB)
constexpr int T5W_STAGES = 5;   // row-side ring (80 KB)
struct T5SmemW {
  uint8_t bst[T5W_MAXKB][T5_TILE_BYTES];
  uint8_t a[T5W_STAGES][T5_TILE_BYTES];
  uint64_t full[T5W_STAGES], empty[T5W_STAGES];
  uint64_t bfull, bempty;
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int32_t abort_flag;
};

// Piece q can reach column tile tc (some row tile).
__device__ __forceinline__ bool piece_hits_col(const TcGeom& g, int q, int64_t tc) {
  return g.c0[q] < (tc + 1) * TO && tc * TO < g.c1[q];
}

// The it-th tile of this CTA, or false past the last.  W = 0: tiles
// blockIdx.x + it * gridDim.x in (batch, row tile, column tile) order.  W = 1:
// CTA c keeps column tile c % ntc and walks, per batch index, the row tiles
// c / ntc, c / ntc + groups, ... (groups = gridDim.x / ntc CTAs share each
// column tile; the CTAs with the same c / ntc read the same row tiles at
// about the same time, so row-side tiles are served from L2).
template <int W>
__device__ __forceinline__ bool tile_at(int64_t it, int64_t ntc, int64_t ntr, int64_t nb,
                                        int64_t& bz, int64_t& tr, int64_t& tc) {
  if (W == 0) {
    const int64_t tile = blockIdx.x + it * gridDim.x;
    if (tile >= ntc * ntr * nb) return false;
    int64_t rest;
    divmod64(tile, ntc, rest, tc);
    divmod64(rest, ntr, bz, tr);
    return true;
  }
  const int64_t groups = gridDim.x / ntc, rg = blockIdx.x / ntc;
  if (rg >= groups || rg >= ntr) return false;
  const int64_t per_b = (ntr - rg + groups - 1) / groups;
  bz = it / per_b;
  if (bz >= nb) return false;
  tr = rg + (it - bz * per_b) * groups;
  tc = blockIdx.x % ntc;
  return true;
}

// N2: 0 the default 128-column tiles with two double-buffered accumulators;
// 1 the 256-column tiles (one accumulator).
template <int S, int W, int N2>
__global__ void __launch_bounds__(T5_THREADS, 2 - W) tc5_gemm_kernel(
    const __grid_constant__ Prog P, int t, const __grid_constant__ TmaMaps maps, TcGeom g,
    const uint2* leafk, uint2* vals, int32_t* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  using Smem = typename std::conditional<
      W != 0, T5SmemW, typename std::conditional<N2 == 1, T5SmemN, T5Smem2>::type>::type;
  constexpr uint32_t NST = W != 0 ? T5W_STAGES : N2 == 1 ? T5N_STAGES : T5_STAGES;
  // outputs per column tile
  constexpr int64_t WC = N2 == 1 ? 2 * TO : TO;
  Smem& sm = *reinterpret_cast<Smem*>(
      (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023));
  const Tensor& T = P.t[t];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t ntc = g.cpad / WC, ntr = g.rpad / TO;
  if (tid == 0) {
    for (uint32_t st = 0; st < NST; ++st) {
      mbar_init(smem_u32(&sm.full[st]), 1);
      mbar_init(smem_u32(&sm.empty[st]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&sm.acc_full[b]), 1);
      mbar_init(smem_u32(&sm.acc_empty[b]), 8);
    }
    if constexpr (W != 0) {
      mbar_init(smem_u32(&sm.bfull), 1);
      mbar_init(smem_u32(&sm.bempty), 1);
    }
    sm.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                     smem_u32(&sm.tmem_base)),
                 "r"(2 * T5_TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
  }
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
  const uint32_t tmem = sm.tmem_base;
  volatile int32_t* abort_flag = &sm.abort_flag;

  // The streaming 128-column kernel has its own producer and MMA loops, kept
  // lean because the per-stage latency of these two single threads bounds the
  // kernel: ring slot and phase as counters, tile coordinates formed once per
  // tile, a thread stops on its own expired wait (the other roles' waits then
  // expire in turn).  The other variants share the general loops below.
  if (warp == 0) {
    if constexpr (W == 0 && N2 == 0) {
      if (lane == 0) {   // ---- TMA producer (streaming, 128-column tiles)
        uint32_t st = 0, ph = 0;
        const int64_t ntl = ntc * ntr * g.batch;
        bool stop = false;
        for (int64_t tile = blockIdx.x; tile < ntl && !stop; tile += gridDim.x) {
          int64_t rest, tc, bz, tr;
          divmod64(tile, ntc, rest, tc);
          divmod64(rest, ntr, bz, tr);
          const int32_t arow = (int32_t)(bz * 4 * g.rpad + 4 * tr * TO);
          const int32_t brow = (int32_t)(bz * 4 * g.cpad + 4 * tc * WC);
          for (int q = 0; q < T.npieces && !stop; ++q) {
            if (!piece_hits(g, q, tr, tc, WC)) continue;
            const int nk = (int)(g.kp[q] / T5_BK);
            const CUtensorMap* ma = &maps.a[q];
            const CUtensorMap* mb = &maps.b[q];
            if (g.conv[q]) {
              int64_t nh, w0, n, h;
              divmod64(tr * TO, g.cv_Wo[q], nh, w0);
              divmod64(nh, g.cv_Ho[q], n, h);
              const int32_t ybase = (int32_t)(((n * g.cv_Hp[q] + h) * g.cv_Wp[q] + w0) * 4);
              const int32_t cbn = g.cv_Cpad[q] / T5_BK, KWq = g.cv_KW[q], Wp4 = g.cv_Wp[q] * 4;
              int32_t cb = 0, kw = 0, yk = ybase;   // yk: ybase + (kh * Wp + kw) * 4
              int32_t yrow = ybase;                  // ybase + kh * Wp * 4
              for (int kk = 0; kk < nk; ++kk) {
                if (!mbar_wait(smem_u32(&sm.empty[st]), ph ^ 1)) {
                  *abort_flag = 1;
                  stop = true;
                  break;
                }
                const uint32_t fb = smem_u32(&sm.full[st]);
                mbar_expect_tx(fb, 2 * T5_TILE_BYTES);
                tma_load_2d(smem_u32(sm.tiles[st][0]), ma, cb * T5_BK, yk, fb);
                tma_load_2d(smem_u32(sm.tiles[st][1]), mb, kk * T5_BK, brow, fb);
                if (++cb == cbn) {
                  cb = 0;
                  if (++kw == KWq) {
                    kw = 0;
                    yrow += Wp4;
                    yk = yrow;
                  } else {
                    yk += 4;
                  }
                }
                if (++st == NST) {
                  st = 0;
                  ph ^= 1;
                }
              }
            } else {
              for (int kk = 0; kk < nk; ++kk) {
                if (!mbar_wait(smem_u32(&sm.empty[st]), ph ^ 1)) {
                  *abort_flag = 1;
                  stop = true;
                  break;
                }
                const uint32_t fb = smem_u32(&sm.full[st]);
                mbar_expect_tx(fb, 2 * T5_TILE_BYTES);
                tma_load_2d(smem_u32(sm.tiles[st][0]), ma, kk * T5_BK, arow, fb);
                tma_load_2d(smem_u32(sm.tiles[st][1]), mb, kk * T5_BK, brow, fb);
                if (++st == NST) {
                  st = 0;
                  ph ^= 1;
                }
              }
            }
          }
        }
      }
    } else if (lane == 0) {   // ---- TMA producer (other variants)
      uint32_t I = 0, Bg = 0;
      int64_t cur_bz = -1;
      for (int64_t it = 0; !*abort_flag; ++it) {
        int64_t bz, tr, tc;
        if (!tile_at<W>(it, ntc, ntr, g.batch, bz, tr, tc)) break;
        const int32_t arow = (int32_t)(bz * 4 * g.rpad + 4 * tr * TO);
        const int32_t brow = (int32_t)(bz * 4 * g.cpad + 4 * tc * WC);
        if constexpr (W != 0) {
          if (bz != cur_bz) {   // the column tile's stationary tiles for this batch index
            if (Bg > 0 && !mbar_wait(smem_u32(&sm.bempty), (Bg - 1) & 1)) {
              *abort_flag = 1;
              break;
            }
            uint32_t nkb = 0;
            for (int q = 0; q < T.npieces; ++q)
              if (piece_hits_col(g, q, tc)) nkb += (uint32_t)(g.kp[q] / T5_BK);
            const uint32_t fb = smem_u32(&sm.bfull);
            mbar_expect_tx(fb, nkb * T5_TILE_BYTES);
            int slot = 0;
            for (int q = 0; q < T.npieces; ++q) {
              if (!piece_hits_col(g, q, tc)) continue;
              for (int64_t k = 0; k < g.kp[q]; k += T5_BK, ++slot)
                tma_load_2d(smem_u32(sm.bst[slot]), &maps.b[q], (int32_t)k, brow, fb);
            }
            ++Bg;
            cur_bz = bz;
          }
        }
        for (int q = 0; q < T.npieces; ++q) {
          // limb-image rows of a convolution piece: the tile's 32 outputs (n, h,
          // w0 .. w0 + 31) start at row ybase; window offset (kh, kw) adds
          // (kh * Wp + kw) * 4 rows, channel block cb selects the columns
          int32_t ybase = 0, cb = 0, kw = 0, kh = 0, cbn = 1;
          if (g.conv[q] && piece_hits(g, q, tr, tc, WC)) {
            int64_t nh, w0, n, h;
            divmod64(tr * TO, g.cv_Wo[q], nh, w0);
            divmod64(nh, g.cv_Ho[q], n, h);
            ybase = (int32_t)(((n * g.cv_Hp[q] + h) * g.cv_Wp[q] + w0) * 4);
            cbn = g.cv_Cpad[q] / T5_BK;
          }
          for (int64_t k = 0; k < g.kp[q] && piece_hits(g, q, tr, tc, WC); k += T5_BK, ++I) {
            uint32_t st = I % NST, ph = (I / NST) & 1;
            if (!mbar_wait(smem_u32(&sm.empty[st]), ph ^ 1)) {
              *abort_flag = 1;
              break;
            }
            uint32_t fb = smem_u32(&sm.full[st]);
            int32_t ax = (int32_t)k, ay = arow;
            if (g.conv[q]) {
              ax = cb * T5_BK;
              ay = ybase + (kh * g.cv_Wp[q] + kw) * 4;
              if (++cb == cbn) {
                cb = 0;
                if (++kw == g.cv_KW[q]) {
                  kw = 0;
                  ++kh;
                }
              }
            }
            if constexpr (W != 0) {
              mbar_expect_tx(fb, T5_TILE_BYTES);
              tma_load_2d(smem_u32(sm.a[st]), &maps.a[q], ax, ay, fb);
            } else if constexpr (N2 == 1) {
              mbar_expect_tx(fb, T5_TILE_BYTES + T5N_B_BYTES);
              tma_load_2d(smem_u32(sm.a[st]), &maps.a[q], ax, ay, fb);
              tma_load_2d(smem_u32(sm.b[st]), &maps.b[q], (int32_t)k, brow, fb);
            } else {
              mbar_expect_tx(fb, 2 * T5_TILE_BYTES);
              tma_load_2d(smem_u32(sm.tiles[st][0]), &maps.a[q], ax, ay, fb);
              tma_load_2d(smem_u32(sm.tiles[st][1]), &maps.b[q], (int32_t)k, brow, fb);
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    if constexpr (W == 0 && N2 == 0) {
      if (lane == 0) {   // ---- MMA issuer (streaming, 128-column tiles)
        uint32_t st = 0, ph = 0, U = 0;
        const int64_t ntl = ntc * ntr * g.batch;
        bool stop = false;
        for (int64_t tile = blockIdx.x; tile < ntl && !stop; tile += gridDim.x) {
          int64_t rest, tc, bz, tr;
          divmod64(tile, ntc, rest, tc);
          divmod64(rest, ntr, bz, tr);
          for (int q = 0; q < T.npieces && !stop; ++q) {
            if (!piece_hits(g, q, tr, tc, WC)) continue;
            const int nk = (int)(g.kp[q] / T5_BK);
            for (int kb = 0; kb < nk && !stop; kb += KBLK / T5_BK, ++U) {
              const uint32_t b = U & 1, acc = tmem + b * T5_TMEM_COLS;
              if (!mbar_wait(smem_u32(&sm.acc_empty[b]), ((U >> 1) & 1) ^ 1)) {
                *abort_flag = 1;
                stop = true;
                break;
              }
              asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
              const int ke = kb + KBLK / T5_BK < nk ? kb + KBLK / T5_BK : nk;
              for (int kk = kb; kk < ke; ++kk) {
                if (!mbar_wait(smem_u32(&sm.full[st]), ph)) {
                  *abort_flag = 1;
                  stop = true;
                  break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
                const uint64_t ad = sw128_desc(smem_u32(sm.tiles[st][0]));
                const uint64_t bd = sw128_desc(smem_u32(sm.tiles[st][1]));
#pragma unroll
                for (int k16 = 0; k16 < T5_BK / 16; ++k16)
                  umma(acc, ad + 2 * k16, bd + 2 * k16, (kk > kb || k16 > 0) ? 1u : 0u, T5_IDESC);
                umma_commit(smem_u32(&sm.empty[st]));
                if (++st == NST) {
                  st = 0;
                  ph ^= 1;
                }
              }
              umma_commit(smem_u32(&sm.acc_full[b]));
            }
          }
        }
      }
    } else if (lane == 0) {   // ---- MMA issuer (other variants)
      uint32_t I = 0, U = 0, Bg = 0;
      int64_t cur_bz = -1;
      for (int64_t it = 0; !*abort_flag; ++it) {
        int64_t bz, tr, tc;
        if (!tile_at<W>(it, ntc, ntr, g.batch, bz, tr, tc)) break;
        if constexpr (W != 0) {
          if (bz != cur_bz) {
            // the previous stationary tiles are free once every MMA so far is done
            if (Bg > 0) umma_commit(smem_u32(&sm.bempty));
            if (!mbar_wait(smem_u32(&sm.bfull), Bg & 1)) {
              *abort_flag = 1;
              break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
            ++Bg;
            cur_bz = bz;
          }
        }
        int slot0 = 0;   // first stationary tile of piece q
        for (int q = 0; q < T.npieces && !*abort_flag; ++q) {
          const bool hq = piece_hits(g, q, tr, tc, WC);
          for (int64_t kb0 = 0; kb0 < g.kp[q] && !*abort_flag && hq; kb0 += KBLK, ++U) {
            // N2: one accumulator, used by every unit in turn
            const uint32_t b = N2 != 0 ? 0u : (U & 1), acc = tmem + b * T5_TMEM_COLS;
            const uint32_t eph = N2 != 0 ? ((U & 1) ^ 1) : (((U >> 1) & 1) ^ 1);
            if (!mbar_wait(smem_u32(&sm.acc_empty[b]), eph)) {
              *abort_flag = 1;
              break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
            const int64_t kb1 = kb0 + KBLK < g.kp[q] ? kb0 + KBLK : g.kp[q];
            for (int64_t k = kb0; k < kb1; k += T5_BK, ++I) {
              uint32_t st = I % NST, ph = (I / NST) & 1;
              if (!mbar_wait(smem_u32(&sm.full[st]), ph)) {
                *abort_flag = 1;
                break;
              }
              asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
              uint64_t ad, bd;
              if constexpr (W != 0) {
                ad = sw128_desc(smem_u32(sm.a[st]));
                bd = sw128_desc(smem_u32(sm.bst[slot0 + (int)(k / T5_BK)]));
              } else if constexpr (N2 == 1) {
                ad = sw128_desc(smem_u32(sm.a[st]));
                bd = sw128_desc(smem_u32(sm.b[st]));
              } else {
                ad = sw128_desc(smem_u32(sm.tiles[st][0]));
                bd = sw128_desc(smem_u32(sm.tiles[st][1]));
              }
#pragma unroll
              for (int k16 = 0; k16 < T5_BK / 16; ++k16)
                umma(acc, ad + 2 * k16, bd + 2 * k16, (k > kb0 || k16 > 0) ? 1u : 0u,
                     N2 == 1 ? T5_IDESC_N256 : T5_IDESC);
              umma_commit(smem_u32(&sm.empty[st]));
            }
            umma_commit(smem_u32(&sm.acc_full[b]));
          }
          if constexpr (W != 0)
            if (piece_hits_col(g, q, tc)) slot0 += (int)(g.kp[q] / T5_BK);
        }
      }
    }
  } else {   // ---- epilogue warps 2..9: TMEM lane quarter (warp % 4), column half
    const int quarter = warp & 3, half = (warp - 2) >> 2;
    const int lrow = quarter * 32 + lane;   // limb row (4m + i) of the tile
    const int my_i = lrow & 3, m = lrow >> 2;
    constexpr uint64_t PS = S ? kP1 : kP0;
    constexpr uint32_t FC = S ? 33u : 3u;    // 2^29 = FC (mod p)
    constexpr uint32_t M29 = (1u << 29) - 1;
    // weight 256^i' of the limb row i' = my_i ^ d held by lane my_i ^ d
    uint32_t wd[4];
#pragma unroll
    for (int d = 0; d < 4; ++d) wd[d] = 1u << (8 * (my_i ^ d));
    uint32_t U = 0;
    for (int64_t it = 0;; ++it) {
      int64_t bz, tr, tc;
      if (W == 0 && g.fd_ok) {
        const int64_t tile = blockIdx.x + it * gridDim.x;
        if (tile >= ntc * ntr * g.batch) break;
        const uint32_t rest = fast_div((uint32_t)tile, g.fd_m[0], g.fd_s[0]);
        tc = (uint32_t)tile - rest * (uint32_t)ntc;
        bz = fast_div(rest, g.fd_m[1], g.fd_s[1]);
        tr = rest - (uint32_t)bz * (uint32_t)ntr;
      } else if (!tile_at<W>(it, ntc, ntr, g.batch, bz, tr, tc)) {
        break;
      }
      // NCH chunks of 32 limb columns per warp: outputs half * HW + 4 k + my_i
      constexpr int NCH = N2 == 1 ? 4 : 2, NK = 2 * NCH, HW = 2 * NCH * 4;
      uint32_t tot[NK];
#pragma unroll
      for (int k = 0; k < NK; ++k) tot[k] = 0;
      // a fused bias add: this thread's bias keys, loaded before the
      // accumulator wait so that their latency overlaps it
      const int64_t row = tr * TO + m;
      uint32_t bk[NK];
#pragma unroll
      for (int k = 0; k < NK; ++k) bk[k] = 0;
      if (g.bsrc && row < g.rsp.count) {
        const int64_t rbias =
            g.brow ? split_offset_w(T, g.bsp, bz, g.bos) + split_offset_w(T, g.rsp, row, g.bos) : 0;
#pragma unroll
        for (int k = 0; k < NK; ++k) {
          const int64_t col = tc * WC + half * HW + 4 * k + my_i;
          if (col < g.csp.count) {
            const uint2 b = g.bsrc[rbias + split_offset_w(T, g.csp, col, g.bos)];
            bk[k] = S ? b.y : b.x;
          }
        }
      }
      bool dead = false;
      for (int q = 0; q < T.npieces; ++q) {
        const uint32_t cf = S ? P.p[T.piece0 + q].coef.k1 : P.p[T.piece0 + q].coef.k0;
        const bool cf1 = cf == 1u;
        for (int64_t kb0 = 0; kb0 < g.kp[q] && piece_hits(g, q, tr, tc, WC); kb0 += KBLK, ++U) {
          const uint32_t b = N2 != 0 ? 0u : (U & 1);
          const uint32_t fph = N2 != 0 ? (U & 1) : ((U >> 1) & 1);
          if (*abort_flag || !mbar_wait(smem_u32(&sm.acc_full[b]), fph)) {
            *abort_flag = 1;
            dead = true;
            break;
          }
          __syncwarp();
          asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
          const uint32_t base = tmem + b * T5_TMEM_COLS + (uint32_t)(half * 32 * NCH) +
                                ((uint32_t)(quarter * 32) << 16);
#pragma unroll
          for (int chunk = 0; chunk < NCH; ++chunk) {
            uint32_t v[32];
            tmem_ld32(base + (uint32_t)(chunk * 32), v);
            if (chunk == NCH - 1) {
              // every chunk is read: the accumulator is free for the next
              // unit's MMAs while this warp still combines the last
              asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
              __syncwarp();
              if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(
                                 smem_u32(&sm.acc_empty[b]))
                             : "memory");
            }
#pragma unroll
            for (int gq = 0; gq < 2; ++gq) {
              // four output columns t = 0..3 (n = 8 chunk + 4 gq + t).  The
              // C'[(m,i),(n,j)] are integers with |C'| <= 1024 * 128^2 = 2^24, so
              // x = sum_j 256^j C'_j + 2^21 p lies in (0, 2^50.4): exact in 64 bits,
              // formed by wide multiply-adds; one fold gives f = x (mod p), f < 2^29.2
              uint32_t f[4];
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                const int c = 4 * (4 * gq + t);
                int64_t x = (int64_t)(PS << 21);
                x = mad_wide_s32(__float2int_rn(__uint_as_float(v[c])), 1, x);
                x = mad_wide_s32(__float2int_rn(__uint_as_float(v[c + 1])), 256, x);
                x = mad_wide_s32(__float2int_rn(__uint_as_float(v[c + 2])), 65536, x);
                x = mad_wide_s32(__float2int_rn(__uint_as_float(v[c + 3])), 16777216, x);
                f[t] = (uint32_t)((uint64_t)x >> 29) * FC + ((uint32_t)x & M29);
              }
              // transpose over the four limb rows (lanes 4m'..4m'+3): in round d
              // lane i sends its f for column i ^ d to lane i ^ d, so lane i
              // collects column t = i from every limb row i' = i ^ d and weights
              // it by 256^i'; z < 4 * 2^29.2 * 2^24 < 2^55.2
              uint64_t z = 0;
#pragma unroll
              for (int d = 0; d < 4; ++d) {
                const int idx = my_i ^ d;
                const uint32_t lo = (idx & 1) ? f[1] : f[0], hi = (idx & 1) ? f[3] : f[2];
                const uint32_t send = (idx & 2) ? hi : lo;
                const uint32_t g = d ? __shfl_xor_sync(0xffffffffu, send, d) : send;
                z = mad_wide_u32(g, wd[d], z);
              }
              // z mod p in 32 bits: (z >> 29) * FC + low < 2^26.2 * 33 + 2^29 < 2^31.6,
              // folded again below 2p and reduced once
              uint32_t rz = (uint32_t)(z >> 29) * FC + ((uint32_t)z & M29);
              rz = (rz >> 29) * FC + (rz & M29);
              rz = rz >= (uint32_t)PS ? rz - (uint32_t)PS : rz;
              tot[2 * chunk + gq] = addmod<S>(tot[2 * chunk + gq], cf1 ? rz : mulmod<S>(rz, cf));
            }
          }
        }
        if (dead) break;
      }
      if (dead) break;
      // write lane S of this thread's outputs: row m, columns half*16 + 4k + my_i
      // (with a fused bias add: plus the bias key, into the sum's array)
      if (row < g.rsp.count) {
        int64_t roff = 0;
        if (g.fd_ok) {   // split_offset(T, g.rsp, row) by multiplies
          uint32_t x = (uint32_t)row;
#pragma unroll
          for (int i = MR - 1; i >= 0; --i) {
            if (i < g.rsp.nd) {
              const int d = g.rsp.dims[i];
              const uint32_t qq = fast_div(x, g.fd_m[2 + i], g.fd_s[2 + i]);
              roff += T.stride[d] * (int64_t)(x - qq * (uint32_t)T.shape[d]);
              x = qq;
            }
          }
        } else {
          roff = split_offset(T, g.rsp, row);
        }
        const int64_t rflat = g.out_ws_off + split_offset(T, g.bsp, bz) + roff;
#pragma unroll
        for (int k = 0; k < NK; ++k) {
          const int64_t col = tc * WC + half * HW + 4 * k + my_i;
          if (col >= g.csp.count) continue;
          reinterpret_cast<uint32_t*>(&vals[rflat + split_offset(T, g.csp, col)])[S] =
              addmod<S>(tot[k], bk[k]);
        }
      }
    }
  }
  __syncthreads();
  if (tid == 0 && sm.abort_flag) atomicOr(status, 1);
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem),
                 "r"(2 * T5_TMEM_COLS));
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
  }
  return fn;
}

// 2-D bf16 map over rows x kp (K contiguous), 64 x box_rows boxes, 128-byte swizzle
bool make_map(CUtensorMap* m, const uint16_t* base, int64_t kp, int64_t rows,
              uint32_t box_rows = 128) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)kp, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)kp * 2};
  cuuint32_t box[2] = {(cuuint32_t)T5_BK, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)base, dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace

static dirigo_status launch_tc5(const Prog& P, int t, const TcGeom& g0, uint16_t* buf,
                                const uint2* leafk, uint2* vals, int32_t* status,
                                cudaStream_t s) {
  const Tensor& T = P.t[t];
  const int64_t ntc = g0.cpad / TO, ntr = g0.rpad / TO;
  int64_t ntiles = ntc * ntr * g0.batch;
  TcGeom g = g0;
  int nsm = 152, dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  // The column-stationary variant (DIRIGO_TC_STATIONARY=1) needs every column
  // tile's column-side tiles to fit in shared memory and a CTA per column
  // tile.  It halves the operand traffic but runs one CTA per SM; the
  // streaming variant with two CTAs per SM overlaps more epilogue work and is
  // the default.
  const char* env = std::getenv("DIRIGO_TC_STATIONARY");
  bool stationary = env && env[0] == '1' && ntc <= nsm;
  for (int64_t tc = 0; tc < ntc && stationary; ++tc) {
    int64_t nkb = 0;
    for (int q = 0; q < T.npieces; ++q)
      if (g.c0[q] < (tc + 1) * TO && tc * TO < g.c1[q]) nkb += g.kp[q] / T5_BK;
    stationary = nkb <= T5W_MAXKB;
  }
  // 256-column tiles (DIRIGO_TC_N=256; two CTAs per SM, each with one 128 x
  // 256 accumulator and two 48 KB stages: twice the work per MMA instruction)
  // where the padded column count allows them.  Slower than the default
  // 128-column tiles on config 4 (1.44 against 1.25 ms per step): each CTA's
  // single accumulator stalls its MMAs for its epilogue.
  const char* env_n = std::getenv("DIRIGO_TC_N");
  const bool n256 = !stationary && g.cpad % (2 * TO) == 0 && env_n &&
                    std::string(env_n) == "256";

  {
    // the epilogue's divisions (the streaming tile walk and the row split)
    // by multiplies, where every dividend fits 31 bits
    const int64_t ntc_k = n256 ? g.cpad / (2 * TO) : ntc;
    fast_div_make(ntc_k, &g.fd_m[0], &g.fd_s[0]);
    fast_div_make(ntr, &g.fd_m[1], &g.fd_s[1]);
    bool ok = ntc_k * ntr * g.batch < (1ll << 31) && g.rpad < (1ll << 31);
    for (int i = 0; i < MR; ++i) {
      g.fd_m[2 + i] = g.fd_s[2 + i] = 0;
      if (i < g.rsp.nd) {
        const int64_t e = T.shape[g.rsp.dims[i]];
        ok = ok && e < (1ll << 31);
        fast_div_make(e, &g.fd_m[2 + i], &g.fd_s[2 + i]);
      }
    }
    g.fd_ok = ok ? 1 : 0;
  }
  dim3 grid;
  size_t shm;
  if (stationary) {
    grid = dim3((unsigned)(nsm / ntc * ntc));
    shm = sizeof(T5SmemW) + 1024;
  } else if (n256) {
    const int64_t nt2 = (g.cpad / (2 * TO)) * ntr * g.batch;
    grid = dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(nt2, 2 * (int64_t)nsm)));
    shm = sizeof(T5SmemN) + 1024;
  } else {
    grid = dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(ntiles, 2 * (int64_t)nsm)));
    shm = sizeof(T5Smem2) + 1024;
  }
  static bool attr_set[64] = {false};
  if (dev < 64 && !attr_set[dev]) {
    const int s2 = (int)(sizeof(T5Smem2) + 1024), sw = (int)(sizeof(T5SmemW) + 1024),
              sn = (int)(sizeof(T5SmemN) + 1024);
    cudaFuncSetAttribute(tc5_gemm_kernel<0, 0, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, s2);
    cudaFuncSetAttribute(tc5_gemm_kernel<1, 0, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, s2);
    cudaFuncSetAttribute(tc5_gemm_kernel<0, 1, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, sw);
    cudaFuncSetAttribute(tc5_gemm_kernel<1, 1, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, sw);
    cudaFuncSetAttribute(tc5_gemm_kernel<0, 0, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sn);
    cudaFuncSetAttribute(tc5_gemm_kernel<1, 0, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sn);

    attr_set[dev] = true;
  }
  for (int lane = 0; lane < 2; ++lane) {
    TmaMaps maps;
    std::memset(&maps, 0, sizeof(maps));
    const uint16_t* lb = buf + (lane ? g.lane_stride : 0);
    for (int q = 0; q < T.npieces; ++q) {
      if (g.kp[q] == 0) continue;
      const bool ok =
          (g.conv[q] ? make_map(&maps.a[q], lb + g.offA[q], g.cv_Cpad[q],
                                (int64_t)g.cv_N[q] * g.cv_Hp[q] * g.cv_Wp[q] * 4)
                     : make_map(&maps.a[q], lb + g.offA[q], g.kp[q], g.batch * 4 * g.rpad)) &&
          make_map(&maps.b[q], lb + g.offB[q], g.kp[q], g.batch * 4 * g.cpad, n256 ? 256 : 128);
      if (!ok) return set_error(DIRIGO_E_CUDA, "tensor map encoding failed");
    }
    if (stationary) {
      if (lane == 0)
        tc5_gemm_kernel<0, 1, 0><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
      else
        tc5_gemm_kernel<1, 1, 0><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
    } else if (n256) {
      if (lane == 0)
        tc5_gemm_kernel<0, 0, 1><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
      else
        tc5_gemm_kernel<1, 0, 1><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
    } else {
      if (lane == 0)
        tc5_gemm_kernel<0, 0, 0><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
      else
        tc5_gemm_kernel<1, 0, 0><<<grid, T5_THREADS, shm, s>>>(P, t, maps, g, leafk, vals, status);
    }
    count_launch();
  }
  return DIRIGO_OK;
}

// The tcgen05 kernel is the default; DIRIGO_TC=mma selects the mma.sync one.
static bool use_tcgen05() {
  const char* e = std::getenv("DIRIGO_TC");
  return !(e && std::string(e) == "mma");
}

// The geometry launch_gemm_keys_tc uses for contraction t, and whether it runs
// the tcgen05 kernel.
static TcGeom dispatch_geom(const Prog& P, const Tensor& T, bool* tc5_out) {
  bool tc5 = use_tcgen05() && T.npieces <= T5_MAXP;
  TcGeom g = tc_geom(P, T, tc5);
  if (tc5 && !(g.batch * 4 * std::max(g.rpad, g.cpad) < (1ll << 31))) {
    tc5 = false;
    g = tc_geom(P, T, false);
  }
  *tc5_out = tc5;
  return g;
}

bool tc_row_side_all_image(const Prog& P, int t) {
  bool tc5 = false;
  const TcGeom g = dispatch_geom(P, P.t[t], &tc5);
  if (!tc5) return false;
  for (int q = 0; q < P.t[t].npieces; ++q)
    if (!g.conv[q]) return false;
  return true;
}

dirigo_status launch_gemm_keys_tc(const Prog& P, int t, const uint2* leafk, uint2* vals,
                                  void* tc_ws, int32_t* status, cudaStream_t s) {
  const Tensor& T = P.t[t];
  bool tc5 = false;
  TcGeom g = dispatch_geom(P, T, &tc5);
  // where the epilogue writes, and the fused bias operand
  g.out_ws_off = T.fused ? P.t[T.fused].ws_off : T.ws_off;
  g.bsrc = nullptr;
  g.brow = 0;
  for (int d = 0; d < MR; ++d) g.bos[d] = 0;
  if (T.fused) {
    const Tensor& U = P.t[T.fused];
    const Tensor& B = P.t[U.args[1]];
    g.bsrc = B.kind == K_INPUT ? leafk + B.gbase : vals + B.ws_off;
    for (int d = 0; d < U.arg_rank[1]; ++d)
      if (B.shape[d] != 1) g.bos[U.axes[1][d]] += B.stride[d];
    for (int d = 0; d < T.rank; ++d)
      if (!((T.col_mask >> d) & 1) && g.bos[d] != 0) g.brow = 1;
  }
  uint16_t* buf = (uint16_t*)tc_ws;
  {
  Prof pr(DIRIGO_K_KEY_LIMBS, s);
  for (int q = 0; q < T.npieces; ++q) {
    if (!g.conv[q] || g.a_src[q] != q) continue;
    const int64_t n = (int64_t)g.cv_N[q] * g.cv_Hp[q] * g.cv_Wp[q] * (g.cv_Cpad[q] / 8);
    if (n > ((int64_t)1 << 40)) return set_error(DIRIGO_E_UNSUPPORTED, "contraction too large");
    tc_limb_image_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(P, t, q, leafk, vals, buf, g);
    count_launch();
  }
  for (int q = 0; q < T.npieces; ++q) {
    // the row-side matrix is another piece's, or a limb image
    const int b_only = g.a_src[q] != q || g.conv[q];
    const int64_t nlb = g.batch * (((b_only ? 0 : g.rpad) + g.cpad) / 32);
    int64_t nb = nlb * ((g.kp[q] + kMatK - 1) / kMatK);
    if (nb == 0) continue;
    if (nb > 0x7fffffff) return set_error(DIRIGO_E_UNSUPPORTED, "contraction too large");
    if (nb < 2 * 152) {   // a small matrix: blocks of 64 steps
      nb = nlb * ((g.kp[q] + 63) / 64);
      tc_materialize_kernel<64><<<(unsigned)nb, 256, 0, s>>>(P, t, q, b_only, leafk, vals, buf, g);
    } else {
      tc_materialize_kernel<kMatK><<<(unsigned)nb, 256, 0, s>>>(P, t, q, b_only, leafk, vals, buf,
                                                                 g);
    }
    count_launch();
  }
  }
  Prof pr(DIRIGO_K_KEY_GEMM, s);
  dim3 grid((unsigned)(g.cpad / TO), (unsigned)(g.rpad / TO), (unsigned)g.batch);
  if (grid.y > 65535 || grid.z > 65535)
    return set_error(DIRIGO_E_UNSUPPORTED, "contraction grid too large");
  if (tc5) return launch_tc5(P, t, g, buf, leafk, vals, status, s);
  size_t shm = sizeof(GemmSmem);
  int dev = 0;
  cudaGetDevice(&dev);
  static bool attr_set[64] = {false};
  if (dev < 64 && !attr_set[dev]) {
    cudaFuncSetAttribute(tc_gemm_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)shm);
    cudaFuncSetAttribute(tc_gemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)shm);
    attr_set[dev] = true;
  }
  tc_gemm_kernel<0><<<grid, NTHR, shm, s>>>(P, t, buf, g, leafk, vals);
  tc_gemm_kernel<1><<<grid, NTHR, shm, s>>>(P, t, buf, g, leafk, vals);
  count_launch();
  count_launch();
  return DIRIGO_OK;
}

}  // namespace dirigo
