// Term keys: forward evaluation of every primitive tensor's per-element
// equation in F_p0 x F_p1, one key pair per element (memoisation per
// (tensor, element) is hash-consing of the shared subterms, Sec. 3.4
// "Back-projection": every T_j[l'] in f_k(l) is resolved once).
//
// Kernels:
//   leaf_keys      key of every global input id (and of bottom, id G)
//   (gemm_tc.cu)   two-operand CONTRACTs on the tensor cores
//   contract_keys  other CONTRACTs (sums, means): G threads per element split
//                  its terms, consecutive elements on consecutive lanes
//   maxset_keys    MAXSET: collect, sort and deduplicate the members' keys in
//                  a register list sized for the tensor's term bound
//   maxset_box_keys  MAXSET of one guard-free piece over the whole output
//                  (a pooling window): the members' offsets from an element's
//                  first member are formed once per thread
// A MAXSET or a non-tensor-core sum whose only reader is a same-shape UNARY
// writes that UNARY's keys itself (the UNARY's own pass is skipped).
//   elem_keys      UNARY / MAXC / AFFINE / BINARY, 4 elements per thread
//   gather_keys    root keys of the queried locations
#include <cstdint>

#include "dev.cuh"
#include "internal.h"
#include "launch.h"

namespace dirigo {

// keys of the global ids [g0, g1)
__global__ void leaf_keys_kernel(int64_t g0, int64_t g1, uint2* leafk) {
  int64_t g = g0 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (; g < g1; g += stride) leafk[g] = make_uint2(leaf_key0((uint64_t)g), leaf_key1((uint64_t)g));
}

// Whether some kernel reads input t's keys from the leaf-key array: every
// reader does, except a tensor-core contraction that reads t only as its row
// side through limb images.
static bool input_keys_read(const Prog& P, int t) {
  for (int u = P.n_inputs; u < P.n_tensors; ++u) {
    const Tensor& U = P.t[u];
    bool reads = false, row_only = true;
    for (int a = 0; a < U.nargs; ++a) {
      if (U.args[a] != t) continue;
      reads = true;
      row_only = row_only && a == 0;
    }
    if (!reads) continue;
    if (!(U.kind == K_CONTRACT && (U.flags & TF_GEMM) && row_only && tc_row_side_all_image(P, u)))
      return true;
  }
  return false;
}

// One operand of an elementwise equation, read once per kernel from the
// program: its key array, its size, and its flat-index stride per output dim
// (zero along broadcast dims).
struct OpSrc {
  const uint2* p;
  uint64_t numel;
  int64_t os[MR];
};

__device__ __forceinline__ OpSrc op_src(const Prog& P, const Tensor& T, int s, bool broadcast,
                                       const uint2* leafk, const uint2* vals) {
  const Tensor& A = P.t[T.args[s]];
  OpSrc r;
  r.p = A.kind == K_INPUT ? leafk + A.gbase : vals + A.ws_off;
  r.numel = (uint64_t)A.numel;
#pragma unroll
  for (int d = 0; d < MR; ++d) r.os[d] = broadcast ? 0 : (d < T.rank ? T.stride[d] : 0);
  if (broadcast) {
#pragma unroll
    for (int d = 0; d < MR; ++d) {
      if (d < T.arg_rank[s] && A.shape[d] != 1) {
        const int od = T.axes[s][d];
#pragma unroll
        for (int e = 0; e < MR; ++e)
          if (e == od) r.os[e] += A.stride[d];
      }
    }
  }
  return r;
}

__device__ __forceinline__ uint2 op_key(const OpSrc& s, const int32_t* o, uint2 bot) {
  int64_t idx = 0;
#pragma unroll
  for (int d = 0; d < MR; ++d) idx += s.os[d] * o[d];
  return (uint64_t)idx < s.numel ? s.p[idx] : bot;
}

constexpr int kElemPerThread = 4;

// kElemPerThread consecutive elements per thread: one coordinate
// decomposition, then the innermost coordinate steps with carries.  The
// equation's operands and constants are read from the program once.
__global__ void elem_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                 uint2* vals) {
  const Tensor& T = P.t[t];
  const int64_t numel = T.numel;
  int64_t e = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * kElemPerThread;
  if (e >= numel) return;
  const int kind = T.kind, fn = T.fn, rank = T.rank;
  int32_t shape[MR];
#pragma unroll
  for (int d = 0; d < MR; ++d) shape[d] = d < rank ? T.shape[d] : 1;
  const uint2 bot = leafk[P.G];
  const bool bin = kind == K_BINARY;
  const OpSrc s0 = op_src(P, T, 0, bin, leafk, vals);
  OpSrc s1 = s0;
  if (bin) s1 = op_src(P, T, 1, true, leafk, vals);
  const KConst ca = T.a, cc = T.c;
  int ufid = fn;
  if (P.axiom_gelu && ufid == F_GELU_TANH) ufid = F_GELU_ERF;
  uint2* out = vals + T.ws_off;
  int32_t o[MR];
  unflatten(e, T, o);
#pragma unroll
  for (int u = 0; u < kElemPerThread; ++u) {
    if (e + u < numel) {
      const uint2 a = op_key(s0, o, bot);
      uint2 r;
      if (bin) {
        const uint2 b = op_key(s1, o, bot);
        if (fn == B_ADD) {
          r = make_uint2(addmod<0>(a.x, b.x), addmod<1>(a.y, b.y));
        } else if (fn == B_SUB) {
          r = make_uint2(submod<0>(a.x, b.x), submod<1>(a.y, b.y));
        } else if (fn == B_MUL) {
          r = make_uint2(mulmod<0>(a.x, b.x), mulmod<1>(a.y, b.y));
        } else {  // a / b = a * recip(b)
          uint32_t r0, r1;
          uf_key(F_RECIP, b.x, b.y, r0, r1);
          r = make_uint2(mulmod<0>(a.x, r0), mulmod<1>(a.y, r1));
        }
      } else if (kind == K_UNARY) {
        uf_key(ufid, a.x, a.y, r.x, r.y);
      } else if (kind == K_AFFINE) {
        r.x = addmod<0>(mulmod<0>(a.x, ca.k0), cc.k0);
        r.y = addmod<1>(mulmod<1>(a.y, ca.k1), cc.k1);
      } else {  // MAXC: Max{a, c}
        uint64_t w[2] = {pack(a), (uint64_t)cc.k0 | ((uint64_t)cc.k1 << 32)};
        if (w[0] > w[1]) {
          const uint64_t x = w[0];
          w[0] = w[1];
          w[1] = x;
        }
        maxset_key_sorted(w, w[0] == w[1] ? 1 : 2, r.x, r.y);
      }
      out[e + u] = r;
    }
    bool carry = true;
#pragma unroll
    for (int d = MR - 1; d >= 0; --d) {
      if (d < rank && carry) {
        if (++o[d] < shape[d])
          carry = false;
        else
          o[d] = 0;
      }
    }
  }
}

// Writes element e's key: its own, or, when its only reader is a UNARY
// (Tensor::unary_next), that UNARY's key of it into the reader's array.
__device__ __forceinline__ void put_key(const Prog& P, const Tensor& T, int64_t e, uint2 k,
                                        uint2* vals) {
  if (T.unary_next) {
    const Tensor& U = P.t[T.unary_next];
    int ufid = U.fn;
    if (P.axiom_gelu && ufid == F_GELU_TANH) ufid = F_GELU_ERF;
    uint2 r;
    uf_key(ufid, k.x, k.y, r.x, r.y);
    vals[U.ws_off + e] = r;
  } else {
    vals[T.ws_off + e] = k;
  }
}

template <int G>
__global__ void contract_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                     uint2* vals) {
  constexpr int W = 32 / G;
  const Tensor& T = P.t[t];
  const int lane = threadIdx.x & 31, j = lane % W, g = lane / W;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t e = warp * W + j;
  const bool valid = e < T.numel;
  if (warp * W >= T.numel) return;   // whole warp past the end (uniform)
  int32_t o[MR], r[MRED];
  unflatten(valid ? e : 0, T, o);
  uint32_t t0 = 0, t1 = 0;
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    if (!valid || !in_box(o, pc, T.rank) || red_empty(pc)) continue;
    int64_t K = 1;
    for (int d = 0; d < pc.nred; ++d) K *= pc.rhi[d] - pc.rlo[d];
    const int64_t ch = (K + G - 1) / G;
    int64_t k0 = g * ch, k1 = k0 + ch < K ? k0 + ch : K;
    if (k0 >= k1) continue;
    {
      int64_t x = k0;
      for (int d = MRED - 1; d >= 0; --d) {
        if (d < pc.nred) {
          int64_t qq, rr;
          divmod64(x, (int64_t)(pc.rhi[d] - pc.rlo[d]), qq, rr);
          r[d] = pc.rlo[d] + (int32_t)rr;
          x = qq;
        } else {
          r[d] = 0;
        }
      }
    }
    uint64_t s0 = 0, s1 = 0;
    if (T.nargs == 1 && pc.nguard == 0 && pc.nred == 1) {
      // a plain sum along one dim (softmax denominators, means): the terms
      // sit at a fixed stride, so eight loads are issued before any is used;
      // fewer than 2^31 terms below 2^29 keep the sums below 2^60
      const int64_t st = pc.acc[0].rs[0];
      int64_t off = access_off(pc.acc[0], o, r, T.rank, pc.nred);
      int64_t k = k0;
      for (; k + 8 <= k1; k += 8, off += 8 * st) {
        uint2 a[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) a[u] = fetch_key(P, T.args[0], off + u * st, leafk, vals);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          s0 += a[u].x;
          s1 += a[u].y;
        }
      }
      for (; k < k1; ++k, off += st) {
        const uint2 a = fetch_key(P, T.args[0], off, leafk, vals);
        s0 += a.x;
        s1 += a.y;
      }
      t0 = addmod<0>(t0, mulmod<0>(reduce<0>(s0), pc.coef.k0));
      t1 = addmod<1>(t1, mulmod<1>(reduce<1>(s1), pc.coef.k1));
      continue;
    }
    int cnt = 0;
    for (int64_t k = k0; k < k1; ++k) {
      if (guards_ok(pc, o, r)) {
        uint2 a = fetch_key(P, T.args[0], access_off(pc.acc[0], o, r, T.rank, pc.nred), leafk, vals);
        if (T.nargs == 2) {
          uint2 b = fetch_key(P, T.args[1], access_off(pc.acc[1], o, r, T.rank, pc.nred), leafk,
                              vals);
          a = make_uint2(mulmod<0>(a.x, b.x), mulmod<1>(a.y, b.y));
        }
        s0 += a.x;
        s1 += a.y;
        if (++cnt == 1 << 20) {
          s0 = fold<0>(s0);
          s1 = fold<1>(s1);
          cnt = 0;
        }
      }
      next_r(r, pc);
    }
    t0 = addmod<0>(t0, mulmod<0>(reduce<0>(s0), pc.coef.k0));
    t1 = addmod<1>(t1, mulmod<1>(reduce<1>(s1), pc.coef.k1));
  }
#pragma unroll
  for (int off = W; off < 32; off <<= 1) {
    t0 = addmod<0>(t0, __shfl_xor_sync(0xffffffffu, t0, off));
    t1 = addmod<1>(t1, __shfl_xor_sync(0xffffffffu, t1, off));
  }
  if (valid && g == 0) put_key(P, T, e, make_uint2(t0, t1), vals);
}

// The member keys are collected into a register list of CAP entries (CAP >=
// the tensor's term bound; free entries hold the largest value), sorted once
// by an odd-even transposition network with compile-time indices, and
// deduplicated while the key chain runs over them.
template <int CAP>
__global__ void maxset_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                   uint2* vals) {
  const Tensor& T = P.t[t];
  int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= T.numel) return;
  int32_t o[MR], r[MRED];
  unflatten(e, T, o);
  uint64_t u[CAP];
#pragma unroll
  for (int i = 0; i < CAP; ++i) u[i] = ~0ull;
  int n = 0;
  const Tensor& A = P.t[T.args[0]];
  const uint2* src = A.kind == K_INPUT ? leafk + A.gbase : vals + A.ws_off;
  const uint64_t anum = (uint64_t)A.numel;
  const uint64_t botk = pack(leafk[P.G]);
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    if (!in_box(o, pc, T.rank) || red_empty(pc)) continue;
    for (int i = 0; i < MRED; ++i) r[i] = pc.rlo[i];
    // the operand offset follows the reduction digits: +rs[e] per step of
    // digit e, -rs[e] * (extent - 1) when it wraps
    int64_t off = access_off(pc.acc[0], o, r, T.rank, pc.nred);
    bool more = true;
    while (more) {
      if ((pc.nguard == 0 || guards_ok(pc, o, r)) && n < CAP) {
        const uint64_t x = (uint64_t)off < anum ? pack(src[off]) : botk;
#pragma unroll
        for (int i = 0; i < CAP; ++i)
          if (i == n) u[i] = x;
        ++n;
      }
      bool carry = true;
#pragma unroll
      for (int d = MRED - 1; d >= 0; --d) {
        if (d < pc.nred && carry) {
          if (++r[d] < pc.rhi[d]) {
            off += pc.acc[0].rs[d];
            carry = false;
          } else {
            off -= pc.acc[0].rs[d] * (int64_t)(pc.rhi[d] - 1 - pc.rlo[d]);
            r[d] = pc.rlo[d];
          }
        }
      }
      more = !carry;
    }
  }
#pragma unroll
  for (int rd = 0; rd < CAP; ++rd) {
#pragma unroll
    for (int i = rd & 1; i + 1 < CAP; i += 2) {
      const uint64_t x = u[i], y = u[i + 1];
      u[i] = x < y ? x : y;
      u[i + 1] = x < y ? y : x;
    }
  }
  uint64_t h = kMaxTag;
  int m = 0;
#pragma unroll
  for (int i = 0; i < CAP; ++i) {
    if (i < n && (i == 0 || u[i] != u[i - 1])) {
      h = mix64(h ^ u[i]);
      ++m;
    }
  }
  uint2 out = make_uint2(0, 0);
  if (m == 1)
    out = make_uint2((uint32_t)(u[0] & 0xffffffffu), (uint32_t)(u[0] >> 32));
  else if (m > 1)
    out = make_uint2(reduce<0>(mix64(h ^ kSigma0)), reduce<1>(mix64(h ^ kSigma1)));
  put_key(P, T, e, out, vals);
}

// MAXSET with more than 32 terms per element (a max over a long dim): one
// block per element.  The block's threads enumerate the element's terms in
// parallel (term j: piece q where the pieces' reduction boxes, in order,
// reach j; reduction digits row-major), load the members' keys into shared
// memory (unused slots hold the largest value, which no key packs to),
// sort them with a bitonic network, and one thread runs the key chain over
// the distinct members in ascending order.
constexpr int kMaxsetLong = 4096;

__global__ void __launch_bounds__(256) maxset_long_keys_kernel(const __grid_constant__ Prog P,
                                                               int t, const uint2* leafk,
                                                               uint2* vals) {
  __shared__ uint64_t su[kMaxsetLong];
  const Tensor& T = P.t[t];
  const Tensor& A = P.t[T.args[0]];
  const uint2* src = A.kind == K_INPUT ? leafk + A.gbase : vals + A.ws_off;
  const uint64_t anum = (uint64_t)A.numel;
  const uint64_t botk = pack(leafk[P.G]);
  int p2 = 1;
  while (p2 < T.max_terms) p2 <<= 1;   // max_terms <= kMaxsetLong (checked by the host)
  for (int64_t e = blockIdx.x; e < T.numel; e += gridDim.x) {
    int32_t o[MR];
    unflatten(e, T, o);
    for (int j = threadIdx.x; j < p2; j += blockDim.x) {
      uint64_t x = ~0ull;
      int64_t jj = j;
      for (int q = 0; q < T.npieces && j < T.max_terms; ++q) {
        const Piece& pc = P.p[T.piece0 + q];
        int64_t vol = 1;
        for (int d = 0; d < pc.nred; ++d) vol *= max(0, pc.rhi[d] - pc.rlo[d]);
        if (jj >= vol) {
          jj -= vol;
          continue;
        }
        if (in_box(o, pc, T.rank)) {
          int32_t r[MRED] = {0, 0, 0, 0};
          int64_t rest = jj;
          for (int d = pc.nred - 1; d >= 0; --d) {
            const int64_t ext = pc.rhi[d] - pc.rlo[d];
            r[d] = pc.rlo[d] + (int32_t)(rest % ext);
            rest /= ext;
          }
          if (pc.nguard == 0 || guards_ok(pc, o, r)) {
            const int64_t off = access_off(pc.acc[0], o, r, T.rank, pc.nred);
            x = (uint64_t)off < anum ? pack(src[off]) : botk;
          }
        }
        break;
      }
      su[j] = x;
    }
    __syncthreads();
    for (int k = 2; k <= p2; k <<= 1) {
      for (int h = k >> 1; h > 0; h >>= 1) {
        for (int i = threadIdx.x; i < p2; i += blockDim.x) {
          const int l = i ^ h;
          if (l > i) {
            const uint64_t a = su[i], b = su[l];
            if ((a > b) == ((i & k) == 0)) {
              su[i] = b;
              su[l] = a;
            }
          }
        }
        __syncthreads();
      }
    }
    if (threadIdx.x == 0) {
      uint64_t hsh = kMaxTag, first = ~0ull, prev = ~0ull;
      int m = 0;
      for (int i = 0; i < p2 && su[i] != ~0ull; ++i) {
        const uint64_t u = su[i];
        if (u == prev) continue;
        if (m == 0) first = u;
        hsh = mix64(hsh ^ u);
        prev = u;
        ++m;
      }
      uint2 out = make_uint2(0, 0);
      if (m == 1)
        out = make_uint2((uint32_t)(first & 0xffffffffu), (uint32_t)(first >> 32));
      else if (m > 1)
        out = make_uint2(reduce<0>(mix64(hsh ^ kSigma0)), reduce<1>(mix64(hsh ^ kSigma1)));
      put_key(P, T, e, out, vals);
    }
    __syncthreads();
  }
}

// MAXSET of one guard-free piece that covers the whole output: the members
// of every element sit at the same offsets relative to the element's first
// member (row-major over the reduction box), so each thread forms those
// offsets once and each element costs its base offset and CAP loads.
template <int CAP>
__device__ __forceinline__ void sort_net(uint64_t* u) {
  if (CAP == 4) {   // the optimal 5-comparator network
    const int pa[5] = {0, 2, 0, 1, 1}, pb[5] = {1, 3, 2, 3, 2};
#pragma unroll
    for (int k = 0; k < 5; ++k) {
      const uint64_t x = u[pa[k]], y = u[pb[k]];
      u[pa[k]] = x < y ? x : y;
      u[pb[k]] = x < y ? y : x;
    }
    return;
  }
#pragma unroll
  for (int rd = 0; rd < CAP; ++rd) {
#pragma unroll
    for (int i = rd & 1; i + 1 < CAP; i += 2) {
      const uint64_t x = u[i], y = u[i + 1];
      u[i] = x < y ? x : y;
      u[i + 1] = x < y ? y : x;
    }
  }
}

// Each thread takes EPT consecutive elements: the members' offsets relative
// to an element's first member are formed once per thread, the coordinates
// of the first element by division and those of the next ones by carrying
// the last coordinate.
template <int CAP, int EPT>
__global__ void __launch_bounds__(256) maxset_box_keys_kernel(const __grid_constant__ Prog P, int t,
                                                              const uint2* leafk, uint2* vals) {
  const Tensor& T = P.t[t];
  const int64_t e_first = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * EPT;
  if (e_first >= T.numel) return;
  const Piece& pc = P.p[T.piece0];
  const int nred = pc.nred;
  int64_t rel[CAP];
  int vol = 0;
  {
    int32_t r[MRED];
    int64_t off = 0;
#pragma unroll
    for (int d = 0; d < MRED; ++d) r[d] = pc.rlo[d];
    bool more = true;
#pragma unroll
    for (int j = 0; j < CAP; ++j) {
      rel[j] = off;
      if (more) ++vol;
      bool carry = more;
#pragma unroll
      for (int d = MRED - 1; d >= 0; --d) {
        if (d < nred && carry) {
          if (++r[d] < pc.rhi[d]) {
            off += pc.acc[0].rs[d];
            carry = false;
          } else {
            off -= pc.acc[0].rs[d] * (int64_t)(pc.rhi[d] - 1 - pc.rlo[d]);
            r[d] = pc.rlo[d];
          }
        }
      }
      more = more && !carry;
    }
  }
  int64_t rbase = pc.acc[0].base;
#pragma unroll
  for (int d = 0; d < MRED; ++d)
    if (d < nred) rbase += pc.acc[0].rs[d] * pc.rlo[d];
  const Tensor& A = P.t[T.args[0]];
  const uint2* src = A.kind == K_INPUT ? leafk + A.gbase : vals + A.ws_off;
  const uint64_t anum = (uint64_t)A.numel;
  const uint64_t botk = pack(leafk[P.G]);
  int32_t o[MR];
  unflatten(e_first, T, o);
#pragma unroll
  for (int q = 0; q < EPT; ++q) {
    const int64_t e = e_first + q;
    if (e >= T.numel) break;
    if (q > 0) {   // next coordinates: carry from the last dim
      bool carry = true;
#pragma unroll
      for (int d = MR - 1; d >= 0; --d) {
        if (d < T.rank && carry) {
          if (++o[d] < T.shape[d]) {
            carry = false;
          } else {
            o[d] = 0;
          }
        }
      }
    }
    int64_t off0 = rbase;
#pragma unroll
    for (int d = 0; d < MR; ++d)
      if (d < T.rank) off0 += pc.acc[0].os[d] * o[d];
    uint64_t u[CAP];
#pragma unroll
    for (int j = 0; j < CAP; ++j) {
      const uint64_t off = (uint64_t)(off0 + rel[j]);
      u[j] = j >= vol ? ~0ull : off < anum ? pack(src[off]) : botk;
    }
    sort_net<CAP>(u);
    uint64_t h = kMaxTag;
    int m = 0;
#pragma unroll
    for (int i = 0; i < CAP; ++i) {
      if (i < vol && (i == 0 || u[i] != u[i - 1])) {
        h = mix64(h ^ u[i]);
        ++m;
      }
    }
    uint2 out = make_uint2(0, 0);
    if (m == 1)
      out = make_uint2((uint32_t)(u[0] & 0xffffffffu), (uint32_t)(u[0] >> 32));
    else if (m > 1)
      out = make_uint2(reduce<0>(mix64(h ^ kSigma0)), reduce<1>(mix64(h ^ kSigma1)));
    put_key(P, T, e, out, vals);
  }
}

// members per element when a MAXSET can use maxset_box_keys_kernel (one
// guard-free piece over the whole output, at most 8 members), else 0
static int64_t maxset_box_members(const Prog& P, const Tensor& T) {
  if (T.npieces != 1 || T.nargs != 1) return 0;
  const Piece& pc = P.p[T.piece0];
  if (pc.nguard != 0 || pc.nred < 1) return 0;
  int64_t vol = 1;
  for (int d = 0; d < pc.nred; ++d) {
    if (pc.rhi[d] <= pc.rlo[d]) return 0;
    vol *= pc.rhi[d] - pc.rlo[d];
  }
  for (int d = 0; d < T.rank; ++d)
    if (pc.lo[d] > 0 || pc.hi[d] < T.shape[d]) return 0;
  return vol <= 8 ? vol : 0;
}

__global__ void gather_keys_kernel(const __grid_constant__ Prog P, const int64_t* locs, int64_t n,
                                   const uint2* vals, uint2* keys) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const Tensor& T = P.t[P.output];
  int64_t l = locs[i];
  keys[i] = (l >= 0 && l < T.numel) ? vals[T.ws_off + l] : make_uint2(0, 0);
}

size_t terms_ws_bytes(const dirigo_graph* g) {
  size_t leaf = ((size_t)(g->prog.G + 1) * 8 + 255) / 256 * 256;
  size_t vals = ((size_t)g->value_elems * 8 + 255) / 256 * 256;
  return leaf + vals + tc_ws_bytes(g->prog) + 256;
}

static unsigned blocks_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  return (unsigned)(b < 1 ? 1 : b);
}

dirigo_status launch_terms(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                           uint32_t* d_keys, void* d_ws, cudaStream_t s) {
  const Prog& P = g->prog;
  char* ws = (char*)d_ws;
  uint2* leafk = (uint2*)ws;
  size_t leaf_bytes = ((size_t)(P.G + 1) * 8 + 255) / 256 * 256;
  uint2* vals = (uint2*)(ws + leaf_bytes);
  void* tc_ws = ws + leaf_bytes + ((size_t)g->value_elems * 8 + 255) / 256 * 256;
  // status word of the contraction kernels (non-zero: a bounded wait expired)
  int32_t* status = (int32_t*)((char*)tc_ws + tc_ws_bytes(P));
  cudaMemsetAsync(status, 0, 4, s);
  {
    // keys of the inputs some kernel reads from the array (merged id ranges),
    // and of bottom
    Prof pr(DIRIGO_K_KEY_LEAF, s);
    int64_t g0 = -1, g1 = -1;
    auto flush = [&]() {
      if (g1 > g0) {
        unsigned nb = blocks_for(g1 - g0, 256);
        if (nb > 152 * 16) nb = 152 * 16;
        leaf_keys_kernel<<<nb, 256, 0, s>>>(g0, g1, leafk);
        count_launch();
      }
      g0 = g1 = -1;
    };
    for (int t = 0; t < P.n_inputs; ++t) {
      if (!input_keys_read(P, t)) continue;
      const int64_t a = P.t[t].gbase, b = a + P.t[t].numel;
      if (a != g1) flush();
      if (g0 < 0) g0 = a;
      g1 = b;
    }
    if (g1 == P.G) {
      g1 = P.G + 1;   // bottom follows the last input
    } else {
      flush();
      g0 = P.G;
      g1 = P.G + 1;
    }
    flush();
  }
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    const Tensor& T = P.t[t];
    if (T.flags & TF_BY_GEMM) continue;       // written by its operand's contraction
    if (T.flags & TF_BY_PRODUCER) continue;   // written by its operand's kernel
    if (T.kind == K_CONTRACT && (T.flags & TF_GEMM)) {
      // timed per kernel class inside (limb matrices, contraction)
      dirigo_status st = launch_gemm_keys_tc(P, t, leafk, vals, tc_ws, status, s);
      if (st != DIRIGO_OK) return st;
      continue;
    } else {
      Prof pr(DIRIGO_K_KEY_ELEM, s);
      unsigned nb = blocks_for(T.numel, 256);
      if (T.kind == K_CONTRACT) {
        // threads per element: enough threads in flight, at most the term bound
        int G = 1;
        while (G < 32 && T.numel * G < (int64_t)1 << 19 && G < T.max_terms) G <<= 1;
        const unsigned cb = blocks_for(T.numel * G, 256);
        switch (G) {
          case 1: contract_keys_kernel<1><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
          case 2: contract_keys_kernel<2><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
          case 4: contract_keys_kernel<4><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
          case 8: contract_keys_kernel<8><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
          case 16: contract_keys_kernel<16><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
          default: contract_keys_kernel<32><<<cb, 256, 0, s>>>(P, t, leafk, vals); break;
        }
      } else if (T.kind == K_MAXSET && maxset_box_members(P, T) > 0) {
        const unsigned nb4 = blocks_for((T.numel + 3) / 4, 256);
        if (maxset_box_members(P, T) <= 4)
          maxset_box_keys_kernel<4, 4><<<nb4, 256, 0, s>>>(P, t, leafk, vals);
        else
          maxset_box_keys_kernel<8, 4><<<nb4, 256, 0, s>>>(P, t, leafk, vals);
      } else if (T.kind == K_MAXSET && T.max_terms > 32) {
        const int64_t lb = std::min<int64_t>(T.numel, 152 * 16);
        maxset_long_keys_kernel<<<(unsigned)std::max<int64_t>(lb, 1), 256, 0, s>>>(P, t, leafk,
                                                                                  vals);
      } else if (T.kind == K_MAXSET) {
        if (T.max_terms <= 4)
          maxset_keys_kernel<4><<<nb, 256, 0, s>>>(P, t, leafk, vals);
        else if (T.max_terms <= 8)
          maxset_keys_kernel<8><<<nb, 256, 0, s>>>(P, t, leafk, vals);
        else if (T.max_terms <= 16)
          maxset_keys_kernel<16><<<nb, 256, 0, s>>>(P, t, leafk, vals);
        else
          maxset_keys_kernel<32><<<nb, 256, 0, s>>>(P, t, leafk, vals);
      } else {
        elem_keys_kernel<<<blocks_for((T.numel + kElemPerThread - 1) / kElemPerThread, 256), 256,
                           0, s>>>(P, t, leafk, vals);
      }
    }
    count_launch();
  }
  {
    Prof pr(DIRIGO_K_KEY_ELEM, s);
    gather_keys_kernel<<<blocks_for(n, 256), 256, 0, s>>>(P, d_locs, n, vals, (uint2*)d_keys);
    count_launch();
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  return DIRIGO_OK;
}

}  // namespace dirigo
