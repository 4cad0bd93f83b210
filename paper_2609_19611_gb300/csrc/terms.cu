// Term keys: forward evaluation of every primitive tensor's per-element
// equation in F_p0 x F_p1, one key pair per element (memoisation per
// (tensor, element) is hash-consing of the shared subterms, Sec. 3.4
// "Back-projection": every T_j[l'] in f_k(l) is resolved once).
//
// Kernels:
//   leaf_keys      key of every global input id (and of bottom, id G)
//   gemm_keys      two-operand CONTRACT as a tiled implicit GEMM over F_p:
//                  operand tiles are gathered through the piece's access map
//                  (guards and pieces masked to zero) into shared memory, and
//                  each thread keeps a 4x4 block of 64-bit lazy accumulators
//                  per lane (products < 2^58, folded every 32 steps)
//   contract_keys  one-operand CONTRACT (sums, means), one thread per element
//   maxset_keys    MAXSET: collect, sort and deduplicate the members' keys
//   elem_keys      UNARY / MAXC / AFFINE / BINARY
//   gather_keys    root keys of the queried locations
#include <cstdint>

#include "dev.cuh"
#include "internal.h"
#include "launch.h"

namespace dirigo {

__global__ void leaf_keys_kernel(int64_t G, uint2* leafk) {
  int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (; g <= G; g += stride) leafk[g] = make_uint2(leaf_key0((uint64_t)g), leaf_key1((uint64_t)g));
}

__global__ void elem_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                 uint2* vals) {
  const Tensor& T = P.t[t];
  int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= T.numel) return;
  int32_t o[MR];
  unflatten(e, T, o);
  uint2 out;
  if (T.kind == K_BINARY) {
    uint2 a = fetch_key(P, T.args[0], bin_index(P, T, 0, o), leafk, vals);
    uint2 b = fetch_key(P, T.args[1], bin_index(P, T, 1, o), leafk, vals);
    switch (T.fn) {
      case B_ADD: out = make_uint2(addmod<0>(a.x, b.x), addmod<1>(a.y, b.y)); break;
      case B_SUB: out = make_uint2(submod<0>(a.x, b.x), submod<1>(a.y, b.y)); break;
      case B_MUL: out = make_uint2(mulmod<0>(a.x, b.x), mulmod<1>(a.y, b.y)); break;
      default: {  // a / b = a * recip(b)
        uint32_t r0, r1;
        uf_key(F_RECIP, b.x, b.y, r0, r1);
        out = make_uint2(mulmod<0>(a.x, r0), mulmod<1>(a.y, r1));
      }
    }
  } else {
    uint2 a = fetch_key(P, T.args[0], e, leafk, vals);
    if (T.kind == K_UNARY) {
      int fid = T.fn;
      if (P.axiom_gelu && fid == F_GELU_TANH) fid = F_GELU_ERF;
      uf_key(fid, a.x, a.y, out.x, out.y);
    } else if (T.kind == K_AFFINE) {
      out.x = addmod<0>(mulmod<0>(a.x, T.a.k0), T.c.k0);
      out.y = addmod<1>(mulmod<1>(a.y, T.a.k1), T.c.k1);
    } else {  // MAXC: Max{a, c}
      uint64_t u[2] = {pack(a), (uint64_t)T.c.k0 | ((uint64_t)T.c.k1 << 32)};
      if (u[0] > u[1]) {
        uint64_t x = u[0];
        u[0] = u[1];
        u[1] = x;
      }
      maxset_key_sorted(u, u[0] == u[1] ? 1 : 2, out.x, out.y);
    }
  }
  vals[T.ws_off + e] = out;
}

__global__ void contract_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                     uint2* vals) {
  const Tensor& T = P.t[t];
  int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= T.numel) return;
  int32_t o[MR], r[MRED];
  unflatten(e, T, o);
  uint32_t t0 = 0, t1 = 0;
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    if (!in_box(o, pc, T.rank) || red_empty(pc)) continue;
    for (int j = 0; j < MRED; ++j) r[j] = pc.rlo[j];
    uint64_t s0 = 0, s1 = 0;
    int cnt = 0;
    do {
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
    } while (next_r(r, pc));
    t0 = addmod<0>(t0, mulmod<0>(reduce<0>(s0), pc.coef.k0));
    t1 = addmod<1>(t1, mulmod<1>(reduce<1>(s1), pc.coef.k1));
  }
  vals[T.ws_off + e] = make_uint2(t0, t1);
}

__global__ void maxset_keys_kernel(const __grid_constant__ Prog P, int t, const uint2* leafk,
                                   uint2* vals) {
  const Tensor& T = P.t[t];
  int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= T.numel) return;
  int32_t o[MR], r[MRED];
  unflatten(e, T, o);
  uint64_t u[32];
  int n = 0;
  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    if (!in_box(o, pc, T.rank) || red_empty(pc)) continue;
    for (int j = 0; j < MRED; ++j) r[j] = pc.rlo[j];
    do {
      if (guards_ok(pc, o, r) && n < 32) {
        uint64_t x = pack(fetch_key(P, T.args[0], access_off(pc.acc[0], o, r, T.rank, pc.nred),
                                    leafk, vals));
        // insertion into the sorted distinct list
        int i = n;
        bool dup = false;
        while (i > 0 && u[i - 1] >= x) {
          if (u[i - 1] == x) {
            dup = true;
            break;
          }
          --i;
        }
        if (!dup) {
          for (int j = n; j > i; --j) u[j] = u[j - 1];
          u[i] = x;
          ++n;
        }
      }
    } while (next_r(r, pc));
  }
  uint2 out = make_uint2(0, 0);
  if (n > 0) maxset_key_sorted(u, n, out.x, out.y);
  vals[T.ws_off + e] = out;
}

// ---------------------------------------------------------------- GEMM over F_p
namespace {

constexpr int GBM = 64, GBN = 64, GBK = 16;

struct DimSplit {
  int nd;
  int dims[MR];
  int64_t count;
};

__device__ __forceinline__ DimSplit split_of(const Tensor& T, int mask) {
  DimSplit s;
  s.nd = 0;
  s.count = 1;
  for (int d = 0; d < T.rank; ++d)
    if (mask & (1 << d)) {
      s.dims[s.nd++] = d;
      s.count *= T.shape[d];
    }
  return s;
}

// write the coordinates of flat index x of a dim split into o
__device__ __forceinline__ void split_coords(const Tensor& T, const DimSplit& s, int64_t x,
                                             int32_t* o) {
  for (int i = s.nd - 1; i >= 0; --i) {
    int d = s.dims[i];
    int64_t q = x / T.shape[d];
    o[d] = (int32_t)(x - q * T.shape[d]);
    x = q;
  }
}

}  // namespace

__global__ void __launch_bounds__(256) gemm_keys_kernel(const __grid_constant__ Prog P, int t,
                                                        const uint2* leafk, uint2* vals) {
  const Tensor& T = P.t[t];
  __shared__ uint2 As[GBK][GBM];
  __shared__ uint2 Bs[GBK][GBN];
  __shared__ int64_t rowoff[GBM], coloff[GBN];
  __shared__ int32_t rowg[MG][GBM];
  __shared__ uint8_t rowok[GBM], colok[GBN];
  __shared__ int64_t koffA[GBK], koffB[GBK];
  __shared__ int32_t kg[MG][GBK];
  __shared__ uint8_t kok[GBK];
  __shared__ int32_t orow[GBM][MR], ocol[GBN][MR];

  const int tid = threadIdx.x;
  const DimSplit rs = split_of(T, T.row_mask), cs = split_of(T, T.col_mask),
                 bs = split_of(T, T.batch_mask);
  const int64_t row0 = (int64_t)blockIdx.x * GBM, col0 = (int64_t)blockIdx.y * GBN;
  int32_t ob[MR] = {0, 0, 0, 0};
  split_coords(T, bs, blockIdx.z, ob);

  // coordinates of the tile's rows and columns (batch dims filled in)
  if (tid < GBM) {
    int32_t o[MR];
    for (int d = 0; d < MR; ++d) o[d] = ob[d];
    int64_t row = row0 + tid;
    if (row < rs.count) split_coords(T, rs, row, o);
    for (int d = 0; d < MR; ++d) orow[tid][d] = o[d];
  } else if (tid < GBM + GBN) {
    int c = tid - GBM;
    int32_t o[MR];
    for (int d = 0; d < MR; ++d) o[d] = ob[d];
    int64_t col = col0 + c;
    if (col < cs.count) split_coords(T, cs, col, o);
    for (int d = 0; d < MR; ++d) ocol[c][d] = o[d];
  }

  const int tm = tid & 15, tn = tid >> 4;   // rows tm + 16 i, cols tn + 16 j
  uint32_t tot0[4][4], tot1[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) tot0[i][j] = tot1[i][j] = 0;

  for (int q = 0; q < T.npieces; ++q) {
    const Piece& pc = P.p[T.piece0 + q];
    // batch coordinates outside the piece: no term for this whole tile
    bool bin = true;
    for (int i = 0; i < bs.nd; ++i) {
      int d = bs.dims[i];
      bin &= ob[d] >= pc.lo[d] && ob[d] < pc.hi[d];
    }
    if (!bin || red_empty(pc)) continue;
    int64_t kvol = 1;
    for (int e = 0; e < pc.nred; ++e) kvol *= pc.rhi[e] - pc.rlo[e];
    __syncthreads();
    if (tid < GBM) {
      const int32_t* o = orow[tid];
      bool ok = row0 + tid < rs.count;
      int64_t off = 0;
      for (int i = 0; i < rs.nd; ++i) {
        int d = rs.dims[i];
        ok &= o[d] >= pc.lo[d] && o[d] < pc.hi[d];
      }
      for (int d = 0; d < T.rank; ++d) off += pc.acc[0].os[d] * o[d];
      rowoff[tid] = off;
      rowok[tid] = ok;
      for (int j = 0; j < MG; ++j) {
        int32_t v = 0;
        if (j < pc.nguard) {
          v = pc.g[j].c;
          if (pc.g[j].od >= 0) v += pc.g[j].oa * o[pc.g[j].od];
        }
        rowg[j][tid] = v;
      }
    } else if (tid < GBM + GBN) {
      int c = tid - GBM;
      const int32_t* o = ocol[c];
      bool ok = col0 + c < cs.count;
      int64_t off = 0;
      for (int i = 0; i < cs.nd; ++i) {
        int d = cs.dims[i];
        ok &= o[d] >= pc.lo[d] && o[d] < pc.hi[d];
      }
      for (int d = 0; d < T.rank; ++d) off += pc.acc[1].os[d] * o[d];
      coloff[c] = off;
      colok[c] = ok;
    }
    uint64_t acc0[4][4], acc1[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc0[i][j] = acc1[i][j] = 0;
    int steps = 0;
    for (int64_t k0 = 0; k0 < kvol; k0 += GBK) {
      __syncthreads();
      if (tid < GBK) {
        int64_t k = k0 + tid;
        int32_t r[MRED];
        bool ok = k < kvol;
        int64_t x = ok ? k : 0;
        for (int e = pc.nred - 1; e >= 0; --e) {
          int64_t ext = pc.rhi[e] - pc.rlo[e];
          int64_t qq = x / ext;
          r[e] = pc.rlo[e] + (int32_t)(x - qq * ext);
          x = qq;
        }
        int64_t a = 0, b = 0;
        for (int e = 0; e < pc.nred; ++e) {
          a += pc.acc[0].rs[e] * r[e];
          b += pc.acc[1].rs[e] * r[e];
        }
        koffA[tid] = a;
        koffB[tid] = b;
        kok[tid] = ok;
        for (int j = 0; j < MG; ++j) kg[j][tid] = (j < pc.nguard && pc.g[j].rd >= 0) ? r[pc.g[j].rd] : 0;
      }
      __syncthreads();
      // gather the operand tiles
      for (int idx = tid; idx < GBK * GBM; idx += 256) {
        int k = idx / GBM, m = idx % GBM;
        bool ok = rowok[m] && kok[k];
        for (int j = 0; j < MG; ++j)
          if (j < pc.nguard) {
            int32_t v = rowg[j][m] + kg[j][k];
            ok &= v >= pc.g[j].lo && v < pc.g[j].hi;
          }
        uint2 val = make_uint2(0, 0);
        if (ok) val = fetch_key(P, T.args[0], pc.acc[0].base + rowoff[m] + koffA[k], leafk, vals);
        As[k][m] = val;
      }
      for (int idx = tid; idx < GBK * GBN; idx += 256) {
        int k = idx / GBN, n = idx % GBN;
        uint2 val = make_uint2(0, 0);
        if (colok[n] && kok[k])
          val = fetch_key(P, T.args[1], pc.acc[1].base + coloff[n] + koffB[k], leafk, vals);
        Bs[k][n] = val;
      }
      __syncthreads();
#pragma unroll 4
      for (int k = 0; k < GBK; ++k) {
        uint2 a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) a[i] = As[k][tm + 16 * i];
#pragma unroll
        for (int j = 0; j < 4; ++j) b[j] = Bs[k][tn + 16 * j];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            acc0[i][j] += (uint64_t)a[i].x * b[j].x;
            acc1[i][j] += (uint64_t)a[i].y * b[j].y;
          }
      }
      steps += GBK;
      if (steps >= 32) {   // 32 products of < 2^58 on top of < 2^41 stay below 2^64
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            acc0[i][j] = fold<0>(acc0[i][j]);
            acc1[i][j] = fold<1>(acc1[i][j]);
          }
        steps = 0;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        tot0[i][j] = addmod<0>(tot0[i][j], mulmod<0>(reduce<0>(acc0[i][j]), pc.coef.k0));
        tot1[i][j] = addmod<1>(tot1[i][j], mulmod<1>(reduce<1>(acc1[i][j]), pc.coef.k1));
      }
  }
  // write back
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int m = tm + 16 * i;
    if (row0 + m >= rs.count) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int n = tn + 16 * j;
      if (col0 + n >= cs.count) continue;
      int64_t flat = 0;
      for (int d = 0; d < T.rank; ++d) {
        int32_t v = ((T.col_mask >> d) & 1) ? ocol[n][d] : orow[m][d];
        flat += T.stride[d] * v;
      }
      vals[T.ws_off + flat] = make_uint2(tot0[i][j], tot1[i][j]);
    }
  }
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
    Prof pr(DIRIGO_K_KEY_LEAF, s);
    int64_t work = P.G + 1;
    unsigned nb = blocks_for(work, 256);
    if (nb > 152 * 16) nb = 152 * 16;
    leaf_keys_kernel<<<nb, 256, 0, s>>>(P.G, leafk);
    count_launch();
  }
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    const Tensor& T = P.t[t];
    if (T.kind == K_CONTRACT && (T.flags & TF_GEMM)) {
      // timed per kernel class inside (limb matrices, contraction)
      dirigo_status st = launch_gemm_keys_tc(P, t, leafk, vals, tc_ws, status, s);
      if (st != DIRIGO_OK) return st;
      continue;
    } else {
      Prof pr(DIRIGO_K_KEY_ELEM, s);
      unsigned nb = blocks_for(T.numel, 256);
      if (T.kind == K_CONTRACT)
        contract_keys_kernel<<<nb, 256, 0, s>>>(P, t, leafk, vals);
      else if (T.kind == K_MAXSET)
        maxset_keys_kernel<<<nb, 256, 0, s>>>(P, t, leafk, vals);
      else
        elem_keys_kernel<<<nb, 256, 0, s>>>(P, t, leafk, vals);
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
