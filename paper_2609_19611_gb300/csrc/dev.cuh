// Device helpers shared by the kernels (library-internal).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "keyspec.cuh"
#include "prog.h"

namespace dirigo {

// q = a / b, r = a % b for a >= 0, b > 0, in 32-bit arithmetic when both fit
__device__ __forceinline__ void divmod64(int64_t a, int64_t b, int64_t& q, int64_t& r) {
  if ((((uint64_t)a) | ((uint64_t)b)) < (1ull << 32)) {
    uint32_t qq = (uint32_t)a / (uint32_t)b;
    q = qq;
    r = (int64_t)((uint32_t)a - qq * (uint32_t)b);
  } else {
    q = a / b;
    r = a - q * b;
  }
}

// flat element index -> coordinates (row-major)
__device__ __forceinline__ void unflatten(int64_t e, const Tensor& T, int32_t* o) {
  if (e < ((int64_t)1 << 32)) {
    uint32_t x = (uint32_t)e;
#pragma unroll
    for (int d = MR - 1; d >= 0; --d) {
      if (d < T.rank) {
        uint32_t q = x / (uint32_t)T.shape[d];
        o[d] = (int32_t)(x - q * (uint32_t)T.shape[d]);
        x = q;
      } else {
        o[d] = 0;
      }
    }
    return;
  }
#pragma unroll
  for (int d = MR - 1; d >= 0; --d) {
    if (d < T.rank) {
      int64_t q = e / T.shape[d];
      o[d] = (int32_t)(e - q * T.shape[d]);
      e = q;
    } else {
      o[d] = 0;
    }
  }
}

__device__ __forceinline__ bool in_box(const int32_t* o, const Piece& pc, int rank) {
  bool in = true;
#pragma unroll
  for (int d = 0; d < MR; ++d)
    if (d < rank) in &= (o[d] >= pc.lo[d]) & (o[d] < pc.hi[d]);
  return in;
}

// flat offset of operand i of a piece at (o, r)
__device__ __forceinline__ int64_t access_off(const Access& a, const int32_t* o, const int32_t* r,
                                              int rank, int nred) {
  int64_t off = a.base;
#pragma unroll
  for (int d = 0; d < MR; ++d)
    if (d < rank) off += a.os[d] * o[d];
#pragma unroll
  for (int e = 0; e < MRED; ++e)
    if (e < nred) off += a.rs[e] * r[e];
  return off;
}

// a[i] for a runtime i < 4 without indexing the array at run time (so a
// register array stays in registers)
__device__ __forceinline__ int32_t sel4(const int32_t* a, int i) {
  int32_t v = a[0];
  v = i == 1 ? a[1] : v;
  v = i == 2 ? a[2] : v;
  v = i == 3 ? a[3] : v;
  return v;
}

// a[i] = v for a runtime i < 4, without indexing the array at run time
__device__ __forceinline__ void set4(int32_t* a, int i, int32_t v) {
  a[0] = i == 0 ? v : a[0];
  a[1] = i == 1 ? v : a[1];
  a[2] = i == 2 ? v : a[2];
  a[3] = i == 3 ? v : a[3];
}

__device__ __forceinline__ bool guards_ok(const Piece& pc, const int32_t* o, const int32_t* r) {
  bool ok = true;
#pragma unroll
  for (int j = 0; j < MG; ++j) {
    if (j < pc.nguard) {
      const Guard& g = pc.g[j];
      int32_t v = g.c;
      if (g.od >= 0) v += g.oa * sel4(o, g.od);
      if (g.rd >= 0) v += sel4(r, g.rd);
      ok &= (v >= g.lo) & (v < g.hi);
    }
  }
  return ok;
}

// advance reduction coordinates row-major; false when the box is exhausted
// next reduction coordinates in row-major order; false after the last.
// Unrolled over MRED so that r stays in registers.
__device__ __forceinline__ bool next_r(int32_t* r, const Piece& pc) {
  bool carry = true;
#pragma unroll
  for (int e = MRED - 1; e >= 0; --e) {
    if (e < pc.nred && carry) {
      if (++r[e] < pc.rhi[e]) {
        carry = false;
      } else {
        r[e] = pc.rlo[e];
      }
    }
  }
  return !carry;
}

__device__ __forceinline__ bool red_empty(const Piece& pc) {
  bool empty = false;
  for (int e = 0; e < pc.nred; ++e) empty |= pc.rlo[e] >= pc.rhi[e];
  return empty;
}

// flat index into operand s of a BINARY op at output coordinates o
__device__ __forceinline__ int64_t bin_index(const Prog& P, const Tensor& T, int s,
                                             const int32_t* o) {
  const Tensor& A = P.t[T.args[s]];
  int64_t idx = 0;
#pragma unroll
  for (int d = 0; d < MR; ++d)
    if (d < T.arg_rank[s] && A.shape[d] != 1) idx += A.stride[d] * sel4(o, T.axes[s][d]);
  return idx;
}

__device__ __forceinline__ uint64_t pack(uint2 k) { return (uint64_t)k.x | ((uint64_t)k.y << 32); }

// key of element `off` of tensor `t` (bottom when off is out of range)
__device__ __forceinline__ uint2 fetch_key(const Prog& P, int t, int64_t off, const uint2* leafk,
                                           const uint2* vals) {
  const Tensor& A = P.t[t];
  if (off < 0 || off >= A.numel) return leafk[P.G];
  if (A.kind == K_INPUT) return leafk[A.gbase + off];
  return vals[A.ws_off + off];
}

}  // namespace dirigo
