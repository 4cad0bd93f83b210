// Concrete fp32 evaluation of every primitive tensor (the semantics
// [[R_y(i)]]_x of Sec. 3.3 "Setup"), then a gather of the queried locations.
// Sums use compensated (Neumaier) fp32 accumulation; transcendentals are
// CUDA's own fp32 functions; a read of bottom gives NaN.
#include <cmath>
#include <cstdint>

#include "dev.cuh"
#include "internal.h"
#include "launch.h"

namespace dirigo {

struct InPtrs {
  const float* p[MT];
};

__device__ __forceinline__ float fetch_val(const Prog& P, const InPtrs& in, int t, int64_t off,
                                          const float* vals) {
  const Tensor& A = P.t[t];
  if (off < 0 || off >= A.numel) return __int_as_float(0x7fc00000);   // NaN: bottom
  if (A.kind == K_INPUT) return in.p[t][off];
  return vals[A.ws_off + off];
}

__device__ __forceinline__ float uf_val(int fid, float x) {
  switch (fid) {
    case F_EXP: return expf(x);
    case F_TANH: return tanhf(x);
    case F_GELU_ERF: return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
    case F_GELU_TANH: {
      float u = 0.79788456080286536f * (x + 0.044715f * x * x * x);
      return 0.5f * x * (1.0f + tanhf(u));
    }
    case F_ERF: return erff(x);
    case F_RSQRT: return 1.0f / sqrtf(x);
    case F_RECIP: return 1.0f / x;
    case F_SQRT: return sqrtf(x);
    case F_LOG: return logf(x);
  }
  return __int_as_float(0x7fc00000);
}

// Neumaier compensated accumulation
struct CSum {
  float s = 0.0f, c = 0.0f;
  __device__ __forceinline__ void add(float x) {
    float t = s + x;
    if (fabsf(s) >= fabsf(x))
      c += (s - t) + x;
    else
      c += (x - t) + s;
    s = t;
  }
  __device__ __forceinline__ float value() const { return s + c; }
};

__global__ void eval_elem_kernel(const __grid_constant__ Prog P, const __grid_constant__ InPtrs in,
                                 int t, float* vals) {
  const Tensor& T = P.t[t];
  int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= T.numel) return;
  int32_t o[MR], r[MRED];
  unflatten(e, T, o);
  float out;
  if (T.kind == K_CONTRACT || T.kind == K_MAXSET) {
    bool mx = T.kind == K_MAXSET;
    CSum acc;
    float m = -INFINITY;
    bool any = false, bot = false;
    for (int q = 0; q < T.npieces; ++q) {
      const Piece& pc = P.p[T.piece0 + q];
      if (!in_box(o, pc, T.rank) || red_empty(pc)) continue;
      for (int j = 0; j < MRED; ++j) r[j] = pc.rlo[j];
      CSum ps;
      do {
        if (guards_ok(pc, o, r)) {
          float a = fetch_val(P, in, T.args[0], access_off(pc.acc[0], o, r, T.rank, pc.nred), vals);
          if (mx) {
            if (isnan(a)) bot = true;
            m = any ? fmaxf(m, a) : a;
            any = true;
          } else {
            if (T.nargs == 2)
              a *= fetch_val(P, in, T.args[1], access_off(pc.acc[1], o, r, T.rank, pc.nred), vals);
            ps.add(a);
          }
        }
      } while (next_r(r, pc));
      if (!mx) acc.add(pc.coef.f * ps.value());
    }
    out = mx ? (bot ? __int_as_float(0x7fc00000) : m) : acc.value();
  } else if (T.kind == K_BINARY) {
    float a = fetch_val(P, in, T.args[0], bin_index(P, T, 0, o), vals);
    float b = fetch_val(P, in, T.args[1], bin_index(P, T, 1, o), vals);
    switch (T.fn) {
      case B_ADD: out = a + b; break;
      case B_SUB: out = a - b; break;
      case B_MUL: out = a * b; break;
      default: out = a / b;
    }
  } else {
    float a = fetch_val(P, in, T.args[0], e, vals);
    if (T.kind == K_UNARY)
      out = uf_val(T.fn, a);
    else if (T.kind == K_AFFINE)
      out = fmaf(T.a.f, a, T.c.f);
    else
      out = isnan(a) ? a : fmaxf(a, T.c.f);
  }
  vals[T.ws_off + e] = out;
}

__global__ void gather_vals_kernel(const __grid_constant__ Prog P, const int64_t* locs, int64_t n,
                                   const float* vals, float* out) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const Tensor& T = P.t[P.output];
  int64_t l = locs[i];
  out[i] = (l >= 0 && l < T.numel) ? vals[T.ws_off + l] : __int_as_float(0x7fc00000);
}

size_t eval_ws_bytes(const dirigo_graph* g) { return (size_t)g->value_elems * 4 + 256; }

dirigo_status launch_eval(const dirigo_graph* g, const float* const* d_inputs,
                          const int64_t* d_locs, int64_t n, float* d_out, void* d_ws,
                          cudaStream_t s) {
  const Prog& P = g->prog;
  InPtrs in;
  for (int t = 0; t < MT; ++t) in.p[t] = t < P.n_inputs ? d_inputs[t] : nullptr;
  float* vals = (float*)d_ws;
  for (int t = P.n_inputs; t < P.n_tensors; ++t) {
    Prof pr(DIRIGO_K_EVAL, s);
    int64_t nb = (P.t[t].numel + 255) / 256;
    eval_elem_kernel<<<(unsigned)nb, 256, 0, s>>>(P, in, t, vals);
    count_launch();
  }
  if (n > 0) {
    gather_vals_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(P, d_locs, n, vals, d_out);
    count_launch();
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  return DIRIGO_OK;
}

}  // namespace dirigo
