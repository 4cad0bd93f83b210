// Integer-ALU peaks of the key arithmetic, measured on the GPU the library
// runs on: the denominators of the rooflines of the key kernels that run on
// the CUDA cores (the paper has no counterpart: it decides equality with a
// solver; these rates only put the key kernels' times in proportion).
//
//   mix64 / s    SplitMix64 output finalisers (keyspec.cuh's mix64, the atom
//                mixing of leaf, function and max-set keys): every thread runs
//                8 independent chains z = mix64(z + c);
//   mad.wide / s 32 x 32 -> 64-bit multiply-adds (the lane multiply-add of a
//                modular dot product, acc += a * b): every thread runs 8
//                independent accumulator chains.
//
// Each rate is the work of one launch of 152 x 8 blocks of 256 threads divided
// by its CUDA-event time on the caller's stream, best of three launches.  The
// results land in a file-scope device word so that no chain is dead code.
#include <cuda_runtime.h>

#include "internal.h"
#include "keyspec.cuh"
#include "launch.h"

namespace dirigo {

namespace {

__device__ unsigned long long g_alu_sink;

constexpr int kAluChains = 8;
constexpr int kAluBlocks = 152 * 8, kAluThreads = 256;

__global__ void __launch_bounds__(kAluThreads) alu_mix_kernel(int iters) {
  uint64_t z[kAluChains];
  const uint64_t t = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
#pragma unroll
  for (int c = 0; c < kAluChains; ++c) z[c] = t * 8 + c;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kAluChains; ++c) z[c] = mix64(z[c] + (uint64_t)c);
  }
  uint64_t x = 0;
#pragma unroll
  for (int c = 0; c < kAluChains; ++c) x ^= z[c];
  if (x == 0x5EED) g_alu_sink = x;   // never true in practice; keeps the chains live
}

__global__ void __launch_bounds__(kAluThreads) alu_mad_kernel(int iters, uint32_t b) {
  uint64_t acc[kAluChains];
  uint32_t a[kAluChains];
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
#pragma unroll
  for (int c = 0; c < kAluChains; ++c) {
    acc[c] = 0;
    a[c] = t * 8u + (uint32_t)c;
  }
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kAluChains; ++c)
      asm volatile("mad.wide.u32 %0, %1, %2, %0;" : "+l"(acc[c]) : "r"(a[c]), "r"(b));
  }
  uint64_t x = 0;
#pragma unroll
  for (int c = 0; c < kAluChains; ++c) x ^= acc[c];
  if (x == 0x5EED) g_alu_sink = x;
}

}  // namespace

}  // namespace dirigo

using namespace dirigo;

extern "C" dirigo_status dirigo_alu_peak(double* mix64_per_s, double* madwide_per_s,
                                         void* stream) {
  if (!mix64_per_s || !madwide_per_s) return set_error(DIRIGO_E_INVALID, "NULL argument");
  cudaStream_t s = (cudaStream_t)stream;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
    if (e0) cudaEventDestroy(e0);
    return set_error(DIRIGO_E_CUDA, cudaGetErrorString(cudaGetLastError()));
  }
  const double per_launch = (double)kAluBlocks * kAluThreads * kAluChains;
  double best[2] = {0, 0};
  cudaError_t e = cudaSuccess;
  for (int which = 0; which < 2 && e == cudaSuccess; ++which) {
    const int iters = which == 0 ? 2048 : 16384;
    for (int rep = 0; rep < 4 && e == cudaSuccess; ++rep) {   // the first is a warm-up
      e = cudaEventRecord(e0, s);
      if (which == 0)
        alu_mix_kernel<<<kAluBlocks, kAluThreads, 0, s>>>(iters);
      else
        alu_mad_kernel<<<kAluBlocks, kAluThreads, 0, s>>>(iters, 0x9E3779B9u);
      count_launch();
      if (e == cudaSuccess) e = cudaGetLastError();
      if (e == cudaSuccess) e = cudaEventRecord(e1, s);
      if (e == cudaSuccess) e = cudaEventSynchronize(e1);
      float ms = 0.0f;
      if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
      if (e == cudaSuccess && rep > 0 && ms > 0.0f) {
        const double rate = per_launch * iters / (ms * 1e-3);
        if (rate > best[which]) best[which] = rate;
      }
    }
  }
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  *mix64_per_s = best[0];
  *madwide_per_s = best[1];
  return DIRIGO_OK;
}
