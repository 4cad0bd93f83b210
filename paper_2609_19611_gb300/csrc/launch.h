// Launch bookkeeping shared by the .cu files (library-internal).
#pragma once
#include <cuda_runtime.h>

#include "internal.h"

namespace dirigo {

// Records CUDA events around a region on `stream` when profiling is enabled.
struct Prof {
  int cls;
  cudaStream_t s;
  int slot;
  Prof(int c, cudaStream_t st);
  ~Prof();
};

void count_launch();

size_t terms_ws_bytes(const dirigo_graph* g);
size_t eval_ws_bytes(const dirigo_graph* g);
size_t cone_ws_bytes(const dirigo_graph* g, int64_t n);
size_t cone_ws_bytes_noplan(int64_t n);
size_t compare_ws_bytes(const dirigo_graph* r, const dirigo_graph* c, int64_t n);

dirigo_status launch_gemm_keys_tc(const Prog& P, int t, const uint2* leafk, uint2* vals,
                                  void* tc_ws, int32_t* status, cudaStream_t s);
size_t tc_ws_bytes(const Prog& P);
// contraction t reads its row side only through limb images (which form an
// input's keys from its global ids), on the tcgen05 path
bool tc_row_side_all_image(const Prog& P, int t);
void tc_work(const Prog& P, double* flops_per_lane, double* limb_bytes);
dirigo_status launch_terms(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                           uint32_t* d_keys, void* d_ws, cudaStream_t s);
dirigo_status launch_eval(const dirigo_graph* g, const float* const* d_inputs,
                          const int64_t* d_locs, int64_t n, float* d_out, void* d_ws,
                          cudaStream_t s);
dirigo_status launch_cone(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                          int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                          uint64_t* d_fp, int64_t* h_total, void* d_ws, cudaStream_t s,
                          bool plan_slots = true);
dirigo_status enqueue_cone(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                           int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                           uint64_t* d_fp, int32_t* status, void* d_ws, cudaStream_t s,
                           bool plan_slots = true);
// Status of a cone's latched error bits (DIRIGO_OK when none), with the message set.
dirigo_status cone_status_error(int32_t bits);
dirigo_status launch_compare(const dirigo_graph* ref, const dirigo_graph* cand,
                             const int64_t* d_locs, int64_t n, const uint32_t* d_kref,
                             const uint32_t* d_kcand, const int64_t* d_off_ref,
                             const uint32_t* d_runs_ref, const uint64_t* d_fp_ref,
                             const int64_t* d_off_cand, const uint32_t* d_runs_cand,
                             const uint64_t* d_fp_cand, const int32_t* d_cone_status,
                             cudaEvent_t cones_ready, uint8_t* d_verdict, uint8_t* d_flags,
                             int64_t budget, uint8_t* d_export, int64_t export_capacity,
                             dirigo_compare_stats* h_stats, void* d_ws, cudaStream_t s,
                             dirigo_compare_stats* async_stats = nullptr,
                             int32_t* async_status = nullptr);
dirigo_status launch_compare_empty(const int32_t* d_cone_status, dirigo_compare_stats* d_stats,
                                   int32_t* d_status, cudaStream_t s);

}  // namespace dirigo
