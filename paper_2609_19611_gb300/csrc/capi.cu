// C ABI entry points (declared in include/dirigo.h): argument checks,
// workspace sizing, error reporting, kernel timing.
#include <algorithm>
#include <atomic>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "cells.h"
#include "internal.h"
#include "launch.h"

namespace dirigo {

namespace {
thread_local std::string g_err;
std::atomic<int64_t> g_launches{0};

// kernel timing (off by default)
std::mutex g_prof_mu;
bool g_prof_on = false;
struct ProfRec {
  int cls;
  cudaEvent_t a, b;
};
std::vector<ProfRec> g_prof_recs;
std::vector<cudaEvent_t> g_event_pool;
double g_prof_ms[DIRIGO_K_COUNT_] = {0};
int64_t g_prof_n[DIRIGO_K_COUNT_] = {0};

cudaEvent_t take_event() {
  if (!g_event_pool.empty()) {
    cudaEvent_t e = g_event_pool.back();
    g_event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

void drain_locked() {
  for (auto& r : g_prof_recs) {
    float ms = 0.0f;
    if (cudaEventSynchronize(r.b) == cudaSuccess && cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess) {
      g_prof_ms[r.cls] += ms;
      g_prof_n[r.cls] += 1;
    }
    g_event_pool.push_back(r.a);
    g_event_pool.push_back(r.b);
  }
  g_prof_recs.clear();
}
}  // namespace

dirigo_status set_error(dirigo_status s, const std::string& msg) {
  g_err = msg;
  return s;
}

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

Prof::Prof(int c, cudaStream_t st) : cls(c), s(st), slot(-1) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof_on) return;
  ProfRec r{c, take_event(), take_event()};
  if (!r.a || !r.b) return;
  cudaEventRecord(r.a, s);
  g_prof_recs.push_back(r);
  slot = (int)g_prof_recs.size() - 1;
}

Prof::~Prof() {
  if (slot < 0) return;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (slot < (int)g_prof_recs.size()) cudaEventRecord(g_prof_recs[slot].b, s);
}

}  // namespace dirigo

using namespace dirigo;

static dirigo_status ws_check(size_t need, void* ws, size_t have) {
  if (need > 0 && !ws) return set_error(DIRIGO_E_INVALID, "workspace pointer is NULL");
  if (have < need)
    return set_error(DIRIGO_E_WORKSPACE, "workspace too small: need " + std::to_string(need) +
                                             " bytes");
  return DIRIGO_OK;
}

extern "C" {

const char* dirigo_last_error(void) { return g_err.c_str(); }

int64_t dirigo_launch_count(void) { return g_launches.load(); }

dirigo_status dirigo_query_order(dirigo_graph_t ref, dirigo_graph_t cand, uint64_t seed,
                                 int64_t* h_order, int64_t* h_prefix) {
  if (!ref || !cand || !h_order) return set_error(DIRIGO_E_INVALID, "NULL argument");
  if (ref->out_rank != cand->out_rank || ref->out_numel != cand->out_numel)
    return set_error(DIRIGO_E_MISMATCH, "reference and candidate outputs differ");
  for (int d = 0; d < ref->out_rank; ++d)
    if (ref->out_shape[d] != cand->out_shape[d])
      return set_error(DIRIGO_E_MISMATCH, "reference and candidate outputs differ");
  const int64_t n = ref->out_numel;
  const int rank = ref->out_rank;
  std::vector<uint8_t> seen((size_t)n, 0);
  int64_t k = 0;
  auto take = [&](int64_t l) {
    if (l >= 0 && l < n && !seen[(size_t)l]) {
      seen[(size_t)l] = 1;
      h_order[k++] = l;
    }
  };
  auto flat = [&](const int64_t* c) {
    int64_t l = 0;
    for (int d = 0; d < rank; ++d) l = l * ref->out_shape[d] + c[d];
    return l;
  };
  // 1. kernel launch corners (later kernels first, candidate first), then the
  //    corners of the output box and the first warp boundary
  for (const dirigo_graph* g : {cand, ref})
    for (auto it = g->kernel_corners.rbegin(); it != g->kernel_corners.rend(); ++it)
      for (int64_t l : *it) take(l);
  for (int m = 0; m < (1 << rank); ++m) {
    int64_t c[DIRIGO_MAX_RANK];
    for (int d = 0; d < rank; ++d) c[d] = ((m >> d) & 1) ? ref->out_shape[d] - 1 : 0;
    take(flat(c));
  }
  take(31);
  take(32);
  // 2. the lowest corner of every cone cell, candidate first
  for (const dirigo_graph* g : {cand, ref}) {
    const dirigo::Prog& P = g->prog;
    if (!P.cell_on) continue;
    const uint16_t* idx = reinterpret_cast<const uint16_t*>(g->cells.data());
    // first coordinate of every interval of every dim
    std::vector<std::vector<int64_t>> starts(rank);
    for (int d = 0; d < rank; ++d)
      for (int64_t x = 0; x < ref->out_shape[d]; ++x)
        if (x == 0 || idx[P.cell_tab[d] + x] != idx[P.cell_tab[d] + x - 1]) starts[d].push_back(x);
    int64_t cells = 1;
    for (int d = 0; d < rank; ++d) cells *= (int64_t)starts[d].size();
    for (int64_t id = 0; id < cells; ++id) {
      int64_t c[DIRIGO_MAX_RANK], x = id;
      for (int d = rank - 1; d >= 0; --d) {
        const int64_t m = (int64_t)starts[d].size();
        c[d] = starts[d][(size_t)(x % m)];
        x /= m;
      }
      take(flat(c));
    }
  }
  // 3. tensor boundaries
  take(0);
  take(n - 1);
  if (h_prefix) *h_prefix = k;
  // the rest in a seeded permutation (Fisher-Yates over the unchecked ones)
  const int64_t first = k;
  for (int64_t l = 0; l < n; ++l)
    if (!seen[(size_t)l]) h_order[k++] = l;
  uint64_t state = seed;
  for (int64_t i = n - 1; i > first; --i) {
    state += 0x9E3779B97F4A7C15ull;
    uint64_t z = state;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    z ^= z >> 31;
    const int64_t j = first + (int64_t)(z % (uint64_t)(i - first + 1));
    std::swap(h_order[i], h_order[j]);
  }
  return DIRIGO_OK;
}

dirigo_status dirigo_graph_create(const dirigo_graph_desc* desc, const dirigo_options* opt,
                                  dirigo_graph_t* out) {
  if (!out) return set_error(DIRIGO_E_INVALID, "out is NULL");
  *out = nullptr;
  dirigo_graph* g = new (std::nothrow) dirigo_graph();
  if (!g) return set_error(DIRIGO_E_NOMEM, "host allocation failed");
  dirigo_status s = compile_graph(desc, opt, g);
  if (s != DIRIGO_OK) {
    delete g;
    return s;
  }
  *out = g;
  return DIRIGO_OK;
}

dirigo_graph::~dirigo_graph() {
  if (cells_pinned) cudaFreeHost(cells_pinned);
}

void dirigo_graph_destroy(dirigo_graph_t g) { delete g; }

dirigo_status dirigo_graph_info_get(dirigo_graph_t g, dirigo_graph_info* info) {
  if (!g || !info) return set_error(DIRIGO_E_INVALID, "NULL argument");
  std::memset(info, 0, sizeof(*info));
  info->n_leaves = g->prog.G;
  info->out_numel = g->out_numel;
  info->out_rank = g->out_rank;
  for (int d = 0; d < DIRIGO_MAX_RANK; ++d) info->out_shape[d] = g->out_shape[d];
  info->n_tensors = g->prog.n_tensors;
  info->n_inputs = g->prog.n_inputs;
  tc_work(g->prog, &info->key_tc_flops, &info->key_limb_bytes);
  // SplitMix64 finalisers the key definition needs per dirigo_terms call: a
  // max-set of m >= 2 members m + 2 (its chain and one per lane), an
  // uninterpreted function 3 (one shared, one per lane)
  for (int t = g->prog.n_inputs; t < g->prog.n_tensors; ++t) {
    const dirigo::Tensor& T = g->prog.t[t];
    if (T.kind == dirigo::K_MAXSET && T.max_terms >= 2)
      info->key_mix_ops += (double)T.numel * (T.max_terms + 2);
    else if (T.kind == dirigo::K_UNARY)
      info->key_mix_ops += 3.0 * (double)T.numel;
  }
  for (int t = g->prog.n_inputs; t < g->prog.n_tensors; ++t)
    info->n_tc_contractions += (g->prog.t[t].flags & dirigo::TF_GEMM) != 0;
  if (g->prog.cell_on) {
    const dirigo::CellRec* rec =
        reinterpret_cast<const dirigo::CellRec*>(g->cells.data() + g->prog.cell_rec_off);
    info->n_cells = g->prog.n_cells;
    int64_t most = 0;
    for (int i = 0; i < g->prog.n_cells; ++i) {
      info->n_fast_cells += rec[i].nseg != dirigo::kCellGeneric;
      most = std::max<int64_t>(most, rec[i].count);
    }
    if (info->n_fast_cells == info->n_cells) info->max_runs_per_location = most;
  }
  return DIRIGO_OK;
}

dirigo_status dirigo_workspace_size(dirigo_graph_t g, int32_t call, int64_t n, size_t* bytes) {
  if (!g || !bytes || n < 0) return set_error(DIRIGO_E_INVALID, "bad argument");
  switch (call) {
    case DIRIGO_CALL_CONE: *bytes = cone_ws_bytes(g, n); break;
    case DIRIGO_CALL_TERMS: *bytes = terms_ws_bytes(g); break;
    case DIRIGO_CALL_EVAL: *bytes = eval_ws_bytes(g); break;
    default: return set_error(DIRIGO_E_INVALID, "unknown call");
  }
  return DIRIGO_OK;
}

dirigo_status dirigo_compare_workspace_size(dirigo_graph_t ref, dirigo_graph_t cand, int64_t n,
                                            size_t* bytes) {
  if (!ref || !cand || !bytes || n < 0) return set_error(DIRIGO_E_INVALID, "bad argument");
  *bytes = compare_ws_bytes(ref, cand, n);
  return DIRIGO_OK;
}

dirigo_status dirigo_cone(dirigo_graph_t g, const int64_t* d_locs, int64_t n, int64_t* d_offsets,
                          uint32_t* d_runs, int64_t run_capacity, uint64_t* d_fp,
                          int64_t* h_total, void* d_ws, size_t ws_bytes, void* stream) {
  if (!g || n < 0 || (n > 0 && !d_locs) || !d_offsets || run_capacity < 0 ||
      (run_capacity > 0 && !d_runs))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  dirigo_status s = ws_check(cone_ws_bytes(g, n), d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  return launch_cone(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, h_total, d_ws,
                     (cudaStream_t)stream);
}

dirigo_status dirigo_cone_async(dirigo_graph_t g, const int64_t* d_locs, int64_t n,
                                int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                                uint64_t* d_fp, int32_t* d_status, void* d_ws, size_t ws_bytes,
                                void* stream) {
  if (!g || n < 0 || (n > 0 && !d_locs) || !d_offsets || !d_status || run_capacity < 0 ||
      (run_capacity > 0 && !d_runs))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  dirigo_status s = ws_check(cone_ws_bytes(g, n), d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  return enqueue_cone(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, d_status, d_ws,
                      (cudaStream_t)stream);
}

dirigo_status dirigo_terms(dirigo_graph_t g, const int64_t* d_locs, int64_t n, uint32_t* d_keys,
                           void* d_ws, size_t ws_bytes, void* stream) {
  if (!g || n < 0 || (n > 0 && (!d_locs || !d_keys)))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  dirigo_status s = ws_check(terms_ws_bytes(g), d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  return launch_terms(g, d_locs, n, d_keys, d_ws, (cudaStream_t)stream);
}

static bool same_io(const dirigo_graph* a, const dirigo_graph* b) {
  if (a->in_shapes != b->in_shapes || a->out_rank != b->out_rank) return false;
  for (int d = 0; d < a->out_rank; ++d)
    if (a->out_shape[d] != b->out_shape[d]) return false;
  return true;
}

static dirigo_status compare_args(dirigo_graph_t ref, dirigo_graph_t cand, const int64_t* d_locs,
                                  int64_t n, const uint32_t* d_kref, const uint32_t* d_kcand,
                                  const int64_t* d_off_ref, const uint32_t* d_runs_ref,
                                  const uint64_t* d_fp_ref, const int64_t* d_off_cand,
                                  const uint32_t* d_runs_cand, const uint64_t* d_fp_cand,
                                  const int32_t* d_cone_status, void* cones_ready,
                                  const uint8_t* d_verdict, const uint8_t* d_flags, int64_t budget,
                                  const uint8_t* d_export, int64_t export_capacity, void* d_ws,
                                  size_t ws_bytes) {
  if (!ref || !cand || n < 0 || (n > 0 && (!d_locs || !d_kref || !d_kcand || !d_verdict || !d_flags)))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  if (!same_io(ref, cand))
    return set_error(DIRIGO_E_MISMATCH, "reference and candidate inputs or output differ");
  // with n = 0 there are no runs to read: the run buffers may then be NULL
  bool cones = d_off_ref || d_runs_ref || d_off_cand || d_runs_cand;
  if (cones && !(d_off_ref && d_off_cand && (n == 0 || (d_runs_ref && d_runs_cand))))
    return set_error(DIRIGO_E_INVALID, "cone arguments must be given together");
  if ((d_cone_status || cones_ready) && !cones)
    return set_error(DIRIGO_E_INVALID, "a cone status word or event without cones");
  if ((d_fp_ref == nullptr) != (d_fp_cand == nullptr))
    return set_error(DIRIGO_E_INVALID, "fingerprints must be given together");
  if (budget < 0 || export_capacity < 0) return set_error(DIRIGO_E_INVALID, "negative budget");
  if (((uintptr_t)d_export & 7) != 0)
    return set_error(DIRIGO_E_INVALID, "export buffer must be 8-byte aligned");
  (void)d_fp_ref;
  return ws_check(compare_ws_bytes(ref, cand, n), d_ws, ws_bytes);
}

dirigo_status dirigo_compare(dirigo_graph_t ref, dirigo_graph_t cand, const int64_t* d_locs,
                             int64_t n, const uint32_t* d_kref, const uint32_t* d_kcand,
                             const int64_t* d_off_ref, const uint32_t* d_runs_ref,
                             const uint64_t* d_fp_ref, const int64_t* d_off_cand,
                             const uint32_t* d_runs_cand, const uint64_t* d_fp_cand,
                             const int32_t* d_cone_status, void* cones_ready,
                             uint8_t* d_verdict, uint8_t* d_flags, int64_t budget,
                             uint8_t* d_export,
                             int64_t export_capacity, dirigo_compare_stats* h_stats,
                             void* d_ws, size_t ws_bytes, void* stream) {
  dirigo_status s = compare_args(ref, cand, d_locs, n, d_kref, d_kcand, d_off_ref, d_runs_ref,
                                 d_fp_ref, d_off_cand, d_runs_cand, d_fp_cand, d_cone_status,
                                 cones_ready, d_verdict, d_flags, budget, d_export,
                                 export_capacity, d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  if (n == 0) {
    if (h_stats) std::memset(h_stats, 0, sizeof(*h_stats));
    if (d_cone_status) {   // the cone calls of an empty batch can still have failed
      int32_t cs = 0;
      cudaError_t e = cones_ready ? cudaStreamWaitEvent((cudaStream_t)stream,
                                                        (cudaEvent_t)cones_ready, 0)
                                  : cudaSuccess;
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(&cs, d_cone_status, 4, cudaMemcpyDeviceToHost, (cudaStream_t)stream);
      if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
      if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
      if (h_stats) h_stats->cone_error = cs;
      if (cs) return cone_status_error(cs);
    }
    return DIRIGO_OK;
  }
  return launch_compare(ref, cand, d_locs, n, d_kref, d_kcand, d_off_ref, d_runs_ref, d_fp_ref,
                        d_off_cand, d_runs_cand, d_fp_cand, d_cone_status,
                        (cudaEvent_t)cones_ready, d_verdict, d_flags,
                        budget, d_export,
                        export_capacity, h_stats, d_ws, (cudaStream_t)stream);
}

dirigo_status dirigo_compare_async(dirigo_graph_t ref, dirigo_graph_t cand, const int64_t* d_locs,
                                   int64_t n, const uint32_t* d_kref, const uint32_t* d_kcand,
                                   const int64_t* d_off_ref, const uint32_t* d_runs_ref,
                                   const uint64_t* d_fp_ref, const int64_t* d_off_cand,
                                   const uint32_t* d_runs_cand, const uint64_t* d_fp_cand,
                                   const int32_t* d_cone_status, void* cones_ready,
                                   uint8_t* d_verdict, uint8_t* d_flags, int64_t budget,
                                   uint8_t* d_export, int64_t export_capacity,
                                   dirigo_compare_stats* d_stats, int32_t* d_status, void* d_ws,
                                   size_t ws_bytes, void* stream) {
  dirigo_status s = compare_args(ref, cand, d_locs, n, d_kref, d_kcand, d_off_ref, d_runs_ref,
                                 d_fp_ref, d_off_cand, d_runs_cand, d_fp_cand, d_cone_status,
                                 cones_ready, d_verdict, d_flags, budget, d_export,
                                 export_capacity, d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  if (!d_stats || (((uintptr_t)d_stats) & 7) != 0)
    return set_error(DIRIGO_E_INVALID, "d_stats must be an 8-byte aligned device pointer");
  if (n == 0) {
    if (cones_ready &&
        cudaStreamWaitEvent((cudaStream_t)stream, (cudaEvent_t)cones_ready, 0) != cudaSuccess)
      return set_error(DIRIGO_E_CUDA, "waiting for the cones");
    return launch_compare_empty(d_cone_status, d_stats, d_status, (cudaStream_t)stream);
  }
  return launch_compare(ref, cand, d_locs, n, d_kref, d_kcand, d_off_ref, d_runs_ref, d_fp_ref,
                        d_off_cand, d_runs_cand, d_fp_cand, d_cone_status,
                        (cudaEvent_t)cones_ready, d_verdict, d_flags, budget, d_export,
                        export_capacity, nullptr, d_ws, (cudaStream_t)stream, d_stats, d_status);
}

dirigo_status dirigo_eval(dirigo_graph_t g, const float* const* d_inputs, const int64_t* d_locs,
                          int64_t n, float* d_out, void* d_ws, size_t ws_bytes, void* stream) {
  if (!g || !d_inputs || n < 0 || (n > 0 && (!d_locs || !d_out)))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  for (int i = 0; i < g->prog.n_inputs; ++i)
    if (!d_inputs[i]) return set_error(DIRIGO_E_INVALID, "input pointer is NULL");
  dirigo_status s = ws_check(eval_ws_bytes(g), d_ws, ws_bytes);
  if (s != DIRIGO_OK) return s;
  return launch_eval(g, d_inputs, d_locs, n, d_out, d_ws, (cudaStream_t)stream);
}

dirigo_status dirigo_profile_enable(int32_t on) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_on = on != 0;
  return DIRIGO_OK;
}

dirigo_status dirigo_profile_read(double* ms, int64_t* launches, int32_t n_classes, int32_t reset) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  drain_locked();
  for (int i = 0; i < n_classes && i < DIRIGO_K_COUNT_; ++i) {
    if (ms) ms[i] = g_prof_ms[i];
    if (launches) launches[i] = g_prof_n[i];
  }
  if (reset) {
    for (int i = 0; i < DIRIGO_K_COUNT_; ++i) {
      g_prof_ms[i] = 0;
      g_prof_n[i] = 0;
    }
  }
  return DIRIGO_OK;
}

}  // extern "C"
