// dirigo_cone_noalloc: the cone call for callers that cannot allocate device
// memory.
//
// dirigo_cone needs a small scratch area (a status word and the prefix-sum
// buffer of the run counts) and takes it from a caller workspace.  Some
// callers cannot provide one: a process whose device memory is owned by a
// memory manager that must not be bypassed, or code under a rule that forbids
// device allocation after start-up (cudaMalloc may also synchronise the whole
// device, which latency-sensitive callers avoid).  This variant takes its
// scratch from a fixed array compiled into the library instead, so the call
// itself allocates nothing; the caller still passes the locations, offsets,
// runs and fingerprints buffers.
//
// The array is a file-scope __device__ variable: every GPU that loads this
// library holds it (17 KB) until the process exits.  Its device address is
// looked up once per device, on the first call made with that device current;
// that first call should therefore come before any stream capture.  Like
// dirigo_cone, each call waits for its stream once, at the end, to read back
// the run total and the status word (errors of the write pass included).  All
// calls share the one array and it keeps the last call's contents (the status
// word is cleared at the start of each call; the prefix sum clears its own
// words), so calls that overlap on the GPU (on different streams, or from
// different host threads) race on it and must not be issued concurrently.
#include <cstring>
#include <mutex>

#include "internal.h"
#include "launch.h"

namespace dirigo {

namespace {

// Largest batch the fixed scratch covers.  The scratch is a 256-byte status
// block, then the prefix sum's words (two, plus one per tile of 4,096 counts:
// 2,050 int64 for 8,388,608 locations) rounded up to 256 bytes, then 256
// bytes of slack, as cone_ws_bytes_noplan() lays it out: 17,152 bytes.  The
// call checks cone_ws_bytes_noplan(n) against the size before every use.
constexpr int64_t kNoAllocMaxLocations = 8388608;
constexpr int64_t kNoAllocScanTile = 4096;
constexpr size_t kNoAllocScratchBytes =
    256 + ((kNoAllocMaxLocations / kNoAllocScanTile + 2) * 8 + 255) / 256 * 256 + 256;
static_assert(kNoAllocScratchBytes == 17152, "fixed scratch size");

static __device__ __align__(256) unsigned char g_cone_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device (set up once).
dirigo_status scratch_for_current_device(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return set_error(DIRIGO_E_UNSUPPORTED, "device index above 63");
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_cone_scratch);
    if (e != cudaSuccess || !p) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return DIRIGO_OK;
}

}  // namespace

}  // namespace dirigo

using namespace dirigo;

extern "C" dirigo_status dirigo_cone_noalloc(dirigo_graph_t g, const int64_t* d_locs, int64_t n,
                                             int64_t* d_offsets, uint32_t* d_runs,
                                             int64_t run_capacity, uint64_t* d_fp,
                                             int64_t* h_total, void* stream) {
  if (!g || n < 0 || (n > 0 && !d_locs) || !d_offsets || run_capacity < 0 ||
      (run_capacity > 0 && !d_runs))
    return set_error(DIRIGO_E_INVALID, "bad argument");
  if (n > kNoAllocMaxLocations)
    return set_error(DIRIGO_E_WORKSPACE,
                     "dirigo_cone_noalloc handles at most 8388608 locations per call");
  if (cone_ws_bytes_noplan(n) > kNoAllocScratchBytes)
    return set_error(DIRIGO_E_WORKSPACE, "fixed scratch smaller than the call needs");
  void* scratch = nullptr;
  dirigo_status s = scratch_for_current_device(&scratch);
  if (s != DIRIGO_OK) return s;
  // the status word at the start of the scratch is cleared by launch_cone,
  // which reads it back after the write pass
  return launch_cone(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, h_total, scratch,
                     (cudaStream_t)stream, /*plan_slots=*/false);
}
