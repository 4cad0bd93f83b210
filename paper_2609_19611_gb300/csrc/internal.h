// Library-internal declarations shared by the translation units.
#pragma once
#include <cstdint>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/dirigo.h"
#include "prog.h"

struct dirigo_graph {
  dirigo::Prog prog;            // compiled program (host copy, passed to kernels by value)
  int64_t out_numel = 0;
  int32_t out_rank = 0;
  int64_t out_shape[DIRIGO_MAX_RANK] = {0, 0, 0, 0};
  int64_t value_elems = 0;      // elements of all primitive (non-input) tensors
  int32_t max_rank_used = 0;
  // input shapes, for dirigo_compare's I/O matching (Sec. 3.2: the inputs and
  // outputs of the two programs are matched)
  std::vector<std::vector<int64_t>> in_shapes;
  // shape of every high-level tensor (inputs, then one per op), for MERGE
  std::vector<std::vector<int64_t>> hl_shapes;
  // output locations written by the corner threads of each kernel op whose
  // output reaches the graph output through index-preserving ops (same-shape
  // elementwise ops), in op order; for the query order
  std::vector<std::vector<int64_t>> kernel_corners;
  // cone cells of the output (cells.h), copied to the device with each cone call
  std::vector<uint8_t> cells;
  int64_t n_generic_cells = 0;
  // pinned copy of `cells`, made by the first cone call that uploads the
  // table: a copy from pageable memory may wait for the stream's earlier
  // work, one from pinned memory is queued like a kernel (freed with the graph)
  mutable uint8_t* cells_pinned = nullptr;
  mutable std::once_flag cells_pinned_once;
  ~dirigo_graph();
};

namespace dirigo {

dirigo_status set_error(dirigo_status s, const std::string& msg);
dirigo_status compile_graph(const dirigo_graph_desc* desc, const dirigo_options* opt,
                            dirigo_graph* g);
// kernel write set -> pieces over output coordinates (kinvert.cpp)
dirigo_status invert_kernel_writes(const dirigo_op_desc& op, std::vector<dirigo_piece>* out,
                                   std::string* err);
// flat locations written by a kernel launch's corner threads (kinvert.cpp)
std::vector<int64_t> kernel_corner_locations(const dirigo_op_desc& op);
KConst encode_const(const dirigo_const& c, bool* ok);

// launch helpers (defined in the .cu files); all enqueue on `stream`
struct KeyWs;
}  // namespace dirigo
