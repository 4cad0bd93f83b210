// MERGE prefix trimming (Sec. 3.2 "MERGE"): when the two programs begin with
// the same operations on the same inputs, that common prefix is cut off and
// the tensors it hands to the rest of either program become the shared inputs
// of both trimmed programs.
//
// Equal canonical terms over the cut tensors stay equal after substituting
// the prefix for them, so a location the trimmed pair discharges is
// discharged by the original pair too: trimming never discharges a location
// wrongly.  It can miss a discharge when the prefix is not surjective (the
// cut tensors are then treated as free values they cannot take), which the
// paper accepts for prefixes (nearly all are surjective).
//
// Host only; nothing here touches the device.
#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

namespace dirigo {
namespace {

bool same_const(const dirigo_const& a, const dirigo_const& b) {
  if (a.den != b.den || a.num != b.num) return false;
  return a.den != 0 || std::memcmp(&a.value, &b.value, sizeof(double)) == 0;
}

// Two op descriptions define the same operation (same kind, arguments and
// every attribute that kind reads, with the lowering's defaults: a conv stride
// of 0 is 1, a pool stride of 0 is the window).  Fields a kind does not read
// are not compared.
bool same_op(const dirigo_op_desc& a, const dirigo_op_desc& b) {
  if (a.kind != b.kind || a.n_args != b.n_args) return false;
  for (int i = 0; i < a.n_args && i < 3; ++i)
    if (a.args[i] != b.args[i]) return false;
  switch (a.kind) {
    case DIRIGO_OP_CONV2D:
      return (a.stride > 0 ? a.stride : 1) == (b.stride > 0 ? b.stride : 1) && a.pad == b.pad;
    case DIRIGO_OP_MAXPOOL2D:
      return a.k == b.k && (a.stride > 0 ? a.stride : a.k) == (b.stride > 0 ? b.stride : b.k);
    case DIRIGO_OP_ADD: case DIRIGO_OP_SUB: case DIRIGO_OP_MUL: case DIRIGO_OP_DIV:
      for (int s = 0; s < 2; ++s) {
        if (a.axes_rank[s] != b.axes_rank[s]) return false;
        for (int d = 0; d < a.axes_rank[s] && d < DIRIGO_MAX_RANK; ++d)
          if (a.axes[s][d] != b.axes[s][d]) return false;
      }
      return true;
    case DIRIGO_OP_SCALE: case DIRIGO_OP_ADD_SCALAR: case DIRIGO_OP_CLAMP_MIN:
    case DIRIGO_OP_LAYERNORM:
      return same_const(a.c, b.c);
    case DIRIGO_OP_SUM: case DIRIGO_OP_MEAN: case DIRIGO_OP_MAX:
      return a.dim == b.dim && (a.keepdim != 0) == (b.keepdim != 0);
    case DIRIGO_OP_SOFTMAX:
      return a.dim == b.dim;
    case DIRIGO_OP_CONTRACT: case DIRIGO_OP_MAXSET:
      if (a.rank != b.rank || a.n_pieces != b.n_pieces) return false;
      for (int d = 0; d < a.rank && d < DIRIGO_MAX_RANK; ++d)
        if (a.shape[d] != b.shape[d]) return false;
      for (int q = 0; q < a.n_pieces; ++q)   // plain structs without padding
        if (std::memcmp(&a.pieces[q], &b.pieces[q], sizeof(dirigo_piece)) != 0) return false;
      return true;
    case DIRIGO_OP_KERNEL_CONTRACT: case DIRIGO_OP_KERNEL_MAXSET:
      if (a.rank != b.rank || a.n_writes != b.n_writes) return false;
      for (int d = 0; d < a.rank && d < DIRIGO_MAX_RANK; ++d)
        if (a.shape[d] != b.shape[d]) return false;
      for (int d = 0; d < 3; ++d)
        if (a.grid[d] != b.grid[d] || a.block[d] != b.block[d]) return false;
      // bytewise: descriptions that differ only in padding bytes count as
      // different, which only trims less
      for (int w = 0; w < a.n_writes; ++w)
        if (std::memcmp(&a.writes[w], &b.writes[w], sizeof(dirigo_kernel_write)) != 0)
          return false;
      return true;
    default:
      return true;
  }
}

// The trimmed description of one program: the cut tensors as inputs (shapes
// from the compiled original), the ops after the prefix with their arguments
// renumbered.
struct Trimmed {
  std::vector<dirigo_tensor_desc> inputs;
  std::vector<dirigo_op_desc> ops;
  dirigo_graph_desc desc;
};

void trim(const dirigo_graph_desc* g, int L, const std::vector<int>& cut,
          const std::vector<std::vector<int64_t>>& shapes, Trimmed* out) {
  const int I = g->n_inputs, ncut = (int)cut.size();
  std::vector<int> newid(I + g->n_ops, -1);
  for (int i = 0; i < ncut; ++i) newid[cut[i]] = i;
  for (int k = L; k < g->n_ops; ++k) newid[I + k] = ncut + (k - L);
  out->inputs.resize(ncut);
  for (int i = 0; i < ncut; ++i) {
    dirigo_tensor_desc& td = out->inputs[i];
    std::memset(&td, 0, sizeof(td));
    const std::vector<int64_t>& sh = shapes[cut[i]];
    td.rank = (int32_t)sh.size();
    for (size_t d = 0; d < sh.size() && d < DIRIGO_MAX_RANK; ++d) td.shape[d] = sh[d];
  }
  out->ops.assign(g->ops + L, g->ops + g->n_ops);
  for (dirigo_op_desc& op : out->ops)
    for (int i = 0; i < op.n_args && i < 3; ++i) op.args[i] = newid[op.args[i]];
  out->desc.n_inputs = ncut;
  out->desc.inputs = out->inputs.data();
  out->desc.n_ops = (int32_t)out->ops.size();
  out->desc.ops = out->ops.data();
  out->desc.output = newid[g->output];
}

}  // namespace
}  // namespace dirigo

using namespace dirigo;

extern "C" dirigo_status dirigo_graph_create_merged(const dirigo_graph_desc* ref,
                                                    const dirigo_graph_desc* cand,
                                                    const dirigo_options* opt,
                                                    dirigo_graph_t* ref_out,
                                                    dirigo_graph_t* cand_out, int32_t* cut_ids,
                                                    int32_t cut_capacity,
                                                    dirigo_merge_info* info) {
  if (!ref || !cand || !ref_out || !cand_out || !info || cut_capacity < 0 ||
      (cut_capacity > 0 && !cut_ids))
    return set_error(DIRIGO_E_INVALID, "NULL argument");
  *ref_out = *cand_out = nullptr;
  std::memset(info, 0, sizeof(*info));
  // the original reference compiled once: it validates the description and
  // gives the shape of every tensor of the prefix
  dirigo_graph full;
  dirigo_status s = compile_graph(ref, opt, &full);
  if (s != DIRIGO_OK) return s;
  if (!cand || cand->n_inputs != ref->n_inputs || !cand->inputs)
    return set_error(DIRIGO_E_MISMATCH, "the programs declare different inputs");
  for (int i = 0; i < ref->n_inputs; ++i) {
    const dirigo_tensor_desc &a = ref->inputs[i], &b = cand->inputs[i];
    if (a.rank != b.rank) return set_error(DIRIGO_E_MISMATCH, "the programs declare different inputs");
    for (int d = 0; d < a.rank && d < DIRIGO_MAX_RANK; ++d)
      if (a.shape[d] != b.shape[d])
        return set_error(DIRIGO_E_MISMATCH, "the programs declare different inputs");
  }
  const int I = ref->n_inputs;
  // longest common prefix; each program keeps the op that computes its output
  const int last = std::min(ref->output - I, cand->output - I);
  int L = 0;
  while (L < ref->n_ops && L < cand->n_ops && L < last && same_op(ref->ops[L], cand->ops[L])) ++L;
  // the cut: tensors before the end of the prefix that the rest of either
  // program reads, in id order (inputs first, then prefix ops in SSA order);
  // with nothing trimmed the inputs stay as declared
  std::vector<int> cut;
  if (L == 0) {
    for (int i = 0; i < I; ++i) cut.push_back(i);
  } else {
    std::vector<char> used(I + L, 0);
    for (const dirigo_graph_desc* g : {ref, cand})
      for (int k = L; k < g->n_ops; ++k)
        for (int i = 0; i < g->ops[k].n_args && i < 3; ++i)
          if (g->ops[k].args[i] >= 0 && g->ops[k].args[i] < I + L) used[g->ops[k].args[i]] = 1;
    for (int id = 0; id < I + L; ++id)
      if (used[id]) cut.push_back(id);
  }
  info->n_shared_ops = L;
  info->n_inputs = (int32_t)cut.size();
  if ((int)cut.size() > cut_capacity) return set_error(DIRIGO_E_CAPACITY, "cut_ids too small");
  for (size_t i = 0; i < cut.size(); ++i) cut_ids[i] = cut[i];
  Trimmed tr, tc;
  trim(ref, L, cut, full.hl_shapes, &tr);
  trim(cand, L, cut, full.hl_shapes, &tc);
  dirigo_graph* gr = new (std::nothrow) dirigo_graph();
  dirigo_graph* gc = new (std::nothrow) dirigo_graph();
  if (!gr || !gc) {
    delete gr;
    delete gc;
    return set_error(DIRIGO_E_NOMEM, "host allocation failed");
  }
  s = compile_graph(&tr.desc, opt, gr);
  if (s == DIRIGO_OK) s = compile_graph(&tc.desc, opt, gc);
  if (s != DIRIGO_OK) {
    delete gr;
    delete gc;
    return s;
  }
  *ref_out = gr;
  *cand_out = gc;
  return DIRIGO_OK;
}
