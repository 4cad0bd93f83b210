// Per-location compare and export (Sec. 3.4 "Solving": the solver is asked
// whether e_A != e_B; identical canonical terms need no solver).
//
//   compare_quick   one thread per slot: keys -> discharged or not; cone
//                   counts, fingerprints and bottom flags; slots whose cones
//                   are equal in count and fingerprint are queued for an
//                   exact check
//   compare_exact   one warp per queued slot: run lists compared in full
//   (scan)          rank of each undischarged slot; the first `budget` are
//                   selected for export
//   export          per program: mark the elements of every tensor that
//                   res() visits from the selected roots (box propagation),
//                   count nodes and their equation terms, scan, write the
//                   "DXP1" records
#include <cstdint>
#include <mutex>

#include "cone_prop.cuh"
#include "internal.h"
#include "launch.h"

namespace dirigo {

void launch_scan(int64_t* data, int64_t n, int64_t* tmp, int32_t* err, cudaStream_t s);
size_t scan_tmp_bytes(int64_t n);

struct DevStats {
  unsigned long long n_disc, n_und, n_cone_diff, n_bot_ref, n_bot_cand;
  unsigned long long n_queue;
  int32_t status;
  int32_t ok;   // the export fits the caller's buffer and is written
  int32_t cone_status;   // the cone calls' latched errors (cones then not read)
  int32_t pad_;
  // export sizes, computed on the device (read by the host once, at the end)
  long long nsel, required, n_nodes[2], n_ent[2], sec_off[2], loc_off;
  unsigned long long n_dirty[2];   // bitmap words with a marked element, per program
  unsigned long long wr_next[2];   // the export writer's next large-node chunk, per program
};

// Sum of one count per thread over the block, added to *dst by one thread
// (256-thread blocks).
__device__ __forceinline__ void block_count(unsigned c, unsigned long long* dst) {
  __shared__ unsigned part[8];
  c = __reduce_add_sync(0xffffffffu, c);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned t = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += part[w];
    if (t) atomicAdd(dst, (unsigned long long)t);
  }
}

// Verdicts from the keys alone: DISCHARGED iff both lanes agree.  Also the
// undischarged indicator the export's ranking scans, the discharged count and
// the location check; with no cones the flags are NO_CONES here.
__global__ void __launch_bounds__(256) verdict_kernel(const int64_t* locs, int64_t n,
                                                      int64_t out_numel, const uint2* kr,
                                                      const uint2* kc, int no_cones,
                                                      uint8_t* verdict, uint8_t* flags,
                                                      int64_t* und, DevStats* st) {
  if (n <= 0) return;
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const bool live = i < n;
  bool eq = false;
  if (live) {
    const int64_t l = locs[i];
    if (l < 0 || l >= out_numel) atomicOr(&st->status, CE_LOCATION);
    const uint2 a = kr[i], b = kc[i];
    eq = a.x == b.x && a.y == b.y;
    verdict[i] = eq ? DIRIGO_DISCHARGED : DIRIGO_DIFFERS_UNEXPORTED;
    und[i] = eq ? 0 : 1;
    if (no_cones) flags[i] = DIRIGO_FLAG_NO_CONES;
  }
  block_count(live && eq, &st->n_disc);
}

// Flags from the cones: CONE_DIFFERS when the run counts or fingerprints
// differ (slots whose counts and fingerprints agree are queued for the exact
// run compare), BOT_REF / BOT_CAND when a cone's last run ends with bottom.
// bot_r / bot_c: whether a cone of that program can contain bottom at all (a
// graph whose output cells all have fast plans reads in range only); the last
// run is read only then.  cone_status: the word asynchronous cone calls
// latched their errors in (NULL: none); when it is nonzero no cone is read
// (their runs may not have been written) and every flag is NO_CONES.
__global__ void __launch_bounds__(256) cone_flags_kernel(
    int64_t n, const int64_t* offr, const uint2* runr, const uint64_t* fpr, const int64_t* offc,
    const uint2* runc, const uint64_t* fpc, const int32_t* cone_status, int64_t Gr, int64_t Gc,
    int bot_r, int bot_c, uint8_t* flags, int64_t* queue, DevStats* st) {
  if (n <= 0) return;
  const int32_t cs = cone_status ? *cone_status : 0;
  if (cs && blockIdx.x == 0 && threadIdx.x == 0) st->cone_status = cs;
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const bool live = i < n;
  uint8_t f = 0;
  if (live) {
    if (cs) {
      f = DIRIGO_FLAG_NO_CONES;
    } else {
      const int64_t r0 = offr[i], r1 = offr[i + 1], c0 = offc[i], c1 = offc[i + 1];
      if (bot_r && r1 > r0) {
        const uint2 last = runr[r1 - 1];
        if ((int64_t)last.x + last.y == Gr + 1) f |= DIRIGO_FLAG_BOT_REF;
      }
      if (bot_c && c1 > c0) {
        const uint2 last = runc[c1 - 1];
        if ((int64_t)last.x + last.y == Gc + 1) f |= DIRIGO_FLAG_BOT_CAND;
      }
      bool differs = (r1 - r0) != (c1 - c0);
      if (!differs && fpr && fpc) differs = fpr[i] != fpc[i];
      if (differs) {
        f |= DIRIGO_FLAG_CONE_DIFFERS;
      } else {
        const unsigned long long k = atomicAdd(&st->n_queue, 1ull);
        queue[k] = i;
      }
    }
    flags[i] = f;
  }
  block_count(live && (f & DIRIGO_FLAG_BOT_REF), &st->n_bot_ref);
  block_count(live && (f & DIRIGO_FLAG_BOT_CAND), &st->n_bot_cand);
}

__global__ void compare_exact_kernel(const int64_t* queue, const DevStats* st, const int64_t* offr,
                                     const uint2* runr, const int64_t* offc, const uint2* runc,
                                     uint8_t* flags) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t nq = (int64_t)st->n_queue;
  for (int64_t q = warp; q < nq; q += nw) {
    int64_t i = queue[q];
    int64_t r0 = offr[i], c0 = offc[i], len = offr[i + 1] - r0;
    bool diff = false;
    for (int64_t kb = 0; kb < len; kb += 32) {
      int64_t k = kb + lane;
      bool d = false;
      if (k < len) {
        uint2 a = runr[r0 + k], b = runc[c0 + k];
        d = a.x != b.x || a.y != b.y;
      }
      if (__any_sync(0xffffffffu, d)) {
        diff = true;
        break;
      }
    }
    if (diff && lane == 0) flags[i] |= DIRIGO_FLAG_CONE_DIFFERS;
  }
}

__global__ void __launch_bounds__(256) count_flags_kernel(const uint8_t* flags, int64_t n,
                                                          DevStats* st) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  block_count(i < n && (flags[i] & DIRIGO_FLAG_CONE_DIFFERS), &st->n_cone_diff);
}

// slots with undischarged rank < budget, in slot order
__global__ void select_kernel(const int64_t* rank, const uint8_t* verdict, int64_t n,
                              int64_t budget, int64_t* sel) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= n) return;
  if (verdict[i] != DIRIGO_DISCHARGED && rank[i] < budget) sel[rank[i]] = i;
}

// ---------------------------------------------------------------- export

// Records every (merged) box that res() visits from one root.
constexpr int kMaxVisits = 24;
struct RecordVisit {
  NBox box[kMaxVisits];
  int n;
  int overflow;
  __device__ void operator()(int t, const NBox& B) {
    if (n < kMaxVisits) {
      box[n] = B;
      box[n].t = t;
      ++n;
    } else {
      overflow = 1;
    }
  }
};

// Marking of the equation nodes that res() visits from the exported roots,
// in two passes over chunks of kMarkChunk roots: one thread per root
// propagates and records the (merged) boxes it visits, then one warp per
// recorded box sets the box's bits.
constexpr int64_t kMarkChunk = 4096;

__global__ void __launch_bounds__(128) record_kernel(const __grid_constant__ Prog P,
                                                     const int64_t* locs, const int64_t* sel,
                                                     int64_t c0, int64_t nroots, NBox* visits,
                                                     int32_t* nvis, DevStats* st) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= nroots) return;
  if (c0 + i >= st->nsel) {   // past the selected roots
    nvis[i] = 0;
    return;
  }
  sel += c0;
  LocState L;
  RecordVisit rv;
  rv.n = 0;
  rv.overflow = 0;
  propagate(P, locs[sel[i]], L, rv);
  if (L.err || rv.overflow) {
    atomicOr(&st->status, L.err | CE_CAPACITY * rv.overflow);
    rv.n = 0;
  }
  for (int b = 0; b < rv.n; ++b) visits[i * kMaxVisits + b] = rv.box[b];
  nvis[i] = rv.n;
}

// Roots that share a subterm record the same boxes (the 16 channels of one
// softmax column share its pooling, exp and convolution boxes), so each box
// is marked once: a warp first claims its box in an open-addressing table of
// visit indices (2x the boxes, linear probing; a probe finds the box, or an
// empty slot it claims, within the table size) and marks only when it
// claimed an empty slot.
constexpr int64_t kBoxTable = 2 * kMarkChunk * kMaxVisits;

__device__ __forceinline__ bool same_box(const NBox& a, const NBox& b) {
  bool eq = a.t == b.t;
#pragma unroll
  for (int d = 0; d < MR; ++d) eq = eq && a.lo[d] == b.lo[d] && a.hi[d] == b.hi[d];
  return eq;
}

__global__ void __launch_bounds__(256) mark_kernel(const __grid_constant__ Prog P,
                                                   const NBox* visits, const int32_t* nvis,
                                                   int64_t nroots, uint32_t* bits, int64_t* dirty,
                                                   unsigned long long* n_dirty,
                                                   int32_t* table) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t root = warp / kMaxVisits;
  const int b = (int)(warp - root * kMaxVisits);
  if (root >= nroots || b >= nvis[root]) return;
  const int32_t me = (int32_t)(root * kMaxVisits + b);
  const NBox& B = visits[me];
  int owner = 0;
  if (lane == 0) {
    uint32_t h = (uint32_t)B.t * 0x9E3779B1u;
#pragma unroll
    for (int d = 0; d < MR; ++d) {
      h = (h ^ (uint32_t)B.lo[d]) * 0x85EBCA6Bu;
      h = (h ^ (uint32_t)B.hi[d]) * 0xC2B2AE35u;
    }
    int64_t slot = (int64_t)(h % (uint32_t)kBoxTable);
    for (int64_t probe = 0; probe < kBoxTable; ++probe) {
      const int32_t cur = atomicCAS(&table[slot], -1, me);
      if (cur == -1) {
        owner = 1;
        break;
      }
      if (same_box(visits[cur], B)) break;   // another warp marks this box
      if (++slot == kBoxTable) slot = 0;
    }
  }
  if (!__shfl_sync(0xffffffffu, owner, 0)) return;
  const Tensor& T = P.t[B.t];
  int32_t lo[MR], ext[MR];
  int64_t total = 1;
  for (int d = 0; d < MR; ++d) {
    lo[d] = B.lo[d];
    ext[d] = B.hi[d] - B.lo[d];
    total *= ext[d];
  }
  const int64_t wbase = T.ws_off / 32;
  uint32_t* w = bits + wbase;
  for (int64_t k = lane; k < total; k += 32) {
    int64_t x = k, flat = 0;
    for (int d = MR - 1; d >= 0; --d) {
      int64_t qq, c;
      divmod64(x, ext[d], qq, c);
      x = qq;
      if (d < T.rank) flat += T.stride[d] * (lo[d] + c);
    }
    // roots that share a subterm mark the same elements: skip bits already set;
    // the thread that sets a word's first bit lists the word
    const uint32_t bit = 1u << (flat & 31);
    if (!(w[flat >> 5] & bit)) {
      const uint32_t old = atomicOr(&w[flat >> 5], bit);
      if (old == 0) dirty[atomicAdd(n_dirty, 1ull)] = wbase + (flat >> 5);
    }
  }
}

// number of selected roots: min(budget, undischarged count)
__global__ void export_init_kernel(const int64_t* n_und, int64_t budget, DevStats* st) {
  const int64_t u = *n_und;
  st->n_und = (unsigned long long)u;
  st->nsel = budget < u ? (budget > 0 ? budget : 0) : u;
}

__device__ __forceinline__ int tensor_of_word(const Prog& P, int64_t w) {
  int t = P.n_inputs;
  for (int u = P.n_inputs + 1; u < P.n_tensors; ++u)
    if (P.t[u].ws_off / 32 <= w) t = u;
  return t;
}

__device__ __forceinline__ uint64_t ref_word(const Prog& P, int arg, int64_t off) {
  const Tensor& A = P.t[arg];
  if (off < 0 || off >= A.numel) return (uint64_t)P.G;
  if (A.kind == K_INPUT) return (uint64_t)(A.gbase + off);
  return (1ull << 63) | ((uint64_t)arg << 40) | (uint64_t)off;
}

// For output coordinates o, the reduction coordinates of a piece whose terms
// exist form a box: each guard restricts one reduction dim to an interval (or
// the whole piece, when it has no reduction dim).  Returns its volume.
__device__ __forceinline__ int64_t valid_box(const Piece& pc, const int32_t* o, int rank,
                                             int32_t* vlo, int32_t* vext) {
  if (!in_box(o, pc, rank)) return 0;
  int32_t vhi[MRED];
  for (int e = 0; e < MRED; ++e) {
    vlo[e] = e < pc.nred ? pc.rlo[e] : 0;
    vhi[e] = e < pc.nred ? pc.rhi[e] : 1;
  }
#pragma unroll
  for (int j = 0; j < MG; ++j) {
    if (j >= pc.nguard) continue;
    const Guard& g = pc.g[j];
    int32_t v0 = g.c + (g.od >= 0 ? g.oa * sel4(o, g.od) : 0);
    if (g.rd < 0) {
      if (v0 < g.lo || v0 >= g.hi) return 0;
    } else {
#pragma unroll
      for (int e = 0; e < MRED; ++e) {
        if (e != g.rd) continue;
        vlo[e] = max(vlo[e], g.lo - v0);
        vhi[e] = min(vhi[e], g.hi - v0);
      }
    }
  }
  int64_t vol = 1;
  for (int e = 0; e < MRED; ++e) {
    vext[e] = max(0, vhi[e] - vlo[e]);
    vol *= vext[e];
  }
  return vol;
}

__device__ __forceinline__ int64_t entry_count(const Prog& P, int t, int64_t e) {
  const Tensor& T = P.t[t];
  if (T.kind == K_CONTRACT || T.kind == K_MAXSET) {
    int32_t o[MR], vlo[MRED], vext[MRED];
    unflatten(e, T, o);
    int64_t n = 0;
    for (int q = 0; q < T.npieces; ++q) n += valid_box(P.p[T.piece0 + q], o, T.rank, vlo, vext);
    return n;
  }
  if (T.kind == K_BINARY) return (T.fn == B_ADD || T.fn == B_SUB) ? 2 : 1;
  if (T.kind == K_MAXC) return 2;
  if (T.kind == K_AFFINE) return T.c.is_zero ? 1 : 2;
  return 1;
}

// Entry j of the per-element equation of element e of tensor t (equation
// order: pieces in order, reduction coordinates row-major).
__device__ __forceinline__ void entry_of(const Prog& P, int t, int64_t e, const int32_t* o,
                                         int64_t j, double& coef, uint64_t& a, uint64_t& b) {
  const Tensor& T = P.t[t];
  const uint64_t NONE = ~0ull;
  b = NONE;
  if (T.kind == K_CONTRACT || T.kind == K_MAXSET) {
    for (int q = 0; q < T.npieces; ++q) {
      const Piece& pc = P.p[T.piece0 + q];
      int32_t vlo[MRED], vext[MRED], r[MRED];
      int64_t vol = valid_box(pc, o, T.rank, vlo, vext);
      if (j >= vol) {
        j -= vol;
        continue;
      }
      int64_t x = j;
      for (int d = MRED - 1; d >= 0; --d) {
        int64_t qq, c;
        divmod64(x, vext[d], qq, c);
        r[d] = vlo[d] + (int32_t)c;
        x = qq;
      }
      coef = T.kind == K_CONTRACT ? pc.coef.d : 1.0;
      a = ref_word(P, T.args[0], access_off(pc.acc[0], o, r, T.rank, pc.nred));
      if (T.nargs > 1) b = ref_word(P, T.args[1], access_off(pc.acc[1], o, r, T.rank, pc.nred));
      return;
    }
    coef = 0.0;
    a = NONE;
    return;
  }
  if (T.kind == K_BINARY) {
    uint64_t ra = ref_word(P, T.args[0], bin_index(P, T, 0, o));
    uint64_t rb = ref_word(P, T.args[1], bin_index(P, T, 1, o));
    if (T.fn == B_ADD || T.fn == B_SUB) {
      coef = j == 0 ? 1.0 : (T.fn == B_ADD ? 1.0 : -1.0);
      a = j == 0 ? ra : rb;
    } else {
      coef = 1.0;
      a = ra;
      b = rb;
    }
    return;
  }
  if (j == 0) {
    coef = T.kind == K_AFFINE ? T.a.d : 1.0;
    a = ref_word(P, T.args[0], e);
  } else {   // the constant of MAXC / AFFINE
    coef = T.c.d;
    a = NONE;
  }
}

// Per listed bitmap word (a word with a marked element): its marked nodes and
// their equation entries, into arrays that are zero elsewhere.  A word never
// spans two tensors (value arrays are 64-element aligned).  One warp per word,
// one lane per bit: the marked elements of a tensor are clustered, so this
// keeps every entry count on its own lane.
__global__ void __launch_bounds__(256) word_count_kernel(const __grid_constant__ Prog P,
                                                         const uint32_t* bits,
                                                         const int64_t* dirty,
                                                         const unsigned long long* n_dirty,
                                                         int64_t* wnodes, int64_t* wents) {
  const int lane = threadIdx.x & 31;
  const int64_t nd = (int64_t)*n_dirty;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < nd; i += nwarps) {
    const int64_t w = dirty[i];
    const uint32_t m = bits[w];
    const int t = tensor_of_word(P, w);
    int64_t c = (m >> lane) & 1 ? entry_count(P, t, (w - P.t[t].ws_off / 32) * 32 + lane) : 0;
#pragma unroll
    for (int s = 16; s >= 1; s >>= 1) c += __shfl_xor_sync(0xffffffffu, c, s);
    if (lane == 0) {
      wnodes[w] = __popc(m);
      wents[w] = c;
    }
  }
}

// Node list (tensor << 40 | elem, in (tensor, elem) order) and the entry
// offset of every node, from the scanned per-word counts (same layout).
__global__ void __launch_bounds__(256) node_list_kernel(const __grid_constant__ Prog P,
                                                        const uint32_t* bits,
                                                        const int64_t* dirty,
                                                        const unsigned long long* n_dirty,
                                                        const int64_t* wnodes,
                                                        const int64_t* wents, uint64_t* nodes,
                                                        int64_t* eoff) {
  const int lane = threadIdx.x & 31;
  const int64_t nd = (int64_t)*n_dirty;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < nd; i += nwarps) {
    const int64_t w = dirty[i];
    const uint32_t m = bits[w];
    const int t = tensor_of_word(P, w);
    const int64_t e = (w - P.t[t].ws_off / 32) * 32 + lane;
    const bool set = (m >> lane) & 1;
    const int64_t c = set ? entry_count(P, t, e) : 0;
    int64_t x = c;   // inclusive scan of the entry counts over the lanes
#pragma unroll
    for (int s = 1; s < 32; s <<= 1) {
      const int64_t y = __shfl_up_sync(0xffffffffu, x, s);
      if (lane >= s) x += y;
    }
    if (set) {
      const int64_t k = wnodes[w] + __popc(m & ((1u << lane) - 1));
      nodes[k] = ((uint64_t)t << 40) | (uint64_t)e;
      eoff[k] = wents[w] + x - c;
    }
  }
}

// Sizes of the export (both programs' node and entry totals, section
// offsets, total bytes); the header and section headers are written when the
// export fits the caller's buffer.
__global__ void export_header_kernel(const int64_t* tot_nodes0, const int64_t* tot_ents0,
                                     const int64_t* tot_nodes1, const int64_t* tot_ents1,
                                     int64_t* eoff0, int64_t* eoff1, uint8_t* exp,
                                     int64_t capacity, DevStats* st) {
  const int64_t nn[2] = {*tot_nodes0, *tot_nodes1}, ne[2] = {*tot_ents0, *tot_ents1};
  eoff0[nn[0]] = ne[0];
  eoff1[nn[1]] = ne[1];
  const int64_t sec0 = 16 + 32 * nn[0] + 24 * ne[0], sec1 = 16 + 32 * nn[1] + 24 * ne[1];
  const int64_t nsel = st->nsel;
  const int64_t required = nsel > 0 ? 32 + sec0 + sec1 + 24 * nsel : 0;
  const bool ok = nsel > 0 && exp != nullptr && required <= capacity;
  for (int p = 0; p < 2; ++p) {
    st->n_nodes[p] = nn[p];
    st->n_ent[p] = ne[p];
  }
  st->sec_off[0] = 32;
  st->sec_off[1] = 32 + sec0;
  st->loc_off = 32 + sec0 + sec1;
  st->required = required;
  st->ok = ok;
  if (!ok) return;
  uint64_t* h = (uint64_t*)exp;
  h[0] = 0x31505844ull | (1ull << 32);   // "DXP1", version 1
  h[1] = (uint64_t)required;
  h[2] = (uint64_t)nsel;
  h[3] = 0;
  uint64_t* h0 = (uint64_t*)(exp + 32);
  h0[0] = (uint64_t)nn[0];
  h0[1] = (uint64_t)ne[0];
  uint64_t* h1 = (uint64_t*)(exp + 32 + sec0);
  h1[0] = (uint64_t)nn[1];
  h1[1] = (uint64_t)ne[1];
}

// Export writer, two grid-stride passes in one launch.  First one thread per
// node writes the node's 32-byte record and the entries of nodes with few
// terms (elementwise equations, small max sets).  Then the entries of larger
// CONTRACT / MAXSET nodes are written by one warp per node: the valid
// reduction box of each piece is computed once, lane i writes entries i,
// i + 32, ..., stepping its reduction digits by 32 in mixed radix (innermost
// dim last).  When the node's operand offsets provably fit in 31
// bits the digits and offsets are 32-bit and branch-free; otherwise each
// offset is formed in 64 bits from the digits.
constexpr int kMaxNodePieces = 8;
constexpr int64_t kLaneNodeMax = 8;   // entries of a node written by one lane

__device__ __forceinline__ int export_kind(const Tensor& T) {
  return T.kind == K_CONTRACT || T.kind == K_AFFINE ? 1
         : T.kind == K_MAXSET || T.kind == K_MAXC   ? 2
         : T.kind == K_UNARY                         ? 3
         : T.fn == B_DIV                             ? 4
                                                     : 1;
}

// operand word of flat offset f into argument `arg`: base + offset in range
// (an input's global id, or a node reference: offsets stay below 2^40),
// bottom outside
__device__ __forceinline__ uint64_t arg_base_word(const Prog& P, int arg) {
  return P.t[arg].kind == K_INPUT ? (uint64_t)P.t[arg].gbase
                                  : (1ull << 63) | ((uint64_t)arg << 40);
}

// Entries of one piece of a CONTRACT / MAXSET node, written by the warp.
__device__ __forceinline__ void warp_piece_entries(const Prog& P, const Tensor& T, const Piece& pc,
                                                   const int32_t* o, const int32_t* vlo,
                                                   const int32_t* vext, int64_t vol, int lane,
                                                   uint64_t* dq) {
  const uint64_t NONE = ~0ull;
  const bool two = T.nargs > 1;
  const int arg0 = T.args[0], arg1 = two ? T.args[1] : T.args[0];
  const uint64_t n0 = (uint64_t)P.t[arg0].numel, n1 = (uint64_t)P.t[arg1].numel;
  const uint64_t w0 = arg_base_word(P, arg0), w1 = arg_base_word(P, arg1);
  const uint64_t bot = (uint64_t)P.G;
  const double cd = T.kind == K_CONTRACT ? pc.coef.d : 1.0;
  const uint64_t cw = (uint64_t)__double_as_longlong(cd);
  // offsets at the box's low corner, and their largest change over the box
  int64_t fa = pc.acc[0].base, fb = pc.acc[1].base, span_a = 0, span_b = 0;
#pragma unroll
  for (int d = 0; d < MR; ++d) {
    if (d < T.rank) {
      fa += pc.acc[0].os[d] * o[d];
      fb += pc.acc[1].os[d] * o[d];
    }
  }
#pragma unroll
  for (int d = 0; d < MRED; ++d) {
    fa += pc.acc[0].rs[d] * vlo[d];
    fb += pc.acc[1].rs[d] * vlo[d];
    const int64_t ra = pc.acc[0].rs[d], rb = pc.acc[1].rs[d];
    span_a += (ra < 0 ? -ra : ra) * (vext[d] - 1);
    span_b += (rb < 0 ? -rb : rb) * (vext[d] - 1);
  }
  // this lane's first digits (entry `lane`) and the digits of the step 32
  int32_t r[MRED], dr[MRED];
  {
    int64_t x = lane, y = 32;
#pragma unroll
    for (int d = MRED - 1; d >= 1; --d) {
      int64_t qq, c;
      divmod64(x, vext[d], qq, c);
      r[d] = (int32_t)c;
      x = qq;
      divmod64(y, vext[d], qq, c);
      dr[d] = (int32_t)c;
      y = qq;
    }
    r[0] = (int32_t)x;
    dr[0] = (int32_t)y;
  }
  const int64_t lim = (int64_t)1 << 31;
  const bool narrow = n0 < (uint64_t)lim && n1 < (uint64_t)lim &&
                      (fa < 0 ? -fa : fa) + span_a < lim && (fb < 0 ? -fb : fb) + span_b < lim &&
                      vol < lim;
  if (narrow) {
    // Entries go out in chunks of 32 (96 words), each store instruction
    // writing 32 consecutive words: store k of lane i writes word 32k + i,
    // field (2k + i) mod 3 of entry (32k + i) / 3.  Over k = 0, 1, 2 a lane
    // writes each field once, so it walks two entries of the chunk: the one
    // whose operand a it writes (digits ra) and the one whose operand b it
    // writes (digits rb).
    int32_t sa[MRED], sb[MRED];
#pragma unroll
    for (int d = 0; d < MRED; ++d) {
      sa[d] = (int32_t)pc.acc[0].rs[d];
      sb[d] = (int32_t)pc.acc[1].rs[d];
    }
    const int m = lane % 3;   // field of store 0; store 1: (m + 2) % 3, store 2: (m + 1) % 3
    const int ka = m == 1 ? 0 : m == 2 ? 1 : 2, kb = m == 2 ? 0 : m == 0 ? 1 : 2;
    const int32_t ba = (int32_t)fa, bb = (int32_t)fb;
    const uint32_t nn0 = (uint32_t)n0, nn1 = (uint32_t)n1;
    const int32_t nwords = 3 * (int32_t)vol;
    int32_t ra[MRED], rb[MRED];
    {
      int64_t xa = (32 * ka + lane) / 3, xb = (32 * kb + lane) / 3;
#pragma unroll
      for (int d = MRED - 1; d >= 1; --d) {
        int64_t qq, c;
        divmod64(xa, vext[d], qq, c);
        ra[d] = (int32_t)c;
        xa = qq;
        divmod64(xb, vext[d], qq, c);
        rb[d] = (int32_t)c;
        xb = qq;
      }
      ra[0] = (int32_t)xa;
      rb[0] = (int32_t)xb;
    }
    uint64_t* q = dq + lane;
    for (int32_t w0i = 0; w0i < nwords; w0i += 96) {
      int32_t oa = ba, ob = bb;
#pragma unroll
      for (int d = 0; d < MRED; ++d) {
        oa += sa[d] * ra[d];
        ob += sb[d] * rb[d];
      }
      const uint64_t va = (uint32_t)oa < nn0 ? w0 + (uint32_t)oa : bot;
      const uint64_t vb = two ? ((uint32_t)ob < nn1 ? w1 + (uint32_t)ob : bot) : NONE;
      const uint64_t x0 = m == 0 ? cw : m == 1 ? va : vb;
      const uint64_t x1 = m == 0 ? vb : m == 1 ? cw : va;   // field (m + 2) % 3
      const uint64_t x2 = m == 0 ? va : m == 1 ? vb : cw;   // field (m + 1) % 3
      const int32_t left = nwords - w0i;
      if (lane < left) q[0] = x0;
      if (32 + lane < left) q[32] = x1;
      if (64 + lane < left) q[64] = x2;
      q += 96;
      int32_t ca = 0, cb = 0;
#pragma unroll
      for (int d = MRED - 1; d >= 1; --d) {
        const int32_t v = ra[d] + dr[d] + ca;
        ca = v >= vext[d] ? 1 : 0;
        ra[d] = v - (ca ? vext[d] : 0);
        const int32_t u = rb[d] + dr[d] + cb;
        cb = u >= vext[d] ? 1 : 0;
        rb[d] = u - (cb ? vext[d] : 0);
      }
      ra[0] += dr[0] + ca;
      rb[0] += dr[0] + cb;
    }
    return;
  }
  for (int64_t jj = lane; jj < vol; jj += 32) {
    int64_t oa = fa, ob = fb;
#pragma unroll
    for (int d = 0; d < MRED; ++d) {
      oa += pc.acc[0].rs[d] * r[d];
      ob += pc.acc[1].rs[d] * r[d];
    }
    uint64_t* q3 = dq + 3 * jj;
    q3[0] = cw;
    q3[1] = (uint64_t)oa < n0 ? w0 + (uint64_t)oa : bot;
    q3[2] = two ? ((uint64_t)ob < n1 ? w1 + (uint64_t)ob : bot) : NONE;
    int carry = 0;
#pragma unroll
    for (int d = MRED - 1; d >= 1; --d) {
      r[d] += dr[d] + carry;
      carry = r[d] >= vext[d];
      if (carry) r[d] -= vext[d];
    }
    r[0] += dr[0] + carry;
  }
}

__device__ __forceinline__ bool coop_node(const Tensor& T, int64_t cnt) {
  return (T.kind == K_CONTRACT || T.kind == K_MAXSET) && T.npieces <= kMaxNodePieces &&
         cnt > kLaneNodeMax;
}

__global__ void __launch_bounds__(256, 3) export_write_kernel(const __grid_constant__ Prog P,
                                                              const uint64_t* nodes,
                                                              const int64_t* eoff,
                                                              DevStats* st, int prog,
                                                              uint8_t* exp) {
  if (!st->ok) return;
  const int64_t n_nodes = st->n_nodes[prog];
  uint8_t* sec = exp + st->sec_off[prog];
  const int lane = threadIdx.x & 31;
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t nthreads = (int64_t)gridDim.x * blockDim.x;
  uint8_t* recs = sec + 16;
  uint8_t* ents = recs + 32 * n_nodes;
  // records, and the entries of small nodes: one thread per node
  for (int64_t k = tid; k < n_nodes; k += nthreads) {
    const uint64_t nd = nodes[k];
    const int t = (int)(nd >> 40);
    const int64_t e = (int64_t)(nd & ((1ull << 40) - 1));
    const Tensor& T = P.t[t];
    const int64_t e0 = eoff[k], cnt = eoff[k + 1] - e0;
    uint64_t* rec = (uint64_t*)(recs + 32 * k);
    rec[0] = (uint64_t)(uint32_t)t | ((uint64_t)export_kind(T) << 32) |
             ((uint64_t)(T.kind == K_UNARY ? (uint8_t)T.fn : 0) << 40);
    rec[1] = (uint64_t)e;
    rec[2] = (uint64_t)e0;
    rec[3] = (uint64_t)cnt;
    if (coop_node(T, cnt)) continue;
    int32_t o[MR];
    unflatten(e, T, o);
    uint64_t* dst = (uint64_t*)(ents + 24 * e0);
    for (int64_t j = 0; j < cnt; ++j) {
      double c;
      uint64_t a, b;
      entry_of(P, t, e, o, j, c, a, b);
      dst[3 * j] = __double_as_longlong(c);
      dst[3 * j + 1] = a;
      dst[3 * j + 2] = b;
    }
  }
  // the entries of large nodes: one warp per node.  A piece whose inner
  // block (the entries of one step of its outermost reduction digit) fits a
  // warp is written in chunks of E = cpo * inner entries (cpo whole inner
  // blocks): the lane's two entries then sit at fixed positions of every
  // chunk, and their offsets advance by cpo steps of the outermost digit per
  // chunk.  Those lane offsets depend only on the piece and the extents of its
  // valid box, so they are kept across the warp's nodes.
  const int m = lane % 3;   // field of store 0; store 1: (m + 2) % 3, store 2: (m + 1) % 3
  const int ja = (32 * (m == 1 ? 0 : m == 2 ? 1 : 2) + lane) / 3;   // entry of field 1
  const int jb = (32 * (m == 2 ? 0 : m == 0 ? 1 : 2) + lane) / 3;   // entry of field 2
  int plan_piece = -1;
  int32_t plan_ext[MRED] = {0, 0, 0, 0};
  int32_t p_cw3 = 0;
  uint32_t p_rela = 0, p_relb = 0, p_stepa = 0, p_stepb = 0;
  // an inner block longer than a warp, along one dim: chunks of 32 entries,
  // p_cpb per block; within a block the offsets advance by p_stepa/b, at a
  // block's end by p_outa/b
  int32_t p_cpb = 0;
  uint32_t p_outa = 0, p_outb = 0;
  int64_t p_spana = 0, p_spanb = 0;
  bool p_ok = false;
  const int64_t lim = (int64_t)1 << 31;
  const uint64_t NONE = ~0ull;
  // Large nodes are handed out at run time, kWrChunk at a time, from a
  // counter in the statistics block: warps on faster SMs take more of them.
  constexpr int64_t kWrChunk = 4;
  int64_t kc = 0, kend = 0;   // this warp's claimed nodes [kc, kend)
  for (;;) {
    if (kc == kend) {
      unsigned long long c0 = 0;
      if (lane == 0) c0 = atomicAdd(&st->wr_next[prog], (unsigned long long)kWrChunk);
      kc = (int64_t)__shfl_sync(0xffffffffu, c0, 0);
      if (kc >= n_nodes) break;
      kend = kc + kWrChunk < n_nodes ? kc + kWrChunk : n_nodes;
    }
    const int64_t k = kc++;
    const uint64_t nd = nodes[k];
    const int t = (int)(nd >> 40);
    const int64_t e = (int64_t)(nd & ((1ull << 40) - 1));
    const Tensor& T = P.t[t];
    const int64_t e0 = eoff[k], cnt = eoff[k + 1] - e0;
    if (!coop_node(T, cnt)) continue;
    int32_t o[MR];
    unflatten(e, T, o);
    uint64_t* dq = (uint64_t*)(ents + 24 * e0);
    for (int q = 0; q < T.npieces; ++q) {
      const int pid = T.piece0 + q;
      const Piece& pc = P.p[pid];
      int32_t vlo[MRED], vext[MRED];
      const int64_t vol = valid_box(pc, o, T.rank, vlo, vext);
      if (vol <= 0) continue;
      bool same = pid == plan_piece;
#pragma unroll
      for (int d = 0; d < MRED; ++d) same = same && plan_ext[d] == vext[d];
      if (!same) {
        plan_piece = pid;
        int32_t inner = 1;
        p_spana = p_spanb = 0;
        bool fits = true;
#pragma unroll
        for (int d = 0; d < MRED; ++d) {
          plan_ext[d] = vext[d];
          if (d > 0) inner *= vext[d];
          const int64_t ra = pc.acc[0].rs[d], rb = pc.acc[1].rs[d];
          p_spana += (ra < 0 ? -ra : ra) * (vext[d] - 1);
          p_spanb += (rb < 0 ? -rb : rb) * (vext[d] - 1);
          fits = fits && ra > -lim && ra < lim && rb > -lim && rb < lim;
        }
        // the dim an inner block longer than a warp runs along (the only
        // dim after the first with more than one step), else -1
        int ld = -1, nbig = 0;
#pragma unroll
        for (int d = 1; d < MRED; ++d)
          if (vext[d] > 1) {
            ld = d;
            ++nbig;
          }
        p_cpb = 0;
        if (fits && inner > 32 && nbig == 1 && inner % 32 == 0 && p_spana < lim && p_spanb < lim) {
          uint32_t ra = 0, rb = 0;
#pragma unroll
          for (int d = 1; d < MRED; ++d)
            if (d == ld) {
              ra = (uint32_t)pc.acc[0].rs[d];
              rb = (uint32_t)pc.acc[1].rs[d];
            }
          p_ok = true;
          p_cpb = inner / 32;
          p_cw3 = 96;
          p_rela = ra * (uint32_t)ja;
          p_relb = rb * (uint32_t)jb;
          p_stepa = 32u * ra;
          p_stepb = 32u * rb;
          p_outa = (uint32_t)pc.acc[0].rs[0] - (uint32_t)(inner - 32) * ra;
          p_outb = (uint32_t)pc.acc[1].rs[0] - (uint32_t)(inner - 32) * rb;
        } else {
          p_ok = fits && inner <= 32 && p_spana < lim && p_spanb < lim;
        }
        if (p_ok && p_cpb == 0) {
          const int32_t cpo = 32 / inner;
          p_cw3 = 3 * cpo * inner;
          uint32_t ra = (uint32_t)pc.acc[0].rs[0] * (uint32_t)(ja / inner);
          uint32_t rb = (uint32_t)pc.acc[1].rs[0] * (uint32_t)(jb / inner);
          int32_t xa = ja % inner, xb = jb % inner;
#pragma unroll
          for (int d = MRED - 1; d >= 1; --d) {
            ra += (uint32_t)pc.acc[0].rs[d] * (uint32_t)(xa % vext[d]);
            xa /= vext[d];
            rb += (uint32_t)pc.acc[1].rs[d] * (uint32_t)(xb % vext[d]);
            xb /= vext[d];
          }
          p_rela = ra;
          p_relb = rb;
          p_stepa = (uint32_t)pc.acc[0].rs[0] * (uint32_t)cpo;
          p_stepb = (uint32_t)pc.acc[1].rs[0] * (uint32_t)cpo;
        }
      }
      if (p_ok) {
        // offsets at the box's low corner
        int64_t fa = pc.acc[0].base, fb = pc.acc[1].base;
#pragma unroll
        for (int d = 0; d < MR; ++d) {
          if (d < T.rank) {
            fa += pc.acc[0].os[d] * o[d];
            fb += pc.acc[1].os[d] * o[d];
          }
        }
#pragma unroll
        for (int d = 0; d < MRED; ++d) {
          fa += pc.acc[0].rs[d] * vlo[d];
          fb += pc.acc[1].rs[d] * vlo[d];
        }
        const bool two = T.nargs > 1;
        const int arg0 = T.args[0], arg1 = two ? T.args[1] : T.args[0];
        const uint64_t n0 = (uint64_t)P.t[arg0].numel, n1 = (uint64_t)P.t[arg1].numel;
        if (n0 < (uint64_t)lim && n1 < (uint64_t)lim && (fa < 0 ? -fa : fa) + p_spana < lim &&
            (fb < 0 ? -fb : fb) + p_spanb < lim && 3 * vol < lim) {
          // every offset of the box fits in 31 bits: 32-bit arithmetic (the
          // words of lanes past the box's end are never stored)
          const uint64_t w0 = arg_base_word(P, arg0), w1 = arg_base_word(P, arg1);
          const uint64_t bot = (uint64_t)P.G;
          const uint64_t cw = (uint64_t)__double_as_longlong(T.kind == K_CONTRACT ? pc.coef.d
                                                                                  : 1.0);
          const uint32_t nn0 = (uint32_t)n0, nn1 = (uint32_t)n1;
          uint32_t oa = (uint32_t)fa + p_rela, ob = (uint32_t)fb + p_relb;
          const int32_t nwords = 3 * (int32_t)vol, cw3 = p_cw3;
          uint64_t* qd = dq + lane;
          int32_t cib = 0;   // chunk within the inner block (p_cpb > 0)
          for (int32_t w0i = 0; w0i < nwords; w0i += cw3) {
            const uint64_t va = oa < nn0 ? w0 + oa : bot;
            const uint64_t vb = two ? (ob < nn1 ? w1 + ob : bot) : NONE;
            const uint64_t x0 = m == 0 ? cw : m == 1 ? va : vb;
            const uint64_t x1 = m == 0 ? vb : m == 1 ? cw : va;
            const uint64_t x2 = m == 0 ? va : m == 1 ? vb : cw;
            const int32_t left = min(cw3, nwords - w0i);
            // written once, read by no later kernel: evict-first stores
            if (lane < left) __stcs(&qd[0], x0);
            if (32 + lane < left) __stcs(&qd[32], x1);
            if (64 + lane < left) __stcs(&qd[64], x2);
            qd += cw3;
            if (p_cpb > 0 && ++cib == p_cpb) {
              cib = 0;
              oa += p_outa;
              ob += p_outb;
            } else {
              oa += p_stepa;
              ob += p_stepb;
            }
          }
          dq += 3 * vol;
          continue;
        }
      }
      warp_piece_entries(P, T, pc, o, vlo, vext, vol, lane, dq);
      dq += 3 * vol;
    }
  }
}

__global__ void export_tail_kernel(int out_r, int out_c, const int64_t* locs, const int64_t* sel,
                                   const DevStats* st, uint8_t* exp, uint8_t* verdict) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (!st->ok || i >= st->nsel) return;
  int64_t s = sel[i], l = locs[s];
  uint64_t* q = (uint64_t*)(exp + st->loc_off + 24 * i);
  q[0] = (uint64_t)s;
  q[1] = (1ull << 63) | ((uint64_t)out_r << 40) | (uint64_t)l;
  q[2] = (1ull << 63) | ((uint64_t)out_c << 40) | (uint64_t)l;
  verdict[s] = DIRIGO_EXPORTED;
}

// ---------------------------------------------------------------- host side

namespace {

struct CmpLayout {
  size_t stats, und, scan_tmp[2], queue, sel, visits[2], nvis[2], boxtab[2], bits[2], wcnt[2],
      went[2], dirty[2], ecnt[2], nodes[2], total;
};

size_t al(size_t x) { return (x + 255) / 256 * 256; }

CmpLayout layout(const dirigo_graph* r, const dirigo_graph* c, int64_t n) {
  CmpLayout L;
  size_t o = 0;
  L.stats = o;
  o += al(sizeof(DevStats));
  L.und = o;
  o += al((size_t)(n + 1) * 8);
  L.queue = o;
  o += al((size_t)(n + 1) * 8);
  L.sel = o;
  o += al((size_t)(n + 1) * 8);
  // per program: the marking scratch (the two programs' export passes run
  // concurrently), then its bitmaps and counts
  for (int p = 0; p < 2; ++p) {
    L.visits[p] = o;
    o += al((size_t)kMarkChunk * kMaxVisits * sizeof(NBox));
    L.nvis[p] = o;
    o += al((size_t)kMarkChunk * 4);
    L.boxtab[p] = o;
    o += al((size_t)kBoxTable * 4);
  }
  const dirigo_graph* gs[2] = {r, c};
  int64_t maxw = 0;
  for (int p = 0; p < 2; ++p) {
    int64_t nw = gs[p]->value_elems / 32;
    maxw = std::max(maxw, std::max(nw, gs[p]->value_elems) + 1);
    L.bits[p] = o;
    o += al((size_t)nw * 4);
    L.wcnt[p] = o;
    o += al((size_t)(nw + 1) * 8);
    L.went[p] = o;
    o += al((size_t)(nw + 1) * 8);
    L.dirty[p] = o;
    o += al((size_t)(nw + 1) * 8);
    L.ecnt[p] = o;
    o += al((size_t)(gs[p]->value_elems + 1) * 8);
    L.nodes[p] = o;
    o += al((size_t)(gs[p]->value_elems + 1) * 8);
  }
  for (int p = 0; p < 2; ++p) {
    L.scan_tmp[p] = o;
    o += al(scan_tmp_bytes(std::max<int64_t>(n, maxw)));
  }
  L.total = o;
  return L;
}

}  // namespace

// A non-blocking stream per device for the candidate's export passes (created
// on first use, kept for the process's lifetime); null if it cannot be made.
cudaStream_t side_stream() {
  static std::mutex mu;
  static cudaStream_t streams[64] = {};
  static bool tried[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if (!tried[dev]) {
    tried[dev] = true;
    if (cudaStreamCreateWithFlags(&streams[dev], cudaStreamNonBlocking) != cudaSuccess)
      streams[dev] = nullptr;
  }
  return streams[dev];
}

// Status and public statistics of a compare from its statistics block (the
// synchronous call maps on the host after its one read, the asynchronous one
// in its last kernel).  *why: 0 the cones' error (they come first; verdicts,
// the export and the counts are still filled in, the flags are NO_CONES),
// 1 a location out of range, 2 an expired bounded wait, 3 an unsupported
// export form, 4 the export did not fit.
__host__ __device__ inline int finish_compare(const DevStats& hs, dirigo_compare_stats* o,
                                              int* why) {
  const bool cone_err = hs.cone_status != 0;
  const int64_t written = hs.ok ? hs.required : 0;
  o->cone_error = hs.cone_status;
  o->n_discharged = (int64_t)hs.n_disc;
  o->n_exported = written ? hs.nsel : 0;
  o->n_unexported = (int64_t)hs.n_und - o->n_exported;
  o->n_cone_differs = cone_err ? 0 : (int64_t)hs.n_cone_diff;
  o->n_bot_ref = cone_err ? 0 : (int64_t)hs.n_bot_ref;
  o->n_bot_cand = cone_err ? 0 : (int64_t)hs.n_bot_cand;
  o->export_bytes = written;
  o->export_required = hs.required;
  if (cone_err) {
    *why = 0;
    return cone_bits_status(hs.cone_status);
  }
  if (hs.status & CE_LOCATION) {
    *why = 1;
    return DIRIGO_E_INVALID;
  }
  if (hs.status & CE_WAIT) {
    *why = 2;
    return DIRIGO_E_CUDA;
  }
  if (hs.status) {
    *why = 3;
    return DIRIGO_E_UNSUPPORTED;
  }
  if (hs.nsel > 0 && !hs.ok) {
    *why = 4;
    return DIRIGO_E_CAPACITY;
  }
  return DIRIGO_OK;
}

__global__ void compare_finish_kernel(const DevStats* st, dirigo_compare_stats* out,
                                      int32_t* status) {
  int why = 0;
  dirigo_compare_stats o;
  const int r = finish_compare(*st, &o, &why);
  *out = o;
  if (status) *status = r;
}

// An empty batch of the asynchronous compare: zero statistics, and the status
// the cone calls' word maps to.
__global__ void compare_empty_kernel(const int32_t* cone_status, dirigo_compare_stats* out,
                                     int32_t* status) {
  dirigo_compare_stats o = {0, 0, 0, 0, 0, 0, 0, 0, 0};
  const int32_t cs = cone_status ? *cone_status : 0;
  o.cone_error = cs;
  *out = o;
  if (status) *status = cone_bits_status(cs);
}

dirigo_status launch_compare_empty(const int32_t* d_cone_status, dirigo_compare_stats* d_stats,
                                   int32_t* d_status, cudaStream_t s) {
  compare_empty_kernel<<<1, 1, 0, s>>>(d_cone_status, d_stats, d_status);
  count_launch();
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? DIRIGO_OK : set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
}

// A second one for the compare's flag passes, which may wait for the cones.
cudaStream_t flag_stream() {
  static std::mutex mu;
  static cudaStream_t streams[64] = {};
  static bool tried[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if (!tried[dev]) {
    tried[dev] = true;
    if (cudaStreamCreateWithFlags(&streams[dev], cudaStreamNonBlocking) != cudaSuccess)
      streams[dev] = nullptr;
  }
  return streams[dev];
}

size_t compare_ws_bytes(const dirigo_graph* r, const dirigo_graph* c, int64_t n) {
  return layout(r, c, n).total;
}

dirigo_status launch_compare(const dirigo_graph* ref, const dirigo_graph* cand,
                             const int64_t* d_locs, int64_t n, const uint32_t* d_kref,
                             const uint32_t* d_kcand, const int64_t* d_off_ref,
                             const uint32_t* d_runs_ref, const uint64_t* d_fp_ref,
                             const int64_t* d_off_cand, const uint32_t* d_runs_cand,
                             const uint64_t* d_fp_cand, const int32_t* d_cone_status,
                             cudaEvent_t cones_ready, uint8_t* d_verdict, uint8_t* d_flags,
                             int64_t budget, uint8_t* d_export, int64_t export_capacity,
                             dirigo_compare_stats* h_stats, void* d_ws, cudaStream_t s,
                             dirigo_compare_stats* async_stats, int32_t* async_status) {
  CmpLayout Lo = layout(ref, cand, n);
  char* ws = (char*)d_ws;
  DevStats* st = (DevStats*)(ws + Lo.stats);
  int64_t* und = (int64_t*)(ws + Lo.und);
  int64_t* queue = (int64_t*)(ws + Lo.queue);
  int64_t* sel = (int64_t*)(ws + Lo.sel);
  int64_t* tmp = (int64_t*)(ws + Lo.scan_tmp[0]);
  cudaError_t e = cudaMemsetAsync(st, 0, sizeof(DevStats), s);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  unsigned nb = (unsigned)((n + 255) / 256);
  if (nb == 0) nb = 1;
  {
    Prof pr(DIRIGO_K_COMPARE, s);
    verdict_kernel<<<nb, 256, 0, s>>>(d_locs, n, ref->out_numel, (const uint2*)d_kref,
                                      (const uint2*)d_kcand, d_off_ref ? 0 : 1, d_verdict,
                                      d_flags, und, st);
    count_launch();
  }
  // The flags need the cones, the verdicts and the export only the keys: the
  // flag passes run on a stream of their own, after the statistics block is
  // cleared and after `cones_ready` (when given), and are joined back before
  // the statistics are read.
  cudaEvent_t flag_join = nullptr;
  if (d_off_ref) {
    cudaStream_t fs = flag_stream();
    cudaEvent_t fork = nullptr;
    bool own = fs != nullptr &&
               cudaEventCreateWithFlags(&fork, cudaEventDisableTiming) == cudaSuccess &&
               cudaEventCreateWithFlags(&flag_join, cudaEventDisableTiming) == cudaSuccess &&
               cudaEventRecord(fork, s) == cudaSuccess &&
               cudaStreamWaitEvent(fs, fork, 0) == cudaSuccess &&
               (cones_ready == nullptr || cudaStreamWaitEvent(fs, cones_ready, 0) == cudaSuccess);
    if (fork) cudaEventDestroy(fork);
    if (!own) {   // everything on the caller's stream, after the cones
      fs = s;
      if (flag_join) cudaEventDestroy(flag_join);
      flag_join = nullptr;
      if (cones_ready && cudaStreamWaitEvent(s, cones_ready, 0) != cudaSuccess)
        return set_error(DIRIGO_E_CUDA, "waiting for the cones");
    }
    Prof pr(DIRIGO_K_COMPARE, fs);
    cone_flags_kernel<<<nb, 256, 0, fs>>>(
        n, d_off_ref, (const uint2*)d_runs_ref, d_fp_ref, d_off_cand, (const uint2*)d_runs_cand,
        d_fp_cand, d_cone_status, ref->prog.G, cand->prog.G,
        !(ref->prog.cell_on && ref->n_generic_cells == 0),
        !(cand->prog.cell_on && cand->n_generic_cells == 0), d_flags, queue, st);
    count_launch();
    const unsigned eb = (unsigned)std::min<int64_t>(152 * 8, (n + 7) / 8 + 1);
    compare_exact_kernel<<<eb, 256, 0, fs>>>(queue, st, d_off_ref, (const uint2*)d_runs_ref,
                                             d_off_cand, (const uint2*)d_runs_cand, d_flags);
    count_launch();
    count_flags_kernel<<<nb, 256, 0, fs>>>(d_flags, n, st);
    count_launch();
    if (flag_join && cudaEventRecord(flag_join, fs) != cudaSuccess)
      return set_error(DIRIGO_E_CUDA, "recording the flag passes' end");
  }
  launch_scan(und, n, tmp, &st->status, s);   // und[i] = undischarged rank of slot i, und[n] = count
  // Export of the first min(budget, undischarged) slots.  Every size is
  // computed on the device, so the call waits for the GPU once, at the end;
  // the host bounds the root count by min(budget, n) and the kernels stop at
  // the device's count.
  export_init_kernel<<<1, 1, 0, s>>>(und + n, budget, st);
  count_launch();
  const int64_t max_roots = std::min<int64_t>(std::max<int64_t>(budget, 0), n);
  if (max_roots > 0) {
    Prof pr(DIRIGO_K_EXPORT, s);
    select_kernel<<<nb, 256, 0, s>>>(und, d_verdict, n, budget, sel);
    count_launch();
    const dirigo_graph* gs[2] = {ref, cand};
    // The two programs' marking and counting passes are independent and made
    // of small, latency-bound kernels: the candidate's run on a side stream
    // forked from (and joined back into) the caller's stream.
    cudaStream_t side = side_stream();
    cudaEvent_t fork = nullptr, join = nullptr;
    if (side) {
      if (cudaEventCreateWithFlags(&fork, cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&join, cudaEventDisableTiming) != cudaSuccess ||
          cudaEventRecord(fork, s) != cudaSuccess || cudaStreamWaitEvent(side, fork, 0) != cudaSuccess)
        side = nullptr;   // run both passes on the caller's stream
    }
    for (int p = 0; p < 2; ++p) {
      const Prog& P = gs[p]->prog;
      const cudaStream_t sp = p == 1 && side ? side : s;
      int64_t* ptmp = (int64_t*)(ws + Lo.scan_tmp[p]);
      uint32_t* bits = (uint32_t*)(ws + Lo.bits[p]);
      const int64_t nw = gs[p]->value_elems / 32;
      int64_t* wcnt = (int64_t*)(ws + Lo.wcnt[p]);
      int64_t* went = (int64_t*)(ws + Lo.went[p]);
      int64_t* dirty = (int64_t*)(ws + Lo.dirty[p]);
      e = cudaMemsetAsync(bits, 0, (size_t)nw * 4, sp);
      if (e == cudaSuccess) e = cudaMemsetAsync(wcnt, 0, (size_t)(nw + 1) * 8, sp);
      if (e == cudaSuccess) e = cudaMemsetAsync(went, 0, (size_t)(nw + 1) * 8, sp);
      if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
      NBox* visits = (NBox*)(ws + Lo.visits[p]);
      int32_t* nvis = (int32_t*)(ws + Lo.nvis[p]);
      for (int64_t c0 = 0; c0 < max_roots; c0 += kMarkChunk) {
        const int64_t nr = std::min(kMarkChunk, max_roots - c0);
        record_kernel<<<(unsigned)((nr + 127) / 128), 128, 0, sp>>>(P, d_locs, sel, c0, nr,
                                                                   visits, nvis, st);
        int32_t* boxtab = (int32_t*)(ws + Lo.boxtab[p]);
        e = cudaMemsetAsync(boxtab, 0xff, (size_t)kBoxTable * 4, sp);   // all slots -1
        if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
        mark_kernel<<<(unsigned)((nr * kMaxVisits + 7) / 8), 256, 0, sp>>>(
            P, visits, nvis, nr, bits, dirty, &st->n_dirty[p], boxtab);
        count_launch();
        count_launch();
      }
      const unsigned wb = (unsigned)std::min<int64_t>((nw + 7) / 8 + 1, 152 * 16);
      word_count_kernel<<<wb, 256, 0, sp>>>(P, bits, dirty, &st->n_dirty[p], wcnt, went);
      count_launch();
      launch_scan(wcnt, nw, ptmp, &st->status, sp);
      launch_scan(went, nw, ptmp, &st->status, sp);
      node_list_kernel<<<wb, 256, 0, sp>>>(P, bits, dirty, &st->n_dirty[p], wcnt, went,
                                           (uint64_t*)(ws + Lo.nodes[p]),
                                           (int64_t*)(ws + Lo.ecnt[p]));
      count_launch();
    }
    if (side) {
      e = cudaEventRecord(join, side);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(s, join, 0);
      cudaEventDestroy(fork);
      cudaEventDestroy(join);
      if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
    } else {
      if (fork) cudaEventDestroy(fork);
      if (join) cudaEventDestroy(join);
    }
    const int64_t nw0 = ref->value_elems / 32, nw1 = cand->value_elems / 32;
    export_header_kernel<<<1, 1, 0, s>>>(
        (int64_t*)(ws + Lo.wcnt[0]) + nw0, (int64_t*)(ws + Lo.went[0]) + nw0,
        (int64_t*)(ws + Lo.wcnt[1]) + nw1, (int64_t*)(ws + Lo.went[1]) + nw1,
        (int64_t*)(ws + Lo.ecnt[0]), (int64_t*)(ws + Lo.ecnt[1]), d_export, export_capacity, st);
    count_launch();
    for (int p = 0; p < 2; ++p) {
      export_write_kernel<<<152 * 32, 256, 0, s>>>(gs[p]->prog, (uint64_t*)(ws + Lo.nodes[p]),
                                                  (int64_t*)(ws + Lo.ecnt[p]), st, p, d_export);
      count_launch();
    }
    export_tail_kernel<<<(unsigned)((max_roots + 255) / 256), 256, 0, s>>>(
        ref->prog.output, cand->prog.output, d_locs, sel, st, d_export, d_verdict);
    count_launch();
  }
  if (flag_join) {
    e = cudaStreamWaitEvent(s, flag_join, 0);
    cudaEventDestroy(flag_join);
    if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  }
  if (async_stats) {
    compare_finish_kernel<<<1, 1, 0, s>>>(st, async_stats, async_status);
    count_launch();
    e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
    return DIRIGO_OK;
  }
  DevStats hs;
  e = cudaMemcpyAsync(&hs, st, sizeof(DevStats), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  dirigo_compare_stats tmp_stats;
  int why = 0;
  const int ret = finish_compare(hs, h_stats ? h_stats : &tmp_stats, &why);
  if (ret == DIRIGO_OK) return DIRIGO_OK;
  if (why == 0) return cone_status_error(hs.cone_status);
  return set_error((dirigo_status)ret, why == 1   ? "a location is outside the output"
                                       : why == 2 ? "prefix sum: a bounded wait expired"
                                       : why == 3 ? "export: an index map outside the supported forms"
                                                  : "export buffer too small");
}

}  // namespace dirigo
