// Cone of influence of each queried location as maximal runs of global ids
// (Sec. 3.4 "Back-projection": the leaves reached by res(y[l])).
//
// Two passes over the batch:
//   cone_count  one thread per location: the run count of the location's
//               cone cell (cells.h), or, in a generic cell, box
//               propagation, then a run plan, then the exact number of
//               maximal runs;
//   (scan)      exclusive prefix sum -> CSR offsets; one host sync to check
//               the capacity;
//   cone_write  one warp per 32 locations: each lane looks up its own
//               location's cell, then the warp writes each location's runs
//               cooperatively (32 consecutive 8-byte runs per store
//               instruction) from the cell's plan with affine starts, or
//               from the plan slot the count pass left for a generic cell.
// Fast plan: the location's run streams are in range, strictly increasing
// with gaps ("regular") and occupy disjoint global-id ranges; maximal runs
// then differ from the streams' runs only where one stream's last run touches
// the next stream's first run, so the plan lists those junction runs and the
// interior run ranges of each stream.  Otherwise (reads past a tensor's end,
// overlapping streams) the owning lane merges the streams serially.
#include <cstdlib>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "cells.h"
#include "cone_prop.cuh"
#include "internal.h"
#include "launch.h"

namespace dirigo {

struct Plan {
  int fast;
  int ns;
  int nbw;
  int64_t count;
  uint32_t gs[NS];                 // global start of each stream (fast plan)
  uint32_t j0[NS], j1[NS], pos[NS];
  uint32_t bw_pos[NS + 1], bw_start[NS + 1], bw_len[NS + 1];
};

__device__ __forceinline__ int64_t stream_last_off(const Stream& s) {
  int64_t x = 0;
  for (int k = 0; k < s.nd; ++k) x += (int64_t)s.step[k] * (s.cnt[k] - 1);
  return x;
}

__device__ __forceinline__ int64_t stream_runs(const Stream& s) {
  int64_t r = 1;
  for (int k = 0; k < s.nd; ++k) r *= s.cnt[k];
  return r;
}

// Serial merge of all streams with clipping to each tensor's range; bottom
// (id G) closes the list when any read falls outside its tensor.  emit(start,
// len) is called for every maximal run in order; returns the run count.
template <class Emit>
__device__ int64_t slow_merge(const Prog& P, LocState& L, Emit& emit) {
  int64_t cur[NS];
  uint32_t idx[NS][MSD];
  bool done[NS];
  for (int s = 0; s < L.nst; ++s) {
    const Stream& S = L.st[s];
    // run starts must not decrease along the stream
    int64_t inner = 0;
    for (int k = 0; k < S.nd; ++k) {
      if ((int64_t)S.step[k] < inner) L.err |= CE_NONMONOTONE;
      inner += (int64_t)S.step[k] * (S.cnt[k] - 1);
    }
    cur[s] = S.start;
    done[s] = false;
    for (int k = 0; k < MSD; ++k) idx[s][k] = 0;
  }
  if (L.err) return 0;
  bool bot = false;
  int64_t ps = -1, pe = -1, count = 0;
  while (true) {
    int best = -1;
    int64_t bs = 0, be = 0;
    for (int s = 0; s < L.nst; ++s) {
      const Stream& S = L.st[s];
      const Tensor& A = P.t[S.t];
      while (!done[s]) {
        int64_t a = cur[s], b = cur[s] + S.L;
        if (a < 0 || b > A.numel) bot = true;
        int64_t ca = a < 0 ? 0 : a, cb = b > A.numel ? A.numel : b;
        if (ca < cb) {
          int64_t gs = A.gbase + ca;
          if (best < 0 || gs < bs) {
            best = s;
            bs = gs;
            be = A.gbase + cb;
          }
          break;
        }
        // entirely outside: skip this run
        int k = 0;
        for (; k < S.nd; ++k) {
          if (++idx[s][k] < S.cnt[k]) {
            cur[s] += S.step[k];
            break;
          }
          cur[s] -= (int64_t)S.step[k] * (S.cnt[k] - 1);
          idx[s][k] = 0;
        }
        if (k == S.nd) done[s] = true;
      }
    }
    if (best < 0) break;
    {  // advance the chosen stream
      const Stream& S = L.st[best];
      int k = 0;
      for (; k < S.nd; ++k) {
        if (++idx[best][k] < S.cnt[k]) {
          cur[best] += S.step[k];
          break;
        }
        cur[best] -= (int64_t)S.step[k] * (S.cnt[k] - 1);
        idx[best][k] = 0;
      }
      if (k == S.nd) done[best] = true;
    }
    if (ps >= 0 && bs <= pe) {
      if (be > pe) pe = be;
    } else {
      if (ps >= 0) {
        emit(count, ps, pe - ps);
        ++count;
      }
      ps = bs;
      pe = be;
    }
  }
  if (bot) {
    if (ps >= 0 && pe == P.G) {
      pe = P.G + 1;
    } else {
      if (ps >= 0) {
        emit(count, ps, pe - ps);
        ++count;
      }
      ps = P.G;
      pe = P.G + 1;
    }
  }
  if (ps >= 0) {
    emit(count, ps, pe - ps);
    ++count;
  }
  return count;
}

struct CountEmit {
  __device__ void operator()(int64_t, int64_t, int64_t) {}
};

// Propagation + run plan for one location.
__device__ void plan_location(const Prog& P, int64_t loc, LocState& L, Plan& pl) {
  NoVisit nv;
  propagate(P, loc, L, nv);
  if (!L.err) boxes_to_streams(P, L);
  pl.fast = 0;
  pl.ns = 0;
  pl.nbw = 0;
  pl.count = 0;
  if (L.err) return;
  bool fast = true;
  for (int s = 0; s < L.nst && fast; ++s) {
    const Stream& S = L.st[s];
    const Tensor& A = P.t[S.t];
    if (S.start < 0 || S.start + stream_last_off(S) + S.L > A.numel) fast = false;
    if (S.nd > 3) fast = false;
    int64_t span = S.L;
    for (int k = 0; k < S.nd; ++k) {
      if ((int64_t)S.step[k] <= span) fast = false;   // adjacency or overlap inside the stream
      span += (int64_t)S.step[k] * (S.cnt[k] - 1);
    }
  }
  if (fast) {
    // global starts; order the streams by start
    uint32_t gs[NS];
    for (int s = 0; s < L.nst; ++s) gs[s] = (uint32_t)(P.t[L.st[s].t].gbase + L.st[s].start);
    for (int i = 1; i < L.nst; ++i) {
      Stream x = L.st[i];
      uint32_t gx = gs[i];
      int j = i;
      while (j > 0 && gs[j - 1] > gx) {
        L.st[j] = L.st[j - 1];
        gs[j] = gs[j - 1];
        --j;
      }
      L.st[j] = x;
      gs[j] = gx;
    }
    // single runs that overlap or touch collapse into one
    int m = 0;
    for (int s = 0; s < L.nst; ++s) {
      if (m > 0 && L.st[m - 1].nd == 0 && L.st[s].nd == 0 &&
          gs[s] <= gs[m - 1] + (int64_t)L.st[m - 1].L) {
        int64_t e = max((int64_t)gs[m - 1] + L.st[m - 1].L, (int64_t)gs[s] + L.st[s].L);
        L.st[m - 1].L = (uint32_t)(e - gs[m - 1]);
        continue;
      }
      L.st[m] = L.st[s];
      gs[m] = gs[s];
      ++m;
    }
    L.nst = m;
    for (int s = 1; s < L.nst; ++s) {
      int64_t prev_end = (int64_t)gs[s - 1] + stream_last_off(L.st[s - 1]) + L.st[s - 1].L;
      if ((int64_t)gs[s] < prev_end) fast = false;
    }
    if (fast) {
      int64_t out = 0;
      bool pend = false;
      int64_t pst = 0, pen = 0;
      for (int s = 0; s < L.nst; ++s) {
        const Stream& S = L.st[s];
        int64_t R = stream_runs(S);
        int64_t first = gs[s], last = gs[s] + stream_last_off(S);
        uint32_t j0 = 0;
        if (pend && pen == first) {
          pen = first + S.L;
          if (R == 1) {
            pl.j0[s] = pl.j1[s] = 0;
            pl.pos[s] = (uint32_t)out;
            pl.gs[s] = gs[s];
            continue;
          }
          pl.bw_pos[pl.nbw] = (uint32_t)out;
          pl.bw_start[pl.nbw] = (uint32_t)pst;
          pl.bw_len[pl.nbw] = (uint32_t)(pen - pst);
          ++pl.nbw;
          ++out;
          j0 = 1;
        } else if (pend) {
          pl.bw_pos[pl.nbw] = (uint32_t)out;
          pl.bw_start[pl.nbw] = (uint32_t)pst;
          pl.bw_len[pl.nbw] = (uint32_t)(pen - pst);
          ++pl.nbw;
          ++out;
        }
        pl.gs[s] = gs[s];
        pl.j0[s] = j0;
        pl.j1[s] = (uint32_t)(R - 1 > j0 ? R - 1 : j0);
        pl.pos[s] = (uint32_t)out;
        out += pl.j1[s] - pl.j0[s];
        pst = last;
        pen = last + S.L;
        pend = true;
      }
      if (pend) {
        pl.bw_pos[pl.nbw] = (uint32_t)out;
        pl.bw_start[pl.nbw] = (uint32_t)pst;
        pl.bw_len[pl.nbw] = (uint32_t)(pen - pst);
        ++pl.nbw;
        ++out;
      }
      pl.fast = 1;
      pl.ns = L.nst;
      pl.count = out;
      return;
    }
  }
  CountEmit ce;
  pl.count = slow_merge(P, L, ce);
}

// Plan slot of one location (kPlanWords 32-bit words), written by the count
// pass and read by the write pass:
//   w0 count of runs, w1 mode | nseg << 8 | nbw << 16 (mode 0: fast plan in
//   the slot; 1: the write pass replans and merges serially),
//   w2.. nseg segments of kSegWords: gs, L, step[3], cnt[2], magic[2], j0, j1,
//   pos (magic = ceil(2^32 / cnt) for division by multiplication, 0: divide),
//   then nbw boundary runs of 3 words: pos, start, len.
constexpr int kSegWords = 12;
constexpr int kMaxSeg = 2;
constexpr int kMaxBw = 4;
constexpr int kPlanWords = 40;   // 2 + 2*12 + 4*3 = 38, padded to 160 bytes

__host__ __device__ __forceinline__ uint32_t div_magic(uint32_t d) {
  return (d > 1 && d < (1u << 27)) ? (uint32_t)(((1ull << 32) + d - 1) / d) : 0u;
}

// q = x / d for x <= 64 (the first runs of a warp's lanes)
__device__ __forceinline__ uint32_t div_small(uint32_t x, uint32_t d, uint32_t magic) {
  return magic ? __umulhi(x, magic) : (d == 1 ? x : x / d);
}

__device__ __forceinline__ bool pack_plan(const LocState& L, const Plan& pl, uint32_t* w) {
  int nseg = 0;
  for (int s = 0; s < pl.ns; ++s)
    if (pl.j1[s] > pl.j0[s]) ++nseg;
  if (!pl.fast || nseg > kMaxSeg || pl.nbw > kMaxBw || pl.count >= ((int64_t)1 << 32))
    return false;
  w[0] = (uint32_t)pl.count;
  w[1] = 0u | ((uint32_t)nseg << 8) | ((uint32_t)pl.nbw << 16);
  int k = 2;
  for (int s = 0; s < pl.ns; ++s) {
    if (pl.j1[s] <= pl.j0[s]) continue;
    const Stream& S = L.st[s];
    w[k + 0] = pl.gs[s];
    w[k + 1] = S.L;
    for (int d = 0; d < 3; ++d) w[k + 2 + d] = d < S.nd ? S.step[d] : 0u;
    for (int d = 0; d < 2; ++d) {
      uint32_t c = d < S.nd ? S.cnt[d] : 1u;
      w[k + 5 + d] = c;
      w[k + 7 + d] = div_magic(c);
    }
    w[k + 9] = pl.j0[s];
    w[k + 10] = pl.j1[s];
    w[k + 11] = pl.pos[s];
    k += kSegWords;
  }
  k = 2 + kMaxSeg * kSegWords;
  for (int b = 0; b < pl.nbw; ++b) {
    w[k + 3 * b] = pl.bw_pos[b];
    w[k + 3 * b + 1] = pl.bw_start[b];
    w[k + 3 * b + 2] = pl.bw_len[b];
  }
  return true;
}

// Cell of output location loc (coordinates in o); -1 when the cell is generic.
__device__ __forceinline__ int cell_of(const Prog& P, const uint8_t* cells, int64_t loc,
                                       int32_t* o) {
  const Tensor& Y = P.t[P.output];
  unflatten(loc, Y, o);
  const uint16_t* idx = reinterpret_cast<const uint16_t*>(cells);
  int c = 0;
#pragma unroll
  for (int d = 0; d < MR; ++d)
    if (d < Y.rank) c += (int)__ldg(idx + P.cell_tab[d] + o[d]) * P.cell_radix[d];
  const CellRec* rec = reinterpret_cast<const CellRec*>(cells + P.cell_rec_off);
  return __ldg(&rec[c].nseg) == kCellGeneric ? -1 : c;
}

__global__ void __launch_bounds__(128) cone_count_kernel(const __grid_constant__ Prog P,
                                                         const int64_t* locs, int64_t n,
                                                         int64_t* counts, uint4* plans,
                                                         const uint8_t* cells,
                                                         int32_t* status) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= n) return;
  if (cells) {
    const int64_t loc = locs[i];
    if (loc < 0 || loc >= P.t[P.output].numel) {
      atomicOr(status, CE_LOCATION);
      counts[i] = 0;
      return;
    }
    int32_t o[MR];
    const int c = cell_of(P, cells, loc, o);
    if (c >= 0) {
      counts[i] = reinterpret_cast<const CellRec*>(cells + P.cell_rec_off)[c].count;
      return;
    }
  }
  LocState L;
  Plan pl;
  plan_location(P, locs[i], L, pl);
  if (L.err) atomicOr(status, L.err);
  counts[i] = L.err ? 0 : pl.count;
  if (!plans) return;
  uint32_t w[kPlanWords];
  if (L.err || !pack_plan(L, pl, w)) {
    w[0] = (uint32_t)pl.count;
    w[1] = 1u;
  }
  uint4* dst = plans + i * (kPlanWords / 4);
#pragma unroll
  for (int q = 0; q < kPlanWords / 4; ++q)
    dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
}

// Counts when every cone cell of the graph has a fast plan: one table lookup
// per location.  Each thread takes kCountPer locations (256 apart, so that
// every load instruction is coalesced) and looks them up side by side, an
// out-of-range location as location 0 with its result discarded, so that the
// lookups' dependent loads overlap; one short block per 256 * kCountPer
// locations (a block loops only past 2^31 - 1 blocks).
constexpr int kCountPer = 4;
__global__ void __launch_bounds__(256) cone_count_cells_kernel(const __grid_constant__ Prog P,
                                                               const int64_t* locs, int64_t n,
                                                               int64_t* counts,
                                                               const uint8_t* cells,
                                                               int32_t* status) {
  const int64_t numel = P.t[P.output].numel;
  const CellRec* rec = reinterpret_cast<const CellRec*>(cells + P.cell_rec_off);
  int bad = 0;
  for (int64_t chunk = blockIdx.x; chunk * (256 * kCountPer) < n; chunk += gridDim.x) {
    const int64_t base = chunk * (256 * kCountPer) + threadIdx.x;
    int64_t lv[kCountPer];
#pragma unroll
    for (int k = 0; k < kCountPer; ++k) {
      const int64_t i = base + 256 * k;
      lv[k] = i < n ? locs[i] : 0;
    }
#pragma unroll
    for (int k = 0; k < kCountPer; ++k) {
      const int64_t i = base + 256 * k;
      const bool ok = lv[k] >= 0 && lv[k] < numel;
      bad |= (i < n && !ok) ? 1 : 0;
      int32_t o[MR];
      const int c = cell_of(P, cells, ok ? lv[k] : 0, o);
      const int64_t cnt = ok && c >= 0 ? (int64_t)__ldg(&rec[c].count) : 0;
      if (i < n) counts[i] = cnt;
    }
  }
  if (bad) atomicOr(status, CE_LOCATION);
}

struct WriteEmit {
  uint2* runs;
  int64_t cap;     // runs reserved for this location by the count pass
  uint64_t fp;
  int bad;
  uint64_t rk = 1;   // kFpR^k for the next run k (runs come in order)
  __device__ void operator()(int64_t k, int64_t s, int64_t len) {
    if (k >= cap) {
      bad = 1;
      return;
    }
    runs[k] = make_uint2((uint32_t)s, (uint32_t)len);
    fp += fp_term((uint32_t)s, (uint32_t)len) * rk;
    rk *= kFpR;
  }
};

// Runs j in [j0, j1) of one segment, 32 per store instruction; with kHash,
// returns the lane's share of the fingerprint (run j sits at position
// pos + j - j0 of the location's list).
template <bool kHash>
__device__ __forceinline__ uint64_t write_segment(uint2* runs, int64_t off, int64_t cnt,
                                                  uint32_t g0, uint32_t Lr, uint32_t st0,
                                                  uint32_t st1, uint32_t st2, uint32_t ct0,
                                                  uint32_t ct1, uint32_t mg0, uint32_t mg1,
                                                  uint32_t j0, uint32_t j1, uint32_t pos,
                                                  int lane, int32_t* status) {
  uint64_t h = 0;
  // digits of this lane's first run and of the stride 32 (all <= 64)
  uint32_t j = j0 + lane;
  uint32_t r1 = div_small(j, ct0, mg0), i0 = j - r1 * ct0;
  uint32_t i2 = div_small(r1, ct1, mg1), i1 = r1 - i2 * ct1;
  uint32_t b1 = div_small(32u, ct0, mg0), a0 = 32u - b1 * ct0;
  uint32_t a2 = div_small(b1, ct1, mg1), a1 = b1 - a2 * ct1;
  uint2* dst = runs + off + pos - j0;
  int64_t lim = cnt - (int64_t)pos + j0;   // j < lim keeps the write in this location
  uint64_t rk = kHash ? fp_pow((uint64_t)pos + lane) : 0;
  const uint64_t r32 = kHash ? fp_pow(32) : 0;
  for (; j < j1; j += 32) {
    uint32_t sv = g0 + st0 * i0 + st1 * i1 + st2 * i2;
    if ((int64_t)j < lim)
      dst[j] = make_uint2(sv, Lr);
    else
      atomicOr(status, CE_CAPACITY);
    if (kHash) {
      h += fp_term(sv, Lr) * rk;
      rk *= r32;
    }
    i0 += a0;
    uint32_t c = i0 >= ct0;
    i0 -= c * ct0;
    i1 += a1 + c;
    c = i1 >= ct1;
    i1 -= c * ct1;
    i2 += a2 + c;
  }
  return h;
}

// Sum over the warp of a 64-bit value, mod 2^64.
__device__ __forceinline__ uint64_t warp_sum64(uint64_t h) {
#pragma unroll
  for (int sh = 16; sh > 0; sh >>= 1) h += __shfl_xor_sync(0xffffffffu, h, sh);
  return h;
}

// Fingerprint of a location in a fast cell: affine in its coordinates.
__device__ __forceinline__ uint64_t cell_fp(const CellRec& rec, const int32_t* o) {
  uint64_t h = rec.fp[0];
#pragma unroll
  for (int d = 0; d < MR; ++d) h += rec.fp[1 + d] * (uint64_t)(uint32_t)o[d];
  return h;
}

__device__ __forceinline__ uint32_t affine_at(int64_t c, const int64_t* a, const int32_t* o) {
  int64_t v = c;
#pragma unroll
  for (int d = 0; d < MR; ++d) v += a[d] * o[d];
  return (uint32_t)v;
}

// Whether a write pass may store runs: nothing latched in the status word
// so far (a location out of range, an unsupported map, an expired wait) and
// the total the prefix sum left in offsets[n] fits the run buffer.  Otherwise
// the whole pass stores nothing; block 0 latches CE_RUNCAP for a total above
// the capacity.  Read once per block.
__device__ __forceinline__ bool write_pass_allowed(const int64_t* offsets, int64_t n,
                                                   int64_t run_cap, int32_t* status) {
  __shared__ int s_ok;
  if (threadIdx.x == 0) {
    const int64_t total = offsets[n];
    const int32_t st = *(volatile int32_t*)status;
    if (total > run_cap && blockIdx.x == 0) atomicOr(status, CE_RUNCAP);
    s_ok = st == 0 && total <= run_cap;
  }
  __syncthreads();
  return s_ok != 0;
}

// Locations in fast cells, one warp per 32 locations.  Each lane resolves its
// own location (cell, CSR range, segment and junction starts at its
// coordinates, fingerprint -- stored at once: it is affine in the
// coordinates) into the warp's shared-memory slots; then the warp writes the
// locations one after another.  A small fast cell (at most two segments and
// four junction runs) is written from a table of its segments' run offsets
// (start minus the segment's start) in the warp's shared memory: a run is the
// table entry plus the location's segment start, and each lane stores two
// adjacent runs with one 16-byte store (a segment that starts on an odd
// 8-byte slot has its first run stored alone).  A table depends only on the
// segment's steps, counts and run range, so neighbouring cells that differ
// in their starts, run lengths or positions (a clipped border column, say)
// share it and it is rebuilt only when that structure changes.  Segments of
// more than kCwRuns runs, and other fast cells, are read from the cell table
// per location.  Locations in generic cells are left to cone_write_kernel.
constexpr int kCwWarps = 8, kCwRuns = 256;
// Table words per segment: entry 1 + t holds run t's offset (t in [0, n));
// entries 0 and n + 1 are read by the edge lanes of the first and last
// rounds, and the last round's idle lanes read at most 1 + 64*4 + 63.
constexpr int kCwTab = kCwRuns + 66;
struct CwWarp {
  uint4 loc[32];                 // {offset low, offset high, cell, run count}
  uint2 g[32];                   // segment starts (small cells)
  uint32_t bv[kMaxBw][32];       // junction starts (small cells)
  int32_t o[MR][32];             // coordinates (other fast cells)
  uint32_t rel[2][kCwTab];
};

__device__ __forceinline__ void cw_build_tab(const CellSeg& g, int lane, uint32_t* rel) {
  const uint32_t n = g.j1 - g.j0;
  for (uint32_t t = lane; t < n; t += 32) {
    const uint32_t j = g.j0 + t;
    const uint32_t r1 = j / g.ct0, i0 = j - r1 * g.ct0;
    const uint32_t i2 = r1 / g.ct1, i1 = r1 - i2 * g.ct1;
    rel[1 + t] = g.st0 * i0 + g.st1 * i1 + g.st2 * i2;
  }
  if (lane == 0) {
    rel[0] = 0u;
    rel[n + 1] = 0u;
  }
}

// The n <= kCwRuns runs of one segment of one location, starting at dst:
// run t is (g0 + rel[1 + t], L).
__device__ __forceinline__ void cw_pairs(uint2* dst, uint32_t n, uint32_t g0, uint32_t L,
                                         const uint32_t* rel, int lane) {
  if (n == 0) return;
  const int s = (int)((reinterpret_cast<uintptr_t>(dst) >> 3) & 1u);
  const int nr = ((int)n + s + 63) >> 6;
  const int t0 = 2 * lane - s;               // this lane's first run of the first round
  const uint32_t* r = rel + 1 + t0;          // >= rel
  uint4* p = reinterpret_cast<uint4*>(dst - s) + lane;
#pragma unroll
  for (int k = 0; k < (kCwRuns + 64) / 64; ++k) {
    if (k < nr) {
      const int t = t0 + 64 * k;
      const uint32_t a = g0 + r[64 * k], b = g0 + r[64 * k + 1];
      if ((uint32_t)t < n - 1u)
        __stcs(p + 32 * k, make_uint4(a, L, b, L));
      else if (t == -1)
        __stcs(reinterpret_cast<uint2*>(p + 32 * k) + 1, make_uint2(b, L));
      else if (t == (int)n - 1)
        __stcs(reinterpret_cast<uint2*>(p + 32 * k), make_uint2(a, L));
    }
  }
}

__global__ void __launch_bounds__(kCwWarps * 32, 4) cone_write_cells_kernel(
    const __grid_constant__ Prog P, const int64_t* locs, int64_t n, const int64_t* offsets,
    const uint8_t* cells, uint2* runs, uint64_t* fp, int64_t run_cap, int32_t* status) {
  if (!write_pass_allowed(offsets, n, run_cap, status)) return;
  __shared__ CwWarp s_w[kCwWarps];
  CwWarp& W = s_w[threadIdx.x >> 5];
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const CellRec* recs = reinterpret_cast<const CellRec*>(cells + P.cell_rec_off);
  const CellSeg* segs = reinterpret_cast<const CellSeg*>(cells + P.cell_seg_off);
  const CellBw* bws = reinterpret_cast<const CellBw*>(cells + P.cell_bw_off);
  // the small cell in use (warp-uniform) and the tables in the two slots
  int cached = -1, cnseg = 0, cnbw = 0;
  uint32_t ccount = 0, cseg0 = 0, big = 0;
  uint32_t tab0 = 0xffffffffu, tab1 = 0xffffffffu;
  uint32_t sL0 = 0, sL1 = 0, sN0 = 0, sN1 = 0, sP0 = 0, sP1 = 0;
  uint32_t bwlen = 0, bwpos = 0;   // this lane's junction run (lane < cnbw)
  for (int64_t base = warp * 32; base < n; base += nwarps * 32) {
    const int64_t mine = base + lane;
    {
      int cid = -1;
      int64_t moff = 0;
      uint32_t cnt = 0;
      if (mine < n) {
        int32_t o[MR] = {0, 0, 0, 0};
        moff = offsets[mine];
        cnt = (uint32_t)(offsets[mine + 1] - moff);
        const int c = cell_of(P, cells, locs[mine], o);
        if (c >= 0) {
          const CellRec& rec = recs[c];
          if (fp) fp[mine] = cell_fp(rec, o);
          if (rec.nseg <= 2 && rec.nbw <= kMaxBw) {
            cid = c;
            uint32_t g2[2] = {0u, 0u};
            for (int sg = 0; sg < (int)rec.nseg; ++sg)
              g2[sg] = affine_at(segs[rec.seg0 + sg].gc, segs[rec.seg0 + sg].ga, o);
            W.g[lane] = make_uint2(g2[0], g2[1]);
            for (int b = 0; b < (int)rec.nbw; ++b)
              W.bv[b][lane] = affine_at(bws[rec.bw0 + b].sc, bws[rec.bw0 + b].sa, o);
          } else {
            cid = -2 - c;
#pragma unroll
            for (int d = 0; d < MR; ++d) W.o[d][lane] = o[d];
          }
        }
      }
      W.loc[lane] = make_uint4((uint32_t)(uint64_t)moff, (uint32_t)((uint64_t)moff >> 32),
                               (uint32_t)cid, cnt);
    }
    __syncwarp();
    const int last = (int)min((int64_t)32, n - base);
    for (int q = 0; q < last; ++q) {
      const uint4 A = W.loc[q];
      const int cq = (int)A.z;
      if (cq == -1) continue;   // generic cell: cone_write_kernel writes it (uniform over the warp)
      const int64_t off = (int64_t)(((uint64_t)A.y << 32) | A.x);
      const uint32_t cnt = A.w;
      if (cq >= 0) {
        if (cq != cached) {
          const CellRec& rec = recs[cq];
          cnseg = rec.nseg;
          cnbw = rec.nbw;
          ccount = rec.count;
          cseg0 = rec.seg0;
          big = 0;
          __syncwarp();
          for (int sg = 0; sg < cnseg; ++sg) {
            const CellSeg& g = segs[cseg0 + sg];
            const uint32_t nr = g.j1 - g.j0;
            if (sg == 0) {
              sL0 = g.L; sN0 = nr; sP0 = g.pos;
            } else {
              sL1 = g.L; sN1 = nr; sP1 = g.pos;
            }
            uint32_t& tb = sg == 0 ? tab0 : tab1;
            if (nr > (uint32_t)kCwRuns) {
              big |= 1u << sg;
              tb = 0xffffffffu;
            } else if (g.tab != tb) {
              cw_build_tab(g, lane, W.rel[sg]);
              tb = g.tab;
            }
          }
          if (lane < cnbw) {
            bwlen = bws[rec.bw0 + lane].len;
            bwpos = bws[rec.bw0 + lane].pos;
          }
          cached = cq;
          __syncwarp();
        }
        if (cnt != ccount) {   // the count pass reserved another size
          if (lane == 0) atomicOr(status, CE_CAPACITY);
          continue;
        }
        const uint2 G = W.g[q];
        if (big & 1u) {
          const CellSeg& g = segs[cseg0];
          write_segment<false>(runs, off, cnt, G.x, g.L, g.st0, g.st1, g.st2, g.ct0, g.ct1,
                               g.mg0, g.mg1, g.j0, g.j1, g.pos, lane, status);
        } else if (cnseg > 0) {
          cw_pairs(runs + off + sP0, sN0, G.x, sL0, W.rel[0], lane);
        }
        if (cnseg > 1) {
          if (big & 2u) {
            const CellSeg& g = segs[cseg0 + 1];
            write_segment<false>(runs, off, cnt, G.y, g.L, g.st0, g.st1, g.st2, g.ct0, g.ct1,
                                 g.mg0, g.mg1, g.j0, g.j1, g.pos, lane, status);
          } else {
            cw_pairs(runs + off + sP1, sN1, G.y, sL1, W.rel[1], lane);
          }
        }
        if (lane < cnbw) __stcs(&runs[off + bwpos], make_uint2(W.bv[lane][q], bwlen));
      } else {
        int32_t oq[MR];
#pragma unroll
        for (int d = 0; d < MR; ++d) oq[d] = W.o[d][q];
        const CellRec& rec = recs[-2 - cq];
        for (int sg = 0; sg < rec.nseg; ++sg) {
          const CellSeg& g = segs[rec.seg0 + sg];
          write_segment<false>(runs, off, cnt, affine_at(g.gc, g.ga, oq), g.L, g.st0, g.st1,
                               g.st2, g.ct0, g.ct1, g.mg0, g.mg1, g.j0, g.j1, g.pos, lane,
                               status);
        }
        for (int b = lane; b < rec.nbw; b += 32) {
          const CellBw& w = bws[rec.bw0 + b];
          const uint32_t sv = affine_at(w.sc, w.sa, oq);
          if ((int64_t)w.pos < (int64_t)cnt)
            __stcs(&runs[off + w.pos], make_uint2(sv, w.len));
          else
            atomicOr(status, CE_CAPACITY);
        }
      }
    }
    __syncwarp();
  }
}

// One warp per location of a generic cell (or every location when the graph
// has no cells): the plan slot is read once (broadcast through shuffles) and
// each segment's runs are written 32 at a time.
__global__ void __launch_bounds__(256) cone_write_kernel(const __grid_constant__ Prog P,
                                                         const int64_t* locs, int64_t n,
                                                         const int64_t* offsets,
                                                         const uint32_t* plans,
                                                         const uint8_t* cells, uint2* runs,
                                                         uint64_t* fp, int64_t run_cap,
                                                         int32_t* status) {
  if (!write_pass_allowed(offsets, n, run_cap, status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = warp; i < n; i += nwarps) {
    if (cells) {
      int32_t o[MR];
      if (cell_of(P, cells, locs[i], o) >= 0) continue;
    }
    const uint32_t* slot = plans + i * kPlanWords;
    uint32_t wl = slot[lane];
    uint32_t wx = lane < kPlanWords - 32 ? slot[32 + lane] : 0u;
    auto W = [&](int k) -> uint32_t {
      uint32_t a = __shfl_sync(0xffffffffu, wl, k & 31);
      uint32_t b = __shfl_sync(0xffffffffu, wx, k & 31);
      return k < 32 ? a : b;
    };
    int64_t off = offsets[i];
    int64_t cnt = offsets[i + 1] - off;
    uint32_t hdr = W(1);
    if (hdr & 0xffu) {   // replan and merge serially on one lane
      if (lane == 0) {
        LocState L;
        Plan pl;
        plan_location(P, locs[i], L, pl);
        if (!L.err) {
          WriteEmit we{runs + off, cnt, 0, 0};
          if (slow_merge(P, L, we) != cnt || we.bad) atomicOr(status, CE_CAPACITY);
          if (fp) fp[i] = we.fp;
        }
      }
      __syncwarp();
      continue;
    }
    int nseg = (hdr >> 8) & 0xff, nbw = (hdr >> 16) & 0xff;
    uint64_t h = 0;
    for (int s = 0; s < nseg; ++s) {
      int k = 2 + s * kSegWords;
      h += write_segment<true>(runs, off, cnt, W(k), W(k + 1), W(k + 2), W(k + 3), W(k + 4),
                               W(k + 5), W(k + 6), W(k + 7), W(k + 8), W(k + 9), W(k + 10),
                               W(k + 11), lane, status);
    }
    int kb = 2 + kMaxSeg * kSegWords;
    uint32_t p = 0, s0 = 0, ln = 0;
    for (int b = 0; b < nbw; ++b) {
      uint32_t pb = W(kb + 3 * b), sb = W(kb + 3 * b + 1), lb = W(kb + 3 * b + 2);
      if (lane == b) {
        p = pb;
        s0 = sb;
        ln = lb;
      }
    }
    if (lane < nbw) {
      if ((int64_t)p < cnt)
        runs[off + p] = make_uint2(s0, ln);
      else
        atomicOr(status, CE_CAPACITY);
      h += fp_term(s0, ln) * fp_pow(p);
    }
    h = warp_sum64(h);
    if (fp && lane == 0) fp[i] = h;
  }
}

// Write pass without plan slots (the fixed-scratch call): one warp per 32
// locations, each lane replans its own location and the warp writes each
// location's runs in turn.
__global__ void __launch_bounds__(128) cone_write_replan_kernel(const __grid_constant__ Prog P,
                                                         const int64_t* locs, int64_t n,
                                                         const int64_t* offsets, uint2* runs,
                                                         uint64_t* fp, int64_t run_cap,
                                                         int32_t* status) {
  if (!write_pass_allowed(offsets, n, run_cap, status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  LocState L;
  Plan pl;
  for (int64_t base = warp * 32; base < n; base += nwarps * 32) {
    int64_t my = base + lane;
    if (my < n) {
      plan_location(P, locs[my], L, pl);
      if (L.err) atomicOr(status, L.err);
    } else {
      pl.fast = 1;
      pl.ns = 0;
      pl.nbw = 0;
      L.err = 0;
    }
    int last = (int)min((int64_t)32, n - base);
    for (int q = 0; q < last; ++q) {
      int fast = __shfl_sync(0xffffffffu, pl.fast && !L.err, q);
      int bad = __shfl_sync(0xffffffffu, L.err, q);
      int64_t off = offsets[base + q];
      int64_t cnt = offsets[base + q + 1] - off;   // runs reserved by the count pass
      if (bad) continue;
      if (!fast) {
        if (lane == q) {
          WriteEmit we{runs + off, cnt, 0, 0};
          if (slow_merge(P, L, we) != cnt || we.bad) atomicOr(status, CE_CAPACITY);
          if (fp) fp[base + q] = we.fp;
        }
        __syncwarp();
        continue;
      }
      uint64_t h = 0;
      int ns = __shfl_sync(0xffffffffu, pl.ns, q);
      for (int s = 0; s < ns; ++s) {
        uint32_t j0 = __shfl_sync(0xffffffffu, pl.j0[s], q);
        uint32_t j1 = __shfl_sync(0xffffffffu, pl.j1[s], q);
        if (j1 <= j0) continue;
        uint32_t g0 = __shfl_sync(0xffffffffu, pl.gs[s], q);
        uint32_t pos = __shfl_sync(0xffffffffu, pl.pos[s], q);
        uint32_t Lr = __shfl_sync(0xffffffffu, L.st[s].L, q);
        int nd = __shfl_sync(0xffffffffu, L.st[s].nd, q);
        uint32_t st[3] = {0, 0, 0}, ct[3] = {1, 1, 1};
        for (int k = 0; k < 3; ++k) {
          uint32_t a = k < L.st[s].nd ? L.st[s].step[k] : 0;
          uint32_t b = k < L.st[s].nd ? L.st[s].cnt[k] : 1;
          st[k] = __shfl_sync(0xffffffffu, a, q);
          ct[k] = __shfl_sync(0xffffffffu, b, q);
        }
        (void)nd;
        // digits of this lane's first run and of the stride 32
        uint32_t j = j0 + lane;
        uint32_t i0 = j % ct[0], r1 = j / ct[0];
        uint32_t i1 = r1 % ct[1], i2 = r1 / ct[1];
        uint32_t a0 = 32 % ct[0], b1 = 32 / ct[0];
        uint32_t a1 = b1 % ct[1], a2 = b1 / ct[1];
        uint2* dst = runs + off + pos - j0;
        int64_t lim = cnt - (int64_t)pos + j0;   // j < lim keeps the write in this location
        uint64_t rk = fp_pow((uint64_t)pos + lane);
        const uint64_t r32 = fp_pow(32);
        for (; j < j1; j += 32) {
          uint32_t sv = g0 + st[0] * i0 + st[1] * i1 + st[2] * i2;
          if ((int64_t)j < lim)
            dst[j] = make_uint2(sv, Lr);
          else
            atomicOr(status, CE_CAPACITY);
          h += fp_term(sv, Lr) * rk;
          rk *= r32;
          i0 += a0;
          uint32_t c = i0 >= ct[0];
          i0 -= c * ct[0];
          i1 += a1 + c;
          c = i1 >= ct[1];
          i1 -= c * ct[1];
          i2 += a2 + c;
        }
      }
      int nbw = __shfl_sync(0xffffffffu, pl.nbw, q);
      for (int b = 0; b < nbw; ++b) {
        uint32_t p = __shfl_sync(0xffffffffu, pl.bw_pos[b], q);
        uint32_t s0 = __shfl_sync(0xffffffffu, pl.bw_start[b], q);
        uint32_t ln = __shfl_sync(0xffffffffu, pl.bw_len[b], q);
        if (lane == (b & 31)) {
          if ((int64_t)p < cnt)
            runs[off + p] = make_uint2(s0, ln);
          else
            atomicOr(status, CE_CAPACITY);
          h += fp_term(s0, ln) * fp_pow(p);
        }
      }
      for (int sh = 16; sh > 0; sh >>= 1) h += __shfl_xor_sync(0xffffffffu, h, sh);
      if (fp && lane == 0) fp[base + q] = h;
    }
  }
}

// ---------------------------------------------------------------- scan
// Exclusive prefix sum of n int64 values in place (data has n + 1 slots;
// data[n] receives the total), in one pass over tiles of 4096 values with
// decoupled look-back.  Each block takes the next tile index from a counter
// (so every earlier tile's block is already running), loads its tile with
// coalesced reads and transposes it through shared memory so that each
// thread holds 16 consecutive values, scans it, publishes the tile's sum, then
// walks back over the published words of the earlier tiles (32 at a time, one
// per lane) until it meets one that carries its inclusive prefix.  A published
// word is the value in the low 62 bits and a state in the top two (1: tile
// sum, 2: inclusive prefix); the values are non-negative counts below 2^62.
// The wait for an unpublished word is bounded (max_polls polls with a short
// sleep): when it expires the block records CE_WAIT in *err and continues.
// stall_tile >= 0 is a test hook: that tile never publishes its word, so the
// next tile's wait runs out (the environment variable DIRIGO_TEST_SCAN_STALL
// sets it, with a short limit, to test how an expired wait is reported).
//
// tmp layout (int64 words, zeroed by launch_scan): [0] tile counter, [1]
// spare, [2 + t] word of tile t.
constexpr int kScanThreads = 256, kScanItems = 16, kScanTile = kScanThreads * kScanItems;
constexpr uint64_t kScanAgg = 1ull << 62, kScanPrefix = 2ull << 62;
constexpr uint64_t kScanValue = (1ull << 62) - 1;
constexpr unsigned kScanMaxPolls = 1u << 20;

// shared-memory slot of tile item i: one pad word per 16 makes both the
// striped (consecutive items per warp) and the blocked (16 per thread)
// accesses conflict-free
__device__ __forceinline__ int scan_slot(int i) { return i + (i >> 4); }

__global__ void __launch_bounds__(kScanThreads) scan_onepass_kernel(int64_t* data, int64_t n,
                                                                    unsigned long long* tmp,
                                                                    int64_t ntiles, int32_t* err,
                                                                    unsigned max_polls,
                                                                    int64_t stall_tile) {
  __shared__ int64_t sm[kScanTile + kScanTile / 16];
  __shared__ int64_t warp_tot[kScanThreads / 32];
  __shared__ int64_t s_before;
  __shared__ unsigned s_tile;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid == 0) s_tile = atomicAdd((unsigned*)tmp, 1u);
  __syncthreads();
  const int64_t t = s_tile;
  const int64_t base = t * kScanTile;
#pragma unroll
  for (int k = 0; k < kScanItems; ++k) {
    const int i = k * kScanThreads + tid;
    sm[scan_slot(i)] = base + i < n ? data[base + i] : 0;
  }
  __syncthreads();
  int64_t v[kScanItems];
  int64_t run = 0;
#pragma unroll
  for (int k = 0; k < kScanItems; ++k) {
    v[k] = run;   // exclusive within the thread
    run += sm[scan_slot(tid * kScanItems + k)];
  }
  int64_t x = run;
#pragma unroll
  for (int s = 1; s < 32; s <<= 1) {
    const int64_t y = __shfl_up_sync(0xffffffffu, x, s);
    if (lane >= s) x += y;
  }
  if (lane == 31) warp_tot[w] = x;
  __syncthreads();
  if (w == 0) {
    int64_t tw = lane < kScanThreads / 32 ? warp_tot[lane] : 0;
#pragma unroll
    for (int s = 1; s < 32; s <<= 1) {
      const int64_t y = __shfl_up_sync(0xffffffffu, tw, s);
      if (lane >= s) tw += y;
    }
    if (lane < kScanThreads / 32) warp_tot[lane] = tw;
    const int64_t agg = __shfl_sync(0xffffffffu, tw, kScanThreads / 32 - 1);   // the tile's sum
    volatile unsigned long long* word = tmp + 2;
    int64_t before = 0;
    if (t == stall_tile) {
      // test hook: publish nothing
    } else if (t == 0) {
      if (lane == 0) word[0] = kScanPrefix | (uint64_t)agg;
    } else {
      if (lane == 0) word[t] = kScanAgg | (uint64_t)agg;
      int64_t j = t - 1;   // nearest earlier tile not yet summed
      unsigned polls = 0;
      while (true) {
        const int64_t idx = j - lane;
        const uint64_t u = idx >= 0 ? (uint64_t)word[idx] : kScanPrefix;
        const uint64_t state = u >> 62;
        const unsigned pre = __ballot_sync(0xffffffffu, state == 2);
        const unsigned none = __ballot_sync(0xffffffffu, state == 0);
        // lanes up to the nearest prefix (all 32 when there is none) must be published
        const int last = pre ? __ffs(pre) - 1 : 31;
        const unsigned need = last == 31 ? 0xffffffffu : ((1u << (last + 1)) - 1);
        if (none & need) {
          if (++polls > max_polls) {
            if (lane == 0) atomicOr(err, (int32_t)CE_WAIT);
            break;
          }
          __nanosleep(32);
          continue;
        }
        int64_t part = lane <= last ? (int64_t)(u & kScanValue) : 0;
#pragma unroll
        for (int s = 16; s >= 1; s >>= 1) part += __shfl_xor_sync(0xffffffffu, part, s);
        before += part;
        if (pre) break;
        j -= 32;
      }
      if (lane == 0) word[t] = kScanPrefix | (uint64_t)(before + agg);
    }
    if (lane == 0) s_before = before;
  }
  __syncthreads();
  const int64_t off = s_before + x - run + (w > 0 ? warp_tot[w - 1] : 0);
#pragma unroll
  for (int k = 0; k < kScanItems; ++k) sm[scan_slot(tid * kScanItems + k)] = off + v[k];
  if (t == ntiles - 1 && tid == kScanThreads - 1) data[n] = off + run;
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kScanItems; ++k) {
    const int i = k * kScanThreads + tid;
    if (base + i < n) data[base + i] = sm[scan_slot(i)];
  }
}

size_t scan_tmp_bytes(int64_t n) { return ((size_t)((n + kScanTile - 1) / kScanTile) + 2) * 8; }

void launch_scan(int64_t* data, int64_t n, int64_t* tmp, int32_t* err, cudaStream_t s) {
  int64_t tiles = (n + kScanTile - 1) / kScanTile;
  if (tiles < 1) tiles = 1;
  // test hook: tile 0 publishes nothing and the waits give up after 4096 polls
  const char* stall = std::getenv("DIRIGO_TEST_SCAN_STALL");
  const bool test_stall = stall && stall[0] == '1' && tiles > 1;
  Prof pr(DIRIGO_K_SCAN, s);
  cudaMemsetAsync(tmp, 0, (size_t)(tiles + 2) * 8, s);
  scan_onepass_kernel<<<(unsigned)tiles, kScanThreads, 0, s>>>(
      data, n, (unsigned long long*)tmp, tiles, err, test_stall ? 4096u : kScanMaxPolls,
      test_stall ? 0 : -1);
  count_launch();
}

size_t cone_ws_bytes(const dirigo_graph* g, int64_t n) {
  size_t scan = (scan_tmp_bytes(n) + 255) / 256 * 256;
  size_t cells = g->prog.cell_on ? (size_t)g->prog.cell_bytes : 0;
  return 256 + scan + cells + (size_t)n * kPlanWords * 4 + 256;
}

size_t cone_ws_bytes_noplan(int64_t n) {
  size_t scan = (scan_tmp_bytes(n) + 255) / 256 * 256;
  return 256 + scan + 256;
}

static_assert((int)CE_UNSUPPORTED == (int)DIRIGO_CONE_ERR_UNSUPPORTED &&
                  (int)CE_CAPACITY == (int)DIRIGO_CONE_ERR_BOXES &&
                  (int)CE_LOCATION == (int)DIRIGO_CONE_ERR_LOCATION &&
                  (int)CE_NONMONOTONE == (int)DIRIGO_CONE_ERR_NONMONOTONE &&
                  (int)CE_WAIT == (int)DIRIGO_CONE_ERR_WAIT &&
                  (int)CE_RUNCAP == (int)DIRIGO_CONE_ERR_RUNS,
              "cone error bits of the C ABI");

// Enqueues count -> prefix sum -> write on `s` without waiting for it.
// Errors are OR-ed into *status (CE_* bits); the write pass stores nothing
// when any bit is set before it or when the total exceeds run_capacity.
dirigo_status enqueue_cone(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                           int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                           uint64_t* d_fp, int32_t* status, void* d_ws, cudaStream_t s,
                           bool plan_slots) {
  const Prog& P = g->prog;
  int64_t* tmp = (int64_t*)((char*)d_ws + 256);
  char* after_scan = (char*)d_ws + 256 + (scan_tmp_bytes(n) + 255) / 256 * 256;
  // the cell table is copied into the workspace with the call (the graph
  // itself holds no device memory); the fixed-scratch call plans every
  // location on its own
  uint8_t* cells = plan_slots && P.cell_on ? (uint8_t*)after_scan : nullptr;
  uint32_t* plans =
      plan_slots ? (uint32_t*)(after_scan + (cells ? (size_t)P.cell_bytes : 0)) : nullptr;
  cudaError_t e = cudaSuccess;
  if (cells && n > 0) {
    std::call_once(g->cells_pinned_once, [g] {
      void* p = nullptr;
      if (cudaHostAlloc(&p, g->cells.size(), cudaHostAllocDefault) == cudaSuccess) {
        std::memcpy(p, g->cells.data(), g->cells.size());
        g->cells_pinned = (uint8_t*)p;
      } else {
        cudaGetLastError();   // no pinned copy: upload from the vector
      }
    });
    const uint8_t* src = g->cells_pinned ? g->cells_pinned : g->cells.data();
    e = cudaMemcpyAsync(cells, src, (size_t)P.cell_bytes, cudaMemcpyHostToDevice, s);
  }
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  if (n > 0) {
    Prof pr(DIRIGO_K_CONE_COUNT, s);
    if (cells && g->n_generic_cells == 0) {
      const int64_t blocks =
          std::min<int64_t>((n + 256 * kCountPer - 1) / (256 * kCountPer), 0x7fffffff);
      cone_count_cells_kernel<<<(unsigned)blocks, 256, 0, s>>>(P, d_locs, n, d_offsets, cells,
                                                              status);
    } else {
      cone_count_kernel<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(P, d_locs, n, d_offsets,
                                                                    (uint4*)plans, cells, status);
    }
    count_launch();
  }
  launch_scan(d_offsets, n, tmp, status, s);
  if (n > 0) {
    Prof pr(DIRIGO_K_CONE_WRITE, s);
    uint2* runs = (uint2*)d_runs;
    if (plans) {
      if (cells) {
        // 8 warps of 32 lanes, 32 locations per warp, one pass per block: a
        // grid of many short blocks lets the block scheduler even out the
        // SMs' store rates (a grid of resident blocks only ends with the
        // slowest SM's share)
        const int64_t blocks = std::min<int64_t>((n + 255) / 256, 0x7fffffff);
        cone_write_cells_kernel<<<(unsigned)blocks, 256, 0, s>>>(P, d_locs, n, d_offsets, cells,
                                                                runs, d_fp, run_capacity, status);
      }
      if (!cells || g->n_generic_cells > 0) {
        int64_t blocks = (n + 7) / 8;   // 8 warps of 32 lanes, one location per warp
        if (blocks > 152 * 32) blocks = 152 * 32;
        cone_write_kernel<<<(unsigned)blocks, 256, 0, s>>>(P, d_locs, n, d_offsets, plans, cells,
                                                          runs, d_fp, run_capacity, status);
        count_launch();
      }
    } else {
      int64_t warps = (n + 31) / 32;
      int64_t blocks = (warps + 3) / 4;
      if (blocks > 152 * 16) blocks = 152 * 16;
      cone_write_replan_kernel<<<(unsigned)blocks, 128, 0, s>>>(P, d_locs, n, d_offsets, runs,
                                                               d_fp, run_capacity, status);
    }
    count_launch();
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  return DIRIGO_OK;
}

dirigo_status cone_status_error(int32_t st) {
  if (st & CE_LOCATION) return set_error(DIRIGO_E_INVALID, "cone: a location is outside the output");
  if (st & (CE_UNSUPPORTED | CE_NONMONOTONE))
    return set_error(DIRIGO_E_UNSUPPORTED, "cone: an index map outside the supported cone forms");
  if (st & CE_CAPACITY)
    return set_error(DIRIGO_E_UNSUPPORTED,
                     "cone: a cone needs more than 12 boxes (8 per tensor) or 6 run streams");
  if (st & CE_WAIT) return set_error(DIRIGO_E_CUDA, "cone: prefix sum: a bounded wait expired");
  if (st & CE_RUNCAP)
    return set_error(DIRIGO_E_CAPACITY, "cone: run buffer too small (offsets[n] holds the runs needed)");
  return DIRIGO_OK;
}

dirigo_status launch_cone(const dirigo_graph* g, const int64_t* d_locs, int64_t n,
                          int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                          uint64_t* d_fp, int64_t* h_total, void* d_ws, cudaStream_t s,
                          bool plan_slots) {
  // the workspace's status word collects this call's errors; the stream is
  // waited for once, at the end, for the total and the status
  int32_t* status = (int32_t*)d_ws;
  cudaError_t e = cudaMemsetAsync(status, 0, 8, s);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  dirigo_status r = enqueue_cone(g, d_locs, n, d_offsets, d_runs, run_capacity, d_fp, status,
                                 d_ws, s, plan_slots);
  if (r != DIRIGO_OK) return r;
  int64_t total = 0;
  int32_t st = 0;
  e = cudaMemcpyAsync(&total, d_offsets + n, 8, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&st, status, 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return set_error(DIRIGO_E_CUDA, cudaGetErrorString(e));
  if (h_total) *h_total = total;
  if (st & CE_RUNCAP) st &= ~CE_RUNCAP;   // reported below with the total
  r = cone_status_error(st);
  if (r != DIRIGO_OK) return r;
  if (total > run_capacity) return set_error(DIRIGO_E_CAPACITY, "run buffer too small");
  return DIRIGO_OK;
}

}  // namespace dirigo
