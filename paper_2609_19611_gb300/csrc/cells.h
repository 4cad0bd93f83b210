// Cone cells (library-internal): a partition of the output index space into
// boxes on which the cone of a location has a fixed run structure.
//
// The box propagation of the cone kernels (reverse SSA order, Sec. 3.4
// "Back-projection") only adds, scales, clips and compares coordinates, so on
// any box of output coordinates where every comparison it makes has one
// outcome, the cone's streams have fixed shapes and their starts are affine
// in the location's coordinates.  The compiler finds such boxes (a product
// grid over the output dims) by running the propagation symbolically, and
// stores per cell the run plan with affine starts; the cone kernels then
// count a location's runs with one table lookup and write them without
// planning.  Cells whose plan is not of that form (reads past a tensor's
// end, overlapping streams, non-affine index arithmetic) are marked generic
// and their locations are planned one by one as before.
//
// Blob layout (bytes, all little-endian, offsets in Prog::cell_*):
//   uint16 idx[sum of output dims]   interval index of each coordinate, per dim
//   CellRec[n_cells]                 row-major over the per-dim intervals
//   CellSeg[]                        run segments of the fast cells
//   CellBw[]                         junction runs of the fast cells
#pragma once
#include <cstdint>
#include <vector>

#include "prog.h"

namespace dirigo {

constexpr uint16_t kCellGeneric = 0xffff;

#if defined(__CUDACC__)
#define DIRIGO_HD __host__ __device__
#else
#define DIRIGO_HD
#endif

// Fingerprint of a run list (start_k, len_k), k = 0 .. m-1 its position in
// the list: the sum over k of (kFpA * start_k + kFpB * len_k + kFpC) * kFpR^k
// mod 2^64 (odd multipliers: SplitMix64's increment and two finaliser
// multipliers, and xorshift64*'s multiplier).  It is affine in the starts, so
// on a cone cell, where every start is affine in the location's coordinates,
// it is an affine function of the coordinates, stored with the cell.
constexpr uint64_t kFpA = 0x9E3779B97F4A7C15ull, kFpB = 0xBF58476D1CE4E5B9ull,
                   kFpC = 0x94D049BB133111EBull, kFpR = 0x2545F4914F6CDD1Dull;
DIRIGO_HD inline uint64_t fp_term(uint64_t start, uint64_t len) {
  return kFpA * start + kFpB * len + kFpC;
}
// kFpR^e mod 2^64
DIRIGO_HD inline uint64_t fp_pow(uint64_t e) {
  uint64_t r = 1, b = kFpR;
  while (e) {
    if (e & 1) r *= b;
    b *= b;
    e >>= 1;
  }
  return r;
}

struct CellRec {
  uint32_t count;   // runs of every location of the cell
  uint16_t nseg;    // kCellGeneric: plan each location on its own
  uint16_t nbw;
  uint32_t seg0, bw0;
  uint32_t pad[2];
  // fingerprint of a location's run list: fp[0] + sum_d fp[1 + d] * o[d]
  uint64_t fp[MR + 1];
};

// Runs j in [j0, j1) of a stream: start gs + st0*i0 + st1*i1 + st2*i2 with
// j = i0 + ct0*(i1 + ct1*i2), length L, written at position pos + j - j0.
// gs = gc + sum_d ga[d] * o[d] for output coordinates o.  tab names the
// table of offsets st0*i0 + st1*i1 + st2*i2 over [j0, j1): the index of the
// first segment of the blob with the same steps, counts, j0 and j1, so that
// a writer can keep one table for cells that differ only in gs, L and pos.
struct CellSeg {
  int64_t gc;
  int64_t ga[MR];
  uint32_t L, st0, st1, st2, ct0, ct1, mg0, mg1, j0, j1, pos, tab;
};

// One run [sc + sum_d sa[d] * o[d], +len) at position pos.
struct CellBw {
  int64_t sc;
  int64_t sa[MR];
  uint32_t len, pos;
};

// Builds the cell blob of program P (fills P.cell_*); returns false (and
// leaves cells off) when the partition would be too fine.
bool build_cells(Prog& P, std::vector<uint8_t>& blob);

}  // namespace dirigo
