// Inversion of a kernel's write set into per-element equations (Sec. 3.4
// "Per-element equations": a kernel yields symbolic writes -- under a path
// condition on (tid, bid) a thread writes a value to an address affine in
// (tid, bid) -- and the equation at output location l is the value of the
// thread whose address is l).
//
// The paper solves a(tid, bid) = l for each concrete l.  Here every location
// is needed at once, so each write is inverted symbolically: its thread box is
// mapped onto a box of output coordinates, and the thread coordinates become
// affine functions of the output coordinates on that box.  That holds when
// every thread coordinate the write varies is one digit of one output
// coordinate (a block row index and a thread row index forming
// row = blockIdx.y * TM + threadIdx.y, for instance): the digits of one output
// coordinate must have address steps S_d * 1, S_d * n1, S_d * n1 * n2, ...
// (S_d the coordinate's row-major stride, n the digits' extents), so that the
// written set is a box and each thread coordinate is (o_d - c_d) / step mod n.
// Reads and guards of the write are then affine in the output coordinates
// when they combine the digits of each output coordinate in the same
// proportion as the address does; a guard may involve one output coordinate.
//
// Host only.
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

namespace dirigo {
namespace {

constexpr int TD = DIRIGO_THREAD_DIMS;

struct OBox {
  int64_t lo[DIRIGO_MAX_RANK], hi[DIRIGO_MAX_RANK];
};

bool overlap(const OBox& a, const OBox& b, int R) {
  for (int d = 0; d < R; ++d)
    if (a.hi[d] <= b.lo[d] || b.hi[d] <= a.lo[d]) return false;
  return true;
}

// One varied thread coordinate j of a write: theta_j = base_j + sign_j * u_j
// with u_j in [0, n_j); it is digit u_j = (o_d - c_d) / gamma mod n_j of
// output coordinate d.
struct Digit {
  int j, d;
  int64_t gamma, n;
};

}  // namespace

dirigo_status invert_kernel_writes(const dirigo_op_desc& op, std::vector<dirigo_piece>* out,
                                   std::string* err) {
  const int R = op.rank;
  auto fail = [&](dirigo_status s, const char* m) {
    *err = m;
    return s;
  };
  if (R < 1 || R > DIRIGO_MAX_RANK) return fail(DIRIGO_E_UNSUPPORTED, "kernel output rank");
  int64_t shape[DIRIGO_MAX_RANK], S[DIRIGO_MAX_RANK], total = 1;
  for (int d = R - 1; d >= 0; --d) {
    shape[d] = op.shape[d];
    if (shape[d] <= 0) return fail(DIRIGO_E_SHAPE, "bad kernel output shape");
    S[d] = total;
    total *= shape[d];
  }
  const int64_t launch[TD] = {op.grid[0], op.grid[1], op.grid[2],
                              op.block[0], op.block[1], op.block[2]};
  for (int j = 0; j < TD; ++j)
    if (launch[j] <= 0) return fail(DIRIGO_E_INVALID, "kernel launch dims must be positive");
  if (op.n_writes < 0 || (op.n_writes > 0 && !op.writes))
    return fail(DIRIGO_E_INVALID, "kernel writes missing");
  std::vector<OBox> boxes;
  for (int w = 0; w < op.n_writes; ++w) {
    const dirigo_kernel_write& kw = op.writes[w];
    if (kw.n_red < 0 || kw.n_red > DIRIGO_MAX_RED || kw.n_guards < 0 ||
        kw.n_guards > DIRIGO_MAX_GUARDS)
      return fail(DIRIGO_E_UNSUPPORTED, "kernel write: too many reduction dims or guards");
    int64_t base[TD], n[TD], sign[TD], A0 = kw.addr_base;
    bool empty = false;
    for (int j = 0; j < TD; ++j) {
      const int64_t lo = std::max<int64_t>(0, kw.when_lo[j]);
      const int64_t hi = std::min<int64_t>(launch[j], kw.when_hi[j]);
      if (hi <= lo) empty = true;
      n[j] = hi - lo;
      sign[j] = kw.addr[j] < 0 ? -1 : 1;
      base[j] = sign[j] > 0 ? lo : hi - 1;
      A0 += kw.addr[j] * base[j];
    }
    if (empty) continue;   // no thread takes this path
    // the write's first location and the digits of each output coordinate
    for (int j = 0; j < TD; ++j)
      if (n[j] > 1 && kw.addr[j] == 0)
        return fail(DIRIGO_E_UNSUPPORTED, "kernel write: threads of one write store to the same location");
    if (A0 < 0 || A0 >= total) return fail(DIRIGO_E_UNSUPPORTED, "kernel write outside its output");
    int64_t c[DIRIGO_MAX_RANK];
    {
      int64_t x = A0;
      for (int d = R - 1; d >= 0; --d) {
        c[d] = x % shape[d];
        x /= shape[d];
      }
    }
    std::vector<Digit> dig;
    for (int j = 0; j < TD; ++j) {
      if (n[j] <= 1) continue;
      const int64_t beta = kw.addr[j] < 0 ? -kw.addr[j] : kw.addr[j];
      int d = 0;
      while (d < R - 1 && S[d] > beta) ++d;   // outermost coordinate with stride <= beta
      if (S[d] > beta || beta % S[d] != 0)
        return fail(DIRIGO_E_UNSUPPORTED, "kernel write: address step not a multiple of an output stride");
      dig.push_back({j, d, beta / S[d], n[j]});
    }
    std::sort(dig.begin(), dig.end(), [](const Digit& a, const Digit& b) {
      return a.d != b.d ? a.d < b.d : a.gamma < b.gamma;
    });
    OBox box;
    for (int d = 0; d < DIRIGO_MAX_RANK; ++d) {
      box.lo[d] = d < R ? c[d] : 0;
      box.hi[d] = d < R ? c[d] + 1 : 1;
    }
    for (size_t i = 0; i < dig.size(); ++i) {
      const bool first = i == 0 || dig[i - 1].d != dig[i].d;
      const int64_t want = first ? 1 : dig[i - 1].gamma * dig[i - 1].n;
      if (dig[i].gamma != want)
        return fail(DIRIGO_E_UNSUPPORTED, "kernel write: written set is not a box of output coordinates");
      box.hi[dig[i].d] = c[dig[i].d] + dig[i].gamma * dig[i].n;
    }
    for (int d = 0; d < R; ++d)
      if (box.hi[d] > shape[d]) return fail(DIRIGO_E_UNSUPPORTED, "kernel write outside its output");
    for (const OBox& b : boxes)
      if (overlap(b, box, R))
        return fail(DIRIGO_E_UNSUPPORTED, "kernel writes: two writes store to the same location");
    boxes.push_back(box);
    // sum_j k_j theta_j = cst + sum_d lam_d o_d on the box, or false
    auto affine = [&](const int64_t* k, int64_t* cst, int64_t* lam) {
      int64_t v0 = 0;
      for (int j = 0; j < TD; ++j) v0 += k[j] * base[j];
      for (int d = 0; d < DIRIGO_MAX_RANK; ++d) lam[d] = 0;
      for (size_t i = 0; i < dig.size(); ++i) {
        const Digit& g = dig[i];
        const int64_t v = k[g.j] * sign[g.j];   // coefficient of u_j
        const bool first = i == 0 || dig[i - 1].d != g.d;
        if (first) lam[g.d] = v;                // gamma of the first digit is 1
        else if (v != lam[g.d] * g.gamma) return false;
      }
      for (int d = 0; d < R; ++d) v0 -= lam[d] * c[d];
      *cst = v0;
      return true;
    };
    dirigo_piece pc;
    std::memset(&pc, 0, sizeof(pc));
    for (int d = 0; d < DIRIGO_MAX_RANK; ++d) {
      pc.lo[d] = box.lo[d];
      pc.hi[d] = box.hi[d];
    }
    pc.n_red = kw.n_red;
    for (int e = 0; e < kw.n_red; ++e) {
      pc.red_lo[e] = kw.red_lo[e];
      pc.red_hi[e] = kw.red_hi[e];
    }
    pc.coef = kw.coef;
    for (int i = 0; i < op.n_args && i < 2; ++i) {
      int64_t cst, lam[DIRIGO_MAX_RANK];
      if (!affine(kw.reads[i].tc, &cst, lam))
        return fail(DIRIGO_E_UNSUPPORTED, "kernel write: a read is not affine in the output coordinates");
      pc.access[i].base = kw.reads[i].base + cst;
      for (int d = 0; d < DIRIGO_MAX_RANK; ++d) pc.access[i].os[d] = lam[d];
      for (int e = 0; e < DIRIGO_MAX_RED; ++e) pc.access[i].rs[e] = kw.reads[i].rs[e];
    }
    pc.n_guards = kw.n_guards;
    for (int q = 0; q < kw.n_guards; ++q) {
      const dirigo_kguard& kg = kw.guards[q];
      int64_t cst, lam[DIRIGO_MAX_RANK];
      if (!affine(kg.tc, &cst, lam))
        return fail(DIRIGO_E_UNSUPPORTED, "kernel write: a guard is not affine in the output coordinates");
      int od = -1;
      for (int d = 0; d < R; ++d) {
        if (lam[d] == 0) continue;
        if (od >= 0) return fail(DIRIGO_E_UNSUPPORTED, "kernel write: a guard spans two output coordinates");
        od = d;
      }
      pc.guards[q] = dirigo_guard{od, kg.rd, od >= 0 ? lam[od] : 0, kg.c + cst, kg.lo, kg.hi};
    }
    out->push_back(pc);
  }
  // Locations no write reaches hold the undefined value: the output cells that
  // no written box covers, cut along every box boundary, each get one term
  // whose operands are all read out of range.
  std::vector<std::vector<int64_t>> cuts(R);
  for (int d = 0; d < R; ++d) {
    cuts[d] = {0, shape[d]};
    for (const OBox& b : boxes) {
      cuts[d].push_back(b.lo[d]);
      cuts[d].push_back(b.hi[d]);
    }
    std::sort(cuts[d].begin(), cuts[d].end());
    cuts[d].erase(std::unique(cuts[d].begin(), cuts[d].end()), cuts[d].end());
  }
  std::vector<size_t> idx(R, 0);
  while (true) {
    OBox cell;
    for (int d = 0; d < DIRIGO_MAX_RANK; ++d) {
      cell.lo[d] = d < R ? cuts[d][idx[d]] : 0;
      cell.hi[d] = d < R ? cuts[d][idx[d] + 1] : 1;
    }
    bool covered = false;
    for (const OBox& b : boxes) covered = covered || overlap(b, cell, R);
    if (!covered) {
      dirigo_piece pc;
      std::memset(&pc, 0, sizeof(pc));
      for (int d = 0; d < DIRIGO_MAX_RANK; ++d) {
        pc.lo[d] = cell.lo[d];
        pc.hi[d] = cell.hi[d];
      }
      pc.n_red = 1;
      pc.red_lo[0] = 0;
      pc.red_hi[0] = 1;
      pc.coef = dirigo_const{1.0, 1, 1};
      for (int i = 0; i < 2; ++i) pc.access[i].base = -1;
      out->push_back(pc);
    }
    int d = R - 1;
    while (d >= 0 && ++idx[d] + 1 >= cuts[d].size()) idx[d--] = 0;
    if (d < 0) break;
  }
  if (out->empty()) return fail(DIRIGO_E_INVALID, "kernel without writes");
  return DIRIGO_OK;
}

// Locations written by the corner threads of a kernel launch (Sec. 4 "Search
// Heuristic", first tier): the first and last thread of the first and last
// block, then threads 31 and 32 of block 0 (the first warp boundary).  Blocks
// and threads are numbered x fastest; a thread that no write's path
// condition admits writes nothing.  In this order, duplicates dropped.
std::vector<int64_t> kernel_corner_locations(const dirigo_op_desc& op) {
  std::vector<int64_t> out;
  const int64_t nb = op.grid[0] * op.grid[1] * op.grid[2];
  const int64_t nt = op.block[0] * op.block[1] * op.block[2];
  if (nb <= 0 || nt <= 0 || op.n_writes <= 0 || !op.writes) return out;
  const int64_t corner[6][2] = {{0, 0}, {nt - 1, 0}, {0, nb - 1}, {nt - 1, nb - 1},
                                {31, 0}, {32, 0}};
  for (const auto& tb : corner) {
    const int64_t t = tb[0], b = tb[1];
    if (t >= nt) continue;
    const int64_t th[6] = {b / (op.grid[1] * op.grid[2]), (b / op.grid[2]) % op.grid[1],
                           b % op.grid[2], t / (op.block[1] * op.block[2]),
                           (t / op.block[2]) % op.block[1], t % op.block[2]};
    for (int w = 0; w < op.n_writes; ++w) {
      const dirigo_kernel_write& kw = op.writes[w];
      bool in = true;
      int64_t a = kw.addr_base;
      for (int j = 0; j < 6; ++j) {
        in = in && th[j] >= kw.when_lo[j] && th[j] < kw.when_hi[j];
        a += kw.addr[j] * th[j];
      }
      if (in && std::find(out.begin(), out.end(), a) == out.end()) out.push_back(a);
    }
  }
  return out;
}

}  // namespace dirigo
