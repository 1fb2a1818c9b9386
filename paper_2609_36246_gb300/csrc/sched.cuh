// sched.cuh -- device-side work decomposition shared by the kernels that
// reduce a row over vocabulary tiles (forward log-sum-exp, divergence).
//
// The row count N_mask lives on the device, so every CTA (and the finalize
// kernels) derive the same decomposition from it: rt row tiles of 128 rows,
// vt vocabulary tiles, split into sv contiguous segments of seg tiles.  A
// unit is one (row tile, segment); its partial (max, sum) per row is merged by
// the finalize kernel.  sv is chosen to minimise the critical path
// ceil(units / ctas) * seg, which removes most of the wave-quantisation loss
// when rt is small compared with the SM count.
#pragma once

#include <cuda_bf16.h>

#include "internal.h"

namespace olive {

struct Split {
  int n;     // valid rows
  int rt;    // row tiles
  int vt;    // vocabulary tiles
  int sv;    // segments
  int seg;   // tiles per segment
  int units; // rt * sv
};

__host__ __device__ inline Split choose_split(int n, int vt, int ctas, int sv_cap = kSvMax) {
  Split s;
  s.n = n;
  s.rt = (n + 127) / 128;
  s.vt = vt;
  int best_sv = 1;
  long long best_cost = -1;
  const int max_sv = vt < sv_cap ? vt : sv_cap;
  for (int sv = 1; sv <= max_sv; ++sv) {
    const int seg = (vt + sv - 1) / sv;
    const int sv_eff = (vt + seg - 1) / seg;
    if (sv_eff != sv) continue;
    const long long units = static_cast<long long>(s.rt) * sv;
    const long long waves = (units + ctas - 1) / ctas;
    // a unit also pays a pipeline fill and a partial write: ~1/8 tile
    const long long cost = waves * (8LL * seg + 1);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best_sv = sv;
    }
  }
  s.sv = best_sv;
  s.seg = (vt + best_sv - 1) / best_sv;
  s.units = s.rt * s.sv;
  return s;
}

// Slabs of the G buffer: n masked rows are cut into n_slabs equal slabs of
// at most tc rows (rps rows each, a multiple of 128); slab s covers compacted
// rows [row0, row0 + in_s).  Shared by every kernel that works on one slab.
struct SlabPlan {
  int n_slabs, rps;
  __host__ __device__ SlabPlan(int n, int tc) {
    n_slabs = n > 0 ? (n + tc - 1) / tc : 1;
    const int per = (n + n_slabs - 1) / n_slabs;
    rps = (per + 127) / 128 * 128;
  }
  __host__ __device__ int rows_in(int n, int s) const {
    const int r = n - s * rps;
    return r < 0 ? 0 : (r > rps ? rps : r);
  }
};

__device__ inline int read_n_rows(const int32_t* n_rows, int T, int32_t* dev_status) {
  int n = *n_rows;
  if (n < 0 || n > T) {
    if (dev_status) atomicOr(dev_status, 1 << OLIVE_ERR_OFFSETS);
    n = n < 0 ? 0 : T;
  }
  return n;
}

}  // namespace olive
