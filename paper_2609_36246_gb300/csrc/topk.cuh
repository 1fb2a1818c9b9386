// topk.cuh -- fixed-length top lists kept in registers by the sweeps that
// report each row's K largest logits (K <= 16).
#pragma once

namespace olive {

constexpr int kTopMax = 16;  // list length kept per row

// True if (cv, ci) belongs before the list's last entry: larger value, or
// the same value with a smaller id.
__device__ __forceinline__ bool topk_beats_last(const float (&tv)[kTopMax],
                                                const int (&ti)[kTopMax], float cv, int ci) {
  return cv > tv[kTopMax - 1] || (cv == tv[kTopMax - 1] && ci < ti[kTopMax - 1]);
}

// Inserts (cv, ci) into a list sorted by value descending, then id ascending;
// the last entry falls off.
__device__ __forceinline__ void topk_insert(float (&tv)[kTopMax], int (&ti)[kTopMax], float cv,
                                            int ci) {
#pragma unroll
  for (int j = 0; j < kTopMax; ++j) {
    const bool before = cv > tv[j] || (cv == tv[j] && ci < ti[j]);
    const float v = tv[j];
    const int i = ti[j];
    tv[j] = before ? cv : v;
    ti[j] = before ? ci : i;
    cv = before ? v : cv;
    ci = before ? i : ci;
  }
}

// The same with a payload value carried along with each entry.
__device__ __forceinline__ void topk_insert3(float (&tv)[kTopMax], int (&ti)[kTopMax],
                                             float (&tx)[kTopMax], float cv, int ci, float cx) {
#pragma unroll
  for (int j = 0; j < kTopMax; ++j) {
    const bool before = cv > tv[j] || (cv == tv[j] && ci < ti[j]);
    const float v = tv[j];
    const int i = ti[j];
    const float x = tx[j];
    tv[j] = before ? cv : v;
    ti[j] = before ? ci : i;
    tx[j] = before ? cx : x;
    cv = before ? v : cv;
    ci = before ? i : ci;
    cx = before ? x : cx;
  }
}

// The same two insertions for a sweep that visits ids in ascending order
// within the list's lifetime: the new id is larger than every id already
// listed, so among equal values it belongs last, and the value alone decides
// its place (no id comparisons).
__device__ __forceinline__ void topk_insert_asc(float (&tv)[kTopMax], int (&ti)[kTopMax], float cv,
                                                int ci) {
#pragma unroll
  for (int j = 0; j < kTopMax; ++j) {
    const bool before = cv > tv[j];
    const float v = tv[j];
    const int i = ti[j];
    tv[j] = before ? cv : v;
    ti[j] = before ? ci : i;
    cv = before ? v : cv;
    ci = before ? i : ci;
  }
}

__device__ __forceinline__ void topk_insert3_asc(float (&tv)[kTopMax], int (&ti)[kTopMax],
                                                 float (&tx)[kTopMax], float cv, int ci, float cx) {
#pragma unroll
  for (int j = 0; j < kTopMax; ++j) {
    const bool before = cv > tv[j];
    const float v = tv[j];
    const int i = ti[j];
    const float x = tx[j];
    tv[j] = before ? cv : v;
    ti[j] = before ? ci : i;
    tx[j] = before ? cx : x;
    cv = before ? v : cv;
    ci = before ? i : ci;
    cx = before ? x : cx;
  }
}

}  // namespace olive
