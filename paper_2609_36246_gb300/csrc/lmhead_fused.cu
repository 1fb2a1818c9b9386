// lmhead_fused.cu -- the slab forms of the LM-head losses' backward passes and
// of their single-pass forward + backward, in one persistent tcgen05 kernel
// (lmhead_fused_kernel) with a static tile schedule: the cross-entropy step
// through an HBM slab of G (olive_token_loss_fwd_bwd_slab) and the top-K KL
// calls (olive_topk_kl_bwd, olive_topk_kl_fwd_bwd).  The on-chip forms are in
// lmhead_group.cu.
//
// Cross-entropy (Eq. (osd-ce), Section 3.1; the sampled sequences are fixed,
// so only hidden and W get gradients).  With p = softmax(z) from the
// forward's lse and G[r, v] = g inv_tau (p[r, v] - [v == y_r]):
//   dH = G . W        (M = rows, N = d, K = V)
//   dW = G^T . hc     (M = V,    N = d, K = rows)
// Top-K truncated reverse KL (OPD's top-16 approximation as read here, the
// student's top-K set S held fixed): with l = log p_s, q = log p_t at the ids
// of S, P_S = sum_S p_s and KL_K the forward value,
//   G[r, u] = g_t inv_tau p_s(u) ([u in S] (l_u - q_u + 1) - KL_K - P_S),
// i.e. a softmax term with the per-row coefficient -g_t inv_tau (KL_K + P_S)
// plus K sparse entries whose full values a prologue kernel computes from the
// forward's top-K lists; the GRAD epilogue writes the softmax term and then
// overwrites the (at most K) entries of S that fall in its tile.  dH and dW
// are then the cross-entropy tiles unchanged.
//
// One-launch form (olive_token_loss_bwd, olive_topk_kl_bwd): the logits are
// recomputed tile by tile and turned into G in the epilogue; G exists only as
// a bf16 slab of at most tc_max compacted rows in the workspace.  The masked rows are split into equal slabs of <= tc_max rows;
// per slab the work is a list of tiles of three kinds, all 128 x 256 fp32
// accumulators in TMEM:
//   GRAD    z = hc . W^T (K = d) -> G tile (bf16) in the slab
//   DH      G . W  (A = G K-major, B = W MN-major, K = V) -> d_hidden rows
//   DW      G^T . hc (A = G MN-major, B = hc MN-major, K = slab rows) -> dW
//           (CE only; stored directly in the output dtype when there is one
//           slab, otherwise through an fp32 accumulator)
// The tiles of all slabs form one list in dependency order and CTA c takes
// tiles c, c+G, c+2G, ... (a static round robin: tiles that share an operand
// run at the same time on neighbouring CTAs, which an atomic work queue was
// measured to lose).  Before loading a tile the producer warp waits (bounded)
// until the tiles it reads have been published through release counters: DH
// of row tile i needs every GRAD tile of row tile i, DW needs every GRAD tile
// of its slab, and GRAD of slab s+1 needs every DH/DW tile of slab s (they
// share the G buffer).  Each CTA walks its tiles in increasing order and a
// tile only waits on tiles with smaller indices, so the lowest unfinished
// tile never waits and all waits end; the cooperative launch keeps every CTA
// resident.
//
// Forward + backward in one call (olive_token_loss_fwd_bwd) avoids the logit
// recomputation: per slab, a launch of ZREF tiles (the first vocabulary tile of
// every row tile) takes each row's reference R = its maximum there; a launch
// of ZSAVE tiles (the forward product) stores e' = 2^(x - R) in bf16 in the G
// slab with each half tile's (R, sum of 2^(x - R)) per row.  Since
// G = g inv_tau (p - [v == y]) = lam e' off the target with one scale per row,
// lam = g inv_tau 2^(R - lse2), the slab is not rewritten: ref_fix_kernel
// merges the partials into lse, writes logp and the row's loss term, puts
// G_y / lam at the target (from the exact fp32 z_y), and stores lam and the
// rows hs = lam hc; the DH and DW launch then computes dH = lam (e' . W) (the
// scale in the DH epilogue) and dW = e'^T . hs.  A half tile whose maximum
// exceeds R by more than kRefMax keeps its own maximum as reference, and its
// row is rewritten in full relative to lse2 by ref_fix_kernel (lam = g
// inv_tau).  The launches are stream ordered, so these phases need no tile
// counters.
#include <climits>
#include <cmath>

#include "gemm_core.cuh"
#include "sched.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kBN = 256;
constexpr int kStages = 4;
// Eight epilogue warps: the two warps of a TMEM lane quadrant (warp % 4) take
// the two 128-column halves (part = warp / 4) of every tile.  Warp 8 is the
// producer, warp 9 the MMA issuer.
constexpr int kFEpiWarps = 8;
constexpr int kFEpi = 32 * kFEpiWarps;
constexpr int kFProducer = kFEpiWarps;
constexpr int kFMma = kFEpiWarps + 1;
constexpr int kFThreads = 32 * (kFEpiWarps + 2);
constexpr int kHalf = kBN / 2;

enum Kind : int { K_NONE = -1, K_GRAD = 0, K_DH = 2, K_DW = 3, K_ZSAVE = 4, K_ZREF = 5 };
// phases: one launch of every tile kind with dependency waits, or one slab's
// forward (ZSAVE) tiles, or one slab's DH and DW tiles, or the first vocabulary
// tile of every row tile of one slab (the rows' reference maxima)
enum Phase : int { PH_ALL = 0, PH_Z = 1, PH_DHDW = 2, PH_R = 3 };

// A half tile whose maximum exceeds the row's reference by more than this
// (base 2) keeps its own maximum as reference: e' = 2^(x - ref) stays below
// 2^64 and the row scale 2^(R - lse2) above 2^-82 (V < 2^18), so neither the
// bf16 operands nor the fp32 sums leave their normal range.
constexpr float kRefMax = 64.f;
// Such a half tile's reference when its small entries are still wanted (the
// top-K candidates): 110 below its maximum, so e' spans 2^-133 .. 2^110 and
// its sum stays below 2^117.
constexpr float kOwnShift = 110.f;

// CE maps: 0 hc K-major 64x128, 1 W K-major 64x256, 2 G K-major 64x128,
//          3 W MN-major 64x64, 4 G MN-major 64x64, 5 hc MN-major 64x64
struct FusedMaps {
  CUtensorMap m[6];
};

struct FusedParams {
  int32_t* dev_status;
  uint64_t wait_limit_ns;
  const int32_t* n_rows;
  const int32_t* rows;
  const int32_t* targets;    // CE
  const float* lse;          // CE, indexed by packed row
  const float* grad_loss;    // CE, device scalar
  const float* sp_coef;      // top-K KL, [T]: softmax coefficient per row
  const float* sp_val;       // top-K KL, [T, sp_k]: full G values at the ids of S
  const int32_t* sp_ids;     // top-K KL, [T, sp_k]: the ids of S
  int32_t sp_k;              // 0: cross-entropy targets; K: top-K KL
  int32_t phase, slab;       // Phase; the slab of PH_Z / PH_DHDW
  float* part_zm;            // PH_Z: [tc, vh] half-tile max (base 2) per slab row
  float* part_zs;            // PH_Z: [tc, vh] half-tile sum of 2^(x - max)
  float* zy_s;               // PH_Z: [tc] target logit (natural units)
  float* zref;               // CE single pass: [tc, 2] per slab row, the maxima (base 2) of the
                             // two halves of its first vocabulary tile (PH_R); null: ZSAVE
                             // tiles store e relative to each half tile's own maximum
  const float* lam;          // CE single pass: [tc] dH row scale (null: none)
  float* part_tm;            // PH_Z: [tc, vh] true half-tile maximum (base 2), when kept
  int32_t dw_coef;           // 1: DW tiles scale by g inv_tau (/ N_mask), the CE single pass
  int32_t T, d, V, reduction, out_dtype, group_rows;
  int32_t tc_max;            // rows of the G buffer (multiple of 128)
  int32_t max_slabs, max_rt; // counter array dimensions
  int64_t ldg;               // G row stride in elements
  float inv_tau, scale2;
  __nv_bfloat16* g;
  void* dh_out;              // [T, d] out_dtype
  void* dw_out;              // [V, d] out_dtype (CE)
  float* dw_acc;             // [V, d] fp32 accumulator used when there are several slabs
  uint32_t* counters;        // [2 max_slabs + max_slabs * max_rt], zeroed before launch
};

struct Plan {
  int n, n_slabs, rps, vt, vh, ntd, mtv, bn_grad;
  float coef;  // CE: g * inv_tau (/ N_mask for the mean)
};

struct Unit {
  int kind, s, i, j, in_s, row0, mt;
};

__device__ __forceinline__ uint32_t* ctr_grad(const FusedParams& p, int s) { return p.counters + s; }
__device__ __forceinline__ uint32_t* ctr_dhdw(const FusedParams& p, int s) {
  return p.counters + p.max_slabs + s;
}
__device__ __forceinline__ uint32_t* ctr_row(const FusedParams& p, int s, int i) {
  return p.counters + 2 * p.max_slabs + static_cast<size_t>(s) * p.max_rt + i;
}

__device__ Plan make_plan(const FusedParams& p) {
  Plan pl;
  pl.n = read_n_rows(p.n_rows, p.T, p.dev_status);
  const SlabPlan sp(pl.n, p.tc_max);
  pl.n_slabs = sp.n_slabs;
  if (pl.n_slabs > p.max_slabs) pl.n_slabs = p.max_slabs;  // cannot happen for n <= T
  pl.rps = sp.rps;
  pl.bn_grad = 256;
  pl.vt = (p.V + pl.bn_grad - 1) / pl.bn_grad;
  pl.vh = (p.V + kHalf - 1) / kHalf;
  pl.ntd = (p.d + kBN - 1) / kBN;
  pl.mtv = (p.V + kBM - 1) / kBM;
  pl.coef = 0.f;
  if (p.sp_k == 0 && (p.phase == PH_ALL || p.dw_coef) && p.grad_loss) {
    float g = *p.grad_loss;
    if (p.reduction == OLIVE_REDUCE_MEAN && pl.n > 0) g = g / static_cast<float>(pl.n);
    pl.coef = g * p.inv_tau;
  }
  return pl;
}

__device__ __forceinline__ int slab_in(const Plan& pl, int s) {
  const int r = pl.n - s * pl.rps;
  return r < 0 ? 0 : (r > pl.rps ? pl.rps : r);
}
__device__ __forceinline__ int units_grad(const Plan& pl, int mt) { return mt * pl.vt; }
__device__ __forceinline__ int units_dh(const Plan& pl, int mt) { return mt * pl.ntd; }
__device__ __forceinline__ int units_dw(const Plan& pl, int s, int in_s) {
  return (s == 0 || in_s > 0) ? pl.mtv * pl.ntd : 0;
}

// slabs a launch covers
__device__ __forceinline__ int slab_lo(const FusedParams& p) { return p.phase == PH_ALL ? 0 : p.slab; }
__device__ __forceinline__ int slab_hi(const FusedParams& p, const Plan& pl) {
  return p.phase == PH_ALL ? pl.n_slabs : (p.slab < pl.n_slabs ? p.slab + 1 : 0);
}

__device__ int total_units(const FusedParams& p, const Plan& pl) {
  int t = 0;
  for (int s = slab_lo(p); s < slab_hi(p, pl); ++s) {
    const int in_s = slab_in(pl, s);
    const int mt = (in_s + 127) / 128;
    if (p.phase == PH_R) {
      t += mt;
      continue;
    }
    if (p.phase != PH_DHDW) t += units_grad(pl, mt);
    if (p.phase != PH_Z) t += units_dh(pl, mt) + units_dw(pl, s, in_s);
  }
  return t;
}

__device__ Unit decode(const FusedParams& p, const Plan& pl, int u) {
  Unit x;
  x.kind = K_NONE;
  for (int s = slab_lo(p); s < slab_hi(p, pl); ++s) {
    const int in_s = slab_in(pl, s);
    const int mt = (in_s + 127) / 128;
    x.s = s;
    x.in_s = in_s;
    x.row0 = s * pl.rps;
    x.mt = mt;
    if (p.phase == PH_R) {
      if (u < mt) {
        x.i = u;
        x.j = 0;
        x.kind = K_ZREF;
        return x;
      }
      u -= mt;
      continue;
    }
    const int ug = p.phase == PH_DHDW ? 0 : units_grad(pl, mt);
    if (u < ug) {
      const Raster r{mt, pl.vt, p.group_rows};
      r.tile(u, x.i, x.j);
      x.kind = p.phase == PH_Z ? K_ZSAVE : K_GRAD;
      return x;
    }
    u -= ug;
    if (p.phase == PH_Z) continue;
    const int uh = units_dh(pl, mt);
    if (u < uh) {
      x.i = u / pl.ntd;
      x.j = u % pl.ntd;
      x.kind = K_DH;
      return x;
    }
    u -= uh;
    const int uw = units_dw(pl, s, in_s);
    if (u < uw) {
      x.i = u / pl.ntd;
      x.j = u % pl.ntd;
      x.kind = K_DW;
      return x;
    }
    u -= uw;
  }
  return x;
}

// K steps of a unit's product
__device__ __forceinline__ int unit_ksteps(const FusedParams& p, const Unit& x) {
  switch (x.kind) {
    case K_GRAD:
    case K_ZSAVE:
    case K_ZREF: return (p.d + kBK - 1) / kBK;
    case K_DH: return (p.V + kBK - 1) / kBK;
    case K_DW: return (x.in_s + kBK - 1) / kBK;
    default: return 0;
  }
}

__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* dst, const float (&g)[32]) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 v;
    v.x = pack_bf16x2(g[8 * q + 0], g[8 * q + 1]);
    v.y = pack_bf16x2(g[8 * q + 2], g[8 * q + 3]);
    v.z = pack_bf16x2(g[8 * q + 4], g[8 * q + 5]);
    v.w = pack_bf16x2(g[8 * q + 6], g[8 * q + 7]);
    d4[q] = v;
  }
}

__device__ __forceinline__ void store_f32x32(float* dst, const float (&g)[32]) {
  float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
  for (int q = 0; q < 8; ++q) d4[q] = make_float4(g[4 * q], g[4 * q + 1], g[4 * q + 2], g[4 * q + 3]);
}

// 32 values -> row segment of `n_valid` (<= 32) elements, bf16 or fp32
__device__ __forceinline__ void store_row32(void* base, size_t off, int dtype, int n_valid,
                                            const float (&g)[32]) {
  if (dtype == OLIVE_DTYPE_BF16) {
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(base) + off;
    if (n_valid >= 32) {
      store_bf16x32(o, g);
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < n_valid) o[k] = __float2bfloat16_rn(g[k]);
    }
  } else {
    float* o = static_cast<float*>(base) + off;
    if (n_valid >= 32) {
      store_f32x32(o, g);
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < n_valid) o[k] = g[k];
    }
  }
}

// ------------------------------------------------------------- epilogues ---
__device__ void epi_grad(const FusedParams& p, const Plan& pl, const Unit& x, int row, int part,
                         uint32_t taddr) {
  const int r_local = x.i * kBM + row;
  const int r = x.row0 + r_local;
  bool valid = r_local < x.in_s;
  int y = -1, t = -1;
  float lse2 = 0.f, coef = pl.coef;
  if (valid) {
    t = p.rows[r];
    if (t >= 0 && t < p.T) {
      if (p.sp_k == 0) y = p.targets[t];
      else coef = p.sp_coef[t];
      lse2 = p.lse[t] * kLog2e;
    } else {
      valid = false;
    }
  }
  __nv_bfloat16* grow = p.g + static_cast<size_t>(r_local) * p.ldg;
  const int n0 = x.j * kBN;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= p.V) break;
    uint32_t a[32];
    tmem_ld_32x32b_x32(taddr + c, a);
    tmem_ld_wait();
    float g[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float pr = fast_exp2(__uint_as_float(a[k]) * p.scale2 - lse2);
      g[k] = valid ? coef * (pr - (col0 + k == y ? 1.f : 0.f)) : 0.f;
    }
    store_row32(grow, col0, OLIVE_DTYPE_BF16, p.V - col0, g);
  }
  if (p.sp_k > 0 && valid) {
    // the entries of S in this half tile: same thread, same addresses, so
    // these stores land after the softmax values written above
    const int h0 = n0 + part * kHalf;
    const int h1 = min(h0 + kHalf, p.V);
    const size_t o = static_cast<size_t>(t) * p.sp_k;
#pragma unroll 1
    for (int k = 0; k < p.sp_k; ++k) {
      const int u = p.sp_ids[o + k];
      if (u >= h0 && u < h1) grow[u] = __float2bfloat16_rn(p.sp_val[o + k]);
    }
  }
}

// forward tile of the fused forward + backward: per row the tile's max and
// sum of 2^(x - max) in base-2 units, e = 2^(x - max) stored in bf16 at the
// row's G slab columns (zeros on padding rows), and the exact target logit
__device__ void epi_zsave(const FusedParams& p, const Plan& pl, const Unit& x, int row, int part,
                          uint32_t taddr) {
  const int r_local = x.i * kBM + row;
  bool valid = r_local < x.in_s;
  int y = -1;
  float R = 0.f;
  if (valid) {
    const int t = p.rows[x.row0 + r_local];
    if (t >= 0 && t < p.T) y = p.targets ? p.targets[t] : -1;  // no targets: top-K KL
    else valid = false;
    if (p.zref) R = fmaxf(p.zref[2 * r_local], p.zref[2 * r_local + 1]);
  }
  const int n0 = x.j * kBN;
  float tm = -INFINITY;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= p.V) break;
    uint32_t a[32];
    tmem_ld_32x32b_x32(taddr + c, a);
    tmem_ld_wait();
    const int nv = p.V - col0;
#pragma unroll
    for (int k = 0; k < 32; ++k)
      if (k < nv) tm = fmaxf(tm, __uint_as_float(a[k]) * p.scale2);
    if (y >= col0 && y < col0 + 32) {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (col0 + k == y) p.zy_s[r_local] = __uint_as_float(a[k]) * p.inv_tau;
    }
  }
  // the reference of the stored e and of the partial sum: the row's reference
  // maximum when one is given and tm does not exceed it by more than kRefMax,
  // else the half tile's own maximum (kOwnShift below it when the true maxima
  // are kept for a top-K selection)
  float ref = tm;
  if (p.zref) ref = !(tm - R > kRefMax) ? R : (p.part_tm ? tm - kOwnShift : tm);
  __nv_bfloat16* grow = p.g + static_cast<size_t>(r_local) * p.ldg;
  float ts = 0.f;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= p.V) break;
    uint32_t a[32];
    tmem_ld_32x32b_x32(taddr + c, a);
    tmem_ld_wait();
    const int nv = p.V - col0;
    float e[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      e[k] = (valid && k < nv) ? fast_exp2(__uint_as_float(a[k]) * p.scale2 - ref) : 0.f;
      ts += e[k];
    }
    store_row32(grow, col0, OLIVE_DTYPE_BF16, nv, e);
  }
  if (valid && n0 + part * kHalf < p.V) {  // a half past V has no partial slot
    const size_t o = static_cast<size_t>(r_local) * pl.vh + 2 * x.j + part;
    p.part_zm[o] = ref;
    p.part_zs[o] = ts;
    if (p.part_tm) p.part_tm[o] = tm;
  }
}

// reference tile (the first vocabulary tile of a row tile): each row's
// maximum over its half, base 2, for the ZSAVE tiles that follow
__device__ void epi_zref(const FusedParams& p, const Unit& x, int row, int part, uint32_t taddr) {
  const int r_local = x.i * kBM + row;
  const bool valid = r_local < x.in_s;
  float tm = -INFINITY;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    if (c >= p.V) break;
    uint32_t a[32];
    tmem_ld_32x32b_x32(taddr + c, a);
    tmem_ld_wait();
    const int nv = p.V - c;
#pragma unroll
    for (int k = 0; k < 32; ++k)
      if (k < nv) tm = fmaxf(tm, __uint_as_float(a[k]) * p.scale2);
  }
  if (valid) p.zref[2 * r_local + part] = tm;
}

__device__ void epi_dh(const FusedParams& p, const Unit& x, int row, int part, uint32_t taddr) {
  const int r_local = x.i * kBM + row;
  int t = -1;
  if (r_local < x.in_s) {
    const int tt = p.rows[x.row0 + r_local];
    if (tt >= 0 && tt < p.T) t = tt;
  }
  const int n0 = x.j * kBN;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= p.d) break;
    uint32_t a[32];
    tmem_ld_32x32b_x32(taddr + c, a);
    tmem_ld_wait();
    if (t < 0) continue;
    const float sc = p.lam ? p.lam[r_local] : 1.f;
    float g[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) g[k] = __uint_as_float(a[k]) * sc;
    store_row32(p.dh_out, static_cast<size_t>(t) * p.d + col0, p.out_dtype, p.d - col0, g);
  }
}

__device__ void epi_dw(const FusedParams& p, const Plan& pl, const Unit& x, int row, int part,
                       uint32_t taddr, int nk) {
  const int v = x.i * kBM + row;
  const bool first = x.s == 0;
  const bool last = x.s == pl.n_slabs - 1;
  const int n0 = x.j * kBN;
  const float sc = p.dw_coef ? pl.coef : 1.f;
#pragma unroll 1
  for (int c = part * kHalf; c < (part + 1) * kHalf; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= p.d) break;
    float g[32];
    if (nk > 0) {
      uint32_t a[32];
      tmem_ld_32x32b_x32(taddr + c, a);
      tmem_ld_wait();
#pragma unroll
      for (int k = 0; k < 32; ++k) g[k] = __uint_as_float(a[k]) * sc;
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k) g[k] = 0.f;
    }
    if (v >= p.V) continue;
    const size_t off = static_cast<size_t>(v) * p.d + col0;
    const int nv = p.d - col0;
    if (!first) {
      const float* acc = p.dw_acc + off;
      if (nv >= 32) {
        const float4* a4 = reinterpret_cast<const float4*>(acc);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 z = a4[q];
          g[4 * q] += z.x;
          g[4 * q + 1] += z.y;
          g[4 * q + 2] += z.z;
          g[4 * q + 3] += z.w;
        }
      } else {
#pragma unroll
        for (int k = 0; k < 32; ++k)
          if (k < nv) g[k] += acc[k];
      }
    }
    if (last) store_row32(p.dw_out, off, p.out_dtype, nv, g);
    else store_row32(p.dw_acc, off, OLIVE_DTYPE_F32, nv, g);
  }
}

// ---------------------------------------------------------------- kernel ---
struct FusedLayout {
  static constexpr int A_BYTES = kBM * kBK * 2;      // 16 KB
  static constexpr int B_BYTES = kBN * kBK * 2;      // 32 KB
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int RING_BYTES = STAGE_BYTES * kStages;
  // full[S], empty[S], tfull[2], tempty[2], drain
  static constexpr int NBARS = 2 * kStages + 5;
  static constexpr int BAR_BYTES = 8 * NBARS;
  static constexpr int MISC_BYTES = 128;
  static constexpr int SMEM_BYTES = 1024 + RING_BYTES + BAR_BYTES + MISC_BYTES;
  static constexpr uint32_t TMEM_COLS = 512;
};

__global__ void __launch_bounds__(kFThreads, 1)
    lmhead_fused_kernel(const __grid_constant__ FusedMaps maps, const FusedParams p) {
  using L = FusedLayout;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t ring = base;
  const uint32_t bar0 = base + L::RING_BYTES;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * kStages + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * kStages + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * kStages + 4);
  uint8_t* misc = gbase + L::RING_BYTES + L::BAR_BYTES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 4);
  Plan* plan_smem = reinterpret_cast<Plan*>(misc + 64);
  static_assert(sizeof(Plan) <= 64, "Plan too large");

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), kFEpi);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    *plan_smem = make_plan(p);
    fence_mbar_init();
  }
  if (warp == kFProducer && lane == 0) {
#pragma unroll
    for (int m = 0; m < 6; ++m) tma_prefetch_desc(&maps.m[m]);
  }
  if (warp == kFMma) {
    tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  const uint32_t tmem_base = *tmem_slot;
  const Plan pl = *plan_smem;
  // two 256-column accumulators: the epilogue of one tile overlaps the next
  // tile's MMAs
  constexpr int nbufs = 2;
  const WaitCtl ctl{abort_flag, p.wait_limit_ns};

  const int total = total_units(p, pl);

  if (warp == kFProducer) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total; u += gridDim.x) {
        const Unit x = decode(p, pl, u);
        // wait until the tiles this one reads are published
        bool dep = true;
        if (p.phase != PH_ALL) {
          // phases are separate launches in stream order: nothing to wait for
        } else if (x.kind == K_GRAD && x.s > 0) {
          const int pin = slab_in(pl, x.s - 1);
          const int pmt = (pin + 127) / 128;
          dep = wait_counter(ctr_dhdw(p, x.s - 1),
                             units_dh(pl, pmt) + units_dw(pl, x.s - 1, pin), ctl);
        } else if (x.kind == K_DH) {
          dep = wait_counter(ctr_row(p, x.s, x.i), pl.vt, ctl);
        } else if (x.kind == K_DW) {
          dep = wait_counter(ctr_grad(p, x.s), units_grad(pl, x.mt), ctl);
        }
        if (!dep) { ok = false; break; }
        fence_proxy_async_global();
        const int nk = unit_ksteps(p, x);
        for (int k = 0; k < nk; ++k) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, ctl)) { ok = false; break; }
          const uint32_t sA = ring + stage * L::STAGE_BYTES;
          const uint32_t sB = sA + L::A_BYTES;
          const uint32_t fb = full_bar(stage);
          mbar_arrive_expect_tx(fb, L::STAGE_BYTES);
          switch (x.kind) {
            case K_GRAD:
            case K_ZSAVE:
            case K_ZREF:
              tma_load_2d(sA, &maps.m[0], fb, k * kBK, x.row0 + x.i * kBM);
              tma_load_2d(sB, &maps.m[1], fb, k * kBK, x.j * kBN);
              break;
            case K_DH:
              tma_load_2d(sA, &maps.m[2], fb, k * kBK, x.i * kBM);
#pragma unroll
              for (int b = 0; b < 4; ++b) tma_load_2d(sB + b * 8192, &maps.m[3], fb, x.j * kBN + 64 * b, k * kBK);
              break;
            case K_DW:
#pragma unroll
              for (int b = 0; b < 2; ++b) tma_load_2d(sA + b * 8192, &maps.m[4], fb, x.i * kBM + 64 * b, k * kBK);
#pragma unroll
              for (int b = 0; b < 4; ++b)
                tma_load_2d(sB + b * 8192, &maps.m[5], fb, x.j * kBN + 64 * b, x.row0 + k * kBK);
              break;
            default: break;
          }
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000) nanosleep_ns(1000);
      }
    }
    __syncwarp();
  } else if (warp == kFMma) {
    if (lane == 0) {
      int stage = 0, buf = 0;
      uint32_t phase = 0, aphase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total; u += gridDim.x) {
        const Unit x = decode(p, pl, u);
        const int nk = unit_ksteps(p, x);
        uint32_t idesc;
        bool a_mn = false, b_mn = false;
        switch (x.kind) {
          case K_DH: idesc = idesc_bf16(kBM, kBN, false, true); b_mn = true; break;
          case K_DW: idesc = idesc_bf16(kBM, kBN, true, true); a_mn = b_mn = true; break;
          default: idesc = idesc_bf16(kBM, kBN, false, false); break;
        }
        if (!mbar_wait(tempty_bar(buf), aphase ^ 1u, ctl)) { ok = false; break; }
        tc_fence_after();
        const uint32_t acc = tmem_base + static_cast<uint32_t>(buf * kBN);
        for (int k = 0; k < nk; ++k) {
          if (!mbar_wait(full_bar(stage), phase, ctl)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sA = ring + stage * L::STAGE_BYTES;
          const uint32_t sB = sA + L::A_BYTES;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = a_mn ? sdesc_sw128(sA + kk * 2048, 8192, 1024)
                                     : sdesc_sw128(sA + kk * 32, 16, 1024);
            const uint64_t bd = b_mn ? sdesc_sw128(sB + kk * 2048, 8192, 1024)
                                     : sdesc_sw128(sB + kk * 32, 16, 1024);
            umma_bf16(acc, ad, bd, idesc, (k > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(empty_bar(stage));
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(tfull_bar(buf));
        if (++buf == nbufs) { buf = 0; aphase ^= 1u; }
      }
      umma_commit(drain_bar);
      volatile int keep_waiting = 0;
      const uint64_t floor_ns = 200ull * 1000 * 1000;  // in-flight MMAs finish in microseconds
      const WaitCtl own{&keep_waiting, p.wait_limit_ns > floor_ns ? p.wait_limit_ns : floor_ns};
      mbar_wait(drain_bar, 0, own);
    }
    __syncwarp();
  } else {
    const int quad = warp & 3;
    const int part = warp >> 2;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16);
    int buf = 0;
    uint32_t aphase = 0;
    // every wait below ends in one group decision (bar.red.and), so the 128
    // epilogue threads always leave the loop together
    for (int u = blockIdx.x; u < total; u += gridDim.x) {
      const Unit x = decode(p, pl, u);
      const int nk = unit_ksteps(p, x);
      if (!named_bar_and(1, kFEpi, mbar_wait(tfull_bar(buf), aphase, ctl))) break;
      tc_fence_after();
      __syncwarp();
      const uint32_t taddr = lane_addr + static_cast<uint32_t>(buf * kBN);
      if (x.kind == K_DW && x.s > 0 && p.phase == PH_ALL) {
        // the fp32 partial of the previous slab must be visible before it is read
        const bool seen =
            threadIdx.x == 0 ? wait_counter(ctr_grad(p, x.s), units_grad(pl, x.mt), ctl) : true;
        if (!named_bar_and(1, kFEpi, seen)) break;
      }
      switch (x.kind) {
        case K_GRAD: epi_grad(p, pl, x, row, part, taddr); break;
        case K_ZSAVE: epi_zsave(p, pl, x, row, part, taddr); break;
        case K_ZREF: epi_zref(p, x, row, part, taddr); break;
        case K_DH: epi_dh(p, x, row, part, taddr); break;
        case K_DW: epi_dw(p, pl, x, row, part, taddr, nk); break;
        default: break;
      }
      tc_fence_before();
      mbar_arrive(tempty_bar(buf));
      if (++buf == nbufs) { buf = 0; aphase ^= 1u; }
      // publish: every epilogue thread's stores, then one release increment
      fence_proxy_async_global();
      __threadfence();
      named_bar_sync(1, kFEpi);
      if (threadIdx.x == 0 && p.phase == PH_ALL) {
        if (x.kind == K_GRAD) {
          red_release_add(ctr_row(p, x.s, x.i), 1u);
          red_release_add(ctr_grad(p, x.s), 1u);
        } else {
          red_release_add(ctr_dhdw(p, x.s), 1u);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.dev_status, kStatusTimeoutBit);
  if (warp == kFMma) {
    tc_fence_after();
    tmem_dealloc(tmem_base, L::TMEM_COLS);
  }
}

// (max, sum) pairs in base 2; an empty side (max = -inf) contributes nothing
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float mn = fmaxf(m, m2);
  s = s * fast_exp2(m - mn) + s2 * fast_exp2(m2 - mn);
  m = mn;
}

// One warp per row tile row of the slab, after ZSAVE tiles with a row
// reference R (base 2): the row's stored e' = 2^(x - R) give G = coef s e'
// off the target, with coef = g inv_tau (/ N_mask) and s = 2^(R - lse2) per
// row, so instead of rewriting the row this merges the partials into lse,
// writes logp, lse and the loss term, puts G_y / (coef s) = expm1(logp) / s at
// the target (G_y from the exact z_y), stores lam = coef s for the dH tiles
// and writes hs = s hc, the dW product's scaled rows (the DW tiles apply
// coef).  A row where some half tile kept its own maximum as reference (it
// exceeded R by more than kRefMax) is rewritten in full relative to lse2
// (e'' = p, s = 1).  Rows past the slab's masked rows get lam = 0 and hs = 0
// up to the row tile's end.
__global__ void __launch_bounds__(256)
    ref_fix_kernel(const int32_t* __restrict__ n_rows, const int32_t* __restrict__ rows,
                   const int32_t* __restrict__ targets, int T, int V, int tc, int slab, int vh,
                   int64_t ldg, float inv_tau, int reduction, const float* __restrict__ grad_loss,
                   const float* __restrict__ part_zm, const float* __restrict__ part_zs,
                   const float* __restrict__ zy_s, const float* __restrict__ zref,
                   const uint4* __restrict__ hc, int d8, __nv_bfloat16* g, float* __restrict__ lam,
                   uint4* __restrict__ hs, float* __restrict__ logp, float* __restrict__ lse,
                   float* __restrict__ nll, int32_t* dev_status) {
  const int n = read_n_rows(n_rows, T, nullptr);
  const SlabPlan sp(n, tc);
  if (slab >= sp.n_slabs) return;
  const int in_s = sp.rows_in(n, slab);
  const int row_end = min((in_s + kBM - 1) / kBM * kBM, tc);
  const int row0 = slab * sp.rps;
  float gs = *grad_loss;
  if (reduction == OLIVE_REDUCE_MEAN && n > 0) gs = gs / static_cast<float>(n);
  const float coef = gs * inv_tau;
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  const int nvec = (V + 7) / 8;
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < row_end; r += warps) {
    const int t = r < in_s ? rows[row0 + r] : -1;
    uint4* hrow = hs + static_cast<size_t>(row0 + r) * d8;
    if (t < 0 || t >= T) {
      // reported by the gather (masked rows); the G row is zero
      if (lane == 0) {
        lam[r] = 0.f;
        if (r < in_s) nll[row0 + r] = 0.f;
      }
      for (int c = lane; c < d8; c += 32) hrow[c] = make_uint4(0u, 0u, 0u, 0u);
      continue;
    }
    const int y = targets[t];
    const float R = fmaxf(zref[2 * r], zref[2 * r + 1]);
    const float* zm = part_zm + static_cast<size_t>(r) * vh;
    const float* zs = part_zs + static_cast<size_t>(r) * vh;
    float m = -INFINITY, sum = 0.f;
    bool own = false;  // some half tile kept its own maximum
    for (int j = lane; j < vh; j += 32) {
      own |= zm[j] != R;
      lse_merge(m, sum, zm[j], zs[j]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float s2 = __shfl_xor_sync(0xffffffffu, sum, o);
      lse_merge(m, sum, m2, s2);
    }
    own = __any_sync(0xffffffffu, own);
    const float lse2 = m + log2f(sum);
    const float l = lse2 * kLn2;
    const bool ybad = y < 0 || y >= V;
    const float lp = ybad ? NAN : zy_s[r] - l;
    if (lane == 0) {
      logp[t] = lp;
      lse[t] = l;
      nll[row0 + r] = -lp;
      if (ybad) atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
    }
    const float sr = own ? 1.f : fast_exp2(R - lse2);
    if (own) {
      // G / coef = e 2^(ref - lse2) = p, in place
      uint4* grow = reinterpret_cast<uint4*>(g + static_cast<size_t>(r) * ldg);
      for (int idx = lane; idx < nvec; idx += 32) {
        uint4 v = grow[idx];
        const float sc = fast_exp2(zm[idx >> 4] - lse2);  // 16 vectors per half tile
        __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 u = __bfloat1622float2(h2[e]);
          const int c = idx * 8 + 2 * e;
          h2[e] = __floats2bfloat162_rn(c < V ? u.x * sc : 0.f, c + 1 < V ? u.y * sc : 0.f);
        }
        grow[idx] = v;
      }
      __syncwarp();  // the dense rewrite precedes the target entry
    }
    if (lane == 0 && !ybad)
      g[static_cast<size_t>(r) * ldg + y] =
          __float2bfloat16_rn(own ? expm1f(lp) : expm1f(lp) * fast_exp2(lse2 - R));
    if (lane == 0) lam[r] = coef * sr;
    const uint4* hin = hc + static_cast<size_t>(row0 + r) * d8;
    for (int c = lane; c < d8; c += 32) {
      uint4 v = hin[c];
      __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 u = __bfloat1622float2(h2[e]);
        h2[e] = __floats2bfloat162_rn(u.x * sr, u.y * sr);
      }
      hrow[c] = v;
    }
  }
}

// ------------------------------------------------ top-K KL in one pass ---
// The student's forward tiles (no targets) leave e' = 2^(x - ref) in bf16 in
// the G slab (ref = the row's reference R, or the half tile's own maximum
// where that exceeds R by more than kRefMax), each half tile's (ref, sum) and
// its true maximum m_half.  Per masked row, topk_kl_rows_kernel then
//   1. merges the partials into lse_s and takes tau, the C-th largest
//      half-tile maximum (C = min(K + 8, 24)): C distinct logits reach tau,
//      so the row's C largest logits all lie in half tiles whose maximum is
//      at least tau, and only those (about C of ~V/128) are read,
//   2. takes from them the C largest approximate logits x ~ log2(e') + ref
//      (bf16 e' resolves x to a few thousandths),
//   3. recomputes those candidates' logits exactly (fp32 dot products
//      h_s . W_s[u]) and keeps the K largest: the student's top-K set S,
//      exact wherever fewer than C - K logits lie within bf16 resolution
//      below the K-th largest,
//   4. takes the teacher's log-probs at S (dot products h_t . W_t[u] minus
//      the teacher's lse) and forms the truncated KL, the overlap with the
//      teacher's top-K ids and the gradient terms of the top-K KL: with
//      g = grad_kl inv_tau, P_S = sum_S p_s and A = KL_K + P_S,
//      G[u] = -g A p_s(u) for every u, plus g p_s(u) (l_u - q_u + 1) on S,
//   5. writes G without rewriting the row: off S, G = lam e' with
//      lam = -g A 2^(R - lse2), so only the K entries of S are stored (as
//      G / lam), lam goes to the dH tiles and hs = lam h_s to the dW tiles.
//      Where lam is out of range (|lam| < 2^-96, |A| < 2^-20) or a half tile
//      kept its own maximum, the row is rewritten as G itself (lam = 1).

constexpr int kTkCand = 24;  // most candidates taken to the exact recomputation (K <= 16)

__device__ __forceinline__ float dot8(uint4 x, uint4 y, float s) {
  const __nv_bfloat162* px = reinterpret_cast<const __nv_bfloat162*>(&x);
  const __nv_bfloat162* py = reinterpret_cast<const __nv_bfloat162*>(&y);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 u = __bfloat1622float2(px[q]);
    const float2 v = __bfloat1622float2(py[q]);
    s = fmaf(u.x, v.x, s);
    s = fmaf(u.y, v.y, s);
  }
  return s;
}

// h . w over d8 16-byte groups, split across the warp; four groups per lane
// in flight
__device__ __forceinline__ float dot_row_bf16(const uint4* __restrict__ h,
                                              const uint4* __restrict__ w, int d8, int lane) {
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
  int c = lane;
  for (; c + 96 < d8; c += 128) {
    const uint4 w0 = __ldg(w + c), w1 = __ldg(w + c + 32), w2 = __ldg(w + c + 64),
                w3 = __ldg(w + c + 96);
    const uint4 h0 = __ldg(h + c), h1 = __ldg(h + c + 32), h2 = __ldg(h + c + 64),
                h3 = __ldg(h + c + 96);
    s0 = dot8(h0, w0, s0);
    s1 = dot8(h1, w1, s1);
    s2 = dot8(h2, w2, s2);
    s3 = dot8(h3, w3, s3);
  }
  for (; c < d8; c += 32) s0 = dot8(__ldg(h + c), __ldg(w + c), s0);
  float s = (s0 + s1) + (s2 + s3);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  return s;
}

// Inserts (v, id) into a lane-local list of N entries sorted by (value
// descending, id ascending).
template <int N>
__device__ __forceinline__ void lane_list_insert(float (&lv)[N], int (&li)[N], float v, int id) {
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const bool before = v > lv[j] || (v == lv[j] && id < li[j]);
    const float tv = lv[j];
    const int ti = li[j];
    lv[j] = before ? v : tv;
    li[j] = before ? id : ti;
    v = before ? tv : v;
    id = before ? ti : id;
  }
}

// Pops the warp's best head of the lanes' sorted lists (value descending,
// id ascending); the lane that held it advances.  Returns the id (INT_MAX
// once every list is exhausted) and the value in *v.
template <int N>
__device__ __forceinline__ int warp_pop(const float (&lv)[N], const int (&li)[N], int& head,
                                        float* v) {
  float bv = -INFINITY;
  int bi = INT_MAX;
#pragma unroll
  for (int j = 0; j < N; ++j)
    if (j == head) {
      bv = lv[j];
      bi = li[j];
    }
  float wv = bv;
  int wi = bi;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, wv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, wi, o);
    if (ov > wv || (ov == wv && oi < wi)) {
      wv = ov;
      wi = oi;
    }
  }
  if (wi != INT_MAX && wi == bi) ++head;  // ids are unique across lanes
  *v = wv;
  return wi;
}

struct TopkKlRows {
  const int32_t* n_rows;
  const int32_t* rows;
  int T, V, tc, slab, vh, K;
  int64_t ldg;
  float inv_tau;
  const float* part_zm;  // [tc, vh] reference of each half tile's e'
  const float* part_zs;  // [tc, vh] sum of 2^(x - ref)
  const float* part_tm;  // [tc, vh] true half-tile maximum
  const float* zref;     // [tc, 2] the row's reference halves
  __nv_bfloat16* g;      // e' of the slab, then G / lam
  float* lam;            // [tc] dH row scale
  uint4* hs;             // [Tpad, ds8] lam h_s rows (dW operand)
  const uint4* h_s;
  const uint4* W_s;
  int ds8;
  const uint4* h_t;
  const uint4* W_t;
  int dt8;
  const float* t_lse;
  const int32_t* t_ids;  // nullable: no overlap
  const float* grad_kl;
  float* s_lse;
  int32_t* s_ids;
  float* s_logp;
  float* t_logp_s;
  float* kl_topk;
  float* overlap;  // nullable
};

__global__ void __launch_bounds__(256) topk_kl_rows_kernel(const TopkKlRows a) {
  const int n = read_n_rows(a.n_rows, a.T, nullptr);
  const SlabPlan sp(n, a.tc);
  if (a.slab >= sp.n_slabs) return;
  const int in_s = sp.rows_in(n, a.slab);
  const int row_end = min((in_s + kBM - 1) / kBM * kBM, a.tc);
  const int row0 = a.slab * sp.rps;
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  const int K = a.K;
  const int C = min(K + 8, kTkCand);
  const int nvec = (a.V + 7) / 8;
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < row_end; r += warps) {
    const int t = r < in_s ? a.rows[row0 + r] : -1;
    uint4* hrow = a.hs + static_cast<size_t>(row0 + r) * a.ds8;
    if (t < 0 || t >= a.T) {
      // reported by the gather (masked rows); the G row is zero
      if (lane == 0) a.lam[r] = 0.f;
      for (int c = lane; c < a.ds8; c += 32) hrow[c] = make_uint4(0u, 0u, 0u, 0u);
      continue;
    }
    const float* zm = a.part_zm + static_cast<size_t>(r) * a.vh;
    const float* zs = a.part_zs + static_cast<size_t>(r) * a.vh;
    const float* tmx = a.part_tm + static_cast<size_t>(r) * a.vh;
    const float R = fmaxf(a.zref[2 * r], a.zref[2 * r + 1]);
    // 1. lse_s, and tau = the C-th largest half-tile maximum: C distinct
    //    logits reach it, so every logit of the row's top C is >= tau and
    //    lies in a half tile whose maximum is >= tau
    float m = -INFINITY, sum = 0.f;
    bool own = false;  // some half tile kept its own maximum as reference
    float tv[kTkCand];
    int ti[kTkCand];
#pragma unroll
    for (int j = 0; j < kTkCand; ++j) {
      tv[j] = -INFINITY;
      ti[j] = INT_MAX;
    }
    for (int j = lane; j < a.vh; j += 32) {
      const float mj = tmx[j];
      own |= mj - R > kRefMax;  // the forward tiles' own test
      lse_merge(m, sum, zm[j], zs[j]);
      if (mj > tv[kTkCand - 1]) lane_list_insert(tv, ti, mj, j);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float s2 = __shfl_xor_sync(0xffffffffu, sum, o);
      lse_merge(m, sum, m2, s2);
    }
    own = __any_sync(0xffffffffu, own);
    const float lse2 = m + log2f(sum);
    const float lse_s = lse2 * kLn2;
    float tau = -INFINITY;
    {
      int head = 0;
      for (int k = 0; k < C; ++k) warp_pop(tv, ti, head, &tau);
    }
    // 2. candidates from the half tiles whose maximum reaches tau: each lane
    //    takes 4 columns of a tile and keeps its 16 best approximate logits
    //    x = log2(e') + ref (bf16 e': x to within a few thousandths)
    float lv[16];
    int li[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      lv[j] = -INFINITY;
      li[j] = INT_MAX;
    }
    __nv_bfloat16* grow = a.g + static_cast<size_t>(r) * a.ldg;
    for (int base = 0; base < a.vh; base += 32) {
      const int j = base + lane;
      unsigned b = __ballot_sync(0xffffffffu, j < a.vh && tmx[j] >= tau);
      while (b) {
        int js[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          js[q] = b ? base + __ffs(b) - 1 : -1;
          b &= b ? b - 1 : 0u;
        }
        uint2 v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          // rows are only vpad(V) wide: columns from V on are not read
          const int c = js[q] * kHalf + 4 * lane;
          v[q] = js[q] >= 0 && c < a.V ? *reinterpret_cast<const uint2*>(grow + c)
                                       : make_uint2(0u, 0u);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (js[q] < 0) continue;
          const float mh = zm[js[q]];
          const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v[q]);
          const int c0 = js[q] * kHalf + 4 * lane;
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float2 u = __bfloat1622float2(h2[e]);
            const float x0 = log2f(u.x) + mh, x1 = log2f(u.y) + mh;
            if (c0 + 2 * e < a.V && x0 >= tau) lane_list_insert(lv, li, x0, c0 + 2 * e);
            if (c0 + 2 * e + 1 < a.V && x1 >= tau) lane_list_insert(lv, li, x1, c0 + 2 * e + 1);
          }
        }
      }
    }
    // the warp's C best: lane k keeps the k-th candidate
    int cid = -1;
    {
      int head = 0;
      float dummy;
      for (int k = 0; k < C; ++k) {
        const int w = warp_pop(lv, li, head, &dummy);
        if (lane == k) cid = w == INT_MAX ? -1 : w;
      }
    }
    // 3. exact logits of the candidates, then the K largest by rank
    const uint4* hs_in = a.h_s + static_cast<size_t>(t) * a.ds8;
    float l = -INFINITY;
    for (int k = 0; k < C; ++k) {
      const int u = __shfl_sync(0xffffffffu, cid, k);
      if (u < 0) break;  // the list ends (fewer columns than candidates)
      const float x = dot_row_bf16(hs_in, a.W_s + static_cast<size_t>(u) * a.ds8, a.ds8, lane);
      if (lane == k) l = x * a.inv_tau - lse_s;
    }
    int rank = 0;
    for (int k = 0; k < C; ++k) {
      const float lk = __shfl_sync(0xffffffffu, l, k);
      const int ik = __shfl_sync(0xffffffffu, cid, k);
      if (ik >= 0 && (lk > l || (lk == l && ik < cid))) ++rank;
    }
    const bool mine = cid >= 0 && rank < K;
    // 4. lane j < K takes the j-th member of S, then the teacher's log-prob there
    int sid = -1;
    float slp = 0.f;
    for (int j = 0; j < K; ++j) {
      const unsigned b = __ballot_sync(0xffffffffu, mine && rank == j);
      const int src = b ? __ffs(b) - 1 : 0;
      const int u = __shfl_sync(0xffffffffu, cid, src);
      const float lu = __shfl_sync(0xffffffffu, l, src);
      if (lane == j && b) {
        sid = u;
        slp = lu;
      }
    }
    const uint4* ht = a.h_t + static_cast<size_t>(t) * a.dt8;
    const float lse_t = a.t_lse[t];
    float q = 0.f;
    for (int j = 0; j < K; ++j) {
      const int u = __shfl_sync(0xffffffffu, sid, j);
      if (u < 0) continue;
      const float x = dot_row_bf16(ht, a.W_t + static_cast<size_t>(u) * a.dt8, a.dt8, lane);
      if (lane == j) q = x * a.inv_tau - lse_t;
    }
    const bool in_k = lane < K && sid >= 0;
    const float p = in_k ? expf(slp) : 0.f;
    float kl = in_k ? p * (slp - q) : 0.f, P = p;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      kl += __shfl_xor_sync(0xffffffffu, kl, o);
      P += __shfl_xor_sync(0xffffffffu, P, o);
    }
    const float gk = a.grad_kl[t] * a.inv_tau;
    const float A = kl + P;
    const float val = in_k ? gk * p * (slp - q + 1.f - A) : 0.f;  // G at the lane's id of S
    const size_t o = static_cast<size_t>(t) * K + lane;
    if (lane < K) {
      a.s_ids[o] = sid;
      a.s_logp[o] = in_k ? slp : -INFINITY;
      a.t_logp_s[o] = in_k ? q : -INFINITY;
    }
    if (a.overlap) {
      const int tid = lane < K ? a.t_ids[static_cast<size_t>(t) * K + lane] : -2;
      bool found = false;
      for (int k = 0; k < K; ++k) found |= __shfl_sync(0xffffffffu, tid, k) == sid;
      const int common = __popc(__ballot_sync(0xffffffffu, in_k && found));
      if (lane == 0) a.overlap[t] = static_cast<float>(common) / static_cast<float>(K);
    }
    if (lane == 0) {
      a.s_lse[t] = lse_s;
      a.kl_topk[t] = kl;
    }
    // 5. G: the scaled form, or the row rewritten as G itself
    const float cf = -gk * A;
    float lm = own ? 0.f : cf * fast_exp2(R - lse2);
    const bool rewrite =
        own || !(fabsf(lm) >= 0x1p-96f) || !(fabsf(lm) < 0x1p96f) || !(fabsf(A) >= 0x1p-20f);
    if (rewrite) {
      lm = 1.f;
      uint4* g4 = reinterpret_cast<uint4*>(grow);
      for (int idx = lane; idx < nvec; idx += 32) {
        uint4 v = g4[idx];
        const float sc = fast_exp2(zm[idx >> 4] - lse2);  // 16 vectors per half tile
        __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 u = __bfloat1622float2(h2[e]);
          const int c = idx * 8 + 2 * e;
          // p = e' 2^(ref - lse2) first, then the row coefficient
          h2[e] = __floats2bfloat162_rn(c < a.V ? (u.x * sc) * cf : 0.f,
                                        c + 1 < a.V ? (u.y * sc) * cf : 0.f);
        }
        g4[idx] = v;
      }
    }
    __syncwarp();  // the candidate reads and any dense rewrite precede the K entries
    if (in_k) grow[sid] = __float2bfloat16_rn(val / lm);
    if (lane == 0) a.lam[r] = lm;
    for (int c = lane; c < a.ds8; c += 32) {
      uint4 v = hs_in[c];
      __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 u = __bfloat1622float2(h2[e]);
        h2[e] = __floats2bfloat162_rn(u.x * lm, u.y * lm);
      }
      hrow[c] = v;
    }
  }
}

olive_status launch_lmhead_fused(const Ctx& c, const FusedMaps& maps, const FusedParams& p) {
  const int smem = FusedLayout::SMEM_BYTES;
  static std::atomic<int> done[kMaxDevices];
  if (!set_smem_once(reinterpret_cast<const void*>(lmhead_fused_kernel), smem, c.device, done))
    return OLIVE_ERR_CUDA;
  // one CTA per SM must fit (the cooperative launch relies on it); checked
  // once per device
  static std::atomic<int> fits[kMaxDevices];
  const bool cached = c.device >= 0 && c.device < kMaxDevices;
  if (!cached || fits[c.device].load(std::memory_order_acquire) == 0) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lmhead_fused_kernel, kFThreads,
                                                      smem) != cudaSuccess ||
        per_sm < 1)
      return OLIVE_ERR_CUDA;
    if (cached) fits[c.device].store(1, std::memory_order_release);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(c.num_sms);
  cfg.blockDim = dim3(kFThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = c.stream;
  // the one-launch form waits across CTAs, so every CTA must be resident: a
  // cooperative launch; the phase launches have no cross-CTA waits
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.phase == PH_ALL ? 1 : 0;
  if (cudaLaunchKernelEx(&cfg, lmhead_fused_kernel, maps, p) != cudaSuccess) {
    cudaGetLastError();
    return OLIVE_ERR_CUDA;
  }
  return OLIVE_OK;
}

FusedParams base_params(const Ctx& c, const int32_t* rows, const int32_t* n_rows, int32_t T,
                      int32_t V, float inv_tau, int32_t* dev_status) {
  FusedParams p = {};
  p.dev_status = dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = n_rows;
  p.rows = rows;
  p.T = T;
  p.V = V;
  p.inv_tau = inv_tau;
  p.scale2 = inv_tau * kLog2e;
  p.group_rows = 16;
  return p;
}

}  // namespace

size_t bwd_counter_words(int64_t Tpad, int64_t tc) {
  const int64_t max_slabs = ceil_div(Tpad, tc) + 1;
  const int64_t max_rt = tc / kRowAlign;
  return static_cast<size_t>(2 * max_slabs + max_slabs * max_rt);
}

olive_status launch_loss_bwd(const Ctx& c, const void* hidden, const void* W,
                             const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                             int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                             const float* lse, const float* grad_loss, void* d_hidden, void* d_W,
                             int grad_dtype, void* ws, int32_t* dev_status,
                             const SparseGrad* sg) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const BwdWs w = carve_bwd(ws, T, d, V, grad_dtype);
  const int64_t ldg = vpad(V);
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;

  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(d_hidden, 0, elt * T * static_cast<size_t>(d), c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;
  const size_t nctr = bwd_counter_words(Tpad, w.tc);
  if (cudaMemsetAsync(w.counters, 0, 4 * nctr, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;

  FusedMaps maps;
  if (!encode_bf16_2d(&maps.m[0], w.hc, d, Tpad, 2ull * d, 64, 128) ||
      !encode_bf16_2d(&maps.m[1], W, d, V, 2ull * d, 64, 256) ||
      !encode_bf16_2d(&maps.m[2], w.g, V, w.tc, 2ull * ldg, 64, 128) ||
      !encode_bf16_2d(&maps.m[3], W, d, V, 2ull * d, 64, 64) ||
      !encode_bf16_2d(&maps.m[4], w.g, V, w.tc, 2ull * ldg, 64, 64) ||
      !encode_bf16_2d(&maps.m[5], w.hc, d, Tpad, 2ull * d, 64, 64))
    return OLIVE_ERR_CUDA;

  FusedParams p = base_params(c, rows, n_rows, T, V, inv_tau, dev_status);
  p.targets = targets;
  p.lse = lse;
  p.grad_loss = grad_loss;
  if (sg) {
    p.sp_coef = sg->coef;
    p.sp_val = sg->val;
    p.sp_ids = sg->ids;
    p.sp_k = sg->K;
  }
  p.d = d;
  p.reduction = reduction;
  p.out_dtype = grad_dtype;
  p.tc_max = static_cast<int32_t>(w.tc);
  p.max_slabs = static_cast<int32_t>(ceil_div(Tpad, w.tc) + 1);
  p.max_rt = static_cast<int32_t>(w.tc / kRowAlign);
  p.ldg = ldg;
  p.g = static_cast<__nv_bfloat16*>(w.g);
  p.dh_out = d_hidden;
  p.dw_out = d_W;
  p.dw_acc = grad_dtype == OLIVE_DTYPE_F32 ? static_cast<float*>(d_W) : w.dw_acc;
  p.counters = w.counters;
  return launch_lmhead_fused(c, maps, p);
}

olive_status launch_loss_fwd_bwd(const Ctx& c, const void* hidden, const void* W,
                                 const int32_t* targets, const int32_t* rows,
                                 const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                 float inv_tau, int reduction, const float* grad_loss, float* logp,
                                 float* lse, float* loss, void* d_hidden, void* d_W, int grad_dtype,
                                 void* ws, int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const FbWs w = carve_fb(ws, T, d, V, grad_dtype);
  const int64_t ldg = vpad(V);
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;
  const int vh = static_cast<int>(ceil_div(V, kHalf));

  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(d_hidden, 0, elt * T * static_cast<size_t>(d), c.stream) != cudaSuccess ||
      cudaMemsetAsync(logp, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      cudaMemsetAsync(lse, 0, sizeof(float) * T, c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;

  FusedMaps maps;
  if (!encode_bf16_2d(&maps.m[0], w.hc, d, Tpad, 2ull * d, 64, 128) ||
      !encode_bf16_2d(&maps.m[1], W, d, V, 2ull * d, 64, 256) ||
      !encode_bf16_2d(&maps.m[2], w.g, V, w.tc, 2ull * ldg, 64, 128) ||
      !encode_bf16_2d(&maps.m[3], W, d, V, 2ull * d, 64, 64) ||
      !encode_bf16_2d(&maps.m[4], w.g, V, w.tc, 2ull * ldg, 64, 64) ||
      !encode_bf16_2d(&maps.m[5], w.hs, d, Tpad, 2ull * d, 64, 64))
    return OLIVE_ERR_CUDA;

  FusedParams p = base_params(c, rows, n_rows, T, V, inv_tau, dev_status);
  p.targets = targets;
  p.d = d;
  p.reduction = reduction;
  p.out_dtype = grad_dtype;
  p.tc_max = static_cast<int32_t>(w.tc);
  const int64_t max_slabs = ceil_div(Tpad, w.tc);
  p.max_slabs = static_cast<int32_t>(max_slabs + 1);
  p.max_rt = static_cast<int32_t>(w.tc / kRowAlign);
  p.ldg = ldg;
  p.g = static_cast<__nv_bfloat16*>(w.g);
  p.dh_out = d_hidden;
  p.dw_out = d_W;
  p.dw_acc = grad_dtype == OLIVE_DTYPE_F32 ? static_cast<float*>(d_W) : w.dw_acc;
  p.part_zm = w.part_zm;
  p.part_zs = w.part_zs;
  p.zy_s = w.zy;
  p.grad_loss = grad_loss;  // the DW tiles' coefficient
  p.zref = w.zref;
  p.lam = w.lam;
  p.dw_coef = 1;

  int conv_blocks = static_cast<int>(ceil_div(w.tc, 8));
  if (conv_blocks > c.num_sms * 16) conv_blocks = c.num_sms * 16;
  for (int s = 0; s < max_slabs; ++s) {
    p.slab = s;
    p.phase = PH_R;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
    p.phase = PH_Z;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
    ref_fix_kernel<<<conv_blocks, 256, 0, c.stream>>>(
        n_rows, rows, targets, T, V, static_cast<int>(w.tc), s, vh, ldg, inv_tau, reduction,
        grad_loss, w.part_zm, w.part_zs, w.zy, w.zref, static_cast<const uint4*>(w.hc), d / 8,
        static_cast<__nv_bfloat16*>(w.g), w.lam, static_cast<uint4*>(w.hs), logp, lse, w.nll,
        dev_status);
    if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
    p.phase = PH_DHDW;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
  }
  return launch_loss_reduce(c, n_rows, T, w.nll, reduction, loss);
}

olive_status launch_topk_kl_fwd_bwd(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                                    const void* h_t, const void* W_t, int32_t d_t,
                                    const int32_t* rows, const int32_t* n_rows, int32_t T,
                                    int32_t V, float inv_tau, int32_t K, const float* t_lse,
                                    const int32_t* t_ids, const float* grad_kl, float* s_lse,
                                    int32_t* s_ids, float* s_logp, float* t_logp_s,
                                    float* kl_topk, float* overlap, void* d_h_s, void* d_W_s,
                                    int grad_dtype, void* ws, int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const FbWs w = carve_fb(ws, T, d_s, V, grad_dtype);
  float* part_tm =
      reinterpret_cast<float*>(static_cast<char*>(ws) + fb_ws_bytes(T, d_s, V, grad_dtype));
  const int64_t ldg = vpad(V);
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;
  const int vh = static_cast<int>(ceil_div(V, kHalf));
  const size_t tk = static_cast<size_t>(T) * K;

  olive_status st = launch_gather_rows(c, h_s, rows, n_rows, T, d_s, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(d_h_s, 0, elt * T * static_cast<size_t>(d_s), c.stream) != cudaSuccess ||
      cudaMemsetAsync(s_lse, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      cudaMemsetAsync(kl_topk, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      (overlap && cudaMemsetAsync(overlap, 0, sizeof(float) * T, c.stream) != cudaSuccess) ||
      cudaMemsetAsync(s_logp, 0, sizeof(float) * tk, c.stream) != cudaSuccess ||
      cudaMemsetAsync(t_logp_s, 0, sizeof(float) * tk, c.stream) != cudaSuccess ||
      cudaMemsetAsync(s_ids, 0xff, sizeof(int32_t) * tk, c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;

  FusedMaps maps;
  if (!encode_bf16_2d(&maps.m[0], w.hc, d_s, Tpad, 2ull * d_s, 64, 128) ||
      !encode_bf16_2d(&maps.m[1], W_s, d_s, V, 2ull * d_s, 64, 256) ||
      !encode_bf16_2d(&maps.m[2], w.g, V, w.tc, 2ull * ldg, 64, 128) ||
      !encode_bf16_2d(&maps.m[3], W_s, d_s, V, 2ull * d_s, 64, 64) ||
      !encode_bf16_2d(&maps.m[4], w.g, V, w.tc, 2ull * ldg, 64, 64) ||
      !encode_bf16_2d(&maps.m[5], w.hs, d_s, Tpad, 2ull * d_s, 64, 64))
    return OLIVE_ERR_CUDA;

  FusedParams p = base_params(c, rows, n_rows, T, V, inv_tau, dev_status);
  p.targets = nullptr;  // the forward tiles keep e and the partials only
  p.d = d_s;
  p.reduction = OLIVE_REDUCE_SUM;
  p.out_dtype = grad_dtype;
  p.tc_max = static_cast<int32_t>(w.tc);
  const int64_t max_slabs = ceil_div(Tpad, w.tc);
  p.max_slabs = static_cast<int32_t>(max_slabs + 1);
  p.max_rt = static_cast<int32_t>(w.tc / kRowAlign);
  p.ldg = ldg;
  p.g = static_cast<__nv_bfloat16*>(w.g);
  p.dh_out = d_h_s;
  p.dw_out = d_W_s;
  p.dw_acc = grad_dtype == OLIVE_DTYPE_F32 ? static_cast<float*>(d_W_s) : w.dw_acc;
  p.part_zm = w.part_zm;
  p.part_zs = w.part_zs;
  p.zy_s = w.zy;
  p.zref = w.zref;
  p.lam = w.lam;
  p.part_tm = part_tm;

  TopkKlRows ra = {};
  ra.n_rows = n_rows;
  ra.rows = rows;
  ra.T = T;
  ra.V = V;
  ra.tc = static_cast<int>(w.tc);
  ra.vh = vh;
  ra.K = K;
  ra.ldg = ldg;
  ra.inv_tau = inv_tau;
  ra.part_zm = w.part_zm;
  ra.part_zs = w.part_zs;
  ra.part_tm = part_tm;
  ra.zref = w.zref;
  ra.g = static_cast<__nv_bfloat16*>(w.g);
  ra.lam = w.lam;
  ra.hs = static_cast<uint4*>(w.hs);
  ra.h_s = static_cast<const uint4*>(h_s);
  ra.W_s = static_cast<const uint4*>(W_s);
  ra.ds8 = d_s / 8;
  ra.h_t = static_cast<const uint4*>(h_t);
  ra.W_t = static_cast<const uint4*>(W_t);
  ra.dt8 = d_t / 8;
  ra.t_lse = t_lse;
  ra.t_ids = t_ids;
  ra.grad_kl = grad_kl;
  ra.s_lse = s_lse;
  ra.s_ids = s_ids;
  ra.s_logp = s_logp;
  ra.t_logp_s = t_logp_s;
  ra.kl_topk = kl_topk;
  ra.overlap = t_ids ? overlap : nullptr;

  int conv_blocks = static_cast<int>(ceil_div(w.tc, 8));
  if (conv_blocks > c.num_sms * 16) conv_blocks = c.num_sms * 16;
  for (int s = 0; s < max_slabs; ++s) {
    p.slab = s;
    p.phase = PH_R;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
    p.phase = PH_Z;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
    ra.slab = s;
    topk_kl_rows_kernel<<<conv_blocks, 256, 0, c.stream>>>(ra);
    if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
    p.phase = PH_DHDW;
    if ((st = launch_lmhead_fused(c, maps, p)) != OLIVE_OK) return st;
  }
  return OLIVE_OK;
}

}  // namespace olive
