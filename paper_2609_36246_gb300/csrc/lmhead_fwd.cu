// lmhead_fwd.cu -- forward of the masked continuation loss (Eq. (osd-ce),
// Section 3.1): LM-head projection, online log-sum-exp and target gather,
// without storing the [T, V] logits; and the same sweep with the per-token
// entropy and the K largest log-probs (Appendix A: OPD reads the student's
// top-16 log-probs).
//
//   gather      hc[r] = hidden[rows[r]]  (compacts the masked rows so TMA can
//               stream 128-row tiles; the last tile is zero-padded)
//   fwd tiles   persistent tcgen05 GEMM, 128 x 256 tiles of z = hc . W^T in
//               TMEM; each epilogue thread owns one row and folds 256 logits
//               per tile into a running (max, sum) in registers, catching
//               z_y when the tile holds the row's target.  The stats variant
//               also folds A = sum 2^(x - m) x (entropy) and keeps the row's
//               16 largest logits: values above the current 16th go to a
//               per-thread shared-memory buffer and are merged into a
//               16-entry register list by a compare-swap network
//   finalize    merges the per-segment partials, writes lse and
//               logp = z_y - lse (or entropy and top-K) on the packed rows
//   loss        one block sums -logp in a fixed order (deterministic)
#include <climits>
#include <cmath>

#include "gemm_core.cuh"
#include "sched.cuh"
#include "topk.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

template <bool kStats>
struct FwdKernT {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = false;
  static constexpr bool kBMn = false;
  static constexpr bool kDual = false;
  static constexpr int kStages = 4;
  static constexpr int kAccBufs = 2;
  static constexpr int kEpiWarps = 4;
  // stats: per-thread candidate buffer of 32 (value, id) pairs, slot-major
  static constexpr int kEpiSmem = kStats ? 32 * kEpiThreads * 8 : 0;

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    const int32_t* rows;
    const int32_t* targets;  // loss variant
    int32_t T, d, V;
    int32_t ctas;        // CTAs the decomposition is computed for (= grid)
    int32_t group_rows;  // row tiles per raster group
    int32_t ld;          // row stride of the partial arrays
    float scale2;        // inv_tau * log2(e): logits in base-2 units
    float inv_tau;
    float* part_m;
    float* part_s;
    float* zy;           // loss variant
    float* part_a;       // stats: [kSvMax][ld]
    float* part_tv;      // stats: [kSvMax][ld][16] raw logits
    int32_t* part_ti;    // stats: [kSvMax][ld][16] vocabulary ids
  };
  struct Sched {
    Split sp;
  };

  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    const int n = read_n_rows(p.n_rows, p.T, p.dev_status);
    s.sp = choose_split(n, (p.V + kBN - 1) / kBN, p.ctas);
    return s;
  }
  static __device__ int num_units(const Params&, const Sched& s) { return s.sp.units; }
  static __device__ void unit_pos(const Params& p, const Sched& s, int u, int& i, int& sg) {
    const Raster r{s.sp.rt, s.sp.sv, p.group_rows};
    r.tile(u, i, sg);
  }
  static __device__ int unit_len(const Params& p, const Sched& s, int u) {
    int i, sg;
    unit_pos(p, s, u, i, sg);
    return min(s.sp.seg, s.sp.vt - sg * s.sp.seg);
  }
  static __device__ TileC tile(const Params& p, const Sched& s, int u, int t) {
    int i, sg;
    unit_pos(p, s, u, i, sg);
    TileC c;
    c.m0 = i * kBM;
    c.n0 = (sg * s.sp.seg + t) * kBN;
    c.ka0 = 0;
    c.kb0 = 0;
    c.nk = (p.d + kBK - 1) / kBK;
    c.nk2 = 0;
    return c;
  }

  struct Epi {
    int r, y, sg;
    float m, s, zy, A;
    bool found;
    float tv[kStats ? kTopMax : 1];
    int ti[kStats ? kTopMax : 1];
    float2* buf;  // stats: this thread's candidate slots, stride kEpiThreads

    __device__ void init(uint8_t* smem, int) {
      buf = reinterpret_cast<float2*>(smem) + threadIdx.x;
    }

    __device__ void begin(const Params& p, const Sched& sc, int u, int row) {
      int i;
      unit_pos(p, sc, u, i, sg);
      r = i * kBM + row;
      y = -1;
      if (!kStats && r < sc.sp.n) {
        const int t = p.rows[r];
        if (t >= 0 && t < p.T) y = p.targets[t];
      }
      m = -INFINITY;
      s = 0.f;
      zy = 0.f;
      A = 0.f;
      found = false;
      if constexpr (kStats) {
#pragma unroll
        for (int j = 0; j < kTopMax; ++j) {
          tv[j] = -INFINITY;
          ti[j] = INT_MAX;
        }
      }
    }

    // fold 32 logits (raw accumulators) starting at vocabulary id col0
    __device__ __forceinline__ void chunk(const Params& p, const uint32_t (&a)[32], int col0) {
      float x[32];
      float cmax = -INFINITY;
      const int nvalid = p.V - col0;
      if (nvalid >= 32) {
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          x[k] = __uint_as_float(a[k]) * p.scale2;
          cmax = fmaxf(cmax, x[k]);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          x[k] = k < nvalid ? __uint_as_float(a[k]) * p.scale2 : -INFINITY;
          cmax = fmaxf(cmax, x[k]);
        }
      }
      if (!kStats && y >= col0 && y < col0 + 32) {
#pragma unroll
        for (int k = 0; k < 32; ++k)
          if (col0 + k == y) zy = __uint_as_float(a[k]) * p.inv_tau;
        found = true;
      }
      const float mn = fmaxf(m, cmax);
      const float rescale = fast_exp2(m - mn);
      float e0 = 0.f, e1 = 0.f, e2 = 0.f, e3 = 0.f;
      if constexpr (kStats) {
        float a0 = 0.f, a1 = 0.f;
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          const float q0 = fast_exp2(x[k] - mn);
          const float q1 = fast_exp2(x[k + 1] - mn);
          e0 += q0;
          e1 += q1;
          a0 += k < nvalid ? q0 * x[k] : 0.f;
          a1 += k + 1 < nvalid ? q1 * x[k + 1] : 0.f;
        }
        A = A * rescale + (a0 + a1);
        // candidates for the top list: raw logits above the current 16th
        const float thr = tv[kTopMax - 1];
        int cnt = 0;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float v = __uint_as_float(a[k]);
          if (k < nvalid && v > thr) {
            buf[cnt * kEpiThreads] = make_float2(v, __int_as_float(col0 + k));
            ++cnt;
          }
        }
#pragma unroll 1
        for (int q = 0; q < cnt; ++q) {
          const float2 e = buf[q * kEpiThreads];
          const float cv = e.x;
          const int ci = __float_as_int(e.y);
          // a unit visits its ids in ascending order: values alone order the list
          if (cv > tv[kTopMax - 1]) topk_insert_asc(tv, ti, cv, ci);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 32; k += 4) {
          e0 += fast_exp2(x[k] - mn);
          e1 += fast_exp2(x[k + 1] - mn);
          e2 += fast_exp2(x[k + 2] - mn);
          e3 += fast_exp2(x[k + 3] - mn);
        }
      }
      s = s * rescale + ((e0 + e1) + (e2 + e3));
      m = mn;
    }

    __device__ void tile(const Params& p, const Sched&, int, int, const TileC& tc, uint32_t taddr) {
#pragma unroll 1
      for (int c = 0; c < kBN; c += 64) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.V) break;
        uint32_t a[32], b[32];
        tmem_ld_32x32b_x32(taddr + c, a);
        tmem_ld_32x32b_x32(taddr + c + 32, b);
        tmem_ld_wait();
        chunk(p, a, col0);
        if (col0 + 32 < p.V) chunk(p, b, col0 + 32);
      }
    }

    __device__ void end(const Params& p, const Sched& sc, int) {
      if (r >= sc.sp.n) return;
      const size_t o = static_cast<size_t>(sg) * p.ld + r;
      p.part_m[o] = m;
      p.part_s[o] = s;
      if constexpr (kStats) {
        p.part_a[o] = A;
        float4* v4 = reinterpret_cast<float4*>(p.part_tv + o * kTopMax);
        int4* i4 = reinterpret_cast<int4*>(p.part_ti + o * kTopMax);
#pragma unroll
        for (int q = 0; q < kTopMax / 4; ++q) {
          v4[q] = make_float4(tv[4 * q], tv[4 * q + 1], tv[4 * q + 2], tv[4 * q + 3]);
          i4[q] = make_int4(ti[4 * q], ti[4 * q + 1], ti[4 * q + 2], ti[4 * q + 3]);
        }
      } else {
        if (found) p.zy[r] = zy;
      }
    }
  };
};

using FwdKern = FwdKernT<false>;
using StatsKern = FwdKernT<true>;

__global__ void gather_rows_kernel(const uint4* __restrict__ hidden, const int32_t* __restrict__ rows,
                                   const int32_t* __restrict__ n_rows, int T, int d8,
                                   uint4* __restrict__ hc, int32_t* dev_status) {
  const int n = read_n_rows(n_rows, T, dev_status);
  const int npad = (n + 127) / 128 * 128;
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < npad; r += warps) {
    int t = -1;
    if (r < n) {
      t = rows[r];
      if (t < 0 || t >= T) {
        if (lane == 0) atomicOr(dev_status, 1 << OLIVE_ERR_OFFSETS);
        t = -1;
      }
    }
    uint4* dst = hc + static_cast<size_t>(r) * d8;
    if (t >= 0) {
      const uint4* src = hidden + static_cast<size_t>(t) * d8;
      for (int c = lane; c < d8; c += 32) dst[c] = __ldg(src + c);
    } else {
      for (int c = lane; c < d8; c += 32) dst[c] = make_uint4(0, 0, 0, 0);
    }
  }
}

__global__ void fwd_finalize_kernel(const int32_t* __restrict__ n_rows, const int32_t* __restrict__ rows,
                                    const int32_t* __restrict__ targets, int T, int V, int vt,
                                    int ctas, int ld, const float* __restrict__ part_m,
                                    const float* __restrict__ part_s, const float* __restrict__ zy,
                                    float* __restrict__ logp, float* __restrict__ lse,
                                    float* __restrict__ nll, int32_t* dev_status) {
  __shared__ int sh_sv;
  const int n = read_n_rows(n_rows, T, nullptr);
  if (threadIdx.x == 0) sh_sv = choose_split(n, vt, ctas).sv;
  __syncthreads();
  const int sv = sh_sv;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x) {
    float M = -INFINITY;
    for (int s = 0; s < sv; ++s) M = fmaxf(M, part_m[static_cast<size_t>(s) * ld + r]);
    float S = 0.f;
    for (int s = 0; s < sv; ++s)
      S += part_s[static_cast<size_t>(s) * ld + r] * exp2f(part_m[static_cast<size_t>(s) * ld + r] - M);
    const float l = (M + log2f(S)) * kLn2;
    const int t = rows[r];
    if (t < 0 || t >= T) {
      nll[r] = 0.f;
      continue;  // reported by the gather kernel
    }
    const int y = targets[t];
    float lp;
    if (y < 0 || y >= V) {
      atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
      lp = NAN;
    } else {
      lp = zy[r] - l;
    }
    logp[t] = lp;
    lse[t] = l;
    nll[r] = -lp;
  }
}

__global__ void stats_finalize_kernel(const int32_t* __restrict__ n_rows,
                                      const int32_t* __restrict__ rows, int T, int vt, int ctas,
                                      int ld, int K, float inv_tau, const float* __restrict__ part_m,
                                      const float* __restrict__ part_s,
                                      const float* __restrict__ part_a,
                                      const float* __restrict__ part_tv,
                                      const int32_t* __restrict__ part_ti,
                                      float* __restrict__ lse, float* __restrict__ entropy,
                                      float* __restrict__ topk_logp, int32_t* __restrict__ topk_ids) {
  __shared__ int sh_sv;
  const int n = read_n_rows(n_rows, T, nullptr);
  if (threadIdx.x == 0) sh_sv = choose_split(n, vt, ctas).sv;
  __syncthreads();
  const int sv = sh_sv;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x) {
    const int t = rows[r];
    if (t < 0 || t >= T) continue;  // reported by the gather kernel
    float M = -INFINITY;
    for (int s = 0; s < sv; ++s) M = fmaxf(M, part_m[static_cast<size_t>(s) * ld + r]);
    float S = 0.f, A = 0.f;
    float tv[kTopMax];
    int ti[kTopMax];
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      tv[j] = -INFINITY;
      ti[j] = INT_MAX;
    }
    for (int s = 0; s < sv; ++s) {
      const size_t o = static_cast<size_t>(s) * ld + r;
      const float w = exp2f(part_m[o] - M);
      S += part_s[o] * w;
      A += part_a[o] * w;
      for (int j = 0; j < kTopMax; ++j) {
        const float cv = part_tv[o * kTopMax + j];
        const int ci = part_ti[o * kTopMax + j];
        if (cv > tv[kTopMax - 1] || (cv == tv[kTopMax - 1] && ci < ti[kTopMax - 1]))
          topk_insert(tv, ti, cv, ci);
      }
    }
    const float l2 = M + log2f(S);
    const float l = l2 * kLn2;
    lse[t] = l;
    entropy[t] = kLn2 * (l2 - A / S);  // lse - E_p[z] in natural units
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      if (j < K) {
        topk_logp[static_cast<size_t>(t) * K + j] = tv[j] * inv_tau - l;
        topk_ids[static_cast<size_t>(t) * K + j] = ti[j];
      }
    }
  }
}

__global__ void loss_reduce_kernel(const int32_t* __restrict__ n_rows, int T, const float* __restrict__ nll,
                                   int reduction, float* __restrict__ loss) {
  const int n = read_n_rows(n_rows, T, nullptr);
  double acc = 0.0;
  for (int r = threadIdx.x; r < n; r += blockDim.x) acc += static_cast<double>(nll[r]);
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  __shared__ double part[32];
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x < 32) {
    double v = threadIdx.x < (blockDim.x >> 5) ? part[threadIdx.x] : 0.0;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) {
      double out = v;
      if (reduction == OLIVE_REDUCE_MEAN) out = n > 0 ? v / n : 0.0;
      *loss = static_cast<float>(out);
    }
  }
}

template <class K>
olive_status launch_fwd_core(const Ctx& c, const CUtensorMap& a, const CUtensorMap& b,
                             const typename K::Params& p) {
  const int smem = core_smem_bytes<K>();
  static std::atomic<int> done[kMaxDevices];
  if (!set_smem_once(reinterpret_cast<const void*>(gemm_persistent<K>), smem, c.device, done))
    return OLIVE_ERR_CUDA;
  gemm_persistent<K><<<c.num_sms, core_threads<K>(), smem, c.stream>>>(a, b, a, b, p);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace

olive_status launch_gather_rows(const Ctx& c, const void* hidden, const int32_t* rows,
                                const int32_t* n_rows, int32_t T, int32_t d, void* hc,
                                int32_t* dev_status) {
  const int blocks = c.num_sms * 8;
  gather_rows_kernel<<<blocks, 256, 0, c.stream>>>(static_cast<const uint4*>(hidden), rows, n_rows,
                                                    T, d / 8, static_cast<uint4*>(hc), dev_status);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

olive_status launch_loss_reduce(const Ctx& c, const int32_t* n_rows, int32_t T, const float* nll,
                                int reduction, float* loss) {
  loss_reduce_kernel<<<1, 1024, 0, c.stream>>>(n_rows, T, nll, reduction, loss);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

olive_status launch_logprob_fwd(const Ctx& c, const void* hidden, const void* W,
                                const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                                int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                                float* logp, float* lse, float* loss, void* ws,
                                int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const FwdWs w = carve_fwd(ws, T, d);
  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(logp, 0, sizeof(float) * T, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;
  if (cudaMemsetAsync(lse, 0, sizeof(float) * T, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;

  CUtensorMap mA, mB;
  if (!encode_bf16_2d(&mA, w.hc, d, Tpad, 2ull * d, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mB, W, d, V, 2ull * d, 64, FwdKern::kBN)) return OLIVE_ERR_CUDA;

  FwdKern::Params p = {};
  p.dev_status = dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = n_rows;
  p.rows = rows;
  p.targets = targets;
  p.T = T;
  p.d = d;
  p.V = V;
  p.ctas = c.num_sms;
  p.group_rows = 16;
  p.ld = static_cast<int32_t>(Tpad);
  p.scale2 = inv_tau * kLog2e;
  p.inv_tau = inv_tau;
  p.part_m = w.part_m;
  p.part_s = w.part_s;
  p.zy = w.zy;
  if ((st = launch_fwd_core<FwdKern>(c, mA, mB, p)) != OLIVE_OK) return st;

  const int vt = (V + FwdKern::kBN - 1) / FwdKern::kBN;
  fwd_finalize_kernel<<<c.num_sms * 4, 256, 0, c.stream>>>(n_rows, rows, targets, T, V, vt,
                                                            c.num_sms, p.ld, w.part_m, w.part_s,
                                                            w.zy, logp, lse, w.nll, dev_status);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  loss_reduce_kernel<<<1, 1024, 0, c.stream>>>(n_rows, T, w.nll, reduction, loss);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  return OLIVE_OK;
}

olive_status launch_topk_fwd(const Ctx& c, const void* hidden, const void* W, const int32_t* rows,
                             const int32_t* n_rows, int32_t T, int32_t d, int32_t V, float inv_tau,
                             int32_t K, float* lse, float* entropy, float* topk_logp,
                             int32_t* topk_ids, void* ws, int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const TopkWs w = carve_topk(ws, T, d);
  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(lse, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      cudaMemsetAsync(entropy, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      cudaMemsetAsync(topk_logp, 0, sizeof(float) * T * static_cast<size_t>(K), c.stream) !=
          cudaSuccess ||
      cudaMemsetAsync(topk_ids, 0xff, sizeof(int32_t) * T * static_cast<size_t>(K), c.stream) !=
          cudaSuccess)
    return OLIVE_ERR_CUDA;

  CUtensorMap mA, mB;
  if (!encode_bf16_2d(&mA, w.hc, d, Tpad, 2ull * d, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mB, W, d, V, 2ull * d, 64, StatsKern::kBN)) return OLIVE_ERR_CUDA;

  StatsKern::Params p = {};
  p.dev_status = dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = n_rows;
  p.rows = rows;
  p.T = T;
  p.d = d;
  p.V = V;
  p.ctas = c.num_sms;
  p.group_rows = 16;
  p.ld = static_cast<int32_t>(Tpad);
  p.scale2 = inv_tau * kLog2e;
  p.inv_tau = inv_tau;
  p.part_m = w.part_m;
  p.part_s = w.part_s;
  p.part_a = w.part_a;
  p.part_tv = w.part_tv;
  p.part_ti = w.part_ti;
  if ((st = launch_fwd_core<StatsKern>(c, mA, mB, p)) != OLIVE_OK) return st;

  const int vt = (V + StatsKern::kBN - 1) / StatsKern::kBN;
  stats_finalize_kernel<<<c.num_sms * 4, 128, 0, c.stream>>>(
      n_rows, rows, T, vt, c.num_sms, p.ld, K, inv_tau, w.part_m, w.part_s, w.part_a, w.part_tv,
      w.part_ti, lse, entropy, topk_logp, topk_ids);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace olive
