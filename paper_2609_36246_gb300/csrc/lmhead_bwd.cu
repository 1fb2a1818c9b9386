// lmhead_bwd.cu -- gradients of the Eq. (osd-ce) loss through the LM head
// (Section 3.1: the sampled sequences are fixed, so only hidden and W get
// gradients).  With p = softmax(z) from the forward's lse,
//   G[r, v] = g * inv_tau * (p[r, v] - [v == y_r]),
//   dH = G . W        (M = rows, N = d, K = V)
//   dW = G^T . hc     (M = V,    N = d, K = rows)
//
// The logits are recomputed tile by tile; the G tiles they produce go to a
// bf16 slab of at most Tc rows in the workspace, which the two gradient GEMMs
// then stream.  Per slab of Tc compacted rows:
//   grad   tcgen05 GEMM hc . W^T (128 x 256 tiles) whose epilogue turns each
//          logit into G (softmax - onehot, scaled) and stores it as bf16
//   dh     tcgen05 GEMM G . W with W read MN-major; epilogue scatters rows
//          to d_hidden[rows[r]]
//   dw     tcgen05 GEMM G^T . hc with both operands MN-major; epilogue
//          accumulates into an fp32 [V, d] buffer (first slab stores)
// then one pass rounds the fp32 dW to bf16 when bf16 output was asked for.
#include <cmath>

#include "gemm_core.cuh"
#include "sched.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

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

// ------------------------------------------------------------------ grad ---
struct GradKern {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = false;
  static constexpr bool kBMn = false;
  static constexpr bool kDual = false;
  static constexpr int kStages = 4;

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    const int32_t* rows;
    const int32_t* targets;
    const float* lse;
    const float* grad_loss;
    int32_t T, d, V, reduction;
    int32_t group_rows;
    int64_t slab_start, tc, ldg;
    float inv_tau, scale2;
    __nv_bfloat16* g;
  };
  struct Sched {
    int n, in_slab, mt, vt, units;
    float coef;
  };
  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    s.n = read_n_rows(p.n_rows, p.T, p.dev_status);
    long long k = s.n - p.slab_start;
    if (k < 0) k = 0;
    if (k > p.tc) k = p.tc;
    s.in_slab = static_cast<int>(k);
    s.mt = (s.in_slab + kBM - 1) / kBM;
    s.vt = (p.V + kBN - 1) / kBN;
    s.units = s.mt * s.vt;
    float g = *p.grad_loss;
    if (p.reduction == OLIVE_REDUCE_MEAN && s.n > 0) g = g / static_cast<float>(s.n);
    s.coef = g * p.inv_tau;
    return s;
  }
  static __device__ int num_units(const Params&, const Sched& s) { return s.units; }
  static __device__ int unit_len(const Params&, const Sched&, int) { return 1; }
  static __device__ void pos(const Params& p, const Sched& s, int u, int& i, int& j) {
    const Raster r{s.mt, s.vt, p.group_rows};
    r.tile(u, i, j);
  }
  static __device__ TileC tile(const Params& p, const Sched& s, int u, int) {
    int i, j;
    pos(p, s, u, i, j);
    TileC c;
    c.m0 = static_cast<int>(p.slab_start) + i * kBM;
    c.n0 = j * kBN;
    c.ka0 = 0;
    c.kb0 = 0;
    c.nk = (p.d + kBK - 1) / kBK;
    c.nk2 = 0;
    return c;
  }
  struct Epi {
    int r_local, y;
    bool valid;
    float lse2;
    __device__ void begin(const Params& p, const Sched& s, int u, int row) {
      int i, j;
      pos(p, s, u, i, j);
      r_local = i * kBM + row;
      const long long r = p.slab_start + r_local;
      valid = r < s.n;
      y = -1;
      lse2 = 0.f;
      if (valid) {
        const int t = p.rows[r];
        if (t >= 0 && t < p.T) {
          y = p.targets[t];
          lse2 = p.lse[t] * kLog2e;
        } else {
          valid = false;
        }
      }
    }
    __device__ void tile(const Params& p, const Sched& s, int, int, const TileC& tc, uint32_t taddr) {
      __nv_bfloat16* grow = p.g + static_cast<size_t>(r_local) * p.ldg;
#pragma unroll 1
      for (int c = 0; c < kBN; c += 32) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.V) break;
        uint32_t a[32];
        tmem_ld_32x32b_x32(taddr + c, a);
        tmem_ld_wait();
        float g[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float pr = fast_exp2(__uint_as_float(a[k]) * p.scale2 - lse2);
          g[k] = valid ? s.coef * (pr - (col0 + k == y ? 1.f : 0.f)) : 0.f;
        }
        if (col0 + 32 <= p.V) {
          store_bf16x32(grow + col0, g);
        } else {
          const int nv = p.V - col0;
#pragma unroll
          for (int k = 0; k < 32; ++k)
            if (k < nv) grow[col0 + k] = __float2bfloat16_rn(g[k]);
        }
      }
    }
    __device__ void end(const Params&, const Sched&, int) {}
  };
};

// -------------------------------------------------------------------- dh ---
struct DhKern {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = false;  // G slab [rows, V]: K = V contiguous
  static constexpr bool kBMn = true;   // W [V, d]: N = d contiguous
  static constexpr bool kDual = false;
  static constexpr int kStages = 4;

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    const int32_t* rows;
    int32_t T, d, V, out_dtype;
    int64_t slab_start, tc;
    void* out;
  };
  struct Sched {
    int n, in_slab, mt, nt, units;
  };
  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    s.n = read_n_rows(p.n_rows, p.T, p.dev_status);
    long long k = s.n - p.slab_start;
    if (k < 0) k = 0;
    if (k > p.tc) k = p.tc;
    s.in_slab = static_cast<int>(k);
    s.mt = (s.in_slab + kBM - 1) / kBM;
    s.nt = (p.d + kBN - 1) / kBN;
    s.units = s.mt * s.nt;
    return s;
  }
  static __device__ int num_units(const Params&, const Sched& s) { return s.units; }
  static __device__ int unit_len(const Params&, const Sched&, int) { return 1; }
  static __device__ TileC tile(const Params& p, const Sched& s, int u, int) {
    TileC c;
    c.m0 = (u / s.nt) * kBM;
    c.n0 = (u % s.nt) * kBN;
    c.ka0 = 0;
    c.kb0 = 0;
    c.nk = (p.V + kBK - 1) / kBK;
    c.nk2 = 0;
    return c;
  }
  struct Epi {
    int t;
    __device__ void begin(const Params& p, const Sched& s, int u, int row) {
      const long long r = p.slab_start + (u / s.nt) * kBM + row;
      t = -1;
      if (r < s.n) {
        const int tt = p.rows[r];
        if (tt >= 0 && tt < p.T) t = tt;
      }
    }
    __device__ void tile(const Params& p, const Sched&, int, int, const TileC& tc, uint32_t taddr) {
#pragma unroll 1
      for (int c = 0; c < kBN; c += 32) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.d) break;
        uint32_t a[32];
        tmem_ld_32x32b_x32(taddr + c, a);
        tmem_ld_wait();
        if (t < 0) continue;
        float g[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) g[k] = __uint_as_float(a[k]);
        const size_t off = static_cast<size_t>(t) * p.d + col0;
        if (p.out_dtype == OLIVE_DTYPE_BF16) {
          __nv_bfloat16* o = static_cast<__nv_bfloat16*>(p.out) + off;
          if (col0 + 32 <= p.d) store_bf16x32(o, g);
          else {
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if (k < p.d - col0) o[k] = __float2bfloat16_rn(g[k]);
          }
        } else {
          float* o = static_cast<float*>(p.out) + off;
          if (col0 + 32 <= p.d) store_f32x32(o, g);
          else {
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if (k < p.d - col0) o[k] = g[k];
          }
        }
      }
    }
    __device__ void end(const Params&, const Sched&, int) {}
  };
};

// -------------------------------------------------------------------- dw ---
struct DwKern {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = true;   // A = G^T: G slab [rows, V], M = V contiguous
  static constexpr bool kBMn = true;   // B = hc [rows, d]: N = d contiguous
  static constexpr bool kDual = false;
  static constexpr int kStages = 4;

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    int32_t T, d, V, first;
    int64_t slab_start, tc;
    float* out;  // fp32 [V, d]
  };
  struct Sched {
    int n, in_slab, nk, mt, nt, units;
  };
  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    s.n = read_n_rows(p.n_rows, p.T, p.dev_status);
    long long k = s.n - p.slab_start;
    if (k < 0) k = 0;
    if (k > p.tc) k = p.tc;
    s.in_slab = static_cast<int>(k);
    s.nk = (s.in_slab + kBK - 1) / kBK;
    s.mt = (p.V + kBM - 1) / kBM;
    s.nt = (p.d + kBN - 1) / kBN;
    s.units = (p.first || s.in_slab > 0) ? s.mt * s.nt : 0;
    return s;
  }
  static __device__ int num_units(const Params&, const Sched& s) { return s.units; }
  static __device__ int unit_len(const Params&, const Sched&, int) { return 1; }
  static __device__ TileC tile(const Params& p, const Sched& s, int u, int) {
    TileC c;
    c.m0 = (u / s.nt) * kBM;
    c.n0 = (u % s.nt) * kBN;
    c.ka0 = 0;
    c.kb0 = static_cast<int>(p.slab_start);
    c.nk = s.nk;
    c.nk2 = 0;
    return c;
  }
  struct Epi {
    int v;
    __device__ void begin(const Params&, const Sched& s, int u, int row) { v = (u / s.nt) * kBM + row; }
    __device__ void tile(const Params& p, const Sched&, int, int, const TileC& tc, uint32_t taddr) {
#pragma unroll 1
      for (int c = 0; c < kBN; c += 32) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.d) break;
        float g[32];
        if (tc.nk > 0) {
          uint32_t a[32];
          tmem_ld_32x32b_x32(taddr + c, a);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 32; ++k) g[k] = __uint_as_float(a[k]);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) g[k] = 0.f;
        }
        if (v >= p.V) continue;
        float* o = p.out + static_cast<size_t>(v) * p.d + col0;
        if (col0 + 32 <= p.d) {
          if (!p.first) {
            const float4* o4 = reinterpret_cast<const float4*>(o);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float4 x = o4[q];
              g[4 * q] += x.x;
              g[4 * q + 1] += x.y;
              g[4 * q + 2] += x.z;
              g[4 * q + 3] += x.w;
            }
          }
          store_f32x32(o, g);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k)
            if (k < p.d - col0) o[k] = p.first ? g[k] : o[k] + g[k];
        }
      }
    }
    __device__ void end(const Params&, const Sched&, int) {}
  };
};

__global__ void f32_to_bf16_kernel(const float4* __restrict__ in, uint2* __restrict__ out, size_t n4) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n4;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const float4 x = in[i];
    out[i] = make_uint2(pack_bf16x2(x.x, x.y), pack_bf16x2(x.z, x.w));
  }
}

template <class K>
olive_status launch_core(const Ctx& c, const CUtensorMap& a, const CUtensorMap& b,
                         const typename K::Params& p) {
  const int smem = core_smem_bytes<K>();
  if (cudaFuncSetAttribute(gemm_persistent<K>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess)
    return OLIVE_ERR_CUDA;
  gemm_persistent<K><<<c.num_sms, kThreads, smem, c.stream>>>(a, b, a, b, p);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace

olive_status launch_dh_slab(const Ctx& c, const void* g, int64_t ldg, int64_t tc, const void* W,
                            int32_t d, int32_t V, const int32_t* rows, const int32_t* n_rows,
                            int32_t T, int64_t slab_start, void* out, int out_dtype,
                            int32_t* dev_status) {
  CUtensorMap mG, mW;
  if (!encode_bf16_2d(&mG, g, V, tc, 2ull * ldg, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mW, W, d, V, 2ull * d, 64, 64)) return OLIVE_ERR_CUDA;
  DhKern::Params p;
  p.dev_status = dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = n_rows;
  p.rows = rows;
  p.T = T;
  p.d = d;
  p.V = V;
  p.out_dtype = out_dtype;
  p.slab_start = slab_start;
  p.tc = tc;
  p.out = out;
  return launch_core<DhKern>(c, mG, mW, p);
}

olive_status launch_loss_bwd(const Ctx& c, const void* hidden, const void* W,
                             const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                             int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                             const float* lse, const float* grad_loss, void* d_hidden, void* d_W,
                             int grad_dtype, void* ws, int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const BwdWs w = carve_bwd(ws, T, d, V, grad_dtype);
  const int64_t ldg = vpad(V);
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;

  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(d_hidden, 0, elt * T * static_cast<size_t>(d), c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;

  CUtensorMap mHcK, mWK, mGmn, mHcMn;
  if (!encode_bf16_2d(&mHcK, w.hc, d, Tpad, 2ull * d, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mWK, W, d, V, 2ull * d, 64, 256)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mGmn, w.g, V, w.tc, 2ull * ldg, 64, 64)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mHcMn, w.hc, d, Tpad, 2ull * d, 64, 64)) return OLIVE_ERR_CUDA;

  float* dw_out = grad_dtype == OLIVE_DTYPE_F32 ? static_cast<float*>(d_W) : w.dw_acc;
  const int64_t n_slabs = ceil_div(Tpad, w.tc);
  for (int64_t sl = 0; sl < n_slabs; ++sl) {
    const int64_t start = sl * w.tc;
    GradKern::Params gp;
    gp.dev_status = dev_status;
    gp.wait_limit_ns = c.wait_limit_ns;
    gp.n_rows = n_rows;
    gp.rows = rows;
    gp.targets = targets;
    gp.lse = lse;
    gp.grad_loss = grad_loss;
    gp.T = T;
    gp.d = d;
    gp.V = V;
    gp.reduction = reduction;
    gp.group_rows = 16;
    gp.slab_start = start;
    gp.tc = w.tc;
    gp.ldg = ldg;
    gp.inv_tau = inv_tau;
    gp.scale2 = inv_tau * kLog2e;
    gp.g = static_cast<__nv_bfloat16*>(w.g);
    if ((st = launch_core<GradKern>(c, mHcK, mWK, gp)) != OLIVE_OK) return st;

    if ((st = launch_dh_slab(c, w.g, ldg, w.tc, W, d, V, rows, n_rows, T, start, d_hidden,
                             grad_dtype, dev_status)) != OLIVE_OK)
      return st;

    DwKern::Params wp;
    wp.dev_status = dev_status;
    wp.wait_limit_ns = c.wait_limit_ns;
    wp.n_rows = n_rows;
    wp.T = T;
    wp.d = d;
    wp.V = V;
    wp.first = sl == 0;
    wp.slab_start = start;
    wp.tc = w.tc;
    wp.out = dw_out;
    if ((st = launch_core<DwKern>(c, mGmn, mHcMn, wp)) != OLIVE_OK) return st;
  }
  if (grad_dtype == OLIVE_DTYPE_BF16) {
    const size_t n4 = static_cast<size_t>(V) * d / 4;
    f32_to_bf16_kernel<<<c.num_sms * 8, 256, 0, c.stream>>>(
        reinterpret_cast<const float4*>(w.dw_acc), static_cast<uint2*>(d_W), n4);
    if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  }
  return OLIVE_OK;
}

}  // namespace olive
