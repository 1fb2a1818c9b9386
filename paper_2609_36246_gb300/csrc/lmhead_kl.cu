// lmhead_kl.cu -- OPD's per-token divergence between student and teacher over
// the full vocabulary (Section 1: OPD scores each rollout token with a reverse
// KL against the teacher), and the gradient of sum_t g_t KL_t with respect to
// the student hidden states.
//
// Forward (one pass over the vocabulary, nothing [T, V] is stored): every
// 128 x 256 tile runs two tcgen05 products into two TMEM accumulators,
// z_s = hs . W_s^T (K = d_s) and z_t = ht . W_t^T (K = d_t).  With the
// "primary" distribution p (the student for the reverse KL, the teacher for
// the forward KL) and the other one q, each epilogue thread keeps, in base-2
// units x = z log2(e),
//   m_p, s_p = sum 2^(x_p - m_p), A = sum 2^(x_p - m_p) (x_p - x_q),
//   m_q, s_q = sum 2^(x_q - m_q)
// so that KL = ln2 * A / s_p - lse_p + lse_q.  Per-segment partials are
// merged by the finalize kernel.
//
// With a gradient request the value sweep runs first, then
//   reverse: G = g_t inv_tau p_s (log p_s - log p_t - KL_t)
//   forward: G = g_t inv_tau (p_s - p_t),   d_h_s = G . W_s
// comes from one pass of the group kernel (lmhead_group.cu), which recomputes
// both heads' logits tile by tile and contracts G with W_s on chip.
#include <cmath>

#include "gemm_core.cuh"
#include "sched.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// 128 x 256 tiles per product (student and teacher), both products in one
// 512-column TMEM accumulator pair: a tile moves the same bytes per FLOP as
// the cross-entropy forward, but the epilogue cannot overlap the next tile's
// MMAs.  Eight epilogue warps shorten it: the two warps of a TMEM lane
// quadrant take the two 128-column halves of every tile, and at the end of a
// unit the second half's (m_p, s_p, A, m_q, s_q) is merged into the first's
// through shared memory.
struct KlFwdKern {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = false;
  static constexpr bool kBMn = false;
  static constexpr bool kDual = true;
  static constexpr int kStages = 4;
  static constexpr int kAccBufs = 1;
  static constexpr int kEpiWarps = 8;
  static constexpr int kEpiT = 32 * kEpiWarps;
  static constexpr int kEpiSmem = 5 * 128 * 4;  // the merge area

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    int32_t T, V, d_s, d_t;
    int32_t ctas, group_rows, ld, reverse;
    float scale2;
    float* part;  // [5][kSvMax][ld]: m_p, s_p, m_q, s_q, A
  };
  struct Sched {
    Split sp;
  };
  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    s.sp = choose_split(read_n_rows(p.n_rows, p.T, p.dev_status), (p.V + kBN - 1) / kBN, p.ctas);
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
    c.nk = (p.d_s + kBK - 1) / kBK;
    c.nk2 = (p.d_t + kBK - 1) / kBK;
    return c;
  }
  struct Epi {
    int r, sg, part;
    float mp, sp, mq, sq, A;
    float* merge;  // [5][128]
    __device__ void init(uint8_t* smem, int prt) {
      merge = reinterpret_cast<float*>(smem);
      part = prt;
    }
    __device__ void begin(const Params& p, const Sched& s, int u, int row) {
      int i;
      unit_pos(p, s, u, i, sg);
      r = i * kBM + row;
      mp = mq = -INFINITY;
      sp = sq = A = 0.f;
    }
    __device__ void chunk(const Params& p, const uint32_t (&a)[32], const uint32_t (&b)[32], int col0) {
      const int nvalid = p.V - col0;
      float xp[32], xq[32];
      float cp = -INFINITY, cq = -INFINITY;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const float xs = __uint_as_float(a[k]) * p.scale2;
        const float xt = __uint_as_float(b[k]) * p.scale2;
        const bool ok = k < nvalid;
        xp[k] = ok ? (p.reverse ? xs : xt) : -INFINITY;
        xq[k] = ok ? (p.reverse ? xt : xs) : -INFINITY;
        cp = fmaxf(cp, xp[k]);
        cq = fmaxf(cq, xq[k]);
      }
      const float mpn = fmaxf(mp, cp);
      const float mqn = fmaxf(mq, cq);
      const float rp = fast_exp2(mp - mpn);
      float es = 0.f, ea = 0.f, eq = 0.f;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const bool ok = k < nvalid;
        const float e = fast_exp2(xp[k] - mpn);
        es += e;
        ea += ok ? e * (xp[k] - xq[k]) : 0.f;
        eq += fast_exp2(xq[k] - mqn);
      }
      sp = sp * rp + es;
      A = A * rp + ea;
      sq = sq * fast_exp2(mq - mqn) + eq;
      mp = mpn;
      mq = mqn;
    }
    __device__ void tile(const Params& p, const Sched&, int, int, const TileC& tc, uint32_t taddr) {
#pragma unroll 1
      for (int c = part * (kBN / 2); c < (part + 1) * (kBN / 2); c += 32) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.V) break;
        uint32_t a[32], b[32];
        tmem_ld_32x32b_x32(taddr + c, a);
        tmem_ld_32x32b_x32(taddr + kBN + c, b);
        tmem_ld_wait();
        chunk(p, a, b, col0);
      }
    }
    // (m, s, a) + (m2, s2, a2) in base 2; an empty side (m = -inf) adds nothing
    static __device__ __forceinline__ void merge3(float& m, float& s, float& a, float m2, float s2,
                                                  float a2) {
      if (m2 == -INFINITY) return;
      if (m == -INFINITY) {
        m = m2;
        s = s2;
        a = a2;
        return;
      }
      const float mn = fmaxf(m, m2);
      const float f1 = fast_exp2(m - mn), f2 = fast_exp2(m2 - mn);
      s = s * f1 + s2 * f2;
      a = a * f1 + a2 * f2;
      m = mn;
    }
    __device__ void end(const Params& p, const Sched& s, int) {
      // the row's two halves meet here; every epilogue thread takes both barriers
      const int row = threadIdx.x & 127;
      named_bar_sync(2, kEpiT);
      if (part == 1) {
        merge[0 * 128 + row] = mp;
        merge[1 * 128 + row] = sp;
        merge[2 * 128 + row] = A;
        merge[3 * 128 + row] = mq;
        merge[4 * 128 + row] = sq;
      }
      named_bar_sync(2, kEpiT);
      if (part == 1) return;
      merge3(mp, sp, A, merge[0 * 128 + row], merge[1 * 128 + row], merge[2 * 128 + row]);
      float unused = 0.f;
      merge3(mq, sq, unused, merge[3 * 128 + row], merge[4 * 128 + row], 0.f);
      if (r >= s.sp.n) return;
      const size_t plane = static_cast<size_t>(kSvMax) * p.ld;
      const size_t o = static_cast<size_t>(sg) * p.ld + r;
      p.part[0 * plane + o] = mp;
      p.part[1 * plane + o] = sp;
      p.part[2 * plane + o] = mq;
      p.part[3 * plane + o] = sq;
      p.part[4 * plane + o] = A;
    }
  };
};

// kl[t] per masked row; with lse_p / lse_q non-null also both heads' lse per
// compact row (p the primary head: the student for the reverse KL)
__global__ void kl_finalize_kernel(const int32_t* __restrict__ n_rows, const int32_t* __restrict__ rows,
                                   int T, int vt, int ctas, int ld,
                                   const float* __restrict__ part, float* __restrict__ kl,
                                   float* __restrict__ lse_p_out, float* __restrict__ lse_q_out) {
  __shared__ int sh_sv;
  const int n = read_n_rows(n_rows, T, nullptr);
  if (threadIdx.x == 0) sh_sv = choose_split(n, vt, ctas).sv;
  __syncthreads();
  const int sv = sh_sv;
  const size_t plane = static_cast<size_t>(kSvMax) * ld;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x) {
    float Mp = -INFINITY, Mq = -INFINITY;
    for (int s = 0; s < sv; ++s) {
      Mp = fmaxf(Mp, part[0 * plane + static_cast<size_t>(s) * ld + r]);
      Mq = fmaxf(Mq, part[2 * plane + static_cast<size_t>(s) * ld + r]);
    }
    float Sp = 0.f, Sq = 0.f, A = 0.f;
    for (int s = 0; s < sv; ++s) {
      const size_t o = static_cast<size_t>(s) * ld + r;
      const float wp = exp2f(part[0 * plane + o] - Mp);
      Sp += part[1 * plane + o] * wp;
      A += part[4 * plane + o] * wp;
      Sq += part[3 * plane + o] * exp2f(part[2 * plane + o] - Mq);
    }
    const float lse_p = (Mp + log2f(Sp)) * kLn2;
    const float lse_q = (Mq + log2f(Sq)) * kLn2;
    const float k = kLn2 * (A / Sp) - lse_p + lse_q;
    const int t = rows[r];
    if (t >= 0 && t < T) kl[t] = k;
    if (lse_p_out) {
      lse_p_out[r] = lse_p;
      lse_q_out[r] = lse_q;
    }
  }
}

template <class K>
olive_status launch_dual(const Ctx& c, const CUtensorMap& a, const CUtensorMap& b,
                         const CUtensorMap& a2, const CUtensorMap& b2, const typename K::Params& p) {
  const int smem = core_smem_bytes<K>();
  static std::atomic<int> done[kMaxDevices];
  if (!set_smem_once(reinterpret_cast<const void*>(gemm_persistent<K>), smem, c.device, done))
    return OLIVE_ERR_CUDA;
  gemm_persistent<K><<<c.num_sms, core_threads<K>(), smem, c.stream>>>(a, b, a2, b2, p);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace

olive_status launch_divergence(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                               const void* h_t, const void* W_t, int32_t d_t, const int32_t* rows,
                               const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                               int direction, float* kl, const float* grad_kl, void* d_h_s,
                               int grad_dtype, void* ws, int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const int grad = d_h_s != nullptr;
  const KlWs w = carve_kl(ws, T, d_s, d_t, V, grad);
  const int reverse = direction == OLIVE_KL_REVERSE;
  olive_status st;
  if ((st = launch_gather_rows(c, h_s, rows, n_rows, T, d_s, w.hcs, dev_status)) != OLIVE_OK) return st;
  if ((st = launch_gather_rows(c, h_t, rows, n_rows, T, d_t, w.hct, dev_status)) != OLIVE_OK) return st;
  if (cudaMemsetAsync(kl, 0, sizeof(float) * T, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;

  CUtensorMap mHs, mWs, mHt, mWt;
  if (!encode_bf16_2d(&mHs, w.hcs, d_s, Tpad, 2ull * d_s, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mWs, W_s, d_s, V, 2ull * d_s, 64, KlFwdKern::kBN)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mHt, w.hct, d_t, Tpad, 2ull * d_t, 64, 128)) return OLIVE_ERR_CUDA;
  if (!encode_bf16_2d(&mWt, W_t, d_t, V, 2ull * d_t, 64, KlFwdKern::kBN)) return OLIVE_ERR_CUDA;

  KlFwdKern::Params p;
  p.dev_status = dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = n_rows;
  p.T = T;
  p.V = V;
  p.d_s = d_s;
  p.d_t = d_t;
  p.ctas = c.num_sms;
  p.group_rows = 16;
  p.ld = static_cast<int32_t>(Tpad);
  p.reverse = reverse;
  p.scale2 = inv_tau * kLog2e;
  p.part = w.part;
  if ((st = launch_dual<KlFwdKern>(c, mHs, mWs, mHt, mWt, p)) != OLIVE_OK) return st;

  const int vt = (V + KlFwdKern::kBN - 1) / KlFwdKern::kBN;
  kl_finalize_kernel<<<c.num_sms * 4, 256, 0, c.stream>>>(n_rows, rows, T, vt, c.num_sms, p.ld,
                                                           w.part, kl, grad ? w.lse_p : nullptr,
                                                           grad ? w.lse_q : nullptr);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  if (!grad) return OLIVE_OK;
  // the gradient: G formed from both heads' logits, recomputed tile by tile
  // and exchanged on chip (lmhead_group.cu); the student's lse is the
  // primary head's for the reverse KL, the other one's for the forward KL
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;
  if (cudaMemsetAsync(d_h_s, 0, elt * T * static_cast<size_t>(d_s), c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;
  return launch_kl_group_grad(c, w.hcs, w.hct, W_s, d_s, W_t, d_t, rows, n_rows, T, V, inv_tau,
                              reverse, kl, reverse ? w.lse_p : w.lse_q, reverse ? w.lse_q : w.lse_p,
                              grad_kl, d_h_s, grad_dtype, w.ring, w.ctr, w.ctr_words, dev_status);
}

}  // namespace olive
