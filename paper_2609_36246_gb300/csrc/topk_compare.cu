// topk_compare.cu -- student/teacher agreement on the top-K tokens of each
// masked row, from the top-K lists of olive_token_topk_fwd:
//   overlap[t] = |top_K(student) intersect top_K(teacher)| / K  (the top-K
//                overlap ratio the paper tracks during OPD, Section 4.1)
//   kl_topk[t] = sum over the student's K most probable tokens v of
//                p_s(v) (log p_s(v) - log p_t(v)), log-probs over the full
//                vocabulary: the reverse KL of Section 1 truncated to its
//                top-K terms (the paper's "top-16 KL approximation"; its exact
//                form is not printed, this is the reading implemented)
//   t_logp_s[t, j] = log p_t at the student's j-th id (optional output, the
//                input of the top-K KL gradient)
// One warp per masked row; the teacher's log-probs at the student's K ids
// need K dot products h_t[t] . W_t[v] (d_t each), which the warp computes with
// 16-byte loads split across lanes and a shuffle reduction.
//
// topk_kl_prep turns those lists into the sparse part of the top-K KL
// gradient (see lmhead_fused.cu): per masked row, with g = grad_kl[t] inv_tau,
// P_S = sum_j exp(l_j) and A = kl_topk[t] + P_S,
//   coef[t]   = -g A                       (multiplies p_s(u) for every u)
//   val[t, j] = g exp(l_j) (l_j - q_j + 1 - A)   (G at the j-th id of S)
#include <cmath>

#include "sched.cuh"

namespace olive {
namespace {

__device__ __forceinline__ float dot_bf16x8(uint4 a, uint4 b) {
  const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
  const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 x = __bfloat1622float2(pa[q]);
    const float2 y = __bfloat1622float2(pb[q]);
    s = fmaf(x.x, y.x, s);
    s = fmaf(x.y, y.y, s);
  }
  return s;
}

__global__ void topk_compare_kernel(const uint4* __restrict__ h_t, const uint4* __restrict__ W_t,
                                    int d8, const int32_t* __restrict__ rows,
                                    const int32_t* __restrict__ n_rows, int T, int V, float inv_tau,
                                    int K, const int32_t* __restrict__ s_ids,
                                    const float* __restrict__ s_logp,
                                    const int32_t* __restrict__ t_ids,
                                    const float* __restrict__ t_lse, float* __restrict__ overlap,
                                    float* __restrict__ kl_topk, float* __restrict__ t_logp_s,
                                    int32_t* dev_status) {
  const int n = read_n_rows(n_rows, T, dev_status);
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < n; r += warps) {
    const int t = rows[r];
    if (t < 0 || t >= T) continue;  // reported by the callers' gathers
    const bool in_k = lane < K;
    const int sid = in_k ? s_ids[static_cast<size_t>(t) * K + lane] : -1;
    const float slp = in_k ? s_logp[static_cast<size_t>(t) * K + lane] : 0.f;
    const int tid = in_k ? t_ids[static_cast<size_t>(t) * K + lane] : -2;
    bool found = false;
    for (int k = 0; k < K; ++k) found |= __shfl_sync(0xffffffffu, tid, k) == sid;
    const int common = __popc(__ballot_sync(0xffffffffu, in_k && found));
    const float lse_t = t_lse[t];
    const uint4* hrow = h_t + static_cast<size_t>(t) * d8;
    float kl = 0.f;
    bool bad = false;
    for (int j = 0; j < K; ++j) {
      const int v = __shfl_sync(0xffffffffu, sid, j);
      const float lps = __shfl_sync(0xffffffffu, slp, j);
      if (v < 0 || v >= V) {
        bad = true;
        if (t_logp_s && lane == 0) t_logp_s[static_cast<size_t>(t) * K + j] = NAN;
        continue;
      }
      const uint4* wrow = W_t + static_cast<size_t>(v) * d8;
      // four 16-byte groups per lane in flight
      float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f;
      int c = lane;
      for (; c + 96 < d8; c += 128) {
        const uint4 w0 = __ldg(wrow + c), w1 = __ldg(wrow + c + 32), w2 = __ldg(wrow + c + 64),
                    w3 = __ldg(wrow + c + 96);
        p0 += dot_bf16x8(__ldg(hrow + c), w0);
        p1 += dot_bf16x8(__ldg(hrow + c + 32), w1);
        p2 += dot_bf16x8(__ldg(hrow + c + 64), w2);
        p3 += dot_bf16x8(__ldg(hrow + c + 96), w3);
      }
      for (; c < d8; c += 32) p0 += dot_bf16x8(__ldg(hrow + c), __ldg(wrow + c));
      float part = (p0 + p1) + (p2 + p3);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      const float lpt = part * inv_tau - lse_t;
      kl += expf(lps) * (lps - lpt);
      if (t_logp_s && lane == 0) t_logp_s[static_cast<size_t>(t) * K + j] = lpt;
    }
    if (lane == 0) {
      overlap[t] = static_cast<float>(common) / static_cast<float>(K);
      kl_topk[t] = bad ? NAN : kl;
      if (bad) atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
    }
  }
}

__global__ void topk_kl_prep_kernel(const int32_t* __restrict__ rows,
                                    const int32_t* __restrict__ n_rows, int T, int V,
                                    float inv_tau, int K, const int32_t* __restrict__ s_ids,
                                    const float* __restrict__ s_logp,
                                    const float* __restrict__ t_logp_s,
                                    const float* __restrict__ kl_topk,
                                    const float* __restrict__ grad_kl, float* __restrict__ coef,
                                    float* __restrict__ val, int32_t* dev_status) {
  const int n = read_n_rows(n_rows, T, dev_status);
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x) {
    const int t = rows[r];
    if (t < 0 || t >= T) continue;  // reported by the backward's gather
    const size_t o = static_cast<size_t>(t) * K;
    const float g = grad_kl[t] * inv_tau;
    float P = 0.f;
    bool bad = false;
    for (int j = 0; j < K; ++j) {
      P += expf(s_logp[o + j]);
      const int v = s_ids[o + j];
      bad |= v < 0 || v >= V;
    }
    const float A = kl_topk[t] + P;
    coef[t] = -g * A;
    for (int j = 0; j < K; ++j) {
      const float l = s_logp[o + j];
      val[o + j] = g * expf(l) * (l - t_logp_s[o + j] + 1.f - A);
    }
    if (bad) atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
  }
}

}  // namespace

olive_status launch_topk_kl_prep(const Ctx& c, const int32_t* rows, const int32_t* n_rows,
                                 int32_t T, int32_t V, float inv_tau, int32_t K,
                                 const int32_t* s_ids, const float* s_logp,
                                 const float* t_logp_s, const float* kl_topk,
                                 const float* grad_kl, float* coef, float* val,
                                 int32_t* dev_status) {
  const int threads = 256;
  int blocks = static_cast<int>(ceil_div(T, threads));
  if (blocks > c.num_sms * 4) blocks = c.num_sms * 4;
  topk_kl_prep_kernel<<<blocks, threads, 0, c.stream>>>(rows, n_rows, T, V, inv_tau, K, s_ids,
                                                        s_logp, t_logp_s, kl_topk, grad_kl, coef,
                                                        val, dev_status);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

olive_status launch_topk_compare(const Ctx& c, const void* h_t, const void* W_t, int32_t d_t,
                                 const int32_t* rows, const int32_t* n_rows, int32_t T, int32_t V,
                                 float inv_tau, int32_t K, const int32_t* s_ids,
                                 const float* s_logp, const int32_t* t_ids, const float* t_lse,
                                 float* overlap, float* kl_topk, float* t_logp_s,
                                 int32_t* dev_status) {
  if (cudaMemsetAsync(overlap, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      cudaMemsetAsync(kl_topk, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
      (t_logp_s &&
       cudaMemsetAsync(t_logp_s, 0, sizeof(float) * T * static_cast<size_t>(K), c.stream) !=
           cudaSuccess))
    return OLIVE_ERR_CUDA;
  topk_compare_kernel<<<c.num_sms * 8, 256, 0, c.stream>>>(
      static_cast<const uint4*>(h_t), static_cast<const uint4*>(W_t), d_t / 8, rows, n_rows, T, V,
      inv_tau, K, s_ids, s_logp, t_ids, t_lse, overlap, kl_topk, t_logp_s, dev_status);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace olive
