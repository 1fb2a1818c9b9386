// opd_stats.cu -- OPD's per-token quantities from one sweep over the
// vocabulary with both LM heads (Section 1: OPD scores each student token
// against the teacher; Appendix A, Table opd-config: top-16 log-probs;
// Section 4.1: the top-K overlap ratio).  Per masked row t:
//   kl[t]            full-vocabulary KL (reverse or forward, as
//                    olive_token_divergence)
//   s_lse, t_lse     log-sum-exp of both heads
//   s_entropy        -sum_v p_s log p_s
//   s_topk_*         the student's K most probable tokens and their log-probs
//   t_logp_s[t, j]   the teacher's log-prob at the student's j-th token
//   overlap[t]       |top_K(p_s) intersect top_K(p_t)| / K
//   kl_topk[t]       sum_j p_s(v_j) (log p_s(v_j) - log p_t(v_j)), the top-K
//                    truncated reverse KL
// Every 128 x 256 tile runs the student and teacher products into the two
// halves of one 512-column TMEM accumulator (as the divergence forward), so
// the epilogue cannot overlap the next tile's MMAs; eight epilogue warps
// shorten it: the two warps of a TMEM lane quadrant take the two 128-column
// halves of every tile.  Each epilogue thread owns a (row, half) and keeps, in
// base-2 units x = z inv_tau log2 e, the online (m_s, s_s, E_s = sum e_s x_s,
// m_t, s_t, A) and two 16-entry top lists of raw logits (the student's carries
// the teacher logit of each entry).
// Per 32-column chunk each thread first marks, in a 32-bit mask per list, the
// columns that beat the list's last entry (after the first tiles of a segment
// few do), then walks the mask in a rolled loop: the value is picked from the
// chunk's registers by a 5-level select tree and the insertion network runs
// once per candidate, so the network exists in one copy (a copy per column
// overflows the instruction cache).  Each half writes its own partial, as
// segment 2 sg + half of the row's vocabulary segment sg (so a row tile has at
// most kSvMax / 2 segments); opd_finalize_kernel merges them.
#include <climits>
#include <cmath>

#include "gemm_core.cuh"
#include "sched.cuh"
#include "topk.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// a[k] for a lane-varying k in [0, 32) without local memory: a select tree
__device__ __forceinline__ uint32_t pick32(const uint32_t (&a)[32], int k) {
  uint32_t l0[16], l1[8], l2[4], l3[2];
#pragma unroll
  for (int i = 0; i < 16; ++i) l0[i] = (k & 1) ? a[2 * i + 1] : a[2 * i];
#pragma unroll
  for (int i = 0; i < 8; ++i) l1[i] = (k & 2) ? l0[2 * i + 1] : l0[2 * i];
#pragma unroll
  for (int i = 0; i < 4; ++i) l2[i] = (k & 4) ? l1[2 * i + 1] : l1[2 * i];
#pragma unroll
  for (int i = 0; i < 2; ++i) l3[i] = (k & 8) ? l2[2 * i + 1] : l2[2 * i];
  return (k & 16) ? l3[1] : l3[0];
}

struct OpdKern {
  static constexpr int kBN = 256;
  static constexpr bool kAMn = false;
  static constexpr bool kBMn = false;
  static constexpr bool kDual = true;
  static constexpr int kStages = 4;
  static constexpr int kAccBufs = 1;
  static constexpr int kEpiWarps = 8;
  static constexpr int kEpiSmem = 0;
  static constexpr int kSvCap = kSvMax / 2;  // segments per row tile (x 2 halves)

  struct Params {
    int32_t* dev_status;
    uint64_t wait_limit_ns;
    const int32_t* n_rows;
    int32_t T, V, d_s, d_t;
    int32_t ctas, group_rows, ld, reverse;
    float scale2;
    float* part;       // [6][kSvMax][ld]: m_s, s_s, E_s, m_t, s_t, A
    float* part_sv;    // [kSvMax][ld][16] student top raw logits
    int32_t* part_si;  // their ids
    float* part_sx;    // the teacher's raw logits at those ids
    float* part_tv;    // [kSvMax][ld][16] teacher top raw logits
    int32_t* part_ti;  // their ids
  };
  struct Sched {
    Split sp;
  };
  static __device__ Sched make_sched(const Params& p) {
    Sched s;
    s.sp = choose_split(read_n_rows(p.n_rows, p.T, p.dev_status), (p.V + kBN - 1) / kBN, p.ctas,
                        kSvCap);
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
    int r, sg, half;
    float ms, ss, es, mt, st, A;
    float sv[kTopMax], sx[kTopMax], tv[kTopMax];
    int si[kTopMax], ti[kTopMax];

    __device__ void init(uint8_t*, int prt) { half = prt; }
    __device__ void begin(const Params& p, const Sched& s, int u, int row) {
      int i;
      unit_pos(p, s, u, i, sg);
      r = i * kBM + row;
      ms = mt = -INFINITY;
      ss = es = st = A = 0.f;
#pragma unroll
      for (int j = 0; j < kTopMax; ++j) {
        sv[j] = tv[j] = sx[j] = -INFINITY;
        si[j] = ti[j] = INT_MAX;
      }
    }

    __device__ __forceinline__ void chunk(const Params& p, const uint32_t (&a)[32],
                                          const uint32_t (&b)[32], int col0) {
      const int nvalid = p.V - col0;
      float cs = -INFINITY, ct = -INFINITY;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        if (k < nvalid) {
          cs = fmaxf(cs, __uint_as_float(a[k]) * p.scale2);
          ct = fmaxf(ct, __uint_as_float(b[k]) * p.scale2);
        }
      }
      const float msn = fmaxf(ms, cs);
      const float mtn = fmaxf(mt, ct);
      float e_s = 0.f, e_e = 0.f, e_t = 0.f, e_a = 0.f;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const bool ok = k < nvalid;
        const float xs = __uint_as_float(a[k]) * p.scale2;
        const float xt = __uint_as_float(b[k]) * p.scale2;
        const float qs = ok ? fast_exp2(xs - msn) : 0.f;
        const float qt = ok ? fast_exp2(xt - mtn) : 0.f;
        e_s += qs;
        e_e += qs * xs;
        e_t += qt;
        e_a += p.reverse ? qs * (xs - xt) : qt * (xt - xs);
      }
      const float rs = fast_exp2(ms - msn);
      const float rt = fast_exp2(mt - mtn);
      ss = ss * rs + e_s;
      es = es * rs + e_e;
      st = st * rt + e_t;
      A = A * (p.reverse ? rs : rt) + e_a;
      ms = msn;
      mt = mtn;
      // a unit visits its ids in ascending order, so a new id is larger than
      // every listed one: values alone decide the candidates and their places
      uint32_t cand_s = 0u, cand_t = 0u;
      const float last_s = sv[kTopMax - 1], last_t = tv[kTopMax - 1];
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const bool ok = k < nvalid;
        if (ok && __uint_as_float(a[k]) > last_s) cand_s |= 1u << k;
        if (ok && __uint_as_float(b[k]) > last_t) cand_t |= 1u << k;
      }
#pragma unroll 1
      while (cand_s) {
        const int k = __ffs(cand_s) - 1;
        cand_s &= cand_s - 1u;
        const float v = __uint_as_float(pick32(a, k));
        if (v > sv[kTopMax - 1]) topk_insert3_asc(sv, si, sx, v, col0 + k, __uint_as_float(pick32(b, k)));
      }
#pragma unroll 1
      while (cand_t) {
        const int k = __ffs(cand_t) - 1;
        cand_t &= cand_t - 1u;
        const float w = __uint_as_float(pick32(b, k));
        if (w > tv[kTopMax - 1]) topk_insert_asc(tv, ti, w, col0 + k);
      }
    }

    __device__ void tile(const Params& p, const Sched&, int, int, const TileC& tc, uint32_t taddr) {
#pragma unroll 1
      for (int c = half * (kBN / 2); c < (half + 1) * (kBN / 2); c += 32) {
        const int col0 = tc.n0 + c;
        if (col0 >= p.V) break;
        uint32_t a[32], b[32];
        tmem_ld_32x32b_x32(taddr + c, a);
        tmem_ld_32x32b_x32(taddr + kBN + c, b);
        tmem_ld_wait();
        chunk(p, a, b, col0);
      }
    }

    __device__ void end(const Params& p, const Sched& s, int) {
      if (r >= s.sp.n) return;
      const size_t plane = static_cast<size_t>(kSvMax) * p.ld;
      const size_t o = static_cast<size_t>(2 * sg + half) * p.ld + r;
      p.part[0 * plane + o] = ms;
      p.part[1 * plane + o] = ss;
      p.part[2 * plane + o] = es;
      p.part[3 * plane + o] = mt;
      p.part[4 * plane + o] = st;
      p.part[5 * plane + o] = A;
      float4* v4 = reinterpret_cast<float4*>(p.part_sv + o * kTopMax);
      float4* x4 = reinterpret_cast<float4*>(p.part_sx + o * kTopMax);
      float4* w4 = reinterpret_cast<float4*>(p.part_tv + o * kTopMax);
      int4* i4 = reinterpret_cast<int4*>(p.part_si + o * kTopMax);
      int4* j4 = reinterpret_cast<int4*>(p.part_ti + o * kTopMax);
#pragma unroll
      for (int q = 0; q < kTopMax / 4; ++q) {
        v4[q] = make_float4(sv[4 * q], sv[4 * q + 1], sv[4 * q + 2], sv[4 * q + 3]);
        x4[q] = make_float4(sx[4 * q], sx[4 * q + 1], sx[4 * q + 2], sx[4 * q + 3]);
        w4[q] = make_float4(tv[4 * q], tv[4 * q + 1], tv[4 * q + 2], tv[4 * q + 3]);
        i4[q] = make_int4(si[4 * q], si[4 * q + 1], si[4 * q + 2], si[4 * q + 3]);
        j4[q] = make_int4(ti[4 * q], ti[4 * q + 1], ti[4 * q + 2], ti[4 * q + 3]);
      }
    }
  };
};

struct OpdOut {
  float *kl, *s_lse, *t_lse, *s_entropy, *s_topk_logp, *t_logp_s, *overlap, *kl_topk;
  int32_t* s_topk_ids;
};

__global__ void opd_finalize_kernel(const int32_t* __restrict__ n_rows,
                                    const int32_t* __restrict__ rows, int T, int vt, int ctas,
                                    int ld, int reverse, int K, float inv_tau,
                                    const float* __restrict__ part,
                                    const float* __restrict__ part_sv,
                                    const int32_t* __restrict__ part_si,
                                    const float* __restrict__ part_sx,
                                    const float* __restrict__ part_tv,
                                    const int32_t* __restrict__ part_ti, OpdOut out) {
  __shared__ int sh_sv;
  const int n = read_n_rows(n_rows, T, nullptr);
  if (threadIdx.x == 0) sh_sv = 2 * choose_split(n, vt, ctas, OpdKern::kSvCap).sv;
  __syncthreads();
  const int nsv = sh_sv;  // two halves per vocabulary segment
  const size_t plane = static_cast<size_t>(kSvMax) * ld;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x) {
    const int t = rows[r];
    if (t < 0 || t >= T) continue;  // reported by the gather kernel
    float Ms = -INFINITY, Mt = -INFINITY;
    for (int s = 0; s < nsv; ++s) {
      Ms = fmaxf(Ms, part[0 * plane + static_cast<size_t>(s) * ld + r]);
      Mt = fmaxf(Mt, part[3 * plane + static_cast<size_t>(s) * ld + r]);
    }
    float Ss = 0.f, Es = 0.f, St = 0.f, A = 0.f;
    float sv[kTopMax], sx[kTopMax], tv[kTopMax];
    int si[kTopMax], ti[kTopMax];
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      sv[j] = tv[j] = sx[j] = -INFINITY;
      si[j] = ti[j] = INT_MAX;
    }
    for (int s = 0; s < nsv; ++s) {
      const size_t o = static_cast<size_t>(s) * ld + r;
      const float ws = exp2f(part[0 * plane + o] - Ms);
      const float wt = exp2f(part[3 * plane + o] - Mt);
      Ss += part[1 * plane + o] * ws;
      Es += part[2 * plane + o] * ws;
      St += part[4 * plane + o] * wt;
      A += part[5 * plane + o] * (reverse ? ws : wt);
      for (int j = 0; j < kTopMax; ++j) {
        const float cv = part_sv[o * kTopMax + j];
        const int ci = part_si[o * kTopMax + j];
        if (topk_beats_last(sv, si, cv, ci)) topk_insert3(sv, si, sx, cv, ci, part_sx[o * kTopMax + j]);
        const float cw = part_tv[o * kTopMax + j];
        const int cj = part_ti[o * kTopMax + j];
        if (topk_beats_last(tv, ti, cw, cj)) topk_insert(tv, ti, cw, cj);
      }
    }
    const float l2s = Ms + log2f(Ss);
    const float l2t = Mt + log2f(St);
    const float ls = l2s * kLn2, lt = l2t * kLn2;
    // KL = ln2 A / S_p - lse_p + lse_q
    const float k = reverse ? kLn2 * (A / Ss) - ls + lt : kLn2 * (A / St) - lt + ls;
    if (out.kl) out.kl[t] = k;
    if (out.s_lse) out.s_lse[t] = ls;
    if (out.t_lse) out.t_lse[t] = lt;
    if (out.s_entropy) out.s_entropy[t] = kLn2 * (l2s - Es / Ss);
    int common = 0;
    float kl_k = 0.f;
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      if (j < K) {
        const float lps = sv[j] * inv_tau - ls;
        const float lpt = sx[j] * inv_tau - lt;
        kl_k += expf(lps) * (lps - lpt);
        bool hit = false;
#pragma unroll
        for (int q = 0; q < kTopMax; ++q) hit |= q < K && ti[q] == si[j];
        common += hit ? 1 : 0;
        const size_t oj = static_cast<size_t>(t) * K + j;
        if (out.s_topk_logp) out.s_topk_logp[oj] = lps;
        if (out.s_topk_ids) out.s_topk_ids[oj] = si[j];
        if (out.t_logp_s) out.t_logp_s[oj] = lpt;
      }
    }
    if (out.overlap) out.overlap[t] = static_cast<float>(common) / static_cast<float>(K);
    if (out.kl_topk) out.kl_topk[t] = kl_k;
  }
}

}  // namespace

olive_status launch_opd_stats(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                              const void* h_t, const void* W_t, int32_t d_t, const int32_t* rows,
                              const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                              int direction, int32_t K, float* kl, float* s_lse, float* t_lse,
                              float* s_entropy, float* s_topk_logp, int32_t* s_topk_ids,
                              float* t_logp_s, float* overlap, float* kl_topk, void* ws,
                              int32_t* dev_status) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const OpdWs w = carve_opd(ws, T, d_s, d_t);
  olive_status st;
  if ((st = launch_gather_rows(c, h_s, rows, n_rows, T, d_s, w.hcs, dev_status)) != OLIVE_OK) return st;
  if ((st = launch_gather_rows(c, h_t, rows, n_rows, T, d_t, w.hct, dev_status)) != OLIVE_OK) return st;
  const size_t tb = sizeof(float) * T, tkb = sizeof(float) * T * static_cast<size_t>(K);
  float* zero_t[] = {kl, s_lse, t_lse, s_entropy, overlap, kl_topk};
  for (float* z : zero_t)
    if (z && cudaMemsetAsync(z, 0, tb, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;
  if ((s_topk_logp && cudaMemsetAsync(s_topk_logp, 0, tkb, c.stream) != cudaSuccess) ||
      (t_logp_s && cudaMemsetAsync(t_logp_s, 0, tkb, c.stream) != cudaSuccess) ||
      (s_topk_ids && cudaMemsetAsync(s_topk_ids, 0xff, tkb, c.stream) != cudaSuccess))
    return OLIVE_ERR_CUDA;

  CUtensorMap mHs, mWs, mHt, mWt;
  if (!encode_bf16_2d(&mHs, w.hcs, d_s, Tpad, 2ull * d_s, 64, 128) ||
      !encode_bf16_2d(&mWs, W_s, d_s, V, 2ull * d_s, 64, OpdKern::kBN) ||
      !encode_bf16_2d(&mHt, w.hct, d_t, Tpad, 2ull * d_t, 64, 128) ||
      !encode_bf16_2d(&mWt, W_t, d_t, V, 2ull * d_t, 64, OpdKern::kBN))
    return OLIVE_ERR_CUDA;

  OpdKern::Params p = {};
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
  p.reverse = direction == OLIVE_KL_REVERSE;
  p.scale2 = inv_tau * kLog2e;
  p.part = w.part;
  p.part_sv = w.part_sv;
  p.part_si = w.part_si;
  p.part_sx = w.part_sx;
  p.part_tv = w.part_tv;
  p.part_ti = w.part_ti;
  const int smem = core_smem_bytes<OpdKern>();
  static std::atomic<int> done[kMaxDevices];
  if (!set_smem_once(reinterpret_cast<const void*>(gemm_persistent<OpdKern>), smem, c.device, done))
    return OLIVE_ERR_CUDA;
  gemm_persistent<OpdKern><<<c.num_sms, core_threads<OpdKern>(), smem, c.stream>>>(mHs, mWs, mHt, mWt, p);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;

  const int vt = (V + OpdKern::kBN - 1) / OpdKern::kBN;
  const OpdOut out{kl, s_lse, t_lse, s_entropy, s_topk_logp, t_logp_s, overlap, kl_topk, s_topk_ids};
  opd_finalize_kernel<<<c.num_sms * 4, 128, 0, c.stream>>>(
      n_rows, rows, T, vt, c.num_sms, p.ld, p.reverse, K, inv_tau, w.part, w.part_sv, w.part_si,
      w.part_sx, w.part_tv, w.part_ti, out);
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace olive
