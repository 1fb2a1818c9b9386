// gemm_core.cuh -- persistent warp-specialised tcgen05 GEMM pipeline shared by
// the LM-head kernels.
//
// One CTA per SM, E = Kern::kEpiWarps epilogue warps (4 or 8) + 2:
//   warps 0..E-1  epilogue: warp w reads TMEM lanes [32 (w % 4), +32), one
//                 accumulator row per thread; with 8 warps the two warps of a
//                 lane quadrant split each tile's columns in halves (part
//                 w / 4), so two threads share a row and the policy merges
//                 their per-row state at the end of a unit.  A kernel-specific
//                 policy turns each finished 128 x BN fp32 tile into its result.
//   warp E        producer: TMA loads of 128 x 64 A and BN x 64 B bf16 tiles
//                 (128-byte swizzle) into a kStages-deep shared-memory ring.
//   warp E+1      MMA issuer: owns the TMEM allocation and issues tcgen05.mma
//                 (M=128, N=BN, K=16) into one of two TMEM accumulators, so
//                 the epilogue of tile n overlaps the MMAs of tile n+1.
// A "dual" policy runs two products per tile (e.g. student and teacher
// logits): K steps [0, nk) use (mapA, mapB) into accumulator columns
// [0, BN), steps [nk, nk+nk2) use (mapA2, mapB2) into columns [BN, 2 BN).
//
// Work comes in "units" (a run of tiles that share epilogue state, e.g. one
// row tile across a vocabulary segment); CTA c takes units c, c+G, c+2G, ...
//
// A Kern policy supplies:
//   Params (with int32_t* dev_status and uint64_t wait_limit_ns), kBN, kAMn,
//   kBMn, kDual, kStages, kEpiWarps, Sched, make_sched(p) (thread 0; may read
//   device counters such as n_rows), num_units(p,s), unit_len(p,s,u),
//   tile(p,s,u,t), kEpiSmem (bytes of shared-memory scratch for the epilogue)
//   and Epi with init(smem, part), begin(p,s,u,row), tile(p,s,u,t,tc,taddr),
//   end(p,s,u).  Every wait of the epilogue ends in one decision of all its
//   warps, so Epi::end may synchronise them (named barrier 2).
#pragma once

#include "sm103.cuh"

namespace olive {

struct TileC {
  int m0;   // A tile origin along M
  int n0;   // B tile origin along N
  int ka0;  // K origin (elements) of A, first product
  int kb0;  // K origin (elements) of B, first product
  int nk;   // 64-wide K steps of the first product (>= 0)
  int nk2;  // 64-wide K steps of the second product (dual policies only)
};

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;
constexpr int kEpiThreads = 128;
constexpr int kProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kStatusTimeoutBit = 1 << 6;  // (1 << OLIVE_ERR_TIMEOUT)

// Thread layout of a policy's CTA.
template <class Kern>
struct CoreThreads {
  static constexpr int kEpiWarps = Kern::kEpiWarps;
  static_assert(kEpiWarps == 4 || kEpiWarps == 8, "4 or 8 epilogue warps");
  static constexpr int kEpi = 32 * kEpiWarps;   // epilogue threads
  static constexpr int kParts = kEpiWarps / 4;  // threads per accumulator row
  static constexpr int kProducer = kEpiWarps;
  static constexpr int kMma = kEpiWarps + 1;
  static constexpr int kAll = 32 * (kEpiWarps + 2);
};

template <class Kern>
struct CoreLayout {
  static constexpr int A_BYTES = kBM * kBK * 2;
  static constexpr int B_BYTES = Kern::kBN * kBK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int RING_BYTES = STAGE_BYTES * Kern::kStages;
  // barriers: full[S], empty[S], tfull[2], tempty[2], drain
  static constexpr int BAR_BYTES = 8 * (2 * Kern::kStages + 5);
  static constexpr int MISC_BYTES = 64;
  static constexpr int EPI_BYTES = Kern::kEpiSmem;  // scratch for the epilogue policy
  static constexpr int SMEM_BYTES =
      1024 /*alignment slack*/ + RING_BYTES + BAR_BYTES + MISC_BYTES + EPI_BYTES;
  static constexpr int ACC_COLS = Kern::kDual ? 2 * Kern::kBN : Kern::kBN;
  static constexpr int ACC_BUFS = Kern::kAccBufs;  // 2: epilogue overlaps the next tile's MMAs
  static constexpr uint32_t TMEM_COLS = ACC_BUFS * ACC_COLS;
  static_assert(ACC_BUFS == 1 || ACC_BUFS == 2, "one or two accumulators");
  static_assert(TMEM_COLS <= 512, "the accumulators must fit in TMEM");
  static_assert(SMEM_BYTES <= 227 * 1024, "shared memory budget");
};

template <class Kern>
__global__ void __launch_bounds__(CoreThreads<Kern>::kAll, 1)
    gemm_persistent(const __grid_constant__ CUtensorMap mapA,
                    const __grid_constant__ CUtensorMap mapB,
                    const __grid_constant__ CUtensorMap mapA2,
                    const __grid_constant__ CUtensorMap mapB2,
                    const typename Kern::Params p) {
  using L = CoreLayout<Kern>;
  using CT = CoreThreads<Kern>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);

  const uint32_t ring = base;
  const uint32_t bar0 = base + L::RING_BYTES;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (Kern::kStages + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * Kern::kStages + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * Kern::kStages + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * Kern::kStages + 4);
  uint8_t* misc = gbase + L::RING_BYTES + L::BAR_BYTES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 4);
  typename Kern::Sched* sched_smem = reinterpret_cast<typename Kern::Sched*>(misc + 16);
  static_assert(sizeof(typename Kern::Sched) <= L::MISC_BYTES - 16, "Sched too large");

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < Kern::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), CT::kEpi);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    *sched_smem = Kern::make_sched(p);
    fence_mbar_init();
  }
  if (warp == CT::kProducer && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    if constexpr (Kern::kDual) {
      tma_prefetch_desc(&mapA2);
      tma_prefetch_desc(&mapB2);
    }
  }
  if (warp == CT::kMma) {
    tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  const uint32_t tmem_base = *tmem_slot;
  const typename Kern::Sched sched = *sched_smem;
  const WaitCtl ctl{abort_flag, p.wait_limit_ns};
  const int n_units = Kern::num_units(p, sched);

  if (warp == CT::kProducer) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const int nt = Kern::unit_len(p, sched, u);
        for (int t = 0; ok && t < nt; ++t) {
          const TileC tc = Kern::tile(p, sched, u, t);
          const int nk_all = tc.nk + (Kern::kDual ? tc.nk2 : 0);
          for (int k = 0; k < nk_all; ++k) {
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, ctl)) { ok = false; break; }
            const uint32_t sA = ring + stage * L::STAGE_BYTES;
            const uint32_t sB = sA + L::A_BYTES;
            const uint32_t fb = full_bar(stage);
            const bool second = Kern::kDual && k >= tc.nk;
            const CUtensorMap* mA = second ? &mapA2 : &mapA;
            const CUtensorMap* mB = second ? &mapB2 : &mapB;
            const int kl = second ? k - tc.nk : k;
            const int ka = (second ? 0 : tc.ka0) + kl * kBK;
            const int kb = (second ? 0 : tc.kb0) + kl * kBK;
            mbar_arrive_expect_tx(fb, L::STAGE_BYTES);
            if constexpr (Kern::kAMn) {
#pragma unroll
              for (int b = 0; b < kBM / 64; ++b) tma_load_2d(sA + b * 8192, mA, fb, tc.m0 + 64 * b, ka);
            } else {
              tma_load_2d(sA, mA, fb, ka, tc.m0);
            }
            if constexpr (Kern::kBMn) {
#pragma unroll
              for (int b = 0; b < Kern::kBN / 64; ++b)
                tma_load_2d(sB + b * 8192, mB, fb, tc.n0 + 64 * b, kb);
            } else {
              tma_load_2d(sB, mB, fb, kb, tc.n0);
            }
            if (++stage == Kern::kStages) { stage = 0; phase ^= 1u; }
          }
        }
      }
      if (!ok) {
        // give copies that were already issued time to land before retiring
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000) nanosleep_ns(1000);
      }
    }
    __syncwarp();
  } else if (warp == CT::kMma) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kBM, Kern::kBN, Kern::kAMn, Kern::kBMn);
      int stage = 0;
      uint32_t phase = 0;
      int buf = 0;
      uint32_t aphase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const int nt = Kern::unit_len(p, sched, u);
        for (int t = 0; ok && t < nt; ++t) {
          const TileC tc = Kern::tile(p, sched, u, t);
          const int nk_all = tc.nk + (Kern::kDual ? tc.nk2 : 0);
          if (!mbar_wait(tempty_bar(buf), aphase ^ 1u, ctl)) { ok = false; break; }
          tc_fence_after();
          const uint32_t acc = tmem_base + static_cast<uint32_t>(buf * L::ACC_COLS);
          for (int k = 0; k < nk_all; ++k) {
            if (!mbar_wait(full_bar(stage), phase, ctl)) { ok = false; break; }
            tc_fence_after();
            const bool second = Kern::kDual && k >= tc.nk;
            const uint32_t dt = second ? acc + Kern::kBN : acc;
            const int kl = second ? k - tc.nk : k;
            const uint32_t sA = ring + stage * L::STAGE_BYTES;
            const uint32_t sB = sA + L::A_BYTES;
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              const uint64_t ad = Kern::kAMn ? sdesc_sw128(sA + kk * 2048, 8192, 1024)
                                             : sdesc_sw128(sA + kk * 32, 16, 1024);
              const uint64_t bd = Kern::kBMn ? sdesc_sw128(sB + kk * 2048, 8192, 1024)
                                             : sdesc_sw128(sB + kk * 32, 16, 1024);
              umma_bf16(dt, ad, bd, idesc, (kl > 0 || kk > 0) ? 1u : 0u);
            }
            umma_commit(empty_bar(stage));
            if (++stage == Kern::kStages) { stage = 0; phase ^= 1u; }
          }
          if (!ok) break;
          umma_commit(tfull_bar(buf));
          if (++buf == L::ACC_BUFS) { buf = 0; aphase ^= 1u; }
        }
      }
      // arrives once every MMA issued above has completed (bounded wait that
      // ignores the abort flag: it only waits for work already in flight)
      umma_commit(drain_bar);
      volatile int keep_waiting = 0;
      const uint64_t floor_ns = 200ull * 1000 * 1000;  // in-flight MMAs finish in microseconds
      const WaitCtl own{&keep_waiting, p.wait_limit_ns > floor_ns ? p.wait_limit_ns : floor_ns};
      mbar_wait(drain_bar, 0, own);
    }
    __syncwarp();
  } else {
    // epilogue warps: thread = accumulator row = TMEM lane (quadrant warp % 4)
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16);
    int buf = 0;
    uint32_t aphase = 0;
    bool ok = true;
    typename Kern::Epi epi;
    epi.init(misc + L::MISC_BYTES, warp >> 2);
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      const int nt = Kern::unit_len(p, sched, u);
      epi.begin(p, sched, u, row);
      for (int t = 0; t < nt; ++t) {
        const TileC tc = Kern::tile(p, sched, u, t);
        // one decision for all epilogue threads: tcgen05.ld below is a warp
        // collective and Epi::end may synchronise the epilogue warps
        if (!named_bar_and(1, CT::kEpi, mbar_wait(tfull_bar(buf), aphase, ctl))) { ok = false; break; }
        tc_fence_after();
        epi.tile(p, sched, u, t, tc, lane_addr + static_cast<uint32_t>(buf * L::ACC_COLS));
        tc_fence_before();
        mbar_arrive(tempty_bar(buf));
        if (++buf == L::ACC_BUFS) { buf = 0; aphase ^= 1u; }
      }
      if (!ok) break;
      epi.end(p, sched, u);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.dev_status, kStatusTimeoutBit);
  if (warp == CT::kMma) {
    tc_fence_after();
    tmem_dealloc(tmem_base, L::TMEM_COLS);
  }
}

template <class Kern>
inline int core_smem_bytes() {
  return CoreLayout<Kern>::SMEM_BYTES;
}

template <class Kern>
inline int core_threads() {
  return CoreThreads<Kern>::kAll;
}

}  // namespace olive
