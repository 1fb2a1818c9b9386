// lmhead_group.cu -- the training step of the Eq. (osd-ce) loss (Section 3.1)
// with its logit gradient formed and consumed on chip.
//
// With z = inv_tau H[rows] W^T, lse per row and G = coef (softmax(z) -
// onehot(y)) (coef = g inv_tau, / N_mask for OLIVE_REDUCE_MEAN):
//   dH = G . W       reduces over the vocabulary  (K = V)
//   dW = G^T . hc    reduces over the masked rows (K = N_mask)
// Either output tile is [128, d] fp32 for a 128-row M tile: 2 MB at d = 4096,
// eight SMs' worth of tensor memory, so one SM cannot hold it.  The CTAs are
// therefore split into GROUPS of g >= ceil(d / 256) members.  Member m owns
// the output columns [c0, c0 + cw) of d (cw <= 256) and keeps their 128 x cw
// fp32 accumulator in TMEM for a whole OUTER tile, while the members take
// turns computing the 128 x 256 logit tiles (Z jobs, K = d) that every member
// needs.  The member that computed a Z tile turns it into a bf16 EXCHANGE
// tile and stores it in its group's ring of R slots of 64 KB; every member
// bulk-copies each exchange tile, 64 K-columns at a time, into shared memory
// as the A operand of its accumulating MMA.  The ring has a fixed size (R
// slots per group, a few tens of MB in all, independent of T and V), each
// slot is rewritten once all g members have read it, and no slot outlives R
// exchange tiles: the logits and G are never stored as a [rows, V] array.
// (The ring is read from the L2; its lines are written back to DRAM when the
// L2 evicts them, about one write of each tile, the size of the exchange.)
//
//   Pass A (outer = 128 masked rows, inner = 256-column vocabulary tile):
//     exchange tile P'[r, v] = 2^(x - R_r), x = z log2(e), R_r a per-row
//     reference (the maximum of the row's first vocabulary tile, from the
//     GM_REF launch, or the row's lse when it is given); the members
//     accumulate acc = P' . W[:, chunk] and keep per-row partial sums of
//     2^(x - R) over their own Z jobs, merged at the end of the outer tile
//     into lse2 = R + log2(sum) (a group barrier through a global counter).
//     The epilogue then applies the softmax-minus-onehot scaling:
//       dH[r, chunk] = coef (2^(R - lse2) acc - W[y_r, chunk]).
//     A row whose maximum exceeds R by more than kRefMax (2^x - R would leave
//     the range the bf16 operand and the fp32 sums are safe in) puts its row
//     tile on a redo list; a second launch recomputes those tiles with R = the
//     rows' maxima from the first launch.
//   Pass B (outer = 128 vocabulary rows, inner = 256 masked rows): exchange
//     tile G^T[v, r] = coef_r (2^(x - lse2_r) - [v == y_r]) from pass A's
//     lse (transposed logit tile z^T = W hc^T, so a TMEM lane is a vocabulary
//     row); member m accumulates dW[v, chunk] = G^T . hc[:, chunk] and stores
//     it when the outer tile ends (every dW element has one owner: no atomics).
//
//   Divergence mode (GM_KL: the gradient of OPD's per-token KL, Section 1,
//   after the value sweep of lmhead_kl.cu has given KL and both heads' lse):
//     the pass A layout with two products per Z job, the student's (K = d_s)
//     and the teacher's (K = d_t) logits of a 128-column vocabulary tile in
//     the two halves of the 256-column Z accumulator; the epilogue forms the
//     exact G (reverse: g inv_tau p_s ((z_s - z_t) - (lse_s - lse_t) - KL),
//     forward: g inv_tau (p_s - p_t)) and the members accumulate
//     d_h_s = G . W_s.
//
// Each pass executes two products per logit (the Z tile and its share of the
// accumulation), so the training step executes 4 GEMM units of 2 N_mask d V
// flops for the 3 it counts.
//
// CTA pairs: the kernel runs as clusters of two CTAs.  Pair m of pair-group
// pg is member m of group 2 pg (its even CTA) and of group 2 pg + 1 (its odd
// CTA); the two groups walk the same inner tiles at the same time, so every
// MMA is a tcgen05.mma.cta_group::2 issued by the even CTA (M = 256: each CTA
// holds 128 rows of A -- its own hc, W or exchange rows -- and half of B's N
// columns, and receives its 128 accumulator rows in its own TMEM).  Each CTA
// loads 32 KB per 64-deep K step instead of 48 KB, and six stages fit.  The
// group size g is chosen between ceil(d / 256) and ~1.25 times that to fill
// the SMs with pair-groups of 2 g CTAs (d = 4096 on 152 SMs: g = 19, members
// of 224 columns, four pair-groups).  When the even group has one more outer
// tile than the odd one, the odd CTAs run a phantom tile whose rows are
// invalid and never stored.
//
// Schedule inside a group (every member derives it from N_mask on the
// device): the exchange tiles of the group's outer tiles form one sequence
// e = 0 .. E-1 (e = i ni + k for the group's i-th outer tile and inner tile
// k), cut into rounds of g tiles; tile e is computed by member e mod g and
// lives in ring slot e mod R (R = 3 g).  Each pair's tensor pipe runs, per
// round r: its Z job of round r, then the accumulation of all g tiles of
// round r - 1, so the epilogue of a Z tile (and the other members'
// epilogues) overlaps the accumulation MMAs, and a single 256-column Z
// accumulator suffices next to the (<= 256)-column output accumulator (512
// TMEM columns).  Waits between members go through global release/acquire
// counters: a slot's `ready` count (tile written) and `cons` count (tile
// copied by all g members); the producer warp checks a whole round's ready
// flags at once and a signal warp posts the cons counts.  Every dependency
// points to a tile of an earlier round, every CTA is resident at once (the
// grid is one CTA per SM; the host checks that the GPU holds all its
// clusters), and every wait is bounded (OLIVE_ERR_TIMEOUT on expiry).  A
// pacing hint keeps the groups within a round of one another, so that one
// DRAM fetch of an inner operand tile (W in pass A, hc in pass B) can serve
// every group from the L2 (how often it does depends on what else the L2
// holds: the call reads the streamed operand several times over).
#include <algorithm>
#include <atomic>
#include <cmath>

#include "sched.cuh"
#include "sm103.cuh"

namespace olive {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kZN = 256;             // logit tile 128 x 256
constexpr int kStages = 6;
constexpr int kSA = kBM * kBK * 2;   // A operand of a stage: this CTA's 128 rows x 64
constexpr int kSB = kBM * kBK * 2;   // B operand: this CTA's half of N (<= 128) x 64
constexpr int kStageBytes = kSA + kSB;
constexpr int kXSlice = kSA;         // one 128 x 64 K-slice of an exchange tile
constexpr int kXTile = 4 * kXSlice;  // 128 x 256 bf16 (64 KB)
constexpr int kEpi = 128;            // epilogue threads: one accumulator row each
constexpr int kProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kSignalWarp = 6;       // posts the members' "tile copied" counts
constexpr int kThreads = 224;
constexpr int kStatusTimeoutBit = 1 << OLIVE_ERR_TIMEOUT;
constexpr float kRefMax = 64.f;
constexpr int kMetaBytes = kZN * 8;  // pass B: lse2 and target of the tile's 256 rows
// Pacing across groups: every group walks the same sequence of inner tiles
// (vocabulary tiles of W in pass A, row pairs of hc in pass B), so while the
// groups stay within kPaceLag rounds of one another one DRAM fetch of a tile
// serves all of them from the L2; a group that runs ahead waits, at most
// kPaceLimitNs per round (a hint: giving up only costs bandwidth).
constexpr int kPaceLag = 1;
constexpr uint64_t kPaceLimitNs = 2000000;
constexpr uint32_t kPaceDone = 0x40000000u;

enum GMode : int { GM_REF = 0, GM_A = 1, GM_B = 2, GM_KL = 3 };

// GM_REF / GM_A: za = hc {64 x 128}, zb = W {64 x 128}, xb = W {64 x 64}
// GM_B:          za = W {64 x 128},  zb = hc {64 x 128}, xb = hc {64 x 64}
// xa: the ring, [slices x 128 rows] of 64 bf16, unswizzled {64 x 128} boxes
// (a slice is stored already swizzled, so the copy is linear)
// GM_KL:         za = hc_s {64 x 128}, zb = W_s {64 x 64}, za2 = hc_t {64 x 128},
//                zb2 = W_t {64 x 64}, xb = W_s {64 x 64} (128-wide vocabulary tiles)
struct GroupMaps {
  CUtensorMap za, zb, xb, xa, za2, zb2;
};

struct GroupParams {
  int32_t* dev_status;
  uint64_t wait_limit_ns;
  const int32_t* n_rows;
  const int32_t* rows;
  const int32_t* targets;
  const __nv_bfloat16* W;   // GM_A: the rows W[y] of the onehot term
  int32_t T, d, V;
  int32_t mode;
  int32_t g, ngroups, R;    // members per group, groups, ring slots per group
  int32_t chunk;            // output columns per member (multiple of 16, <= 256)
  int32_t c_base, c_end;    // output columns [c_base, c_end) of this launch
  int32_t reduction;
  float inv_tau, scale2;    // 1 / tau, log2(e) / tau
  const float* grad_loss;   // device scalar g
  int32_t lse_known;        // GM_A: R = lse2 from lse_in (backward of a given forward)
  int32_t redo;             // GM_A: outer tiles from redo_list, R = rmax
  int32_t write_fwd;        // GM_A: write lse, logp, nll
  const float* lse_in;      // [T] natural lse per packed row (GM_A lse_known, GM_B)
  float* rref;              // [Tpad] base-2 reference per compact row (GM_REF writes)
  float* rmax;              // [Tpad] base-2 row maximum (GM_A writes for redo rows)
  float* part_s;            // [g][Tpad] per-member sums of 2^(x - R)
  float* part_m;            // [g][Tpad] per-member maxima (base 2)
  float* zy;                // [Tpad] target logit z_y (natural units)
  float* pyb;               // [Tpad] P'_y as rounded to bf16 in the exchange tile
  float* logp;              // [T]
  float* lse;               // [T]
  float* nll;               // [Tpad] per-row loss terms
  uint32_t* redo_list;      // [1 + rt]: count, then row tiles
  uint32_t* outer_ctr;      // [rt] pass A group barrier (one array per GM_A launch)
  __nv_bfloat16* ring;      // [ngroups][R][128 x 256] exchange tiles (swizzled images)
  uint32_t* ready;          // [ngroups][R]
  uint32_t* cons;           // [ngroups][R]
  uint32_t* pace;           // [ngroups] rounds each group has begun (a pacing hint)
  void* out;                // GM_A: d_hidden [T, d]; GM_B: d_W [V, d]
  int32_t out_dtype;
  int64_t ring_tiles;       // exchange tiles the ring holds (debug checks)
  int32_t part_groups;      // rows of part_s / part_m (debug checks)
  int32_t zn;               // width of an inner vocabulary tile: 256 (CE), 128 (GM_KL)
  // GM_KL (divergence gradient): per compact row the lse of both heads from the
  // value sweep, per packed row the KL and the weights g_t
  int32_t d2;               // teacher width
  int32_t reverse;          // KL direction
  const float* lse_sc;      // [Tpad] student lse (natural)
  const float* lse_tc;      // [Tpad] teacher lse (natural)
  const float* kl;          // [T]
  const float* grad_kl;     // [T]
};

// per-CTA schedule, the same in every CTA of a group
struct GSched {
  int n;      // masked rows
  int rank;   // 0: the pair's even CTA (issues the MMAs), 1: its peer
  int ph;     // outer index standing for "no outer tile" (past the last)
  int no;     // outer tiles in all
  int ni;     // inner tiles per outer tile
  int nk;     // 64-wide K steps of a Z job
  int q, m;   // group, member
  int myo;    // outer tiles of this group
  int E;      // exchange tiles of this group
  int c0, cw; // output columns of this member
  int nbox;   // 64-column boxes of this CTA's half of the accumulation's B
  int nacc;   // N of the accumulation MMA (cw rounded up to 16)
  int b0;     // first column of this CTA's half of B
  int kcount; // inner extent: V (pass A) or n (pass B)
  int zn;     // inner tile width
  int nk2;    // 64-wide K steps of a Z job's second product (GM_KL: the teacher)
  float coef;
};

// CTAs come in pairs (clusters of 2): pair-group pg of g pairs runs groups
// 2 pg (even CTAs) and 2 pg + 1 (odd CTAs) in lockstep, pair m being member m
// of both; the two groups walk the same inner tiles at the same time, so
// each pair's MMAs share the B operand (W or hc tiles), half from each CTA.
__device__ GSched make_gsched(const GroupParams& p) {
  GSched s;
  s.n = read_n_rows(p.n_rows, p.T, p.dev_status);
  s.rank = static_cast<int>(cluster_rank());
  const int rt = (s.n + kBM - 1) / kBM;
  if (p.mode == GM_B) {
    s.no = (p.V + kBM - 1) / kBM;
    s.ph = s.no;
    s.ni = (s.n + kZN - 1) / kZN;
    s.kcount = s.n;
  } else {
    s.no = (p.mode == GM_A && p.redo) ? static_cast<int>(min(p.redo_list[0], static_cast<uint32_t>(rt))) : rt;
    s.ph = rt;
    s.ni = p.mode == GM_REF ? 1 : (p.V + p.zn - 1) / p.zn;
    s.kcount = p.V;
  }
  s.zn = p.zn;
  s.nk = (p.d + kBK - 1) / kBK;
  s.nk2 = p.mode == GM_KL ? (p.d2 + kBK - 1) / kBK : 0;
  const int pair = blockIdx.x >> 1;
  s.m = pair % p.g;
  const int pg = pair / p.g;
  s.q = 2 * pg + s.rank;
  // both groups of a pair-group run as many outer tiles as the even one
  // (which has at least as many); the odd one's extra tile, if any, is a
  // phantom whose rows are invalid
  const int qe = 2 * pg;
  s.myo = qe < s.no ? (s.no - qe + p.ngroups - 1) / p.ngroups : 0;
  s.E = s.myo * s.ni;
  s.c0 = p.c_base + s.m * p.chunk;
  s.cw = min(p.chunk, p.c_end - s.c0);
  if (s.cw < 0) s.cw = 0;
  s.nacc = (s.cw + 15) / 16 * 16;
  if (s.nacc < 16) s.nacc = 16;
  s.b0 = s.c0 + s.rank * (s.nacc / 2);
  s.nbox = (s.nacc / 2 + 63) / 64;
  s.coef = 0.f;
  if (p.grad_loss) {
    float gl = *p.grad_loss;
    if (p.reduction == OLIVE_REDUCE_MEAN && s.n > 0) gl = gl / static_cast<float>(s.n);
    s.coef = gl * p.inv_tau;
  }
  return s;
}

// global index of the group's i-th outer tile (s.ph for a phantom)
__device__ __forceinline__ bool phantom(const GroupParams& p, const GSched& s, int i) {
  return s.q + i * p.ngroups >= s.no;
}
__device__ __forceinline__ int outer_of(const GroupParams& p, const GSched& s, int i) {
  const int k = s.q + i * p.ngroups;
  if (k >= s.no) return s.ph;
  return (p.mode == GM_A && p.redo) ? static_cast<int>(p.redo_list[1 + k]) : k;
}
__device__ __forceinline__ int kvalid_of(const GSched& s, int k) {
  return min(s.zn, s.kcount - k * s.zn);
}
// 64-wide K slices of inner tile k that hold valid columns
__device__ __forceinline__ int slices_of(const GSched& s, int k) {
  return (kvalid_of(s, k) + kBK - 1) / kBK;
}
// does member m compute a Z job of the group's i-th outer tile?
__device__ __forceinline__ bool member_has_job(const GSched& s, int g, int i) {
  const int lo = i * s.ni;
  const int first = lo + (((s.m - lo) % g) + g) % g;
  return first < lo + s.ni;
}

// byte offset of 16-byte chunk c (0..7) of row r in K-slice sl of an exchange
// tile: the 128-byte-swizzled K-major layout a TMA load of a 64 x 128 box
// produces (row r at r * 128, chunk c at position c ^ (r & 7)), so a linear
// copy of a slice to a 1024-byte-aligned stage is a valid UMMA operand
__device__ __forceinline__ uint32_t img_off(int r, int sl, int c) {
  return static_cast<uint32_t>(sl * kXSlice + (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ void store_out32(void* base, size_t off, int dtype, int n_valid,
                                            const float (&v)[32]) {
  if (dtype == OLIVE_DTYPE_BF16) {
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(base) + off;
    if (n_valid >= 32) {
      uint4* d4 = reinterpret_cast<uint4*>(o);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        d4[q] = make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                           pack_bf16x2(v[8 * q + 4], v[8 * q + 5]), pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < n_valid) o[k] = __float2bfloat16_rn(v[k]);
    }
  } else {
    float* o = static_cast<float*>(base) + off;
    if (n_valid >= 32) {
      float4* d4 = reinterpret_cast<float4*>(o);
#pragma unroll
      for (int q = 0; q < 8; ++q) d4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < n_valid) o[k] = v[k];
    }
  }
}

// 32 fp32 values -> four 16-byte chunks of row r of the exchange image
__device__ __forceinline__ void store_img32(uint8_t* img, int r, int h, const float (&v)[32]) {
  const int sl = h >> 1;
  const int c0 = (h & 1) * 4;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint4 u = make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                               pack_bf16x2(v[8 * q + 4], v[8 * q + 5]), pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
    *reinterpret_cast<uint4*>(img + img_off(r, sl, c0 + q)) = u;
  }
}

// per-row values of pass A (and GM_REF) for compact row rc
struct RowA {
  bool valid;   // rc < n and rows[rc] in [0, T)
  int t, y;     // packed row, target (-1 when none)
  float R;      // reference (base 2)
};

__device__ __forceinline__ RowA load_row_a(const GroupParams& p, const GSched& s, int rc) {
  RowA a;
  a.valid = false;
  a.t = -1;
  a.y = -1;
  a.R = 0.f;
  if (rc < s.n) {
    const int t = p.rows[rc];
    if (t >= 0 && t < p.T) {
      a.valid = true;
      a.t = t;
      a.y = p.targets[t];
      if (p.mode == GM_A) {
        if (p.lse_known) a.R = p.lse_in[t] * kLog2e;
        else if (p.redo) a.R = p.rmax[rc];
        else a.R = p.rref[rc];
      }
    }
  }
  return a;
}

// All lanes of a warp: wait until the exchange tiles [e_lo, e_end) of a
// round are written (ready[e mod R] > e / R), lane i checking tiles i, i+32,
// ...  Returns the warp's common decision (false: limit ran out or abort).
__device__ bool wait_round_ready(const uint32_t* ready, int R, int e_lo, int e_end, int lane,
                                 const WaitCtl& ctl) {
  const uint64_t t0 = global_timer_ns();
  while (true) {
    bool mine = true;
    for (int e = e_lo + lane; e < e_end; e += 32)
      mine = mine && ld_acquire(ready + e % R) >= static_cast<uint32_t>(e / R + 1);
    if (__all_sync(0xffffffffu, mine)) return true;
    bool stop = *ctl.abort != 0;
    if (!stop && global_timer_ns() - t0 > ctl.limit_ns) {
      if (lane == 0) *ctl.abort = 1;
      stop = true;
    }
    if (__any_sync(0xffffffffu, stop)) return false;
    nanosleep_ns(64);
  }
}

// All lanes of a warp: wait (at most kPaceLimitNs) until every group has
// begun round `need` (pace[q] >= need), lane i checking groups i, i+32, ...
__device__ void pace_wait(const uint32_t* pace, int ngroups, int need, int lane) {
  if (need <= 0) return;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    bool mine = true;
    for (int q = lane; q < ngroups; q += 32)
      mine = mine && *reinterpret_cast<const volatile uint32_t*>(pace + q) >= static_cast<uint32_t>(need);
    if (__all_sync(0xffffffffu, mine)) return;
    if (global_timer_ns() - t0 > kPaceLimitNs) return;
    nanosleep_ns(128);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    lmhead_group_kernel(const __grid_constant__ GroupMaps maps, const GroupParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);

  // the same layout in both CTAs of a pair: the MMA reads both at these offsets
  const uint32_t stages = base;
  const uint32_t bar0 = base + kStages * kStageBytes;
  auto full_bar = [&](int st) { return bar0 + 8u * st; };
  auto empty_bar = [&](int st) { return bar0 + 8u * (kStages + st); };
  const uint32_t zfull = bar0 + 8u * (2 * kStages);
  const uint32_t zempty = zfull + 8;
  const uint32_t ofull = zfull + 16;
  const uint32_t oempty = zfull + 24;
  const uint32_t drain = zfull + 32;
  uint8_t* misc = gbase + kStages * kStageBytes + 8 * (2 * kStages + 5);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 4);
  volatile uint32_t* copied = reinterpret_cast<volatile uint32_t*>(misc + 8);  // tiles copied
  GSched* sched_smem = reinterpret_cast<GSched*>(misc + 16);
  float* meta_l = reinterpret_cast<float*>(misc + 128);                 // [256] lse2 (GM_B)
  int* meta_y = reinterpret_cast<int*>(misc + 128 + kMetaBytes / 2);    // [256] targets (GM_B)

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();

  if (threadIdx.x == 0) {
    for (int st = 0; st < kStages; ++st) {
      mbar_init(full_bar(st), 1);   // the even CTA's producer (both CTAs' bytes)
      mbar_init(empty_bar(st), 1);  // the even CTA's MMA commit (multicast)
    }
    mbar_init(zfull, 1);
    mbar_init(zempty, 8);           // the four epilogue warps of both CTAs
    mbar_init(ofull, 1);
    mbar_init(oempty, 8);
    mbar_init(drain, 1);
    *abort_flag = 0;
    *copied = 0;
    *sched_smem = make_gsched(p);
    fence_mbar_init();
  }
  if (warp == kProducerWarp && lane == 0) {
    tma_prefetch_desc(&maps.za);
    tma_prefetch_desc(&maps.zb);
    tma_prefetch_desc(&maps.xb);
    tma_prefetch_desc(&maps.xa);
  }
  if (warp == kMmaWarp) {
    tmem_alloc_pair(smem_u32(tmem_slot), 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  // barriers of both CTAs initialised and TMEM allocated before any CTA
  // touches its peer's
  cluster_sync_all();
  tc_fence_after();

  const uint32_t tmem_base = *tmem_slot;
  const GSched s = *sched_smem;
  const WaitCtl ctl{abort_flag, p.wait_limit_ns};
  const int g = p.g;
  const bool consume = p.mode != GM_REF;
  const int nr = (s.E + g - 1) / g;  // rounds
  const size_t ring0 = static_cast<size_t>(s.q) * p.R;

  if (warp == kProducerWarp) {
    // lane 0 issues every copy (this CTA's 128 rows of A and its half of B;
    // completion counted on the even CTA's full barrier, whose producer
    // announces both CTAs' bytes: the odd CTA's copies may land first, the
    // transaction count then dips below zero within the phase, which mbarriers
    // allow; no phase can mix with the next, since a CTA refills a stage only
    // after the MMAs that read it have committed); the whole warp checks the
    // `ready` flags of a round's g exchange tiles at once
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    const bool paced = consume && p.ngroups > 2;
    // the streamed operand of a Z job (W rows in pass A, hc rows in pass B)
    // is read again by the accumulation a round later: keep it in the L2
    // ahead of other lines (ncu at 16384 rows: DRAM reads 196 -> 149 GB per
    // call, time level)
    const uint64_t keep = l2_policy_evict_last();
    for (int r = 0; ok && r <= nr; ++r) {
      const int j = r * g + s.m;
      if (paced && r < nr) {
        pace_wait(p.pace, p.ngroups, r - kPaceLag, lane);
        if (s.m == 0 && lane == 0)
          *reinterpret_cast<volatile uint32_t*>(p.pace + s.q) = static_cast<uint32_t>(r + 1);
      }
      if (r < nr && j < s.E) {
        if (lane == 0) {
          const int o = outer_of(p, s, j / s.ni);
          const int k = j % s.ni;
          // K steps [0, nk): the (first) product, za x zb; [nk, nk + nk2):
          // GM_KL's teacher product, za2 x zb2; B rows of this CTA's half of
          // the zn-wide vocabulary (or row) tile
          const int half = s.zn / 2;
          const uint32_t zbytes = 2 * (kSA + half * kBK * 2);
          for (int ks = 0; ks < s.nk + s.nk2; ++ks) {
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, ctl)) { ok = false; break; }
            const uint32_t sA = stages + stage * kStageBytes;
            const uint32_t fb = map_shared(full_bar(stage), 0);
            if (rank == 0) mbar_arrive_expect_tx(full_bar(stage), zbytes);
            const bool second = ks >= s.nk;
            const int kx = (second ? ks - s.nk : ks) * kBK;
            // (a skipped copy leaves its stage short: the MMA's wait then runs
            // out and the call reports OLIVE_ERR_TIMEOUT as well)
            if (OLIVE_DCHECK(p.dev_status, o >= 0 && o <= s.ph && k >= 0 && k < s.ni)) {
              tma_load_2d_pair(sA, second ? &maps.za2 : &maps.za, fb, kx, o * kBM);
              tma_load_2d_pair_hint(sA + kSA, second ? &maps.zb2 : &maps.zb, fb, kx,
                                    k * s.zn + static_cast<int>(rank) * half, keep);
            }
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
      }
      if (!ok || !consume || r == 0) continue;
      const int e_lo = (r - 1) * g;
      const int e_end = min(r * g, s.E);
      ok = wait_round_ready(p.ready + ring0, p.R, e_lo, e_end, lane, ctl);
      if (!ok) break;
      if (lane == 0) {
        fence_proxy_async_global();
        for (int e = e_lo; ok && e < e_end; ++e) {
          const int slot = e % p.R;
          const int k = e % s.ni;
          const int nsl = slices_of(s, k);
          for (int sl = 0; sl < nsl; ++sl) {
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, ctl)) { ok = false; break; }
            const uint32_t sA = stages + stage * kStageBytes;
            const uint32_t fb = map_shared(full_bar(stage), 0);
            if (rank == 0) mbar_arrive_expect_tx(full_bar(stage), 2 * (kXSlice + s.nbox * 8192));
            // TMA x coordinates must be 16-byte aligned (8 bf16)
            if (OLIVE_DCHECK(p.dev_status, static_cast<int64_t>(ring0 + slot) < p.ring_tiles &&
                                               s.b0 % 8 == 0 && s.b0 >= 0 && s.b0 < p.d + 64)) {
              tma_load_2d_pair(sA, &maps.xa, fb, 0, static_cast<int>(((ring0 + slot) * 4 + sl) * kBM));
              for (int b = 0; b < s.nbox; ++b)
                tma_load_2d_pair(sA + kSA + b * 8192, &maps.xb, fb, s.b0 + 64 * b, k * s.zn + sl * kBK);
            }
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    if (paced && s.m == 0 && lane == 0) *reinterpret_cast<volatile uint32_t*>(p.pace + s.q) = kPaceDone;
    if (!ok && lane == 0) {
      // let copies already issued land before the CTA retires
      const uint64_t t0 = global_timer_ns();
      while (global_timer_ns() - t0 < 50000) nanosleep_ns(1000);
    }
    __syncwarp();
  } else if (warp == kSignalWarp) {
    // for every exchange tile, in order, once the pair's MMA thread has seen
    // all its slices land: one release increment of the slot's `cons` count
    if (lane == 0 && consume) {
      uint32_t sent = 0;
      const uint32_t total = static_cast<uint32_t>(s.E);
      uint64_t last = global_timer_ns();
      while (sent < total) {
        const uint32_t c = *copied;
        if (c > sent) {
          for (; sent < c; ++sent) red_release_add(p.cons + ring0 + sent % p.R, 1u);
          last = global_timer_ns();
          continue;
        }
        if (*abort_flag) break;
        nanosleep_ns(100);
        if (global_timer_ns() - last > p.wait_limit_ns) {
          *abort_flag = 1;
          break;
        }
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // the even CTA's lane 0 issues the pair's MMAs (M = 256: 128 rows in each
    // CTA's TMEM); the odd CTA's MMA warp only holds its TMEM allocation
    if (lane == 0 && rank == 0) {
      const uint32_t zacc = tmem_base;
      const uint32_t oacc = tmem_base + 256;
      const uint32_t idz = idesc_bf16(2 * kBM, s.zn, false, false);
      const uint32_t idx = idesc_bf16(2 * kBM, s.nacc, false, true);
      const uint32_t copied_peer = map_shared(smem_u32(const_cast<uint32_t*>(copied)), 1);
      int stage = 0;
      uint32_t phase = 0, zph = 0, oph = 0;
      bool ok = true;
      for (int r = 0; ok && r <= nr; ++r) {
        const int j = r * g + s.m;
        if (r < nr && j < s.E) {
          if (!mbar_wait(zempty, zph ^ 1u, ctl)) { ok = false; break; }
          tc_fence_after();
          for (int ks = 0; ks < s.nk + s.nk2; ++ks) {
            if (!mbar_wait(full_bar(stage), phase, ctl)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sA = stages + stage * kStageBytes;
            const uint32_t sB = sA + kSA;
            // GM_KL: the teacher's product goes to the next zn columns
            const bool second = ks >= s.nk;
            const uint32_t dz = second ? zacc + static_cast<uint32_t>(s.zn) : zacc;
            const int kl = second ? ks - s.nk : ks;
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
              umma_bf16_pair(dz, sdesc_sw128(sA + kk * 32, 16, 1024), sdesc_sw128(sB + kk * 32, 16, 1024),
                             idz, (kl > 0 || kk > 0) ? 1u : 0u);
            umma_commit_pair(empty_bar(stage));
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
          }
          if (!ok) break;
          umma_commit_pair(zfull);
          zph ^= 1u;
        }
        if (!consume || r == 0) continue;
        const int e_end = min(r * g, s.E);
        for (int e = (r - 1) * g; ok && e < e_end; ++e) {
          const int k = e % s.ni;
          if (k == 0) {
            if (!mbar_wait(oempty, oph ^ 1u, ctl)) { ok = false; break; }
            tc_fence_after();
          }
          const int nsl = slices_of(s, k);
          for (int sl = 0; sl < nsl; ++sl) {
            if (!mbar_wait(full_bar(stage), phase, ctl)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sA = stages + stage * kStageBytes;
            const uint32_t sB = sA + kSA;
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
              umma_bf16_pair(oacc, sdesc_sw128(sA + kk * 32, 16, 1024),
                             sdesc_sw128(sB + kk * 2048, 8192, 1024), idx,
                             (k > 0 || sl > 0 || kk > 0) ? 1u : 0u);
            umma_commit_pair(empty_bar(stage));
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
          }
          if (!ok) break;
          // every slice of tile e has landed in both CTAs: their signal warps
          // tell the two groups (a slot may be rewritten once all of its
          // group's members have said so)
          *copied = static_cast<uint32_t>(e + 1);
          st_shared_cluster(copied_peer, static_cast<uint32_t>(e + 1));
          if (k == s.ni - 1) {
            umma_commit_pair(ofull);
            oph ^= 1u;
          }
        }
      }
      // arrives once every MMA issued above has completed (bounded wait that
      // ignores the abort flag: it only waits for work already in flight)
      umma_commit_pair(drain);
      volatile int keep_waiting = 0;
      const uint64_t floor_ns = 200ull * 1000 * 1000;
      const WaitCtl own{&keep_waiting, p.wait_limit_ns > floor_ns ? p.wait_limit_ns : floor_ns};
      mbar_wait(drain, 0, own);
    }
    __syncwarp();
  } else {
    // epilogue warps 0..3: thread = accumulator row = TMEM lane
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(warp * 32) << 16);
    uint8_t* ring_bytes = reinterpret_cast<uint8_t*>(p.ring);
    // the even CTA's MMA thread waits until both CTAs' epilogues are done with
    // an accumulator: one arrival per epilogue warp on its barriers
    const uint32_t zempty_lead = map_shared(zempty, 0);
    const uint32_t oempty_lead = map_shared(oempty, 0);
    const uint32_t zaddr = lane_addr;
    const uint32_t oaddr = lane_addr + 256;
    uint32_t zph = 0, oph = 0;
    bool ok = true;
    const size_t Tpad = static_cast<size_t>((p.T + kBM - 1) / kBM) * kBM;

    if (p.mode == GM_B && s.ni == 0) {
      // no masked rows: dW is zero on this member's columns of its outer tiles
      float zero[32];
#pragma unroll
      for (int k = 0; k < 32; ++k) zero[k] = 0.f;
      for (int i = 0; i < s.myo; ++i) {
        const int v = outer_of(p, s, i) * kBM + row;
        if (v >= p.V) continue;
        for (int c = 0; c < s.cw; c += 32)
          store_out32(p.out, static_cast<size_t>(v) * p.d + s.c0 + c, p.out_dtype, min(32, s.cw - c), zero);
      }
    }

    int cur_o = -1;             // pass A: the outer tile of the running partials
    RowA ra{false, -1, -1, 0.f};
    float run_s = 0.f, run_m = -INFINITY;
    for (int r = 0; ok && r <= nr; ++r) {
      const int j = r * g + s.m;
      if (r < nr && j < s.E) {
        // ---------------------------------------------------- Z epilogue
        const int i = j / s.ni;
        const int k = j % s.ni;
        const int o = outer_of(p, s, i);
        const int slot = j % p.R;
        const int kv = kvalid_of(s, k);
        // 32-column blocks to read: every block of the slices the members
        // copy, so columns >= kv are written as zeros, never left stale
        const int hend = 2 * slices_of(s, k);
        if (consume) {
          // the slot's previous tile must have been copied by every member
          const bool free_ok =
              threadIdx.x == 0
                  ? wait_counter(p.cons + ring0 + slot, static_cast<uint32_t>(g * (j / p.R)), ctl)
                  : true;
          if (!named_bar_and(1, kEpi, free_ok)) { ok = false; break; }
        }
        if (p.mode == GM_B) {
          // lse2 and target of the tile's 256 masked rows (+inf / -1 beyond n)
          for (int c = threadIdx.x; c < kZN; c += kEpi) {
            const int rc = k * kZN + c;
            float l2 = INFINITY;
            int yy = -1;
            if (rc < s.n) {
              const int t = p.rows[rc];
              if (t >= 0 && t < p.T) {
                l2 = p.lse_in[t] * kLog2e;
                yy = p.targets[t];
              }
            }
            meta_l[c] = l2;
            meta_y[c] = yy;
          }
        }
        if (!named_bar_and(1, kEpi, mbar_wait(zfull, zph, ctl))) { ok = false; break; }
        zph ^= 1u;
        tc_fence_after();
        uint8_t* img = ring_bytes + (ring0 + slot) * static_cast<size_t>(kXTile);
        if (!OLIVE_DCHECK(p.dev_status, !consume || static_cast<int64_t>(ring0 + slot) < p.ring_tiles))
          img = nullptr;
        if (p.mode == GM_B) {
          const int v = o * kBM + row;
#pragma unroll 1
          for (int h = 0; h < hend; ++h) {
            uint32_t a[32];
            tmem_ld_32x32b_x32(zaddr + h * 32, a);
            tmem_ld_wait();
            float gv[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const int col = h * 32 + c;
              const float xl = fmaf(__uint_as_float(a[c]), p.scale2, -meta_l[col]);
              // the target entry p - 1 from expm1, exact where p is near 1
              const float pm = meta_y[col] == v ? expm1f(xl * kLn2) : fast_exp2(xl);
              gv[c] = col < kv ? s.coef * pm : 0.f;
            }
            if (img) store_img32(img, row, h, gv);
          }
        } else if (p.mode == GM_KL) {
          // G of the divergence for this 128 x 128 tile from both heads'
          // fp32 logits (zn columns each) and the row's lse of each head and
          // KL from the value sweep: reverse g inv_tau p_s (log p_s - log p_t
          // - KL), forward g inv_tau (p_s - p_t)
          const int rc = o * kBM + row;
          bool valid = false;
          float ls0 = 0.f, lt0 = 0.f, klv = 0.f, cf = 0.f;
          if (rc < s.n) {
            const int t = p.rows[rc];
            if (t >= 0 && t < p.T) {
              valid = true;
              ls0 = p.lse_sc[rc];
              lt0 = p.lse_tc[rc];
              klv = p.kl[t];
              cf = p.grad_kl[t] * p.inv_tau;
            }
          }
#pragma unroll 1
          for (int h = 0; h < hend; ++h) {
            uint32_t a[32], b[32];
            tmem_ld_32x32b_x32(zaddr + h * 32, a);
            tmem_ld_32x32b_x32(zaddr + static_cast<uint32_t>(s.zn) + h * 32, b);
            tmem_ld_wait();
            float gv[32];
            // log p_s - log p_t as (z_s - z_t) - (lse_s - lse_t): a teacher
            // shifted by a constant per row cancels before the large terms meet
            const float dl = ls0 - lt0;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float zs = __uint_as_float(a[c]) * p.inv_tau;
              const float zt = __uint_as_float(b[c]) * p.inv_tau;
              const float ps = fast_exp2((zs - ls0) * kLog2e);
              const float gg = p.reverse ? cf * ps * (((zs - zt) - dl) - klv)
                                         : cf * (ps - fast_exp2((zt - lt0) * kLog2e));
              gv[c] = (valid && h * 32 + c < kv) ? gg : 0.f;
            }
            if (img) store_img32(img, row, h, gv);
          }
        } else {
          if (o != cur_o) {
            cur_o = o;
            ra = load_row_a(p, s, o * kBM + row);
            run_s = 0.f;
            run_m = -INFINITY;
          }
          const int v0 = k * s.zn;
#pragma unroll 1
          for (int h = 0; h < hend; ++h) {
            uint32_t a[32];
            tmem_ld_32x32b_x32(zaddr + h * 32, a);
            tmem_ld_wait();
            float pv[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const int col = h * 32 + c;
              const float x = __uint_as_float(a[c]) * p.scale2;
              const bool in = col < kv;
              run_m = in ? fmaxf(run_m, x) : run_m;
              const float e = fast_exp2(x - ra.R);
              pv[c] = in ? e : 0.f;
              run_s += pv[c];
            }
            const int yo = ra.y - (v0 + h * 32);
            if (p.mode == GM_A && yo >= 0 && yo < 32) {
              // the target's exact logit and the bf16 value of P'_y the MMA
              // sees: the epilogue replaces that term by p_y - 1 from the
              // logit, so rows with p_y near 1 keep their accuracy
#pragma unroll
              for (int c = 0; c < 32; ++c)
                if (c == yo) {
                  p.zy[o * kBM + row] = __uint_as_float(a[c]) * p.inv_tau;
                  p.pyb[o * kBM + row] = __bfloat162float(__float2bfloat16_rn(pv[c]));
                }
            }
            if (p.mode == GM_A && img) store_img32(img, row, h, pv);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(zempty_lead);
        if (p.mode == GM_REF) {
          if (o * kBM + row < s.n) p.rref[o * kBM + row] = run_m;
        } else {
          if (p.mode == GM_A && ra.valid &&
              OLIVE_DCHECK(p.dev_status, s.m < p.part_groups && o * kBM + row < static_cast<int>(Tpad))) {
            p.part_s[static_cast<size_t>(s.m) * Tpad + o * kBM + row] = run_s;
            p.part_m[static_cast<size_t>(s.m) * Tpad + o * kBM + row] = run_m;
          }
          // publish the tile: every thread's stores, then one release
          fence_proxy_async_global();
          __threadfence();
          named_bar_sync(1, kEpi);
          if (threadIdx.x == 0) red_release_add(p.ready + ring0 + slot, 1u);
        }
      }
      if (!consume || r == 0) continue;
      // ------------------------------------------- outer tiles completed
      const int e_end = min(r * g, s.E);
      for (int e = (r - 1) * g; ok && e < e_end; ++e) {
        if (e % s.ni != s.ni - 1) continue;
        const int i = e / s.ni;
        const int o = outer_of(p, s, i);
        if (p.mode == GM_B) {
          if (!named_bar_and(1, kEpi, mbar_wait(ofull, oph, ctl))) { ok = false; break; }
          oph ^= 1u;
          tc_fence_after();
          const int v = o * kBM + row;
#pragma unroll 1
          for (int c = 0; c < s.cw; c += 32) {
            uint32_t a[32];
            tmem_ld_32x32b_x32(oaddr + c, a);
            tmem_ld_wait();
            float ov[32];
#pragma unroll
            for (int q = 0; q < 32; ++q) ov[q] = __uint_as_float(a[q]);
            if (v < p.V && OLIVE_DCHECK(p.dev_status, v >= 0 && s.c0 + c + min(32, s.cw - c) <= p.d))
              store_out32(p.out, static_cast<size_t>(v) * p.d + s.c0 + c, p.out_dtype,
                          min(32, s.cw - c), ov);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(oempty_lead);
          continue;
        }
        if (p.mode == GM_KL) {
          // the divergence gradient: G carried g inv_tau, so d_h_s is the sum
          if (!named_bar_and(1, kEpi, mbar_wait(ofull, oph, ctl))) { ok = false; break; }
          oph ^= 1u;
          tc_fence_after();
          const int rc = o * kBM + row;
          const int t = rc < s.n ? p.rows[rc] : -1;
#pragma unroll 1
          for (int c = 0; c < s.cw; c += 32) {
            uint32_t a[32];
            tmem_ld_32x32b_x32(oaddr + c, a);
            tmem_ld_wait();
            float ov[32];
#pragma unroll
            for (int q = 0; q < 32; ++q) ov[q] = __uint_as_float(a[q]);
            const int nv = min(32, s.cw - c);
            if (t >= 0 && t < p.T && OLIVE_DCHECK(p.dev_status, s.c0 + c + nv <= p.d))
              store_out32(p.out, static_cast<size_t>(t) * p.d + s.c0 + c, p.out_dtype, nv, ov);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(oempty_lead);
          continue;
        }
        // pass A: merge the members' partials, then dH
        const int rc = o * kBM + row;
        const RowA rw = load_row_a(p, s, rc);
        // every member's partials (and the target's z_y, P'_y from the
        // member that met it) are published before any member reads them
        if (rw.valid && !member_has_job(s, g, i)) {
          p.part_s[static_cast<size_t>(s.m) * Tpad + rc] = 0.f;
          p.part_m[static_cast<size_t>(s.m) * Tpad + rc] = -INFINITY;
        }
        if (!phantom(p, s, i) && OLIVE_DCHECK(p.dev_status, o >= 0 && o * kBM < static_cast<int>(Tpad))) {
          __threadfence();
          named_bar_sync(1, kEpi);
          if (threadIdx.x == 0) red_release_add(p.outer_ctr + o, 1u);
          const bool seen =
              threadIdx.x == 0 ? wait_counter(p.outer_ctr + o, static_cast<uint32_t>(g), ctl) : true;
          if (!named_bar_and(1, kEpi, seen)) { ok = false; break; }
        }
        if (!named_bar_and(1, kEpi, mbar_wait(ofull, oph, ctl))) { ok = false; break; }
        oph ^= 1u;
        tc_fence_after();
        float lse2 = rw.R, mx = -INFINITY;
        if (!p.lse_known && rw.valid) {
          float sum = 0.f;
          for (int mm = 0; mm < g; ++mm) {
            sum += __ldcg(p.part_s + static_cast<size_t>(mm) * Tpad + rc);
            mx = fmaxf(mx, __ldcg(p.part_m + static_cast<size_t>(mm) * Tpad + rc));
          }
          lse2 = rw.R + log2f(sum);
        }
        // (the redo launch, with R = the rows' maxima, never flags)
        const bool row_ok = !rw.valid || p.lse_known || p.redo ||
                            (mx - rw.R <= kRefMax && isfinite(lse2));
        const bool tile_ok = named_bar_and(1, kEpi, row_ok);
        if (!tile_ok) {
          // the reference was too low for some row: the redo launch
          // recomputes this row tile with R = the rows' maxima
          if (s.m == 0) {
            if (rw.valid) p.rmax[rc] = mx;
            if (threadIdx.x == 0) {
              const uint32_t at = atomicAdd(p.redo_list, 1u);
              p.redo_list[1 + at] = static_cast<uint32_t>(o);
            }
          }
        } else {
          const bool has_y = rw.valid && rw.y >= 0 && rw.y < p.V;
          if (s.m == 0 && rw.valid) {
            if (!has_y) atomicOr(p.dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
            if (p.write_fwd) {
              const float l = lse2 * kLn2;
              const float lp = has_y ? __ldcg(p.zy + rc) - l : NAN;
              p.lse[rw.t] = l;
              p.logp[rw.t] = lp;
              p.nll[rc] = -lp;
            }
          }
          const float scale = fast_exp2(rw.R - lse2);
          // dH = coef (scale acc - W[y]) with the target's term taken out of
          // acc (scale P'_y, P'_y as the MMA saw it) and put back as p_y W[y]:
          // together coef (scale acc + corr W[y]), corr = (p_y - 1) - scale P'_y
          float corr = 0.f;
          if (has_y) {
            const float lnat = p.lse_known ? p.lse_in[rw.t] : lse2 * kLn2;
            corr = expm1f(__ldcg(p.zy + rc) - lnat) - scale * __ldcg(p.pyb + rc);
          }
          const uint4* wy =
              has_y ? reinterpret_cast<const uint4*>(p.W + static_cast<size_t>(rw.y) * p.d + s.c0) : nullptr;
#pragma unroll 1
          for (int c = 0; c < s.cw; c += 32) {
            uint32_t a[32];
            tmem_ld_32x32b_x32(oaddr + c, a);
            tmem_ld_wait();
            float dv[32];
            const int nv = min(32, s.cw - c);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint4 w4 = make_uint4(0, 0, 0, 0);
              if (wy && 8 * q < nv) w4 = __ldg(wy + c / 8 + q);
              const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&w4);
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const float2 wf = __bfloat1622float2(w2[u]);
                dv[8 * q + 2 * u] = s.coef * fmaf(scale, __uint_as_float(a[8 * q + 2 * u]), corr * wf.x);
                dv[8 * q + 2 * u + 1] =
                    s.coef * fmaf(scale, __uint_as_float(a[8 * q + 2 * u + 1]), corr * wf.y);
              }
            }
            if (rw.valid && OLIVE_DCHECK(p.dev_status, rw.t >= 0 && rw.t < p.T && s.c0 + c + nv <= p.d))
              store_out32(p.out, static_cast<size_t>(rw.t) * p.d + s.c0 + c, p.out_dtype, nv, dv);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(oempty_lead);
      }
    }
  }

  tc_fence_before();
  // the pair's MMAs (all complete: the even CTA waited for them) and every
  // access to the peer's barriers are over before either CTA frees its TMEM
  cluster_sync_all();
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.dev_status, kStatusTimeoutBit);
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, 512);
  }
}

constexpr int kGroupSmem = 1024 + kStages * kStageBytes + 8 * (2 * kStages + 5) + 128 + kMetaBytes;
static_assert(kGroupSmem <= 227 * 1024, "shared memory budget");

int ring_slots_for(int g) { return 3 * g > 4 ? 3 * g : 4; }

// fewest members a group of `cols` output columns can have, and the most the
// shape search below may pick
int g_min_for(int cols) { return cols > kZN ? (cols + kZN - 1) / kZN : 1; }
int g_hi_for(int cols) { return g_min_for(cols) + g_min_for(cols) / 4 + 1; }

// Groups of g members, run as pair-groups of 2 g CTAs.  g is the member count
// between ceil(cols / 256) and ~1.25 times that which puts the most CTAs to
// work (d = 4096 at 152 SMs: g = 19, four pair-groups fill all 152), the
// smaller g on ties; members hold ceil(cols / g) columns rounded up to 16.
struct GroupShape {
  int g, chunk, ngroups, R;
};

GroupShape group_shape(int cols, int sms) {
  GroupShape gs{0, 0, 0, 0};
  int best_used = 0;
  for (int g = g_min_for(cols); g <= g_hi_for(cols); ++g) {
    const int used = 2 * g * (sms / (2 * g));
    if (used > best_used) {
      best_used = used;
      gs.g = g;
    }
  }
  if (gs.g == 0) return gs;
  gs.chunk = ((cols + gs.g - 1) / gs.g + 15) / 16 * 16;
  gs.ngroups = 2 * (sms / (2 * gs.g));
  gs.R = ring_slots_for(gs.g);
  return gs;
}

// output columns one sweep covers: the widest whose fewest members still
// form one pair-group
int sweep_cols_for(int sms) { return (sms / 2) * kZN; }

}  // namespace

// the widest group a launch may form for width d (ring and partials are
// sized for it)
int group_g_max(int64_t d) {
  const int64_t cap = static_cast<int64_t>(sweep_cols_for(kGroupMaxSms));
  return g_hi_for(static_cast<int>(d < cap ? d : cap));
}

int ring_slots(int g) { return ring_slots_for(g); }

// groups a launch forms at most (an even number): as many as the SMs hold,
// and no more than the outer tiles of either pass (row tiles of T rows,
// vocabulary tiles) rounded up to a pair
int group_count_max(int64_t T, int64_t d, int64_t V) {
  const int64_t cap = static_cast<int64_t>(sweep_cols_for(kGroupMaxSms));
  const int gmin = g_min_for(static_cast<int>(d < cap ? d : cap));
  const int64_t outer = std::max<int64_t>(std::max(ceil_div(T, kBM), ceil_div(V, kBM)), 2);
  return static_cast<int>(std::min<int64_t>(2 * (kGroupMaxSms / (2 * gmin)), (outer + 1) / 2 * 2));
}

size_t group_ring_words(int64_t T, int64_t d, int64_t V) {
  return static_cast<size_t>(group_count_max(T, d, V)) * ring_slots_for(group_g_max(d));
}

size_t group_ring_bytes(int64_t T, int64_t d, int64_t V) { return group_ring_words(T, d, V) * kXTile; }

// counter words of one launch: ready and cons per ring slot, pace per group
size_t group_ctr_words(int64_t T, int64_t d, int64_t V) {
  return 2 * group_ring_words(T, d, V) + static_cast<size_t>(group_count_max(T, d, V));
}

int group_sweep_cols(int sms) { return sweep_cols_for(sms < kGroupMaxSms ? sms : kGroupMaxSms); }

olive_status launch_group(const Ctx& c, int mode, const void* hc, const void* W, int32_t T,
                          int32_t d, int32_t V, const GroupArgs& a, int c_base, int c_end,
                          uint32_t* ring_ctr) {
  const int sms = c.num_sms < kGroupMaxSms ? c.num_sms : kGroupMaxSms;
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  GroupShape gs;
  if (mode == GM_REF) {
    gs.g = 1;
    gs.chunk = kZN;
    gs.ngroups = sms / 2 * 2;
    gs.R = 1;
  } else {
    gs = group_shape(c_end - c_base, sms);
    gs.ngroups = std::min(gs.ngroups, group_count_max(T, d, V));
    if (gs.ngroups < 2 || gs.g * gs.ngroups > sms) return OLIVE_ERR_SHAPE;
  }
  GroupMaps maps;
  const bool rowsA = mode != GM_B;
  const void* zaBase = rowsA ? hc : W;
  const void* zbBase = rowsA ? W : hc;
  const uint64_t zaRows = rowsA ? Tpad : V;
  const uint64_t zbRows = rowsA ? V : Tpad;
  // the ring viewed as rows of 64 bf16 (one 128-byte row of a slice image)
  const uint64_t ring_rows = group_ring_bytes(T, d, V) / 128;
  // inner tiles of 256 vocabulary entries (rows in pass B), 128 for the
  // divergence, whose Z jobs hold both heads' logits in the Z accumulator;
  // each CTA of a pair loads half of them as its B rows
  const int zn = mode == GM_KL ? 128 : kZN;
  if (!encode_bf16_2d(&maps.za, zaBase, d, zaRows, 2ull * d, 64, 128) ||
      !encode_bf16_2d(&maps.zb, zbBase, d, zbRows, 2ull * d, 64, zn / 2) ||
      !encode_bf16_2d(&maps.xb, zbBase, d, zbRows, 2ull * d, 64, 64) ||
      !encode_bf16_2d_plain(&maps.xa, a.ring, 64, ring_rows, 128, 64, 128))
    return OLIVE_ERR_CUDA;
  if (mode == GM_KL) {
    if (!encode_bf16_2d(&maps.za2, a.hc2, a.d2, Tpad, 2ull * a.d2, 64, 128) ||
        !encode_bf16_2d(&maps.zb2, a.W2, a.d2, V, 2ull * a.d2, 64, zn / 2))
      return OLIVE_ERR_CUDA;
  } else {
    maps.za2 = maps.za;
    maps.zb2 = maps.zb;
  }

  GroupParams p = {};
  p.dev_status = a.dev_status;
  p.wait_limit_ns = c.wait_limit_ns;
  p.n_rows = a.n_rows;
  p.rows = a.rows;
  p.targets = a.targets;
  p.W = static_cast<const __nv_bfloat16*>(W);
  p.T = T;
  p.d = d;
  p.V = V;
  p.mode = mode;
  p.g = gs.g;
  p.ngroups = gs.ngroups;
  p.R = gs.R;
  p.chunk = gs.chunk;
  p.c_base = c_base;
  p.c_end = c_end;
  p.reduction = a.reduction;
  p.inv_tau = a.inv_tau;
  p.scale2 = a.inv_tau * kLog2e;
  p.grad_loss = a.grad_loss;
  p.lse_known = a.lse_known;
  p.redo = a.redo;
  p.write_fwd = a.write_fwd;
  p.lse_in = a.lse_in;
  p.rref = a.rref;
  p.rmax = a.rmax;
  p.part_s = a.part_s;
  p.part_m = a.part_m;
  p.zy = a.zy;
  p.pyb = a.pyb;
  p.logp = a.logp;
  p.lse = a.lse;
  p.nll = a.nll;
  p.redo_list = a.redo_list;
  p.outer_ctr = a.outer_ctr + (mode == GM_A && a.redo ? (T + kBM - 1) / kBM : 0);
  p.ring = static_cast<__nv_bfloat16*>(a.ring);
  p.ready = ring_ctr;
  p.cons = ring_ctr ? ring_ctr + static_cast<size_t>(gs.ngroups) * gs.R : nullptr;
  p.pace = ring_ctr ? ring_ctr + 2 * static_cast<size_t>(gs.ngroups) * gs.R : nullptr;
  p.out = mode == GM_B ? a.d_W : a.d_hidden;  // GM_KL: d_h_s
  p.out_dtype = a.out_dtype;
  p.ring_tiles = static_cast<int64_t>(group_ring_words(T, d, V));
  p.part_groups = group_g_max(d);
  p.zn = zn;
  p.d2 = a.d2;
  p.reverse = a.reverse;
  p.lse_sc = a.lse_sc;
  p.lse_tc = a.lse_tc;
  p.kl = a.kl;
  p.grad_kl = a.grad_kl;

  static std::atomic<int> done[kMaxDevices];
  if (!set_smem_once(reinterpret_cast<const void*>(lmhead_group_kernel), kGroupSmem, c.device, done))
    return OLIVE_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(gs.ngroups * gs.g);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kGroupSmem;
  cfg.stream = c.stream;
  // clusters of two CTAs (the MMA pairs).  Members of a group wait on one
  // another, so every CTA must be resident at once: the grid is at most one
  // CTA per SM, and the first launch on each device checks that the GPU holds
  // all of its clusters together (cudaOccupancyMaxActiveClusters), else the
  // call is refused.  The launch is not marked cooperative: profilers (ncu)
  // cannot launch cooperative grids of clusters, and a grid that fits starts
  // whole on an idle GPU; if another stream's kernel holds SMs, the waits are
  // bounded and report OLIVE_ERR_TIMEOUT.
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  static std::atomic<int> fits[kMaxDevices];  // clusters the device holds at once, + 1
  const bool cached = c.device >= 0 && c.device < kMaxDevices;
  int held = cached ? fits[c.device].load(std::memory_order_acquire) - 1 : -1;
  if (held < 0) {
    cudaLaunchConfig_t q = cfg;
    q.gridDim = dim3(2 * (sms / 2));
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, lmhead_group_kernel, &q) != cudaSuccess) {
      cudaGetLastError();
      return OLIVE_ERR_CUDA;
    }
    held = n;
    if (cached) fits[c.device].store(n + 1, std::memory_order_release);
  }
  if (static_cast<int>(cfg.gridDim.x) > 2 * held) return OLIVE_ERR_UNSUPPORTED_DEVICE;
  if (cudaLaunchKernelEx(&cfg, lmhead_group_kernel, maps, p) != cudaSuccess) {
    cudaGetLastError();
    return OLIVE_ERR_CUDA;
  }
  return OLIVE_OK;
}

}  // namespace olive

namespace olive {

olive_status launch_loss_group(const Ctx& c, const void* hidden, const void* W,
                               const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                               int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                               const float* grad_loss, const float* lse_given, float* logp,
                               float* lse, float* loss, void* d_hidden, void* d_W, int grad_dtype,
                               void* ws, int32_t* dev_status) {
  const bool fwd = lse_given == nullptr;
  const GroupWs w = carve_group(ws, T, d, V);
  const size_t elt = grad_dtype == OLIVE_DTYPE_BF16 ? 2 : 4;
  olive_status st = launch_gather_rows(c, hidden, rows, n_rows, T, d, w.hc, dev_status);
  if (st != OLIVE_OK) return st;
  if (cudaMemsetAsync(d_hidden, 0, elt * T * static_cast<size_t>(d), c.stream) != cudaSuccess ||
      cudaMemsetAsync(w.outer, 0, 4 * w.ctr_words, c.stream) != cudaSuccess)
    return OLIVE_ERR_CUDA;
  if (fwd && (cudaMemsetAsync(logp, 0, sizeof(float) * T, c.stream) != cudaSuccess ||
              cudaMemsetAsync(lse, 0, sizeof(float) * T, c.stream) != cudaSuccess))
    return OLIVE_ERR_CUDA;

  GroupArgs a = {};
  a.dev_status = dev_status;
  a.n_rows = n_rows;
  a.rows = rows;
  a.targets = targets;
  a.reduction = reduction;
  a.inv_tau = inv_tau;
  a.grad_loss = grad_loss;
  a.lse_in = fwd ? lse : lse_given;
  a.rref = w.rref;
  a.rmax = w.rmax;
  a.part_s = w.part_s;
  a.part_m = w.part_m;
  a.zy = w.zy;
  a.pyb = w.pyb;
  a.logp = logp;
  a.lse = lse;
  a.nll = w.nll;
  a.redo_list = w.redo;
  a.outer_ctr = w.outer;
  a.ring = w.ring;
  a.d_hidden = d_hidden;
  a.d_W = d_W;
  a.out_dtype = grad_dtype;

  if (fwd && (st = launch_group(c, GM_REF, w.hc, W, T, d, V, a, 0, d, nullptr)) != OLIVE_OK)
    return st;
  // one sweep of both passes per range of output columns the SMs can hold
  // (every d up to 19456 at 152 SMs takes one)
  const int cols = group_sweep_cols(c.num_sms);
  const size_t rw = group_ctr_words(T, d, V);
  for (int cb = 0; cb < d; cb += cols) {
    const int ce = d - cb < cols ? d : cb + cols;
    if (cb > 0 && cudaMemsetAsync(w.outer, 0, 4 * w.ctr_words, c.stream) != cudaSuccess)
      return OLIVE_ERR_CUDA;
    a.lse_known = (!fwd || cb > 0) ? 1 : 0;
    a.write_fwd = (fwd && cb == 0) ? 1 : 0;
    a.redo = 0;
    if ((st = launch_group(c, GM_A, w.hc, W, T, d, V, a, cb, ce, w.ring_ctr)) != OLIVE_OK) return st;
    if (fwd && cb == 0) {
      a.redo = 1;
      if ((st = launch_group(c, GM_A, w.hc, W, T, d, V, a, cb, ce, w.ring_ctr + rw)) != OLIVE_OK)
        return st;
      a.redo = 0;
    }
    if ((st = launch_group(c, GM_B, w.hc, W, T, d, V, a, cb, ce, w.ring_ctr + 2 * rw)) != OLIVE_OK)
      return st;
  }
  return fwd ? launch_loss_reduce(c, n_rows, T, w.nll, reduction, loss) : OLIVE_OK;
}

}  // namespace olive

namespace olive {

olive_status launch_kl_group_grad(const Ctx& c, const void* hcs, const void* hct, const void* W_s,
                                  int32_t d_s, const void* W_t, int32_t d_t, const int32_t* rows,
                                  const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                                  int reverse, const float* kl, const float* lse_s,
                                  const float* lse_t, const float* grad_kl, void* d_h_s,
                                  int grad_dtype, void* ring, uint32_t* ctr, size_t ctr_words,
                                  int32_t* dev_status) {
  const int64_t rt = align_up(static_cast<size_t>(T), kRowAlign) / kRowAlign;
  GroupArgs a = {};
  a.dev_status = dev_status;
  a.n_rows = n_rows;
  a.rows = rows;
  a.inv_tau = inv_tau;
  a.ring = ring;
  a.d_hidden = d_h_s;
  a.out_dtype = grad_dtype;
  a.hc2 = hct;
  a.W2 = W_t;
  a.d2 = d_t;
  a.reverse = reverse;
  a.lse_sc = lse_s;
  a.lse_tc = lse_t;
  a.kl = kl;
  a.grad_kl = grad_kl;
  uint32_t* ring_ctr = ctr + 3 * rt + 1;
  const int cols = group_sweep_cols(c.num_sms);
  for (int cb = 0; cb < d_s; cb += cols) {
    const int ce = d_s - cb < cols ? d_s : cb + cols;
    if (cudaMemsetAsync(ctr, 0, 4 * ctr_words, c.stream) != cudaSuccess) return OLIVE_ERR_CUDA;
    const olive_status st = launch_group(c, GM_KL, hcs, W_s, T, d_s, V, a, cb, ce, ring_ctr);
    if (st != OLIVE_OK) return st;
  }
  return OLIVE_OK;
}

}  // namespace olive
