// internal.h -- host-side declarations shared by the translation units of
// libolive.so.  Not part of the public ABI (include/olive.h is).
#pragma once

#include <atomic>
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/olive.h"

namespace olive {

constexpr int kSvMax = 64;        // most vocabulary segments per row tile
constexpr int kRowAlign = 128;    // row tiles of the compacted hidden copy
constexpr size_t kWsAlign = 256;  // alignment of every workspace region

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Launch context gathered once per API call.
struct Ctx {
  cudaStream_t stream;
  int device;
  int num_sms;
  uint64_t wait_limit_ns;
};

// Fills ctx for the current device; checks compute capability 10.3.
olive_status make_ctx(void* stream, Ctx* ctx);

// Raises a kernel's dynamic shared-memory limit to `smem` once per device
// and process (`done` is the call site's per-device flag array of
// kMaxDevices entries), so later calls issue no attribute call and can be
// captured into a CUDA graph.  Returns false if the attribute call fails.
constexpr int kMaxDevices = 64;
bool set_smem_once(const void* func, int smem, int device, std::atomic<int>* done);

// Encodes a 2-D bf16 tensor map (row-major [outer, inner], row pitch in
// bytes) with 128-byte swizzle and the given box.  Returns false on failure.
bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                    uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer);
// The same without swizzling (a box lands in shared memory row after row).
bool encode_bf16_2d_plain(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer);

// Rows of the G slab used by the backward passes for vocabulary size V.
int64_t slab_rows(int64_t Tpad, int64_t V);
inline int64_t vpad(int64_t V) { return align_up(static_cast<size_t>(V), 8); }

// ---- workspace carving (sizes in bytes; every region 256-byte aligned) ----
struct FwdWs {
  void* hc;       // bf16 [Tpad, d] compacted hidden rows
  float* part_m;  // [kSvMax, Tpad]
  float* part_s;  // [kSvMax, Tpad]
  float* zy;      // [Tpad]
  float* nll;     // [Tpad]
};
size_t fwd_ws_bytes(int64_t T, int64_t d);
FwdWs carve_fwd(void* ws, int64_t T, int64_t d);

struct TopkWs {
  void* hc;          // bf16 [Tpad, d]
  float* part_m;     // [kSvMax, Tpad]
  float* part_s;     // [kSvMax, Tpad]
  float* part_a;     // [kSvMax, Tpad] entropy numerators
  float* part_tv;    // [kSvMax, Tpad, 16] per-segment top logits
  int32_t* part_ti;  // [kSvMax, Tpad, 16] their vocabulary ids
};
size_t topk_ws_bytes(int64_t T, int64_t d);
TopkWs carve_topk(void* ws, int64_t T, int64_t d);

struct BwdWs {
  void* hc;       // bf16 [Tpad, d]
  void* g;        // bf16 [Tc, Vpad]
  float* dw_acc;  // fp32 [V, d] (bf16 output only)
  uint32_t* counters;  // tile-scheduler counters of the fused backward
  int64_t tc;     // slab rows
};
size_t bwd_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype);
BwdWs carve_bwd(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype);
size_t topk_kl_bwd_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype);

// OPD per-token stats sweep (dual product with two top lists)
struct OpdWs {
  void* hcs;         // bf16 [Tpad, d_s]
  void* hct;         // bf16 [Tpad, d_t]
  float* part;       // [6, kSvMax, Tpad]
  float* part_sv;    // [kSvMax, Tpad, 16]
  int32_t* part_si;  // [kSvMax, Tpad, 16]
  float* part_sx;    // [kSvMax, Tpad, 16]
  float* part_tv;    // [kSvMax, Tpad, 16]
  int32_t* part_ti;  // [kSvMax, Tpad, 16]
};
size_t opd_ws_bytes(int64_t T, int64_t ds, int64_t dt);
OpdWs carve_opd(void* ws, int64_t T, int64_t ds, int64_t dt);

// fused forward + backward: the backward's regions plus the ZSAVE partials
struct FbWs {
  void* hc;        // bf16 [Tpad, d]
  void* g;         // bf16 [Tc, Vpad]: e = 2^(x - m_tile), then G
  float* part_zm;  // [Tc, ceil(V/128)] half-tile max (base 2)
  float* part_zs;  // [Tc, ceil(V/128)] half-tile sums
  float* zy;       // [Tc] target logits of the slab
  float* nll;      // [Tpad] per-row loss terms
  float* dw_acc;   // fp32 [V, d] (bf16 output only)
  float* zref;     // [Tc, 2] reference maxima of the slab rows (base 2)
  float* lam;      // [Tc] dH row scale of the slab rows
  void* hs;        // bf16 [Tpad, d]: hc rows scaled by their lam (dW operand)
  int64_t tc;
};
size_t fb_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype);
FbWs carve_fb(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype);

struct KlWs {
  void* hcs;      // bf16 [Tpad, d_s]
  void* hct;      // bf16 [Tpad, d_t]
  float* part;    // [5, kSvMax, Tpad] value-sweep partials
  // gradient only: both heads' lse per compact row (p the primary head), the
  // exchange ring of the on-chip gradient pass and its counters
  float* lse_p;   // [Tpad]
  float* lse_q;   // [Tpad]
  void* ring;     // group_ring_bytes(T, d_s, V)
  uint32_t* ctr;  // ctr_words words
  size_t ctr_words;
};
size_t kl_ws_bytes(int64_t T, int64_t ds, int64_t dt, int64_t V, int grad);
KlWs carve_kl(void* ws, int64_t T, int64_t ds, int64_t dt, int64_t V, int grad);

// On-chip training step (lmhead_group.cu): groups of ceil(d / 256) CTAs
// exchange 128 x 256 bf16 logit-gradient tiles through a ring of fixed size.
constexpr int kGroupMaxSms = 192;  // ring and counters are sized for up to this many SMs
struct GroupWs {
  void* hc;          // bf16 [Tpad, d]
  float* rref;       // [Tpad] reference (base 2) per compact row
  float* rmax;       // [Tpad] row maxima of tiles that are redone
  float* zy;         // [Tpad] target logits
  float* pyb;        // [Tpad] the targets' bf16 exchange-tile entries
  float* nll;        // [Tpad] per-row loss terms
  float* part_s;     // [g_max, Tpad] per-member partial sums
  float* part_m;     // [g_max, Tpad] per-member partial maxima
  void* ring;        // group_ring_bytes(T, d, V)
  uint32_t* outer;   // [2 rt] pass-A group barriers (first launch, redo launch)
  uint32_t* redo;    // [1 + rt] redo list
  uint32_t* ring_ctr;  // 3 launches x group_ctr_words(T, d, V)
  size_t ctr_words;  // words from `outer` to the end of ring_ctr
};
size_t group_ws_bytes(int64_t T, int64_t d, int64_t V);
GroupWs carve_group(void* ws, int64_t T, int64_t d, int64_t V);
int group_g_max(int64_t d);
int group_count_max(int64_t T, int64_t d, int64_t V);
size_t group_ring_words(int64_t T, int64_t d, int64_t V);
size_t group_ring_bytes(int64_t T, int64_t d, int64_t V);
size_t group_ctr_words(int64_t T, int64_t d, int64_t V);
int group_sweep_cols(int sms);

struct GroupArgs {
  int32_t* dev_status;
  const int32_t* n_rows;
  const int32_t* rows;
  const int32_t* targets;
  int reduction;
  float inv_tau;
  const float* grad_loss;
  int lse_known, redo, write_fwd;
  const float* lse_in;
  float *rref, *rmax, *part_s, *part_m, *zy, *pyb, *logp, *lse, *nll;
  uint32_t* redo_list;
  uint32_t* outer_ctr;
  void* ring;
  void* d_hidden;
  void* d_W;
  int out_dtype;
  // mode 3 (divergence gradient) only
  const void* hc2;      // teacher rows, bf16 [Tpad, d2]
  const void* W2;       // teacher head, bf16 [V, d2]
  int d2, reverse;
  const float *lse_sc, *lse_tc, *kl, *grad_kl;
};
// mode 0: reference maxima, 1: pass A (lse, logp, dH), 2: pass B (dW),
// 3: divergence gradient (d_hidden = G . W with G from both heads)
olive_status launch_group(const Ctx& c, int mode, const void* hc, const void* W, int32_t T,
                          int32_t d, int32_t V, const GroupArgs& a, int c_base, int c_end,
                          uint32_t* ring_ctr);
// The divergence gradient on chip: d_h_s = G . W_s with G from both heads'
// logits (recomputed tile by tile by groups of CTA pairs, 128-wide vocabulary
// tiles) and the value sweep's kl, lse_s, lse_t; ctr (ctr_words) is zeroed here.
olive_status launch_kl_group_grad(const Ctx& c, const void* hcs, const void* hct, const void* W_s,
                                  int32_t d_s, const void* W_t, int32_t d_t, const int32_t* rows,
                                  const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                                  int reverse, const float* kl, const float* lse_s,
                                  const float* lse_t, const float* grad_kl, void* d_h_s,
                                  int grad_dtype, void* ring, uint32_t* ctr, size_t ctr_words,
                                  int32_t* dev_status);
// The whole step: forward + backward when lse_given is null (logp, lse, loss
// written), else the backward of that forward.
olive_status launch_loss_group(const Ctx& c, const void* hidden, const void* W,
                               const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                               int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                               const float* grad_loss, const float* lse_given, float* logp,
                               float* lse, float* loss, void* d_hidden, void* d_W, int grad_dtype,
                               void* ws, int32_t* dev_status);

// ---- launchers (validated arguments; return OLIVE_OK or OLIVE_ERR_CUDA) ----
olive_status launch_splice_pack(const Ctx& c, const int32_t* prefix_ids, const int32_t* prefix_off,
                                const int32_t* cont_ids, const int32_t* cont_off, int32_t S,
                                int32_t V, int32_t T_cap, int32_t* ids, int32_t* targets,
                                uint8_t* loss_mask, int32_t* cu_seqlens, int32_t* cut_offsets,
                                int32_t* rows, int32_t* n_rows, int32_t* dev_status);

// Multi-turn variant: the loss flag of every continuation token selects the
// rows; ws holds one int per 2048 packed positions.
size_t splice_masked_ws_bytes(int64_t T_cap);
olive_status launch_splice_pack_masked(const Ctx& c, const int32_t* prefix_ids,
                                       const int32_t* prefix_off, const int32_t* cont_ids,
                                       const int32_t* cont_off, const uint8_t* cont_loss, int32_t S,
                                       int32_t V, int32_t T_cap, int32_t* ids, int32_t* targets,
                                       uint8_t* loss_mask, int32_t* cu_seqlens,
                                       int32_t* cut_offsets, int32_t* rows, int32_t* n_rows,
                                       void* ws, int32_t* dev_status);

// Copies hidden[rows[r]] to hc[r] for r < n_rows and zero-fills the rest of
// the last 128-row tile.
olive_status launch_gather_rows(const Ctx& c, const void* hidden, const int32_t* rows,
                                const int32_t* n_rows, int32_t T, int32_t d, void* hc,
                                int32_t* dev_status);

olive_status launch_logprob_fwd(const Ctx& c, const void* hidden, const void* W,
                                const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                                int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                                float* logp, float* lse, float* loss, void* ws,
                                int32_t* dev_status);

// y = x * (*scale) on n bf16 or fp32 elements (x == y allowed).
olive_status launch_scale(const Ctx& c, const void* x, void* y, size_t n, int dtype,
                          const float* scale);

// One block sums the per-row loss terms nll[0, n) in a fixed order (fp64).
olive_status launch_loss_reduce(const Ctx& c, const int32_t* n_rows, int32_t T, const float* nll,
                                int reduction, float* loss);

// Forward and backward of the Eq. (osd-ce) loss in one pass over the logits
// (grad_loss is read on the device before the gradients are formed).
olive_status launch_loss_fwd_bwd(const Ctx& c, const void* hidden, const void* W,
                                 const int32_t* targets, const int32_t* rows,
                                 const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                 float inv_tau, int reduction, const float* grad_loss, float* logp,
                                 float* lse, float* loss, void* d_hidden, void* d_W, int grad_dtype,
                                 void* ws, int32_t* dev_status);

olive_status launch_topk_fwd(const Ctx& c, const void* hidden, const void* W, const int32_t* rows,
                             const int32_t* n_rows, int32_t T, int32_t d, int32_t V, float inv_tau,
                             int32_t K, float* lse, float* entropy, float* topk_logp,
                             int32_t* topk_ids, void* ws, int32_t* dev_status);

olive_status launch_topk_compare(const Ctx& c, const void* h_t, const void* W_t, int32_t d_t,
                                 const int32_t* rows, const int32_t* n_rows, int32_t T, int32_t V,
                                 float inv_tau, int32_t K, const int32_t* s_ids,
                                 const float* s_logp, const int32_t* t_ids, const float* t_lse,
                                 float* overlap, float* kl_topk, float* t_logp_s,
                                 int32_t* dev_status);

// Top-K KL gradient in place of the cross-entropy one: per masked row t the
// softmax coefficient coef[t] and the full gradient values val[t, k] at the
// ids[t, k] of the student's top-K set (K <= 16).
struct SparseGrad {
  const float* coef;
  const float* val;
  const int32_t* ids;
  int32_t K;
};

// Cross-entropy backward (sg == nullptr: targets, grad_loss, reduction used)
// or, with sg, the top-K KL backward (targets, grad_loss unused; lse is the
// student's).
olive_status launch_opd_stats(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                              const void* h_t, const void* W_t, int32_t d_t, const int32_t* rows,
                              const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                              int direction, int32_t K, float* kl, float* s_lse, float* t_lse,
                              float* s_entropy, float* s_topk_logp, int32_t* s_topk_ids,
                              float* t_logp_s, float* overlap, float* kl_topk, void* ws,
                              int32_t* dev_status);

olive_status launch_loss_bwd(const Ctx& c, const void* hidden, const void* W,
                             const int32_t* targets, const int32_t* rows, const int32_t* n_rows,
                             int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
                             const float* lse, const float* grad_loss, void* d_hidden, void* d_W,
                             int grad_dtype, void* ws, int32_t* dev_status,
                             const SparseGrad* sg = nullptr);

// Fills coef [T] and val [T, K] of the top-K KL gradient on the masked rows
// from the forward's top-K lists, the teacher's log-probs at the student's
// ids (t_logp_s), kl_topk and the weights grad_kl.
olive_status launch_topk_kl_prep(const Ctx& c, const int32_t* rows, const int32_t* n_rows,
                                 int32_t T, int32_t V, float inv_tau, int32_t K,
                                 const int32_t* s_ids, const float* s_logp,
                                 const float* t_logp_s, const float* kl_topk,
                                 const float* grad_kl, float* coef, float* val,
                                 int32_t* dev_status);

olive_status launch_divergence(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                               const void* h_t, const void* W_t, int32_t d_t, const int32_t* rows,
                               const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                               int direction, float* kl, const float* grad_kl, void* d_h_s,
                               int grad_dtype, void* ws, int32_t* dev_status);

// Words of tile-scheduler counters the fused backward needs.
size_t bwd_counter_words(int64_t Tpad, int64_t tc);

// Top-K KL forward and backward over one sweep of the student's logits
// (lmhead_fused.cu): workspace = the fused forward + backward regions, then
// the slab rows' true half-tile maxima [tc, ceil(V/128)].
size_t topk_kl_fb_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype);
olive_status launch_topk_kl_fwd_bwd(const Ctx& c, const void* h_s, const void* W_s, int32_t d_s,
                                    const void* h_t, const void* W_t, int32_t d_t,
                                    const int32_t* rows, const int32_t* n_rows, int32_t T,
                                    int32_t V, float inv_tau, int32_t K, const float* t_lse,
                                    const int32_t* t_ids, const float* grad_kl, float* s_lse,
                                    int32_t* s_ids, float* s_logp, float* t_logp_s,
                                    float* kl_topk, float* overlap, void* d_h_s, void* d_W_s,
                                    int grad_dtype, void* ws, int32_t* dev_status);

}  // namespace olive
