/*
 * olive.h -- C ABI of libolive.so, the GB300 (sm_103a) implementation of the
 * per-token scoring path of OLIVE ("Learning from Teacher Continuations at
 * Student States").
 *
 * The path: a student prefix (prompt x and student tokens y_{1:k}) is cut at a
 * student state and followed by a teacher continuation y~_{1:l}; the student
 * is trained with the masked cross-entropy of Eq. (osd-ce) (Section 3.1) on the
 * continuation tokens only.  The OPD baseline (Section 1) scores tokens with a
 * per-token reverse KL against the teacher instead.  Four calls cover it:
 *
 *   olive_splice_pack        packs the spliced sequences and builds the loss mask
 *   olive_token_logprob_fwd  LM-head projection + online log-sum-exp + masked
 *                            target log-prob and loss (the [T,V] logits are
 *                            never stored)
 *   olive_token_loss_bwd     d loss / d hidden and d loss / d W
 *   olive_token_divergence   full-vocabulary per-token KL (+ d KL / d h_s)
 *
 * and these extend it:
 *
 *   olive_token_loss_fwd_bwd the forward and backward of a training step in
 *                            one call, G formed and consumed on chip
 *   olive_token_loss_fwd_bwd_slab  the same step through an HBM slab of G
 *                            (no logit recomputation)
 *   olive_splice_pack_masked multi-turn packing, loss only on teacher actions
 *                            (Section 3.2)
 *   olive_token_topk_fwd     per-token entropy and top-K log-probs
 *   olive_topk_compare       student/teacher top-K overlap and top-K KL
 *   olive_topk_kl_bwd        gradient of the top-K KL
 *   olive_topk_kl_fwd_bwd    the student's top-K lists, the top-K KL and its
 *                            gradient from one sweep of the student's logits
 *   olive_opd_token_stats    OPD's per-token KL, entropy, top-K lists, overlap
 *                            and top-K KL from one sweep with both heads
 *   olive_token_logprob_fwd_noalloc  the forward without a workspace
 *
 * Conventions shared by every call
 *   - Every pointer argument is a DEVICE pointer unless stated otherwise.  The
 *     caller owns every buffer; no call allocates device memory.  Scratch
 *     memory comes from the caller's `workspace` (size from
 *     olive_workspace_size, 256-byte aligned).  Three things outlive a call:
 *     the OLIVE_NOALLOC_SCRATCH_BYTES array that olive_token_logprob_fwd_noalloc
 *     uses (compiled into the library, held by every GPU that loads it); the
 *     per-device kernel attributes (shared-memory limits), set on the first
 *     call on each device so that later calls issue no attribute call and can
 *     be captured in a CUDA graph (the on-chip training step also checks
 *     there, once, that the device holds its whole grid of CTA pairs at
 *     once); and two environment variables, read at each call:
 *     OLIVE_WAIT_LIMIT_MS (wall-clock limit of every internal wait, default
 *     1000; on expiry the call sets OLIVE_ERR_TIMEOUT) and OLIVE_SLAB_ROWS
 *     (lowers the slab of the slab forms, see olive_slab_rows).
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  All calls
 *     are asynchronous on it; none synchronises the host.
 *   - The returned olive_status covers what the host can check before any
 *     launch (null pointers, shapes, alignment, device).  On any non-OK
 *     return nothing was launched.
 *   - Errors in device data (a token id outside [0,V), offsets that do not
 *     describe the batch, an internal wait that ran out of time) are OR-ed
 *     into *dev_status as bits (1u << code), code from olive_status.  The
 *     caller zeroes *dev_status and reads it whenever it synchronises.
 *   - Row counts such as N_mask stay on the device (`n_rows`), so the three
 *     compute calls can follow olive_splice_pack without a host round trip;
 *     grids are sized from the host-side upper bound T.
 *   - Tensors are row-major and contiguous.  bf16 is IEEE bfloat16.  Base
 *     pointers of hidden, W, d_hidden and d_W must be 16-byte aligned, and
 *     d (every hidden width) must be a multiple of 8.
 *   - The library runs only on compute capability 10.3 (sm_103a).
 */
#ifndef OLIVE_H_
#define OLIVE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define OLIVE_API __attribute__((visibility("default")))
#else
#define OLIVE_API
#endif

#define OLIVE_ABI_VERSION 1

typedef enum {
  OLIVE_OK = 0,
  OLIVE_ERR_INVALID_ARG = 1,       /* null pointer, bad enum value            */
  OLIVE_ERR_SHAPE = 2,             /* non-positive or too large size          */
  OLIVE_ERR_ALIGNMENT = 3,         /* pointer or width breaks the 16-B rule   */
  OLIVE_ERR_TOKEN_RANGE = 4,       /* (device) an id or target outside [0,V)  */
  OLIVE_ERR_OFFSETS = 5,           /* (device) offsets / row list malformed   */
  OLIVE_ERR_TIMEOUT = 6,           /* (device) an internal wait ran out       */
  OLIVE_ERR_UNSUPPORTED_DEVICE = 7,/* current device is not sm_103           */
  OLIVE_ERR_CUDA = 8,              /* a CUDA runtime/driver call failed       */
  OLIVE_ERR_WORKSPACE = 9,         /* workspace null, misaligned or too small */
  OLIVE_ERR_BOUNDS = 10            /* (device, OLIVE_DEBUG builds only) an index
                                      check failed; the access was skipped      */
} olive_status;

enum { OLIVE_REDUCE_SUM = 0, OLIVE_REDUCE_MEAN = 1 };
enum { OLIVE_KL_REVERSE = 0, OLIVE_KL_FORWARD = 1 };
enum { OLIVE_DTYPE_BF16 = 0, OLIVE_DTYPE_F32 = 1 };
enum { OLIVE_OP_LOGPROB_FWD = 0, OLIVE_OP_LOSS_BWD = 1, OLIVE_OP_DIVERGENCE = 2,
       OLIVE_OP_TOPK_FWD = 3, OLIVE_OP_SPLICE_MASKED = 4, OLIVE_OP_TOPK_KL_BWD = 5,
       OLIVE_OP_LOSS_FWD_BWD = 6, OLIVE_OP_OPD_STATS = 7, OLIVE_OP_TOPK_KL_FWD_BWD = 8,
       OLIVE_OP_LOSS_FWD_BWD_SLAB = 9 };

/*
 * Rows of the G slab that the slab forms (olive_token_loss_fwd_bwd_slab,
 * olive_topk_kl_bwd, olive_topk_kl_fwd_bwd) hold at a time for T packed rows
 * and V vocabulary
 * entries: about 5.6 GB of bf16 G in whole 128-row tiles, at most 32768 rows
 * and at most T rounded up to 128, lowered by OLIVE_SLAB_ROWS (a multiple of
 * 128).  A call on more masked rows runs ceil(N_mask / rows) slabs.  Returns 0
 * for T < 1 or V < 1.  The paper has no counterpart.
 */
OLIVE_API int32_t olive_slab_rows(int32_t T, int32_t V);

/* ABI version of the loaded library (OLIVE_ABI_VERSION). */
OLIVE_API int olive_abi_version(void);

/* Static text for a status code. Never NULL. */
OLIVE_API const char* olive_status_string(olive_status s);

/*
 * Workspace bytes a compute call needs for host-side upper bound T rows.
 *   op  OLIVE_OP_LOGPROB_FWD / OLIVE_OP_LOSS_BWD: d = hidden width, d_t ignored.
 *   op  OLIVE_OP_DIVERGENCE: d = student width d_s, d_t = teacher width.
 *   op  OLIVE_OP_TOPK_FWD: d = hidden width, d_t ignored.
 *   op  OLIVE_OP_SPLICE_MASKED: T = T_cap; d, d_t, V ignored.
 *   op  OLIVE_OP_OPD_STATS: d = student width d_s, d_t = teacher width.
 *   op  OLIVE_OP_TOPK_KL_BWD, OLIVE_OP_LOSS_FWD_BWD,
 *       OLIVE_OP_TOPK_KL_FWD_BWD: d = (student) hidden width, grad_dtype as
 *       for OLIVE_OP_LOSS_BWD, d_t ignored.
 *   `grad` (bwd / divergence): non-zero when gradients are requested
 *   (OLIVE_OP_LOSS_BWD always computes them); `grad_dtype` is the dtype of
 *   d_W for OLIVE_OP_LOSS_BWD (bf16 output needs an fp32 accumulator).
 * Returns 0 for invalid arguments.
 */
OLIVE_API size_t olive_workspace_size(int op, int32_t T, int32_t d, int32_t d_t, int32_t V,
                            int grad, int grad_dtype);

/*
 * olive_splice_pack -- builds the packed student-update batch of Section 3.1:
 * for each sequence s the spliced sequence (x, y_{1:k}, y~_{1:l}) =
 * prefix_s || continuation_s, laid back to back, with the loss of Eq. (osd-ce)
 * on the continuation tokens only ("the prompt and student prefix remain in
 * the conditioning context but are masked out of the loss").
 *
 * Inputs (device, int32):
 *   prefix_ids  all prefixes (prompt + student prefix) back to back;
 *   prefix_off  [S+1] CSR offsets, prefix_off[0] = 0, non-decreasing;
 *               every prefix holds >= 1 id;
 *   cont_ids    all continuations (already in student tokens) back to back;
 *   cont_off    [S+1] CSR offsets, cont_off[0] = 0, non-decreasing (a
 *               continuation may be empty);
 *   S >= 1 sequences, V >= 1 vocabulary size, T_cap >= 1 capacity of the
 *   packed outputs.
 * Outputs (device), with T = sum_s (P_s + C_s) packed tokens:
 *   ids[T_cap]        packed ids; positions >= T are set to 0;
 *   targets[T_cap]    ids[t+1] when t+1 belongs to the same sequence, else -1
 *                     (row t of the hidden states predicts token t+1);
 *   loss_mask[T_cap]  1 where targets[t] is a continuation token y~_j, else 0;
 *   cu_seqlens[S+1]   packed start of every sequence, cu_seqlens[S] = T;
 *   cut_offsets[S]    packed index of y~_1 (= cu_seqlens[s] + P_s);
 *   rows[T_cap]       the masked rows in ascending order (first n_rows valid);
 *   n_rows[1]         N_mask = sum_s C_s.
 * Device errors: OFFSETS (malformed offsets, empty prefix, T > T_cap: then
 * n_rows = 0 and the outputs are cleared), TOKEN_RANGE (an id outside [0,V);
 * the ids are still copied).
 */
OLIVE_API olive_status olive_splice_pack(const int32_t* prefix_ids, const int32_t* prefix_off,
                               const int32_t* cont_ids, const int32_t* cont_off,
                               int32_t S, int32_t V, int32_t T_cap,
                               int32_t* ids, int32_t* targets, uint8_t* loss_mask,
                               int32_t* cu_seqlens, int32_t* cut_offsets,
                               int32_t* rows, int32_t* n_rows,
                               int32_t* dev_status, void* stream);

/*
 * olive_splice_pack_masked -- olive_splice_pack for multi-turn OLIVE
 * (Section 3.2): the whole interaction (student turns, environment
 * observations, teacher turns) is kept as context, and the loss applies only
 * to the teacher's actions.  cont_loss (device, uint8, one flag per
 * continuation id, same CSR as cont_ids) marks the continuation tokens that
 * are teacher actions; row t is masked when targets[t] is such a token.
 * Outputs and device errors as in olive_splice_pack, with
 * n_rows = number of flagged continuation tokens and rows ascending.
 * workspace: olive_workspace_size(OLIVE_OP_SPLICE_MASKED, T_cap, ...) bytes.
 */
OLIVE_API olive_status olive_splice_pack_masked(const int32_t* prefix_ids,
                                                const int32_t* prefix_off, const int32_t* cont_ids,
                                                const int32_t* cont_off, const uint8_t* cont_loss,
                                                int32_t S, int32_t V, int32_t T_cap, int32_t* ids,
                                                int32_t* targets, uint8_t* loss_mask,
                                                int32_t* cu_seqlens, int32_t* cut_offsets,
                                                int32_t* rows, int32_t* n_rows, void* workspace,
                                                size_t ws_bytes, int32_t* dev_status,
                                                void* stream);

/*
 * olive_token_logprob_fwd -- Eq. (osd-ce): for every masked row r (t = rows[r],
 * r < *n_rows) with target y = targets[t],
 *   z_v    = inv_tau * <hidden[t,:], W[v,:]>          (v = 0..V-1, fp32 accumulate)
 *   lse[t] = log sum_v exp(z_v)
 *   logp[t]= z_y - lse[t]
 *   loss   = -sum_r logp[rows[r]]            (OLIVE_REDUCE_SUM, Eq. (osd-ce))
 *          = that / N_mask                   (OLIVE_REDUCE_MEAN; 0 if N_mask = 0)
 * inv_tau is the inverse sampling temperature (1.0 in Appendix A).
 *   hidden  bf16 [T, d]     W bf16 [V, d]     targets int32 [T]
 *   rows    int32 [>= *n_rows] ascending or not, each in [0,T)
 *   logp, lse  fp32 [T]: written on every row, 0 on rows not in `rows`
 *   loss    fp32 [1]
 * The [T,V] logits are never stored: vocabulary tiles are reduced on chip.
 * Device errors: TOKEN_RANGE (target outside [0,V); that row's logp is NaN),
 * OFFSETS (*n_rows > T or a row outside [0,T)), TIMEOUT.
 */
OLIVE_API olive_status olive_token_logprob_fwd(const void* hidden, const void* W,
                                     const int32_t* targets, const int32_t* rows,
                                     const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                     float inv_tau, int reduction,
                                     float* logp, float* lse, float* loss,
                                     void* workspace, size_t ws_bytes,
                                     int32_t* dev_status, void* stream);

/*
 * olive_token_topk_fwd -- per-token entropy and the K largest log-probs of
 * the student, from the same LM-head sweep as olive_token_logprob_fwd.  OPD
 * consumes the student's top-16 log-probs per token (Appendix A, Table
 * opd-config, "LogProb top-K 16"); the entropy is -sum_v p_v log p_v.  On
 * every masked row r (t = rows[r], r < *n_rows), with z = inv_tau h[t] W^T:
 *   lse[t]           = log sum_v exp(z_v)
 *   entropy[t]       = lse[t] - sum_v p_v z_v
 *   topk_logp[t, j]  = z_(j) - lse[t], the j-th largest, j = 0..K-1
 *   topk_ids[t, j]   = its vocabulary id (equal log-probs: smaller id first)
 * 1 <= K <= 16.  Rows not in `rows` get 0 (ids -1).  lse, entropy fp32 [T];
 * topk_logp fp32 [T, K]; topk_ids int32 [T, K].  The logits are not stored.
 */
OLIVE_API olive_status olive_token_topk_fwd(const void* hidden, const void* W,
                                            const int32_t* rows, const int32_t* n_rows,
                                            int32_t T, int32_t d, int32_t V, float inv_tau,
                                            int32_t K, float* lse, float* entropy,
                                            float* topk_logp, int32_t* topk_ids,
                                            void* workspace, size_t ws_bytes,
                                            int32_t* dev_status, void* stream);

/*
 * olive_topk_compare -- student/teacher agreement on each masked row's top-K
 * tokens, from two olive_token_topk_fwd outputs (student: s_ids, s_logp;
 * teacher: t_ids, t_lse) and the teacher's LM head (h_t [T, d_t], W_t
 * [V, d_t], bf16):
 *   overlap[t] = |top_K(p_s) intersect top_K(p_t)| / K  (the top-K overlap
 *                ratio tracked during OPD, Section 4.1)
 *   kl_topk[t] = sum_{j<K} p_s(v_j) (log p_s(v_j) - log p_t(v_j)) over the
 *                student's top-K ids v_j, with log p_t(v) = inv_tau
 *                h_t[t] . W_t[v] - t_lse[t]: the reverse KL of Section 1
 *                truncated to the student's K most probable tokens (the
 *                paper's "top-16 KL approximation" is not printed in full;
 *                this is the reading implemented, no renormalisation).
 *   t_logp_s[t, j] = log p_t(v_j), the teacher's log-prob at the student's
 *                j-th id (optional: NULL skips it; the input of
 *                olive_topk_kl_bwd)
 * 1 <= K <= 16; s_ids, t_ids int32 [T, K]; s_logp fp32 [T, K]; t_lse fp32
 * [T]; overlap, kl_topk fp32 [T], t_logp_s fp32 [T, K] (0 on rows not in
 * `rows`).  An id outside [0, V) gives NaN and OLIVE_ERR_TOKEN_RANGE.
 */
OLIVE_API olive_status olive_topk_compare(const void* h_t, const void* W_t, int32_t d_t,
                                          const int32_t* rows, const int32_t* n_rows, int32_t T,
                                          int32_t V, float inv_tau, int32_t K,
                                          const int32_t* s_ids, const float* s_logp,
                                          const int32_t* t_ids, const float* t_lse,
                                          float* overlap, float* kl_topk, float* t_logp_s,
                                          int32_t* dev_status, void* stream);

/*
 * olive_opd_token_stats -- everything OPD reads per token from one sweep over
 * the vocabulary with the student (h_s [T, d_s], W_s [V, d_s]) and teacher
 * (h_t [T, d_t], W_t [V, d_t]) heads, bf16 (Section 1, the per-token KL;
 * Appendix A, Table opd-config, top-16 log-probs; Section 4.1, the top-K
 * overlap ratio).  On every masked row t (z = inv_tau h W^T for each head):
 *   kl[t]               full-vocabulary KL, direction as in
 *                       olive_token_divergence
 *   s_lse[t], t_lse[t]  log sum_v exp(z_v) of each head
 *   s_entropy[t]        -sum_v p_s log p_s
 *   s_topk_logp[t, j], s_topk_ids[t, j]
 *                       the student's K most probable tokens (as
 *                       olive_token_topk_fwd: equal logits, smaller id first)
 *   t_logp_s[t, j]      log p_t at s_topk_ids[t, j]
 *   overlap[t], kl_topk[t]
 *                       as olive_topk_compare (kl_topk: the reverse KL
 *                       truncated to the student's K tokens)
 * Every output pointer may be NULL (not written) but not all of them; fp32
 * [T] or [T, K], ids int32 [T, K]; 0 (ids -1) on rows not in `rows`.
 * 1 <= K <= 16.  The outputs feed olive_topk_kl_bwd directly.  workspace:
 * olive_workspace_size(OLIVE_OP_OPD_STATS, T, d_s, d_t, V, 0, 0) bytes.
 */
OLIVE_API olive_status olive_opd_token_stats(const void* h_s, const void* W_s, int32_t d_s,
                                             const void* h_t, const void* W_t, int32_t d_t,
                                             const int32_t* rows, const int32_t* n_rows,
                                             int32_t T, int32_t V, float inv_tau, int direction,
                                             int32_t K, float* kl, float* s_lse, float* t_lse,
                                             float* s_entropy, float* s_topk_logp,
                                             int32_t* s_topk_ids, float* t_logp_s,
                                             float* overlap, float* kl_topk, void* workspace,
                                             size_t ws_bytes, int32_t* dev_status, void* stream);

/*
 * olive_topk_kl_bwd -- gradient of sum_t g_t kl_topk[t] (the truncated
 * reverse KL of olive_topk_compare) with respect to the student's hidden rows
 * and LM head, the student's top-K set S_t held fixed (it is selected, not
 * differentiated).  With l = log p_s, q = log p_t at the ids of S_t,
 * P_S = sum_{v in S_t} p_s(v) and KL_K = kl_topk[t]:
 *   G[t, u]  = g_t inv_tau p_s(u) ([u in S_t] (l_u - q_u + 1) - KL_K - P_S)
 *   d_h_s[t] = sum_u G[t, u] W_s[u]     (0 on rows not in `rows`)
 *   d_W_s[u] = sum_t G[t, u] h_s[t]
 * Inputs: h_s [T, d], W_s [V, d] bf16; s_lse fp32 [T], s_ids int32 [T, K],
 * s_logp fp32 [T, K] from olive_token_topk_fwd on the student; t_logp_s
 * fp32 [T, K] and kl_topk fp32 [T] from olive_topk_compare (or all five from
 * olive_opd_token_stats); grad_kl fp32 [T]
 * the weights g_t.  d_h_s [T, d] and d_W_s [V, d] of grad_dtype as in
 * olive_token_loss_bwd.  The softmax term is recomputed tile by tile as in
 * that backward; the K entries of S_t per row are written over it.  1 <= K
 * <= 16; an id outside [0, V) sets OLIVE_ERR_TOKEN_RANGE.  workspace:
 * olive_workspace_size(OLIVE_OP_TOPK_KL_BWD, T, d, 0, V, 1, grad_dtype) bytes.
 */
OLIVE_API olive_status olive_topk_kl_bwd(const void* h_s, const void* W_s, const int32_t* rows,
                                         const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                         float inv_tau, int32_t K, const float* s_lse,
                                         const int32_t* s_ids, const float* s_logp,
                                         const float* t_logp_s, const float* kl_topk,
                                         const float* grad_kl, void* d_h_s, void* d_W_s,
                                         int grad_dtype, void* workspace, size_t ws_bytes,
                                         int32_t* dev_status, void* stream);

/*
 * olive_token_loss_bwd -- gradients of the Eq. (osd-ce) loss through the LM
 * head (the sampled sequences are fixed, Section 3.1, so ids get none):
 *   G[r,v]    = g * inv_tau * (exp(z_v - lse[t]) - [v == y])
 *               with g = *grad_loss, divided by N_mask for OLIVE_REDUCE_MEAN
 *   d_hidden[t,:] = sum_v G[r,v] W[v,:]   on masked rows, 0 on all other rows
 *   d_W[v,:]      = sum_r G[r,v] hidden[t,:]
 * Arguments as in olive_token_logprob_fwd; lse fp32 [T] is the forward's
 * output; grad_loss fp32 [1] (device); d_hidden [T,d] and d_W [V,d] of
 * grad_dtype (OLIVE_DTYPE_BF16: fp32 accumulation, round-to-nearest-even
 * store; OLIVE_DTYPE_F32).  The logits are recomputed tile by tile and G is
 * formed and consumed on chip: groups of ceil(d / 256) CTAs each hold a
 * 128 x 256 column block of the d_hidden (then d_W) accumulator in tensor
 * memory and pass 128 x 256 bf16 tiles of G to one another through a ring of
 * fixed size in the workspace (3 ceil(d/256) tiles of 64 KB per group, tens
 * of MB in all, independent of T and V); no [rows, V] array is stored.  The
 * bf16 tile carries one rounding of G (relative 2^-9).  workspace:
 * olive_workspace_size(OLIVE_OP_LOSS_BWD, T, d, 0, V, 1, grad_dtype) bytes.
 */
OLIVE_API olive_status olive_token_loss_bwd(const void* hidden, const void* W,
                                  const int32_t* targets, const int32_t* rows,
                                  const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                  float inv_tau, int reduction,
                                  const float* lse, const float* grad_loss,
                                  void* d_hidden, void* d_W, int grad_dtype,
                                  void* workspace, size_t ws_bytes,
                                  int32_t* dev_status, void* stream);

/*
 * olive_token_loss_fwd_bwd -- olive_token_logprob_fwd and olive_token_loss_bwd
 * of one training step in a single call, for callers that know the loss
 * gradient before the forward runs (*grad_loss is read on the device, e.g. 1
 * for a loss that is the objective itself).  Outputs and arguments as in
 * those two calls: logp, lse fp32 [T], loss fp32 [1], d_hidden [T, d] and
 * d_W [V, d] of grad_dtype.  Nothing of size [rows, V] is stored: the first
 * pass walks each 128-row tile across the vocabulary, forms P = exp(z - R)
 * against a per-row reference R (the maximum of the row's first vocabulary
 * tile) in bf16 tiles that a group of CTAs shares through a fixed-size ring
 * (see olive_token_loss_bwd), and accumulates P . W and the row sums, from
 * which lse, logp and d_hidden = g inv_tau (exp(R - lse) P.W - W[y]) follow;
 * the second pass walks each 128-row vocabulary tile across the masked rows,
 * recomputes the logits and accumulates d_W = G^T hidden with G formed on
 * chip from that lse.  A row whose maximum logit exceeds R by more than 64
 * log2 units has its row tile recomputed with R = its maximum (exact, only
 * slower).  The training step executes four products of 2 N_mask d V flops
 * for the three it needs.  workspace: olive_workspace_size(
 * OLIVE_OP_LOSS_FWD_BWD, T, d, 0, V, 1, grad_dtype) bytes.
 */
OLIVE_API olive_status olive_token_loss_fwd_bwd(const void* hidden, const void* W,
                                                const int32_t* targets, const int32_t* rows,
                                                const int32_t* n_rows, int32_t T, int32_t d,
                                                int32_t V, float inv_tau, int reduction,
                                                const float* grad_loss, float* logp, float* lse,
                                                float* loss, void* d_hidden, void* d_W,
                                                int grad_dtype, void* workspace, size_t ws_bytes,
                                                int32_t* dev_status, void* stream);

/*
 * olive_token_loss_fwd_bwd_slab -- the same step, arguments and outputs as
 * olive_token_loss_fwd_bwd, computing each logit tile once instead of twice
 * by keeping it in HBM: the forward product stores e' = 2^(x - R) in bf16
 * (R = the row's maximum over its first vocabulary tile) in a slab of the
 * workspace of at most min(T, 32768, ~5.6 GB / (2 V)) rows -- at the
 * 8 x 4096-token, V = 151936 batch that slab holds every masked row, about
 * 5 GB -- a per-row pass merges the tile partials into lse and writes logp,
 * the target entry of G and the row scale lam = g inv_tau 2^(R - lse2), and
 * the d_hidden and d_W products read the slab (d_hidden = lam (e' . W) with
 * lam in the epilogue; d_W = e'^T . (lam hidden)).  Faster where HBM capacity
 * allows (three products instead of four) but the G of up to 32768 rows is
 * materialised; olive_token_loss_fwd_bwd is the on-chip form.  The paper has
 * no counterpart (an implementation alternative).  workspace:
 * olive_workspace_size(OLIVE_OP_LOSS_FWD_BWD_SLAB, T, d, 0, V, 1, grad_dtype)
 * bytes.
 */
OLIVE_API olive_status olive_token_loss_fwd_bwd_slab(const void* hidden, const void* W,
                                                     const int32_t* targets, const int32_t* rows,
                                                     const int32_t* n_rows, int32_t T, int32_t d,
                                                     int32_t V, float inv_tau, int reduction,
                                                     const float* grad_loss, float* logp,
                                                     float* lse, float* loss, void* d_hidden,
                                                     void* d_W, int grad_dtype, void* workspace,
                                                     size_t ws_bytes, int32_t* dev_status,
                                                     void* stream);

/*
 * olive_topk_kl_fwd_bwd -- olive_token_topk_fwd on the student,
 * olive_topk_compare and olive_topk_kl_bwd of one OPD training step in a
 * single call, for callers that know the weights g_t = grad_kl[t] before the
 * forward runs and have the teacher's lse (and top-K ids) from
 * olive_token_topk_fwd on the teacher.  Each student logit tile is computed
 * once: the forward product stores e = exp(z - tile max) in bf16 in the G
 * slab of the workspace; per masked row the C = min(K + 8, 24) largest
 * entries of e (read only in the 128-column blocks whose maximum can hold
 * one) are the candidates whose logits are recomputed exactly (fp32 dot
 * products), S_t is the K largest of those, and the teacher's log-probs at
 * S_t come from h_t . W_t[v] - t_lse[t]; a bandwidth-bound pass writes G
 * (the formula of olive_topk_kl_bwd) and the dH and dW products follow.
 * Inputs: h_s [T, d_s], W_s [V, d_s], h_t [T, d_t], W_t [V, d_t] bf16 (d_s,
 * d_t multiples of 8); t_lse fp32 [T]; t_ids int32 [T, K] (nullable: no
 * overlap); grad_kl fp32 [T].  Outputs: s_lse fp32 [T]; s_ids int32 [T, K] and
 * s_logp fp32 [T, K] (S_t by decreasing log-prob, ties by id); t_logp_s fp32
 * [T, K]; kl_topk fp32 [T]; overlap fp32 [T] (written when t_ids is given;
 * may be NULL otherwise); d_h_s [T, d_s] and d_W_s [V, d_s] of grad_dtype.
 * Rows not in `rows` get 0 (ids -1).  S_t differs from the exact top-K only
 * where C - K or more logits lie within bf16 resolution (~2^-8 relative of
 * exp) below the K-th largest.  1 <= K <= min(16, V).  workspace:
 * olive_workspace_size(OLIVE_OP_TOPK_KL_FWD_BWD, T, d_s, 0, V, 1, grad_dtype)
 * bytes.
 */
OLIVE_API olive_status olive_topk_kl_fwd_bwd(const void* h_s, const void* W_s, int32_t d_s,
                                             const void* h_t, const void* W_t, int32_t d_t,
                                             const int32_t* rows, const int32_t* n_rows,
                                             int32_t T, int32_t V, float inv_tau, int32_t K,
                                             const float* t_lse, const int32_t* t_ids,
                                             const float* grad_kl, float* s_lse, int32_t* s_ids,
                                             float* s_logp, float* t_logp_s, float* kl_topk,
                                             float* overlap, void* d_h_s, void* d_W_s,
                                             int grad_dtype, void* workspace, size_t ws_bytes,
                                             int32_t* dev_status, void* stream);

/*
 * olive_scale -- y[i] = x[i] * (*scale) for i < n, x and y of `dtype`
 * (OLIVE_DTYPE_BF16: fp32 product, round to nearest even; OLIVE_DTYPE_F32),
 * x == y allowed, both 16-byte aligned; scale fp32 [1] on the device.  The
 * paper has no counterpart: this lets a caller that learns the loss gradient
 * g only after olive_token_loss_fwd_bwd (an autograd backward) run that call
 * with *grad_loss = 1 and scale d_hidden and d_W by g afterwards.
 */
OLIVE_API olive_status olive_scale(const void* x, void* y, size_t n, int dtype,
                                   const float* scale, void* stream);

/*
 * olive_token_divergence -- OPD's per-token divergence between the student
 * pi_theta and the teacher pi_T over the full vocabulary (Section 1; the
 * paper's top-16 approximation is not used): on masked row t,
 *   p_s = softmax(inv_tau * h_s[t] W_s^T)   (width d_s)
 *   p_t = softmax(inv_tau * h_t[t] W_t^T)   (width d_t, same V)
 *   OLIVE_KL_REVERSE: kl[t] = sum_v p_s (log p_s - log p_t)
 *   OLIVE_KL_FORWARD: kl[t] = sum_v p_t (log p_t - log p_s)
 * kl fp32 [T] (0 on rows not in `rows`).  If grad_kl (fp32 [T], weights g_t)
 * and d_h_s ([T, d_s] of grad_dtype) are both non-NULL, also writes the
 * gradient of sum_t g_t kl[t] with respect to h_s:
 *   reverse: d_h_s[t] = g_t inv_tau sum_v p_s (log p_s - log p_t - kl[t]) W_s[v]
 *   forward: d_h_s[t] = g_t inv_tau sum_v (p_s - p_t) W_s[v]
 * (0 on rows not in `rows`; the teacher receives no gradient).
 * With the gradient the call makes two sweeps over the vocabulary: the first
 * gives kl[t] and both log-sum-exps, the second recomputes both heads' logits
 * tile by tile and contracts G against W_s on chip (G is never written to
 * device memory); its counters and exchange ring are in the workspace.
 */
OLIVE_API olive_status olive_token_divergence(const void* h_s, const void* W_s, int32_t d_s,
                                    const void* h_t, const void* W_t, int32_t d_t,
                                    const int32_t* rows, const int32_t* n_rows,
                                    int32_t T, int32_t V, float inv_tau, int direction,
                                    float* kl, const float* grad_kl, void* d_h_s,
                                    int grad_dtype, void* workspace, size_t ws_bytes,
                                    int32_t* dev_status, void* stream);

/*
 * olive_token_logprob_fwd_noalloc -- the same computation, arguments and
 * outputs as olive_token_logprob_fwd, for callers that cannot provide a
 * workspace: code hosted by another framework whose allocator owns all
 * device memory and lends none, or code that must not call cudaMalloc (it
 * can synchronise the device).  The paper has no counterpart; this is a
 * deployment convenience of this library.
 *
 * Scratch comes from one array of OLIVE_NOALLOC_SCRATCH_BYTES compiled into
 * the library, which every GPU that loads the library keeps until the process
 * exits.  Limit: the call is rejected with OLIVE_ERR_SHAPE, before any
 * launch, when olive_workspace_size(OLIVE_OP_LOGPROB_FWD, T, d, 0, V, 0, 0)
 * exceeds that size (for example T = 2048 rows at d = 4096 fit, T = 4096 rows
 * at d = 4096 do not).  The first call on each device looks up the array's
 * device address; make that first call before any stream capture.  Every
 * call shares the array: calls whose work may overlap on the GPU (other
 * streams, other host threads) race on it, so the caller must serialise
 * them.  The call allocates no device or host memory.
 */
#define OLIVE_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)
OLIVE_API olive_status olive_token_logprob_fwd_noalloc(const void* hidden, const void* W,
                                                       const int32_t* targets, const int32_t* rows,
                                                       const int32_t* n_rows, int32_t T, int32_t d,
                                                       int32_t V, float inv_tau, int reduction,
                                                       float* logp, float* lse, float* loss,
                                                       int32_t* dev_status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* OLIVE_H_ */
