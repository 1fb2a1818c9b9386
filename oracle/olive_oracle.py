"""Plain fp64 CPU oracle for the OLIVE per-token scoring path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, calls or
executes this module: only the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` do.  It shares no
code with the CUDA library (no kernels, headers, helpers or constants): it is
written straight from the paper's definitions so that a reader can check it
against the paper by eye.

What it computes (paper: "OLIVE: Learning from Teacher Continuations at
Student States", Section 3.1 "Main Algorithm", Eq. (osd-ce); OPD baseline,
Section 1; temperature, Appendix A, Table opd-config):

* ``splice_pack``      -- the spliced sequence (x, y_{1:k}, y~_{1:l}) packed
                          back to back, with the continuation-only loss mask
                          (Section 3.1: prompt and student prefix stay in the
                          context but are masked out of the loss).
* ``token_logprob``    -- log pi_theta(y~_j | x, y_{1:k}, y~_{<j}) for every
                          masked row and the loss of Eq. (osd-ce).
* ``token_loss_bwd``   -- d loss / d hidden and d loss / d W of Eq. (osd-ce)
                          through the LM head (sequences held fixed,
                          Section 3.1, so no gradient flows through the ids).
* ``token_topk``       -- per-token entropy and the student's K largest
                          log-probs (Appendix A: OPD reads the top-16).
* ``token_topk_compare`` -- student/teacher top-K overlap and the top-K
                          truncation of the reverse KL.
* ``token_topk_kl_bwd`` -- gradients of the top-K truncated KL (top-K set
                          held fixed).
* ``token_divergence`` -- OPD's per-token reverse KL between student and
                          teacher over the full vocabulary (Section 1), the
                          forward direction as an option, and the gradient of
                          sum_t g_t KL_t with respect to the student hidden.

Readings where the paper is silent:
  - causal shift: row t of ``hidden`` predicts packed token t+1 of the same
    sequence, so y~_1 is scored from the last prefix row and the last row of
    every sequence has no target;
  - the prefix is prompt || student prefix and must hold at least one id;
  - reduction "sum" is Eq. (osd-ce) literally; "mean" divides by N_mask; an
    empty mask gives loss 0 and zero gradients;
  - logits are z = inv_tau * h . W_v with inv_tau = 1 by default
    (training temperature 1.0, Appendix A);
  - the KL is taken over the full vocabulary (the "top-16 approximation" of
    Section 1 is not defined in the paper).

Parity pins for every function live in ``tests/test_oracle_pins.py``; none of
the functions here is "parity unpinned".

All floating point work is float64.  Inputs may be float32 or float64 arrays
(bf16 values widen exactly to both); ``bf16_bits_to_f64`` widens raw bf16 bit
patterns exactly.
"""

from __future__ import annotations

import numpy as np

REDUCTIONS = ("sum", "mean")
DIRECTIONS = ("reverse", "forward")

# Rows of logits are formed this many at a time.  Rows are independent in
# every quantity below, so the grouping only bounds memory; it changes no sum.
_ROW_CHUNK = 256
# Vocabulary rows of W are widened to float64 this many at a time (memory
# bound only: each logit is the same dot product whichever chunk it falls in).
_VOCAB_CHUNK = 16384


class OracleError(ValueError):
    """Raised for inputs the paper's problem statement rules out."""


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Widen raw bf16 bit patterns (uint16) exactly to float64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# Splice / pack  (Section 3.1, Eq. (osd-ce) and the masking sentence after it)
# --------------------------------------------------------------------------
def splice_pack(prefix_ids, prefix_off, cont_ids, cont_off, V: int, cont_loss=None) -> dict:
    """Pack S spliced sequences prefix_s || continuation_s back to back.

    prefix_s is x || y_{1:k} (prompt and student prefix), continuation_s is
    the teacher continuation y~_{1:l} re-tokenised in the student vocabulary
    (Section 3.1).  Both come in CSR form: sequence s owns
    ``prefix_ids[prefix_off[s]:prefix_off[s+1]]`` and likewise for ``cont``.

    Returns a dict of int64 numpy arrays:
      ids[T]         packed token ids,
      targets[T]     ids[t+1] when t+1 is in the same sequence, else -1,
      loss_mask[T]   1 where targets[t] is a continuation token y~_j
                     (those rows carry the terms of Eq. (osd-ce)), else 0,
      cu_seqlens[S+1], cut_offsets[S] (packed index of y~_1),
      rows[N_mask]   the masked t in ascending order, n_rows = N_mask,
      token_range_ok whether every id lies in [0, V).
    Multi-turn OLIVE (Section 3.2) keeps the whole interaction as context but
    applies the loss only to the teacher's actions: ``cont_loss`` (optional,
    one flag per continuation id) marks the continuation tokens that are
    teacher actions; a row is then masked only when its target is such a
    token (environment observations inside the continuation stay unmasked).
    Raises OracleError for offsets that do not describe S sequences with a
    non-empty prefix.
    """
    prefix_ids = np.asarray(prefix_ids, dtype=np.int64)
    cont_ids = np.asarray(cont_ids, dtype=np.int64)
    prefix_off = np.asarray(prefix_off, dtype=np.int64)
    cont_off = np.asarray(cont_off, dtype=np.int64)
    S = len(prefix_off) - 1
    if S < 0 or len(cont_off) != S + 1:
        raise OracleError("offset arrays must both have S+1 entries")
    if prefix_off[0] != 0 or cont_off[0] != 0:
        raise OracleError("offsets must start at 0")
    if prefix_off[-1] != len(prefix_ids) or cont_off[-1] != len(cont_ids):
        raise OracleError("last offset must equal the number of ids")
    if cont_loss is not None:
        cont_loss = np.asarray(cont_loss).astype(bool)
        if len(cont_loss) != len(cont_ids):
            raise OracleError("cont_loss needs one flag per continuation id")

    ids, targets, mask, cu, cut = [], [], [], [0], []
    for s in range(S):
        pre = prefix_ids[prefix_off[s]:prefix_off[s + 1]]
        con = cont_ids[cont_off[s]:cont_off[s + 1]]
        P = prefix_off[s + 1] - prefix_off[s]
        C = cont_off[s + 1] - cont_off[s]
        if P < 1 or C < 0:
            raise OracleError("every sequence needs a prefix of >= 1 id and C >= 0")
        seq = list(pre) + list(con)
        L = P + C
        cut.append(cu[-1] + P)
        for i in range(L):
            ids.append(seq[i])
            if i + 1 < L:
                targets.append(seq[i + 1])
                # the target of row i is seq[i+1]; it is a teacher token
                # y~_j exactly when i+1 >= P (and, with cont_loss, a
                # teacher action rather than an observation)
                in_loss = i + 1 >= P
                if in_loss and cont_loss is not None:
                    in_loss = bool(cont_loss[cont_off[s] + (i + 1 - P)])
                mask.append(1 if in_loss else 0)
            else:
                targets.append(-1)
                mask.append(0)
        cu.append(cu[-1] + L)

    ids = np.array(ids, dtype=np.int64)
    mask = np.array(mask, dtype=np.int64)
    rows = np.nonzero(mask)[0].astype(np.int64)
    all_ids = np.concatenate([prefix_ids, cont_ids])
    return {
        "ids": ids,
        "targets": np.array(targets, dtype=np.int64),
        "loss_mask": mask,
        "cu_seqlens": np.array(cu, dtype=np.int64),
        "cut_offsets": np.array(cut, dtype=np.int64),
        "rows": rows,
        "n_rows": int(len(rows)),
        "token_range_ok": bool(np.all((all_ids >= 0) & (all_ids < V))),
    }


# --------------------------------------------------------------------------
# Logits and log-softmax of one group of rows
# --------------------------------------------------------------------------
def _as_f64_rows(hidden, rows) -> np.ndarray:
    return np.asarray(hidden)[np.asarray(rows, dtype=np.int64)].astype(np.float64)


def logits(h_rows: np.ndarray, W, inv_tau: float) -> np.ndarray:
    """z[r, v] = inv_tau * sum_k h[r, k] W[v, k]  (the student's LM head)."""
    W = np.asarray(W)
    V = W.shape[0]
    z = np.empty((h_rows.shape[0], V), dtype=np.float64)
    for v0 in range(0, V, _VOCAB_CHUNK):
        v1 = min(V, v0 + _VOCAB_CHUNK)
        z[:, v0:v1] = h_rows @ W[v0:v1].astype(np.float64).T
    z *= float(inv_tau)
    return z


def log_softmax_rows(z: np.ndarray):
    """log p = z - lse with lse = m + ln sum_v exp(z_v - m), m = max_v z_v."""
    m = z.max(axis=1)
    lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    return z - lse[:, None], lse


def _check_reduction(reduction):
    if reduction not in REDUCTIONS:
        raise OracleError(f"reduction must be one of {REDUCTIONS}")


# --------------------------------------------------------------------------
# Eq. (osd-ce): per-token log-probabilities and the masked loss
# --------------------------------------------------------------------------
def token_logprob(hidden, W, targets, rows, inv_tau: float = 1.0,
                  reduction: str = "sum"):
    """Per-token log pi_theta(y~_j | context) on the masked rows.

    hidden [T, d], W [V, d], targets [T] (target id of every row), rows the
    masked rows.  Returns (logp[T], lse[T], loss): logp = z_y - lse on the
    masked rows and 0 elsewhere, lse likewise, and
    loss = -sum_rows logp  ("sum", Eq. (osd-ce))  or that / N_mask ("mean").
    """
    _check_reduction(reduction)
    T = np.asarray(hidden).shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    targets = np.asarray(targets, dtype=np.int64)
    logp = np.zeros(T, dtype=np.float64)
    lse = np.zeros(T, dtype=np.float64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        z = logits(_as_f64_rows(hidden, rr), W, inv_tau)
        lp, l = log_softmax_rows(z)
        y = targets[rr]
        logp[rr] = lp[np.arange(len(rr)), y]
        lse[rr] = l
    loss = -logp[rows].sum()
    if reduction == "mean":
        loss = loss / len(rows) if len(rows) else 0.0
    return logp, lse, float(loss)


def token_loss_bwd(hidden, W, targets, rows, inv_tau: float = 1.0,
                   reduction: str = "sum", grad_loss: float = 1.0):
    """Gradients of the Eq. (osd-ce) loss through the LM head.

    With p = softmax(z) per masked row and y its target,
      G[r, v] = g * inv_tau * (p[r, v] - [v == y_r])   (g = grad_loss, / N_mask for "mean")
      dH[t]   = sum_v G[t, v] W[v]       (zero on unmasked rows)
      dW[v]   = sum_t G[t, v] h[t]
    Returns (dH [T, d], dW [V, d]) in float64.
    """
    _check_reduction(reduction)
    hidden = np.asarray(hidden)
    W = np.asarray(W)
    T, d = hidden.shape
    V = W.shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    targets = np.asarray(targets, dtype=np.int64)
    g = float(grad_loss)
    if reduction == "mean" and len(rows):
        g = g / len(rows)
    dH = np.zeros((T, d), dtype=np.float64)
    dW = np.zeros((V, d), dtype=np.float64)
    W64 = W.astype(np.float64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        h = _as_f64_rows(hidden, rr)
        z = logits(h, W, inv_tau)
        lp, _ = log_softmax_rows(z)
        G = np.exp(lp)
        G[np.arange(len(rr)), targets[rr]] -= 1.0
        G *= g * float(inv_tau)
        dH[rr] = G @ W64
        dW += G.T @ h
    return dH, dW


def token_loss_bwd_rows(hidden, W, targets, rows, inv_tau: float = 1.0,
                        reduction: str = "sum", grad_loss: float = 1.0,
                        n_mask: int | None = None):
    """dH for a subset ``rows`` of the masked rows only (sampled checks).

    ``n_mask`` is the full N_mask, needed for the "mean" scale.  Returns
    dH_rows [len(rows), d] with the same definition as ``token_loss_bwd``.
    """
    _check_reduction(reduction)
    rows = np.asarray(rows, dtype=np.int64)
    targets = np.asarray(targets, dtype=np.int64)
    g = float(grad_loss)
    if reduction == "mean":
        n = len(rows) if n_mask is None else n_mask
        g = g / n if n else g
    W = np.asarray(W)
    out = np.zeros((len(rows), W.shape[1]), dtype=np.float64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        z = logits(_as_f64_rows(hidden, rr), W, inv_tau)
        lp, _ = log_softmax_rows(z)
        G = np.exp(lp)
        G[np.arange(len(rr)), targets[rr]] -= 1.0
        G *= g * float(inv_tau)
        for v0 in range(0, W.shape[0], _VOCAB_CHUNK):
            v1 = min(W.shape[0], v0 + _VOCAB_CHUNK)
            out[r0:r0 + len(rr)] += G[:, v0:v1] @ W[v0:v1].astype(np.float64)
    return out


def token_loss_bwd_vocab(hidden, W, targets, rows, vocab, inv_tau: float = 1.0,
                         reduction: str = "sum", grad_loss: float = 1.0):
    """dW for a subset ``vocab`` of vocabulary rows only (sampled checks).

    Same definition as ``token_loss_bwd``: every masked row's full softmax is
    formed (its lse needs all V logits), then
    dW[v] = sum_t g inv_tau (p[t, v] - [v == y_t]) h[t] for v in ``vocab``.
    Returns dW_vocab [len(vocab), d].
    """
    _check_reduction(reduction)
    rows = np.asarray(rows, dtype=np.int64)
    vocab = np.asarray(vocab, dtype=np.int64)
    targets = np.asarray(targets, dtype=np.int64)
    g = float(grad_loss)
    if reduction == "mean" and len(rows):
        g = g / len(rows)
    out = np.zeros((len(vocab), np.asarray(W).shape[1]), dtype=np.float64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        h = _as_f64_rows(hidden, rr)
        lp, _ = log_softmax_rows(logits(h, W, inv_tau))
        G = np.exp(lp[:, vocab])
        G -= (targets[rr][:, None] == vocab[None, :])
        G *= g * float(inv_tau)
        out += G.T @ h
    return out


# --------------------------------------------------------------------------
# Per-token entropy and top-K log-probs of the student (Appendix A, Table
# opd-config: OPD consumes the student's top-16 log-probs per token)
# --------------------------------------------------------------------------
def token_topk(hidden, W, rows, K: int, inv_tau: float = 1.0):
    """Entropy and the K largest log-probabilities of pi_theta per masked row.

    For each row in ``rows``: lse, H = -sum_v p_v log p_v, and the K largest
    log p_v in descending order with their vocabulary ids; equal log-probs are
    ordered by ascending id.  Returns (lse [T], H [T], topk_logp [T, K],
    topk_ids [T, K]) with 0 / -1 off ``rows``.
    """
    hidden = np.asarray(hidden)
    T = hidden.shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    lse = np.zeros(T, dtype=np.float64)
    H = np.zeros(T, dtype=np.float64)
    tv = np.zeros((T, K), dtype=np.float64)
    ti = np.full((T, K), -1, dtype=np.int64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        lp, l = log_softmax_rows(logits(_as_f64_rows(hidden, rr), W, inv_tau))
        lse[rr] = l
        H[rr] = -(np.exp(lp) * lp).sum(axis=1)
        ids = np.arange(lp.shape[1])
        for k, r in enumerate(rr):
            order = np.lexsort((ids, -lp[k]))[:K]
            tv[r] = lp[k, order]
            ti[r] = order
    return lse, H, tv, ti


def token_topk_compare(h_s, W_s, h_t, W_t, rows, K: int, inv_tau: float = 1.0):
    """Top-K agreement between student and teacher per masked row.

    overlap[t]  = |top_K(p_s) intersect top_K(p_t)| / K   (the student/teacher
                  top-K overlap ratio tracked during OPD, Section 4.1)
    kl_topk[t]  = sum over the student's K most probable tokens v of
                  p_s(v) (log p_s(v) - log p_t(v)), both log-probs over the
                  full vocabulary: the reverse KL of Section 1 truncated to
                  the top-K terms (the paper's "top-16 KL approximation",
                  whose exact form it does not print; this is the reading
                  used here).
    Also returns the gaps between the K-th and (K+1)-th largest log-probs of
    the student and of the teacher (0 / inf off ``rows``), which tell a test
    where top-K membership is decided by more than rounding.
    """
    T = np.asarray(h_s).shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    overlap = np.zeros(T)
    kl = np.zeros(T)
    gap_s = np.full(T, np.inf)
    gap_t = np.full(T, np.inf)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        lps, _ = log_softmax_rows(logits(_as_f64_rows(h_s, rr), W_s, inv_tau))
        lpt, _ = log_softmax_rows(logits(_as_f64_rows(h_t, rr), W_t, inv_tau))
        ids = np.arange(lps.shape[1])
        for k, r in enumerate(rr):
            os_ = np.lexsort((ids, -lps[k]))
            ot_ = np.lexsort((ids, -lpt[k]))
            S, Tk = os_[:K], ot_[:K]
            overlap[r] = len(set(S.tolist()) & set(Tk.tolist())) / K
            kl[r] = float((np.exp(lps[k, S]) * (lps[k, S] - lpt[k, S])).sum())
            if len(ids) > K:
                gap_s[r] = lps[k, os_[K - 1]] - lps[k, os_[K]]
                gap_t[r] = lpt[k, ot_[K - 1]] - lpt[k, ot_[K]]
    return overlap, kl, gap_s, gap_t


def token_topk_kl_bwd(h_s, W_s, h_t, W_t, rows, K: int, inv_tau: float = 1.0, grad=None,
                      with_dW: bool = True):
    """Gradient of sum_t g_t kl_topk[t] (see ``token_topk_compare``) with
    respect to the student's hidden rows and LM head, the top-K set S_t of
    the student held fixed (it is selected, not differentiated):
      with l = log p_s, q = log p_t, P_S = sum_{v in S} p_s(v) and
      KL_K = sum_{v in S} p_s(v) (l_v - q_v),
      dz_u = p_s(u) ([u in S] (l_u - q_u + 1) - KL_K - P_S)
      G[t, u] = g_t inv_tau dz_u,  dH_s[t] = G[t] W_s,  dW_s = G^T h_s.
    Returns (dH_s [T, d_s], dW_s [V, d_s] or None without ``with_dW``).
    """
    h_s = np.asarray(h_s)
    W_s = np.asarray(W_s)
    T = h_s.shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    g = np.ones(T) if grad is None else np.asarray(grad, dtype=np.float64)
    dH = np.zeros((T, h_s.shape[1]))
    dW = np.zeros(W_s.shape) if with_dW else None
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        hs = _as_f64_rows(h_s, rr)
        lps, _ = log_softmax_rows(logits(hs, W_s, inv_tau))
        lpt, _ = log_softmax_rows(logits(_as_f64_rows(h_t, rr), W_t, inv_tau))
        ps = np.exp(lps)
        ids = np.arange(lps.shape[1])
        G = np.zeros_like(lps)
        for k in range(len(rr)):
            S = np.lexsort((ids, -lps[k]))[:K]
            kl = float((ps[k, S] * (lps[k, S] - lpt[k, S])).sum())
            P_S = float(ps[k, S].sum())
            G[k] = -ps[k] * (kl + P_S)
            G[k, S] += ps[k, S] * (lps[k, S] - lpt[k, S] + 1.0)
        G *= (g[rr] * float(inv_tau))[:, None]
        for v0 in range(0, W_s.shape[0], _VOCAB_CHUNK):
            v1 = min(W_s.shape[0], v0 + _VOCAB_CHUNK)
            dH[rr] += G[:, v0:v1] @ W_s[v0:v1].astype(np.float64)
        if with_dW:
            dW += G.T @ hs
    return dH, dW


# --------------------------------------------------------------------------
# OPD per-token divergence over the full vocabulary (Section 1)
# --------------------------------------------------------------------------
def token_divergence(h_s, W_s, h_t, W_t, rows, inv_tau: float = 1.0,
                     direction: str = "reverse", grad_kl=None):
    """Per-token KL between the student and teacher next-token distributions.

    p_s = softmax(inv_tau * h_s W_s^T), p_t = softmax(inv_tau * h_t W_t^T) on
    each row in ``rows`` (student width d_s, teacher width d_t, shared V).
      reverse: KL_t = sum_v p_s (log p_s - log p_t)     (OPD, Section 1)
      forward: KL_t = sum_v p_t (log p_t - log p_s)
    If ``grad_kl`` ([T] weights g_t) is given, also returns the gradient of
    sum_t g_t KL_t with respect to h_s:
      reverse: dz_s = p_s * (log p_s - log p_t - KL_t)
      forward: dz_s = p_s - p_t
      dH_s[t] = g_t * inv_tau * dz_s W_s   (teacher side gets no gradient).
    Returns (kl [T] (0 off ``rows``), dH_s [T, d_s] or None).
    """
    if direction not in DIRECTIONS:
        raise OracleError(f"direction must be one of {DIRECTIONS}")
    h_s = np.asarray(h_s)
    T = h_s.shape[0]
    rows = np.asarray(rows, dtype=np.int64)
    kl = np.zeros(T, dtype=np.float64)
    dHs = None
    if grad_kl is not None:
        grad_kl = np.asarray(grad_kl, dtype=np.float64)
        dHs = np.zeros((T, h_s.shape[1]), dtype=np.float64)
        Ws64 = np.asarray(W_s).astype(np.float64)
    for r0 in range(0, len(rows), _ROW_CHUNK):
        rr = rows[r0:r0 + _ROW_CHUNK]
        lps, _ = log_softmax_rows(logits(_as_f64_rows(h_s, rr), W_s, inv_tau))
        lpt, _ = log_softmax_rows(logits(_as_f64_rows(h_t, rr), W_t, inv_tau))
        ps, pt = np.exp(lps), np.exp(lpt)
        if direction == "reverse":
            k = (ps * (lps - lpt)).sum(axis=1)
        else:
            k = (pt * (lpt - lps)).sum(axis=1)
        kl[rr] = k
        if grad_kl is not None:
            if direction == "reverse":
                dz = ps * (lps - lpt - k[:, None])
            else:
                dz = ps - pt
            dz *= (grad_kl[rr] * float(inv_tau))[:, None]
            dHs[rr] = dz @ Ws64
    return kl, dHs
