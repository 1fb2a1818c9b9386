"""Pins for the fp64 oracle: each check ties it to something other than itself.

Closed forms and special cases (uniform logits, a dominant logit, two classes,
identical teacher/student), library routines that compute the same quantity
by another route (scipy's log_softmax, torch's cross_entropy / kl_div and
autograd in float64), finite differences, invariants (gradient rows summing
to zero, shift and permutation invariance) and a hand-worked splice/pack
fixture.  All run on the CPU.
"""

import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle
from paper_2609_36246_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _case(seed, T=12, d=16, V=37, std_h=1.0, std_w=0.3):
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((T, d))
    W = rng.standard_normal((V, d)) * std_w
    targets = rng.integers(0, V, size=T)
    rows = np.sort(rng.choice(T, size=max(1, T // 2), replace=False))
    return h * std_h, W, targets, rows


# --------------------------------------------------------------------------
# splice / pack
# --------------------------------------------------------------------------
def test_splice_pack_golden():
    with open(os.path.join(GOLDEN, "splice_pack_small.json")) as f:
        g = json.load(f)
    out = oracle.splice_pack(g["prefix_ids"], g["prefix_off"], g["cont_ids"], g["cont_off"], g["V"])
    for k, v in g["expect"].items():
        got = out[k]
        if isinstance(v, list):
            assert list(map(int, got)) == v, k
        else:
            assert int(got) == v, k
    assert out["token_range_ok"]


@pytest.mark.parametrize("seed", range(5))
def test_splice_pack_invariants(seed):
    rng = np.random.default_rng(seed)
    S = int(rng.integers(1, 9))
    P = rng.integers(1, 30, size=S)
    C = rng.integers(0, 30, size=S)
    b = synth.batch_from_lengths(rng, P, C, 1000)
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)
    assert o["n_rows"] == int(C.sum()) == int(o["loss_mask"].sum())
    assert len(o["ids"]) == int(P.sum() + C.sum())
    # the targets of the masked rows are exactly the continuation ids, in order
    assert np.array_equal(o["targets"][o["rows"]], b.cont_ids)
    assert np.all(np.diff(o["rows"]) > 0)
    # each sequence: prefix then continuation, cut at cu + P
    for s in range(S):
        cu = o["cu_seqlens"][s]
        assert o["cut_offsets"][s] == cu + P[s]
        seq = o["ids"][cu:o["cu_seqlens"][s + 1]]
        assert np.array_equal(seq[:P[s]], b.prefix_ids[b.prefix_off[s]:b.prefix_off[s + 1]])
        assert np.array_equal(seq[P[s]:], b.cont_ids[b.cont_off[s]:b.cont_off[s + 1]])
        assert o["targets"][o["cu_seqlens"][s + 1] - 1] == -1


def test_splice_pack_turns_golden():
    with open(os.path.join(GOLDEN, "splice_pack_turns.json")) as f:
        g = json.load(f)
    out = oracle.splice_pack(g["prefix_ids"], g["prefix_off"], g["cont_ids"], g["cont_off"], g["V"],
                             cont_loss=g["cont_loss"])
    for k, v in g["expect"].items():
        got = out[k]
        assert (list(map(int, got)) if isinstance(v, list) else int(got)) == v, k


@pytest.mark.parametrize("seed", range(3))
def test_splice_pack_turn_flags_invariants(seed):
    rng = np.random.default_rng(50 + seed)
    S = int(rng.integers(1, 7))
    b = synth.batch_from_lengths(rng, rng.integers(1, 20, size=S), rng.integers(0, 20, size=S), 500)
    flags = rng.integers(0, 2, size=len(b.cont_ids))
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V, cont_loss=flags)
    plain = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)
    assert o["n_rows"] == int(flags.sum())
    # the masked rows are a subset of the plain ones whose targets are flagged actions
    assert set(o["rows"]).issubset(set(plain["rows"]))
    assert np.array_equal(o["targets"][o["rows"]], b.cont_ids[flags.astype(bool)])
    ones = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V,
                              cont_loss=np.ones(len(b.cont_ids)))
    assert np.array_equal(ones["rows"], plain["rows"])


def test_splice_pack_rejects_empty_prefix_and_flags_range():
    with pytest.raises(oracle.OracleError):
        oracle.splice_pack([], [0, 0], [1, 2], [0, 2], 10)
    o = oracle.splice_pack([3, 12], [0, 2], [1], [0, 1], 10)
    assert not o["token_range_ok"]


# --------------------------------------------------------------------------
# forward: closed forms and library routines
# --------------------------------------------------------------------------
@pytest.mark.parametrize("V", [4096, 151936])
def test_uniform_logits_give_minus_log_V(V):
    T, d = 6, 8
    h = np.random.default_rng(0).standard_normal((T, d))
    W = np.zeros((V, d), dtype=np.float32)
    targets = np.arange(T) * 7 % V
    rows = np.arange(T)
    logp, lse, loss = oracle.token_logprob(h, W, targets, rows)
    assert np.allclose(logp, -math.log(V), rtol=0, atol=1e-12)
    assert np.allclose(lse, math.log(V), rtol=0, atol=1e-12)
    assert loss == pytest.approx(T * math.log(V), rel=1e-13)
    # hidden = 0 gives the same
    logp0, _, _ = oracle.token_logprob(np.zeros((T, d)), np.ones((V, d)), targets, rows)
    assert np.allclose(logp0, -math.log(V), atol=1e-12)


def test_dominant_logit():
    V, d = 4096, 4
    W = np.zeros((V, d))
    y = 1234
    W[y, 0] = 30.0
    h = np.zeros((1, d))
    h[0, 0] = 1.0
    logp, _, _ = oracle.token_logprob(h, W, [y], [0])
    expect = -math.log1p((V - 1) * math.exp(-30.0))
    # z_y - lse cancels at |lse| ~ 30: the result is exact to a few ulp(30)
    assert logp[0] == pytest.approx(expect, rel=0, abs=2e-14)
    assert -1.6e-9 < logp[0] < 0


def test_two_class_is_log_sigmoid():
    rng = np.random.default_rng(3)
    T, d = 10, 5
    h = rng.standard_normal((T, d))
    W = rng.standard_normal((2, d))
    targets = rng.integers(0, 2, size=T)
    logp, _, _ = oracle.token_logprob(h, W, targets, np.arange(T), inv_tau=0.7)
    for t in range(T):
        zy = 0.7 * float(np.dot(h[t], W[targets[t]]))
        zo = 0.7 * float(np.dot(h[t], W[1 - targets[t]]))
        # log sigmoid(a) = -log(1 + e^{-a})
        assert logp[t] == pytest.approx(-math.log1p(math.exp(-(zy - zo))), rel=1e-12)


def test_logprob_matches_scipy_log_softmax():
    h, W, targets, rows = _case(4, T=20, d=24, V=101)
    logp, lse, loss = oracle.token_logprob(h, W, targets, rows, inv_tau=1.3)
    z = 1.3 * np.einsum("td,vd->tv", h, W)
    ref = scipy.special.log_softmax(z, axis=1)
    assert np.allclose(logp[rows], ref[rows, targets[rows]], rtol=1e-12, atol=1e-12)
    assert np.allclose(lse[rows], scipy.special.logsumexp(z, axis=1)[rows], rtol=1e-12)
    off = np.setdiff1d(np.arange(len(h)), rows)
    assert np.all(logp[off] == 0) and np.all(lse[off] == 0)
    assert loss == pytest.approx(-ref[rows, targets[rows]].sum(), rel=1e-12)


@pytest.mark.parametrize("reduction", ["sum", "mean"])
def test_loss_matches_torch_cross_entropy(reduction):
    h, W, targets, rows = _case(5, T=16, d=12, V=53)
    _, _, loss = oracle.token_logprob(h, W, targets, rows, inv_tau=0.8, reduction=reduction)
    z = 0.8 * (torch.from_numpy(h[rows]) @ torch.from_numpy(W).T)
    ref = F.cross_entropy(z, torch.from_numpy(targets[rows]), reduction=reduction)
    assert loss == pytest.approx(ref.item(), rel=1e-12)


def test_logprob_nonpositive_and_loss_is_minus_sum():
    h, W, targets, rows = _case(6, T=30, d=8, V=40, std_h=3.0, std_w=2.0)
    logp, _, loss = oracle.token_logprob(h, W, targets, rows)
    assert np.all(logp <= 0)
    assert loss == pytest.approx(-logp.sum(), rel=1e-13)


def test_shift_and_permutation_invariance():
    h, W, targets, rows = _case(7, T=14, d=10, V=64)
    base, _, _ = oracle.token_logprob(h, W, targets, rows)
    # a constant logit offset (h[:, -1] = 1, W[:, -1] = c) changes nothing
    h2, W2 = h.copy(), W.copy()
    h2[:, -1] = 1.0
    W2[:, -1] = 2.5
    h3, W3 = h.copy(), W.copy()
    h3[:, -1] = 0.0
    a, _, _ = oracle.token_logprob(h2, W2, targets, rows)
    b, _, _ = oracle.token_logprob(h3, W3, targets, rows)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)
    # permuting the vocabulary and remapping targets changes nothing
    perm = np.random.default_rng(1).permutation(W.shape[0])
    inv = np.argsort(perm)
    c, _, _ = oracle.token_logprob(h, W[perm], inv[targets], rows)
    assert np.allclose(c, base, rtol=1e-12, atol=1e-12)


def test_temperature_scales_logits():
    h, W, targets, rows = _case(8)
    a, _, _ = oracle.token_logprob(h, W, targets, rows, inv_tau=2.0)
    b, _, _ = oracle.token_logprob(2.0 * h, W, targets, rows, inv_tau=1.0)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)


def test_statistical_band_rms_hidden():
    # z ~ N(0, (0.02 sqrt d)^2): mean log p ~ -ln V - sigma^2 / 2 (sanity band)
    rng = np.random.default_rng(11)
    T, d, V = 600, 256, 4096
    h = synth.rms_hidden_bf16(rng, (T, d)).double().numpy()
    W = synth.normal_bf16(rng, (V, d), 0.02).double().numpy()
    targets = rng.integers(0, V, size=T)
    logp, _, _ = oracle.token_logprob(h, W, targets, np.arange(T))
    sigma2 = (0.02 ** 2) * d
    assert abs(logp.mean() - (-math.log(V) - sigma2 / 2)) < 0.05


# --------------------------------------------------------------------------
# backward
# --------------------------------------------------------------------------
@pytest.mark.parametrize("reduction", ["sum", "mean"])
def test_bwd_matches_torch_autograd(reduction):
    h, W, targets, rows = _case(9, T=10, d=12, V=41)
    dH, dW = oracle.token_loss_bwd(h, W, targets, rows, inv_tau=1.5,
                                   reduction=reduction, grad_loss=0.7)
    ht = torch.from_numpy(h).requires_grad_(True)
    Wt = torch.from_numpy(W).requires_grad_(True)
    z = 1.5 * (ht[torch.from_numpy(rows)] @ Wt.T)
    loss = 0.7 * F.cross_entropy(z, torch.from_numpy(targets[rows]), reduction=reduction)
    loss.backward()
    assert np.allclose(dH, ht.grad.numpy(), rtol=1e-11, atol=1e-14)
    assert np.allclose(dW, Wt.grad.numpy(), rtol=1e-11, atol=1e-14)


def test_bwd_finite_differences():
    h, W, targets, rows = _case(10, T=8, d=16, V=37)
    dH, dW = oracle.token_loss_bwd(h, W, targets, rows, inv_tau=0.9)
    eps = 1e-6

    def f(hh, WW):
        return oracle.token_logprob(hh, WW, targets, rows, inv_tau=0.9)[2]

    rng = np.random.default_rng(0)
    for _ in range(12):
        t, k = int(rng.integers(0, 8)), int(rng.integers(0, 16))
        hp, hm = h.copy(), h.copy()
        hp[t, k] += eps
        hm[t, k] -= eps
        fd = (f(hp, W) - f(hm, W)) / (2 * eps)
        assert fd == pytest.approx(dH[t, k], rel=1e-6, abs=1e-8)
        v = int(rng.integers(0, 37))
        Wp, Wm = W.copy(), W.copy()
        Wp[v, k] += eps
        Wm[v, k] -= eps
        fd = (f(h, Wp) - f(h, Wm)) / (2 * eps)
        assert fd == pytest.approx(dW[v, k], rel=1e-6, abs=1e-8)


def test_bwd_invariants_and_row_sampler():
    h, W, targets, rows = _case(12, T=20, d=9, V=30)
    dH, dW = oracle.token_loss_bwd(h, W, targets, rows, reduction="mean")
    # softmax - onehot rows sum to zero, so the vocabulary sum of dW vanishes
    assert np.allclose(dW.sum(axis=0), 0, atol=1e-13)
    off = np.setdiff1d(np.arange(len(h)), rows)
    assert np.all(dH[off] == 0)
    sub = rows[::2]
    part = oracle.token_loss_bwd_rows(h, W, targets, sub, reduction="mean", n_mask=len(rows))
    assert np.allclose(part, dH[sub], rtol=1e-12, atol=1e-15)
    vs = np.array([0, 7, 29])
    partw = oracle.token_loss_bwd_vocab(h, W, targets, rows, vs, reduction="mean")
    assert np.allclose(partw, dW[vs], rtol=1e-12, atol=1e-15)


def test_empty_mask():
    h, W, targets, _ = _case(13)
    rows = np.zeros(0, dtype=np.int64)
    for red in ("sum", "mean"):
        logp, lse, loss = oracle.token_logprob(h, W, targets, rows, reduction=red)
        assert loss == 0 and not logp.any() and not lse.any()
        dH, dW = oracle.token_loss_bwd(h, W, targets, rows, reduction=red)
        assert not dH.any() and not dW.any()


# --------------------------------------------------------------------------
# divergence
# --------------------------------------------------------------------------
def test_kl_identical_is_zero():
    h, W, _, rows = _case(14, T=10, d=8, V=50)
    for direction in ("reverse", "forward"):
        kl, dHs = oracle.token_divergence(h, W, h, W, rows, direction=direction,
                                          grad_kl=np.ones(len(h)))
        assert np.allclose(kl, 0, atol=1e-14)
        assert np.allclose(dHs, 0, atol=1e-14)


@pytest.mark.parametrize("direction", ["reverse", "forward"])
def test_kl_matches_torch_and_autograd(direction):
    rng = np.random.default_rng(15)
    T, ds, dt, V = 9, 10, 14, 33
    hs, Ws = rng.standard_normal((T, ds)), rng.standard_normal((V, ds)) * 0.4
    ht, Wt = rng.standard_normal((T, dt)), rng.standard_normal((V, dt)) * 0.4
    rows = np.array([0, 2, 3, 5, 8])
    g = rng.uniform(0.5, 2.0, size=T)
    kl, dHs = oracle.token_divergence(hs, Ws, ht, Wt, rows, inv_tau=1.2,
                                      direction=direction, grad_kl=g)
    assert np.all(kl[rows] >= 0)
    hs_t = torch.from_numpy(hs).requires_grad_(True)
    r = torch.from_numpy(rows)
    lps = F.log_softmax(1.2 * (hs_t[r] @ torch.from_numpy(Ws).T), dim=1)
    lpt = F.log_softmax(1.2 * (torch.from_numpy(ht)[r] @ torch.from_numpy(Wt).T), dim=1)
    if direction == "reverse":   # KL(p_s || p_t)
        ref = F.kl_div(lpt, lps, log_target=True, reduction="none").sum(1)
    else:                        # KL(p_t || p_s)
        ref = F.kl_div(lps, lpt, log_target=True, reduction="none").sum(1)
    assert np.allclose(kl[rows], ref.detach().numpy(), rtol=1e-11, atol=1e-14)
    (ref * torch.from_numpy(g)[r]).sum().backward()
    assert np.allclose(dHs, hs_t.grad.numpy(), rtol=1e-10, atol=1e-14)


def test_kl_finite_differences():
    rng = np.random.default_rng(16)
    T, ds, dt, V = 4, 6, 7, 37
    hs, Ws = rng.standard_normal((T, ds)), rng.standard_normal((V, ds))
    ht, Wt = rng.standard_normal((T, dt)), rng.standard_normal((V, dt))
    rows = np.arange(T)
    g = np.ones(T)
    for direction in ("reverse", "forward"):
        kl, dHs = oracle.token_divergence(hs, Ws, ht, Wt, rows, direction=direction, grad_kl=g)
        eps = 1e-6
        for t in range(T):
            for k in (0, ds - 1):
                hp, hm = hs.copy(), hs.copy()
                hp[t, k] += eps
                hm[t, k] -= eps
                fp = oracle.token_divergence(hp, Ws, ht, Wt, rows, direction=direction)[0].sum()
                fm = oracle.token_divergence(hm, Ws, ht, Wt, rows, direction=direction)[0].sum()
                assert (fp - fm) / (2 * eps) == pytest.approx(dHs[t, k], rel=1e-6, abs=1e-8)


def test_bf16_widening_exact():
    x = torch.randn(1000, generator=torch.Generator().manual_seed(0)).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.bf16_bits_to_f64(bits), x.double().numpy())


# --------------------------------------------------------------------------
# entropy and top-K
# --------------------------------------------------------------------------
def test_topk_matches_torch_and_entropy_matches_scipy():
    import scipy.stats
    h, W, targets, rows = _case(17, T=15, d=10, V=90)
    lse, H, tv, ti = oracle.token_topk(h, W, rows, 16, inv_tau=0.9)
    z = torch.from_numpy(0.9 * h @ W.T)
    lp = torch.log_softmax(z, dim=1)
    ref_v, ref_i = torch.topk(lp, 16, dim=1)
    assert np.allclose(tv[rows], ref_v.numpy()[rows], atol=1e-12)
    assert np.array_equal(ti[rows], ref_i.numpy()[rows])
    p = np.exp(lp.numpy())
    assert np.allclose(H[rows], scipy.stats.entropy(p[rows], axis=1), atol=1e-12)
    off = np.setdiff1d(np.arange(len(h)), rows)
    assert np.all(ti[off] == -1) and not tv[off].any() and not H[off].any()


def test_topk_closed_forms():
    V, d = 100, 4
    h = np.random.default_rng(0).standard_normal((3, d))
    lse, H, tv, ti = oracle.token_topk(h, np.zeros((V, d)), [0, 1, 2], 5)
    # uniform: H = ln V, every log-prob = -ln V, ties ordered by ascending id
    assert np.allclose(H, math.log(V), atol=1e-12)
    assert np.allclose(tv, -math.log(V), atol=1e-12)
    assert np.array_equal(ti, np.tile(np.arange(5), (3, 1)))
    # a dominant entry: entropy -> 0, top-1 is that id with log-prob -> 0
    W = np.zeros((V, d))
    W[37, 0] = 40.0
    h1 = np.zeros((1, d))
    h1[0, 0] = 1.0
    _, H1, tv1, ti1 = oracle.token_topk(h1, W, [0], 3)
    a = (V - 1) * math.exp(-40.0)
    # H = ln Z - 40 e^40 / Z with Z = e^40 + V - 1, i.e. a + 40 a / (1 + a)
    assert ti1[0, 0] == 37 and abs(tv1[0, 0]) < 1e-15
    assert H1[0] == pytest.approx(a + 40 * a / (1 + a), rel=1e-3)
    assert np.array_equal(ti1[0, 1:], [0, 1])


def test_topk_compare_pins():
    rng = np.random.default_rng(18)
    T, d, V, K = 6, 9, 60, 8
    hs, Ws = rng.standard_normal((T, d)), rng.standard_normal((V, d)) * 0.8
    ht, Wt = rng.standard_normal((T, d + 3)), rng.standard_normal((V, d + 3)) * 0.8
    rows = np.array([0, 2, 3, 5])
    # identical models: full overlap, zero truncated KL
    ov, kl, _, _ = oracle.token_topk_compare(hs, Ws, hs, Ws, rows, K)
    assert np.all(ov[rows] == 1.0) and np.allclose(kl[rows], 0, atol=1e-14)
    # K = V: the truncation is the full reverse KL, and the overlap is 1
    ovV, klV, _, _ = oracle.token_topk_compare(hs, Ws, ht, Wt, rows, V)
    full, _ = oracle.token_divergence(hs, Ws, ht, Wt, rows)
    assert np.allclose(klV[rows], full[rows], rtol=1e-12, atol=1e-14) and np.all(ovV[rows] == 1.0)
    # against torch.topk on independently formed log-probs
    ov, kl, gs, gt = oracle.token_topk_compare(hs, Ws, ht, Wt, rows, K)
    lps = torch.log_softmax(torch.from_numpy(hs @ Ws.T), 1)
    lpt = torch.log_softmax(torch.from_numpy(ht @ Wt.T), 1)
    for r in rows:
        S = torch.topk(lps[r], K).indices
        Tk = torch.topk(lpt[r], K).indices
        assert ov[r] == len(set(S.tolist()) & set(Tk.tolist())) / K
        ref = (lps[r, S].exp() * (lps[r, S] - lpt[r, S])).sum().item()
        assert kl[r] == pytest.approx(ref, rel=1e-12, abs=1e-14)
        assert gs[r] > 0 and gt[r] > 0


def test_topk_compare_three_token_closed_form():
    """V = 3, student logits (2, 1, 0), teacher logits (0, 1, 2): both rows have the same
    log-sum-exp Z = ln(e^2 + e + 1), so log p_s(v) - log p_t(v) = z_s(v) - z_t(v) = (2, 0, -2).
    K = 1: S = {0}, teacher top-1 = {2}: overlap 0, KL_1 = 2 p_s(0).
    K = 2: S = {0, 1}, teacher {2, 1}: overlap 1/2, KL_2 = 2 p_s(0) + 0 p_s(1) = KL_1.
    K = 3: overlap 1, KL_3 = 2 p_s(0) - 2 p_s(2), the full reverse KL.
    Without renormalisation over S the truncated terms keep the full-vocabulary p_s."""
    hs, ht = np.ones((1, 1)), np.ones((1, 1))
    Ws = np.array([[2.0], [1.0], [0.0]])
    Wt = np.array([[0.0], [1.0], [2.0]])
    Z = math.e ** 2 + math.e + 1
    p0, p2 = math.e ** 2 / Z, 1 / Z
    expect = {1: (0.0, 2 * p0), 2: (0.5, 2 * p0), 3: (1.0, 2 * p0 - 2 * p2)}
    for K, (ov_ref, kl_ref) in expect.items():
        ov, kl, _, _ = oracle.token_topk_compare(hs, Ws, ht, Wt, [0], K)
        assert ov[0] == ov_ref
        assert kl[0] == pytest.approx(kl_ref, rel=1e-13)
    # the top-K lists themselves: descending log-probs with their ids
    _, H, tv, ti = oracle.token_topk(hs, Ws, [0], 2)
    assert ti[0].tolist() == [0, 1]
    assert tv[0] == pytest.approx([2 - math.log(Z), 1 - math.log(Z)], rel=1e-13)
    # entropy: ln Z - sum_v p_v z_v
    assert H[0] == pytest.approx(math.log(Z) - (2 * math.e ** 2 + math.e) / Z, rel=1e-13)


def test_topk_kl_bwd_matches_autograd_with_fixed_set():
    rng = np.random.default_rng(19)
    T, ds, dt, V, K = 5, 7, 9, 40, 6
    hs, Ws = rng.standard_normal((T, ds)), rng.standard_normal((V, ds)) * 0.7
    ht, Wt = rng.standard_normal((T, dt)), rng.standard_normal((V, dt)) * 0.7
    rows = np.array([0, 1, 3, 4])
    g = rng.uniform(0.5, 2.0, size=T)
    dH, dW = oracle.token_topk_kl_bwd(hs, Ws, ht, Wt, rows, K, inv_tau=1.2, grad=g)
    hs_t = torch.from_numpy(hs).requires_grad_(True)
    Ws_t = torch.from_numpy(Ws).requires_grad_(True)
    r = torch.from_numpy(rows)
    lps = torch.log_softmax(1.2 * (hs_t[r] @ Ws_t.T), 1)
    lpt = torch.log_softmax(1.2 * (torch.from_numpy(ht)[r] @ torch.from_numpy(Wt).T), 1)
    S = torch.topk(lps.detach(), K, dim=1).indices          # the set is selected, not differentiated
    ls, lt = lps.gather(1, S), lpt.gather(1, S)
    kl = (ls.exp() * (ls - lt)).sum(1)
    (kl * torch.from_numpy(g)[r]).sum().backward()
    assert np.allclose(dH, hs_t.grad.numpy(), rtol=1e-10, atol=1e-13)
    assert np.allclose(dW, Ws_t.grad.numpy(), rtol=1e-10, atol=1e-13)
    # K = V: the gradient of the full reverse KL
    dHV, _ = oracle.token_topk_kl_bwd(hs, Ws, ht, Wt, rows, V, inv_tau=1.2, grad=g)
    _, full = oracle.token_divergence(hs, Ws, ht, Wt, rows, 1.2, "reverse", grad_kl=g)
    assert np.allclose(dHV, full, rtol=1e-10, atol=1e-13)
