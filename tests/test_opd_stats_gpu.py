"""olive_opd_token_stats (CUDA: one sweep with both heads) against the
oracle's token_divergence, token_topk and token_topk_compare, and against the
separate entry points that compute the same quantities in three sweeps."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (LOGP_ATOL, LOGP_RTOL, assert_close_grad, assert_close_logp, sample_rows,
                          to_f32, to_f64)
from tests.test_topk_gpu import _check_rows, _oracle_full

pytestmark = pytest.mark.gpu

DECIDE = 1e-3  # log-prob gap above which top-K membership is not a rounding decision


def _models(rng, T, ds, dt, V, std_w=0.4):
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), std_w)
    # the teacher shares part of the student's structure, so the overlap is not trivial
    ht = torch.cat([hs, synth.normal_bf16(rng, (T, dt - ds), 1.0)], 1) if dt > ds else hs[:, :dt].contiguous()
    Wt = torch.cat([Ws, synth.normal_bf16(rng, (V, dt - ds), std_w)], 1) if dt > ds else Ws[:, :dt].contiguous()
    return hs, Ws, ht, Wt


def _gpu(hs, Ws, ht, Wt, rows, K, inv_tau=1.0, direction="reverse"):
    r = torch.from_numpy(np.asarray(rows, dtype=np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    out = B.olive_opd_token_stats(hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda(), r, n, K, inv_tau,
                                  direction, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return {k: v.cpu().numpy() for k, v in out.items()}


def _check_against_oracle(hs, Ws, ht, Wt, rows, K, inv_tau, direction, g, min_decided=0.8):
    f = to_f64
    T = hs.shape[0]
    rkl, _ = oracle.token_divergence(f(hs), f(Ws), f(ht), f(Wt), rows, inv_tau, direction)
    assert_close_logp(g["kl"], rkl, "kl")
    # student lse, entropy and top-K list (ids valid, exact where separated)
    lse_s, H_s, lp_s = _oracle_full(hs, Ws, rows, inv_tau)
    _check_rows(rows, K, (g["s_lse"], g["s_entropy"], g["s_topk_logp"], g["s_topk_ids"]),
                lse_s, H_s, lp_s)
    lse_t, _, lp_t = _oracle_full(ht, Wt, rows, inv_tau)
    assert_close_logp(g["t_lse"][rows], lse_t, "t_lse")
    # teacher log-probs at the returned student ids
    for k, t in enumerate(rows):
        ids = g["s_topk_ids"][t].astype(np.int64)
        assert_close_logp(g["t_logp_s"][t], lp_t[k][ids], f"t_logp_s row {t}")
    # overlap and top-K KL where both top-K sets are decided
    rov, rklk, gs, gt = oracle.token_topk_compare(f(hs), f(Ws), f(ht), f(Wt), rows, K, inv_tau)
    decided = 0
    for t in rows:
        if gs[t] > DECIDE and gt[t] > DECIDE:
            decided += 1
            assert g["overlap"][t] == pytest.approx(rov[t], abs=1e-6), t
            assert abs(g["kl_topk"][t] - rklk[t]) <= LOGP_ATOL + LOGP_RTOL * abs(rklk[t]), t
    assert decided >= min_decided * len(rows)
    off = np.setdiff1d(np.arange(T), rows)
    for k in ("kl", "s_lse", "t_lse", "s_entropy", "overlap", "kl_topk"):
        assert not g[k][off].any(), k
    assert (g["s_topk_ids"][off] == -1).all()


@pytest.mark.parametrize("T,ds,dt,V,K,inv_tau,direction", [
    (200, 64, 96, 3000, 16, 1.0, "reverse"),
    (150, 128, 64, 800, 4, 0.8, "forward"),
    (260, 64, 64, 20000, 16, 1.2, "reverse"),
    (130, 96, 128, 1000, 1, 1.0, "forward"),
])
def test_small_shapes(T, ds, dt, V, K, inv_tau, direction):
    rng = np.random.default_rng(T + V + K)
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False))
    g = _gpu(hs, Ws, ht, Wt, rows, K, inv_tau, direction)
    _check_against_oracle(hs, Ws, ht, Wt, rows, K, inv_tau, direction, g)


def test_full_set_and_identical_models():
    """K = V = 16: overlap 1 and the truncated KL is the full KL; identical
    heads: KL 0, overlap 1."""
    rng = np.random.default_rng(3)
    hs, Ws, ht, Wt = _models(rng, 140, 64, 96, 16, std_w=0.5)
    rows = np.arange(0, 140, 2)
    g = _gpu(hs, Ws, ht, Wt, rows, 16)
    assert np.all(g["overlap"][rows] == 1.0)
    assert np.abs(g["kl_topk"][rows] - g["kl"][rows]).max() <= 1e-5
    g = _gpu(hs, Ws, hs, Ws, rows, 16)
    assert np.abs(g["kl"]).max() <= 1e-5 and np.all(g["overlap"][rows] == 1.0)


def test_matches_the_three_sweep_path():
    """Same quantities through olive_token_divergence, two
    olive_token_topk_fwd sweeps and olive_topk_compare."""
    rng = np.random.default_rng(17)
    hs, Ws, ht, Wt = _models(rng, 300, 128, 160, 5001)
    rows = np.arange(300)
    g = _gpu(hs, Ws, ht, Wt, rows, 16)
    r = torch.from_numpy(rows.astype(np.int32)).cuda()
    n = torch.tensor([300], dtype=torch.int32, device="cuda")
    hs, Ws, ht, Wt = hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda()
    kl, _ = B.olive_token_divergence(hs, Ws, ht, Wt, r, n)
    s_lse, s_ent, s_lp, s_id = B.olive_token_topk_fwd(hs, Ws, r, n, 16)
    t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, r, n, 16)
    ov, klk, tlp = B.olive_topk_compare(ht, Wt, r, n, s_id, s_lp, t_id, t_lse, want_t_logp=True)
    np.testing.assert_allclose(g["kl"], kl.cpu().numpy(), atol=2e-5, rtol=1e-4)
    np.testing.assert_allclose(g["s_lse"], s_lse.cpu().numpy(), atol=2e-5)
    np.testing.assert_allclose(g["t_lse"], t_lse.cpu().numpy(), atol=2e-5)
    np.testing.assert_allclose(g["s_entropy"], s_ent.cpu().numpy(), atol=5e-5)
    same = (g["s_topk_ids"] == s_id.cpu().numpy()).all(axis=1)
    assert same.mean() > 0.95
    np.testing.assert_allclose(g["s_topk_logp"][same], s_lp.cpu().numpy()[same], atol=2e-5)
    np.testing.assert_allclose(g["t_logp_s"][same], tlp.cpu().numpy()[same], atol=5e-5)
    np.testing.assert_allclose(g["kl_topk"][same], klk.cpu().numpy()[same], atol=5e-5)


def test_feeds_the_topk_kl_gradient():
    """olive_topk_kl_bwd on the sweep's outputs against the oracle's gradient
    (rows whose top-K set is decided)."""
    rng = np.random.default_rng(23)
    T, ds, dt, V, K = 200, 64, 96, 3000, 16
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    cand = np.arange(T)
    _, _, gs, _ = oracle.token_topk_compare(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), cand, K)
    rows = cand[gs[cand] > DECIDE]
    gk = rng.uniform(0.5, 2.0, size=T)
    r = torch.from_numpy(rows.astype(np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    hsc, Wsc = hs.cuda(), Ws.cuda()
    o = B.olive_opd_token_stats(hsc, Wsc, ht.cuda(), Wt.cuda(), r, n, K,
                                want=("s_lse", "s_topk_logp", "s_topk_ids", "t_logp_s", "kl_topk"),
                                dev_status=st)
    dh, dw = B.olive_topk_kl_bwd(hsc, Wsc, r, n, o["s_lse"], o["s_topk_ids"], o["s_topk_logp"],
                                 o["t_logp_s"], o["kl_topk"],
                                 torch.from_numpy(gk.astype(np.float32)).cuda(),
                                 grad_dtype=torch.float32, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    rdh, rdw = oracle.token_topk_kl_bwd(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, K,
                                        grad=gk)
    assert_close_grad(dh.cpu().numpy()[rows], rdh[rows], "dH_s")
    assert_close_grad(dw.cpu().numpy(), rdw, "dW_s")


@pytest.mark.slow
def test_kl_workload_sampled():
    """16384 rows, student d = 4096, teacher d = 5120, V = 151936, K = 16; KL, lse,
    entropy and the student's top-16 log-probs on 256 sampled rows."""
    T = 16384
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rows = np.arange(T)
    g = _gpu(hs, Ws, ht, Wt, rows, 16)
    pick = sample_rows(rows, 256, seed=6)
    rkl, _ = oracle.token_divergence(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick)
    assert_close_logp(g["kl"][pick], rkl[pick], "kl")
    rl, rH, rv, _ = oracle.token_topk(to_f32(hs), to_f32(Ws), pick, 16)
    assert_close_logp(g["s_lse"][pick], rl[pick], "s_lse")
    assert_close_logp(g["s_entropy"][pick], rH[pick], "s_entropy")
    assert_close_logp(g["s_topk_logp"][pick], rv[pick], "s_topk_logp")
    assert np.all(g["kl"] >= -1e-3) and np.all((g["overlap"] >= 0) & (g["overlap"] <= 1))
