"""olive_topk_kl_bwd (CUDA) against the oracle's token_topk_kl_bwd: the
gradient of the top-K truncated reverse KL with the student's top-K set held
fixed.

The set is a selection: the GPU (fp32 logits of bf16 products) and the oracle
(fp64) agree on it only where the K-th and (K+1)-th student log-probs are
separated by more than rounding.  The rows handed to both sides are therefore
the rows whose oracle gap exceeds DECIDE (a choice made from oracle values
only), so both sides differentiate the same objective."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_grad, assert_close_logp, sample_rows, to_f32, to_f64

pytestmark = pytest.mark.gpu

DECIDE = 1e-3


def _gpu(hs, Ws, ht, Wt, rows, K, g, inv_tau=1.0, grad_dtype=torch.float32):
    r = torch.from_numpy(np.asarray(rows, dtype=np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    hs, Ws, ht, Wt = hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda()
    s_lse, _, s_lp, s_id = B.olive_token_topk_fwd(hs, Ws, r, n, K, inv_tau, dev_status=st)
    t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, r, n, K, inv_tau, dev_status=st)
    _, kl, tlp = B.olive_topk_compare(ht, Wt, r, n, s_id, s_lp, t_id, t_lse, inv_tau,
                                      dev_status=st, want_t_logp=True)
    gk = torch.from_numpy(np.asarray(g, dtype=np.float32)).cuda()
    dh, dw = B.olive_topk_kl_bwd(hs, Ws, r, n, s_lse, s_id, s_lp, tlp, kl, gk, inv_tau,
                                 grad_dtype=grad_dtype, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return (dh.float().cpu().numpy(), dw.float().cpu().numpy(), s_id.cpu().numpy(),
            tlp.cpu().numpy(), kl.cpu().numpy())


def _models(rng, T, ds, dt, V, std_w=0.4):
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), std_w)
    # the teacher shares part of the student's structure, as in the overlap tests
    ht = torch.cat([hs, synth.normal_bf16(rng, (T, dt - ds), 1.0)], 1) if dt > ds else hs[:, :dt].contiguous()
    Wt = torch.cat([Ws, synth.normal_bf16(rng, (V, dt - ds), std_w)], 1) if dt > ds else Ws[:, :dt].contiguous()
    return hs, Ws, ht, Wt


def _decided_rows(hs, Ws, ht, Wt, cand, K, inv_tau):
    _, _, gs, _ = oracle.token_topk_compare(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), cand, K,
                                            inv_tau)
    rows = np.array([t for t in cand if gs[t] > DECIDE], dtype=np.int64)
    assert len(rows) >= 0.8 * len(cand)
    return rows


@pytest.mark.parametrize("T,ds,dt,V,K,inv_tau,grad_dtype", [
    (200, 64, 96, 3000, 16, 1.0, torch.float32),
    (150, 128, 64, 800, 4, 0.8, torch.bfloat16),
    (300, 64, 64, 1000, 1, 1.0, torch.float32),
])
def test_small_shapes(T, ds, dt, V, K, inv_tau, grad_dtype):
    rng = np.random.default_rng(T + V + 31 * K)
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    cand = np.sort(rng.choice(T, size=T * 2 // 3, replace=False))
    rows = _decided_rows(hs, Ws, ht, Wt, cand, K, inv_tau)
    g = rng.uniform(0.5, 2.0, size=T)
    dh, dw, s_id, tlp, _ = _gpu(hs, Ws, ht, Wt, rows, K, g, inv_tau, grad_dtype)
    rdh, rdw = oracle.token_topk_kl_bwd(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, K,
                                        inv_tau, grad=g)
    assert_close_grad(dh[rows], rdh[rows], "dH_s")
    assert_close_grad(dw, rdw, "dW_s")
    off = np.setdiff1d(np.arange(T), rows)
    assert not dh[off].any()
    # the teacher log-probs at the student's ids that feed the gradient
    lpt, _ = oracle.log_softmax_rows(oracle.logits(to_f64(ht)[rows], to_f64(Wt), inv_tau))
    assert_close_logp(tlp[rows], np.take_along_axis(lpt, s_id[rows].astype(np.int64), 1), "t_logp_s")
    assert not tlp[off].any()


def test_full_set_equals_full_kl_gradient():
    """K = V: the truncation keeps every term, P_S = 1 and the gradient is the
    full reverse-KL gradient (dH through olive_token_divergence's formula)."""
    rng = np.random.default_rng(12)
    T, d, V = 140, 64, 16
    hs, Ws, ht, Wt = _models(rng, T, d, d + 32, V, std_w=0.5)
    rows = np.arange(0, T, 2)
    g = rng.uniform(0.5, 2.0, size=T)
    dh, dw, _, _, kl = _gpu(hs, Ws, ht, Wt, rows, V, g)
    _, rfull = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, 1.0,
                                       "reverse", grad_kl=g)
    assert_close_grad(dh[rows], rfull[rows], "dH_s")
    rkl, _ = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows)
    assert_close_logp(kl[rows], rkl[rows], "kl")
    _, rdw = oracle.token_topk_kl_bwd(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, V, grad=g)
    assert_close_grad(dw, rdw, "dW_s")


@pytest.mark.slow
def test_kl_workload_sampled():
    """Student d = 4096 / teacher d = 5120, V = 151936, K = 16; dH_s on
    sampled decided rows (dH_s[t] depends on row t alone)."""
    T = 2048
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rng = np.random.default_rng(3)
    g = rng.uniform(0.5, 2.0, size=T)
    dh, dw, _, _, _ = _gpu(hs, Ws, ht, Wt, np.arange(T), 16, g, grad_dtype=torch.bfloat16)
    assert np.isfinite(dw).all()
    pick = sample_rows(np.arange(T), 256, seed=5)
    _, _, gs, _ = oracle.token_topk_compare(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick, 16)
    pick = np.array([t for t in pick if gs[t] > DECIDE])
    assert len(pick) >= 128
    rdh, _ = oracle.token_topk_kl_bwd(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick, 16, grad=g,
                                      with_dW=False)
    for t in pick:
        assert_close_grad(dh[t], rdh[t], f"dH_s[{t}]")


def test_several_slabs(monkeypatch):
    """The slab cap lowered to 128 rows: the sparse correction and dW's fp32
    accumulation run across slabs of the one-launch backward."""
    monkeypatch.setenv("OLIVE_SLAB_ROWS", "128")
    rng = np.random.default_rng(61)
    T, ds, dt, V, K = 700, 64, 96, 1500, 8
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(T), K, 1.0)
    assert len(rows) > 4 * 128
    g = rng.uniform(0.5, 2.0, size=T)
    dh, dw, _, _, _ = _gpu(hs, Ws, ht, Wt, rows, K, g, grad_dtype=torch.bfloat16)
    rdh, rdw = oracle.token_topk_kl_bwd(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, K, grad=g)
    assert_close_grad(dh[rows], rdh[rows], "dH_s")
    assert_close_grad(dw, rdw, "dW_s")
