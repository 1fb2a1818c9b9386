"""olive_topk_compare (CUDA) on top of two olive_token_topk_fwd sweeps,
against the oracle's token_topk_compare.

Top-K membership is unique only where the K-th and (K+1)-th log-probs are
separated by more than the GPU's own log-prob error (fp32 accumulation of
bf16 products: ~1e-5 here; the margin used is 1e-3); on those rows the overlap
must match exactly and the truncated KL within the parity tolerance.  Rows
decided by rounding are only checked for range, and most rows must be
decidable."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import LOGP_ATOL, LOGP_RTOL, sample_rows, to_f32, to_f64

pytestmark = pytest.mark.gpu

DECIDE = 1e-3  # log-prob gap above which top-K membership is not a rounding decision


def _gpu(hs, Ws, ht, Wt, rows, K, inv_tau=1.0):
    r = torch.from_numpy(np.asarray(rows, dtype=np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    hs, Ws, ht, Wt = hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda()
    _, _, s_lp, s_id = B.olive_token_topk_fwd(hs, Ws, r, n, K, inv_tau, dev_status=st)
    t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, r, n, K, inv_tau, dev_status=st)
    ov, kl = B.olive_topk_compare(ht, Wt, r, n, s_id, s_lp, t_id, t_lse, inv_tau, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return ov.cpu().numpy(), kl.cpu().numpy()


def _check(ov, kl, ref, rows, min_decided=0.8):
    rov, rkl, gs, gt = ref
    decided = 0
    for t in rows:
        assert 0.0 <= ov[t] <= 1.0
        if gs[t] > DECIDE and gt[t] > DECIDE:
            decided += 1
            assert ov[t] == pytest.approx(rov[t], abs=1e-6), t
            assert abs(kl[t] - rkl[t]) <= LOGP_ATOL + LOGP_RTOL * abs(rkl[t]), (t, kl[t], rkl[t])
    assert decided >= min_decided * len(rows), (decided, len(rows))


@pytest.mark.parametrize("T,ds,dt,V,K,inv_tau", [
    (200, 64, 96, 3000, 16, 1.0),
    (150, 128, 64, 800, 4, 0.8),
])
def test_small_shapes(T, ds, dt, V, K, inv_tau):
    rng = np.random.default_rng(T + V + K)
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), 0.4)
    # the teacher shares part of the student's structure, so the overlap is not trivial
    ht = torch.cat([hs, synth.normal_bf16(rng, (T, dt - ds), 1.0)], 1) if dt > ds else hs[:, :dt].contiguous()
    Wt = torch.cat([Ws, synth.normal_bf16(rng, (V, dt - ds), 0.4)], 1) if dt > ds else Ws[:, :dt].contiguous()
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False))
    ov, kl = _gpu(hs, Ws, ht, Wt, rows, K, inv_tau)
    ref = oracle.token_topk_compare(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, K, inv_tau)
    _check(ov, kl, ref, rows)
    off = np.setdiff1d(np.arange(T), rows)
    assert not ov[off].any() and not kl[off].any()
    assert 0.0 < ov[rows].mean() < 1.0


def test_identical_models_full_overlap_zero_kl():
    rng = np.random.default_rng(5)
    h = synth.normal_bf16(rng, (130, 64), 1.0)
    W = synth.normal_bf16(rng, (2000, 64), 0.4)
    rows = np.arange(130)
    ov, kl = _gpu(h, W, h, W, rows, 16)
    assert np.all(ov == 1.0)
    assert np.abs(kl).max() <= 1e-5


@pytest.mark.slow
def test_kl_workload_sampled():
    """Student d = 4096 / teacher d = 5120, V = 151936, K = 16, sampled rows."""
    T = 2048
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rows = np.arange(T)
    ov, kl = _gpu(hs, Ws, ht, Wt, rows, 16)
    pick = sample_rows(rows, 256, seed=8)
    ref = oracle.token_topk_compare(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick, 16)
    _check(ov, kl, ref, pick, min_decided=0.5)
