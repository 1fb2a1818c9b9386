"""olive_token_divergence (CUDA) against the oracle's full-vocabulary KL."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_grad, assert_close_logp, rel_frob, sample_rows, to_f32, to_f64

pytestmark = pytest.mark.gpu


def _case(seed, T, ds, dt, V, std=0.1):
    rng = np.random.default_rng(seed)
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), std)
    ht = synth.normal_bf16(rng, (T, dt), 1.0)
    Wt = synth.normal_bf16(rng, (V, dt), std)
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False)).astype(np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    return hs, Ws, ht, Wt, rows, gk


def _gpu(hs, Ws, ht, Wt, rows, gk, direction, inv_tau=1.0, grad_dtype=torch.float32):
    r = torch.from_numpy(rows).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    g = torch.from_numpy(gk).cuda() if gk is not None else None
    kl, dhs = B.olive_token_divergence(hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda(), r, n, inv_tau,
                                       direction, g, grad_dtype, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return kl.cpu().numpy(), (dhs.float().cpu().numpy() if dhs is not None else None)


@pytest.mark.parametrize("direction", ["reverse", "forward"])
@pytest.mark.parametrize("T,ds,dt,V,inv_tau", [
    (200, 64, 72, 1000, 1.0),
    (300, 128, 192, 4097, 0.8),
    (150, 256, 64, 300, 1.0),
])
def test_small_shapes(direction, T, ds, dt, V, inv_tau):
    hs, Ws, ht, Wt, rows, gk = _case(T + V, T, ds, dt, V)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction, inv_tau)
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows,
                                        inv_tau, direction, grad_kl=gk.astype(np.float64))
    assert_close_logp(kl, rkl, "kl")
    assert_close_grad(dhs, rdhs, "dH_s")
    assert np.all(kl[rows] >= -1e-4)
    off = np.setdiff1d(np.arange(T), rows)
    assert not kl[off].any() and not dhs[off].any()


def test_identical_student_teacher_is_zero():
    hs, Ws, _, _, rows, gk = _case(3, 256, 128, 128, 2000)
    for direction in ("reverse", "forward"):
        kl, dhs = _gpu(hs, Ws, hs, Ws, rows, gk, direction)
        assert np.abs(kl).max() <= 1e-5
        assert np.abs(dhs).max() <= 1e-6


def test_no_gradient_requested_bf16():
    hs, Ws, ht, Wt, rows, _ = _case(4, 130, 64, 64, 513)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, None, "reverse")
    assert dhs is None
    rkl, _ = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows)
    assert_close_logp(kl, rkl, "kl")


@pytest.mark.slow
def test_kl_workload_sampled_rows():
    """16384 rows, d_s = 4096, d_t = 5120, V = 151936: sampled oracle rows."""
    T = 16384
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rows = np.arange(T, dtype=np.int32)
    gk = np.ones(T, dtype=np.float32)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, "reverse", grad_dtype=torch.bfloat16)
    pick = sample_rows(rows, 16, seed=2)
    rkl, rdhs = oracle.token_divergence(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick,
                                        grad_kl=np.ones(T))
    assert_close_logp(kl[pick], rkl[pick], "kl")
    assert rel_frob(dhs[pick], rdhs[pick]) <= 1e-2
    assert np.all(kl >= -1e-3)
