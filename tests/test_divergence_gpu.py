"""olive_token_divergence (CUDA) against the oracle's full-vocabulary KL."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (FULL_SIZE_ROWS, assert_close_grad, assert_close_logp, rel_frob, sample_rows,
                          to_f32, to_f64)

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
    """16384 rows, d_s = 4096, d_t = 5120, V = 151936: KL and dH_s on 2048
    sampled rows."""
    T = 16384
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rows = np.arange(T, dtype=np.int32)
    gk = np.ones(T, dtype=np.float32)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, "reverse", grad_dtype=torch.bfloat16)
    pick = sample_rows(rows, FULL_SIZE_ROWS, seed=2)
    rkl, rdhs = oracle.token_divergence(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick,
                                        grad_kl=np.ones(T))
    assert_close_logp(kl[pick], rkl[pick], "kl")
    assert rel_frob(dhs[pick], rdhs[pick]) <= 1e-2
    assert np.all(kl >= -1e-3)


@pytest.mark.parametrize("direction", ["reverse", "forward"])
def test_many_outer_tiles(direction):
    """~1.3k masked rows, d_s = 4096: groups of ~16 CTAs that each run several
    row tiles, so the exchange ring wraps many times; the last row tile and
    the last vocabulary tile are partial."""
    rng = np.random.default_rng(8)
    T, ds, dt, V = 2000, 4096, 96, 1500
    hs = synth.rms_hidden_bf16(rng, (T, ds))
    Ws = synth.normal_bf16(rng, (V, ds), 0.02)
    ht = synth.normal_bf16(rng, (T, dt), 1.0)
    Wt = synth.normal_bf16(rng, (V, dt), 0.1)
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False)).astype(np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction, grad_dtype=torch.bfloat16)
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows,
                                        1.0, direction, grad_kl=gk.astype(np.float64))
    assert_close_logp(kl, rkl, "kl")
    assert_close_grad(dhs, rdhs, "dH_s")


def test_two_column_sweeps():
    """d_s one 64-column tail wider than one sweep of the on-chip gradient:
    the group pass runs twice over the same logits."""
    rng = np.random.default_rng(18)
    sms = min(torch.cuda.get_device_properties(0).multi_processor_count, 192)
    T, ds, dt, V = 300, sms // 2 * 256 + 64, 64, 700
    hs = synth.rms_hidden_bf16(rng, (T, ds))
    Ws = synth.normal_bf16(rng, (V, ds), 0.01)
    ht = synth.normal_bf16(rng, (T, dt), 1.0)
    Wt = synth.normal_bf16(rng, (V, dt), 0.3)
    rows = np.arange(0, T, 2, dtype=np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    for direction in ("reverse", "forward"):
        kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction)
        rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows,
                                            1.0, direction, grad_kl=gk.astype(np.float64))
        assert_close_logp(kl, rkl, "kl")
        assert_close_grad(dhs, rdhs, "dH_s")


def test_value_with_and_without_gradient_agree():
    """KL from the value-only call and from the call with the gradient (whose
    first sweep is the same value sweep) agree."""
    hs, Ws, ht, Wt, rows, gk = _case(9, 400, 128, 64, 3001)
    for direction in ("reverse", "forward"):
        k1, _ = _gpu(hs, Ws, ht, Wt, rows, None, direction)
        k2, _ = _gpu(hs, Ws, ht, Wt, rows, gk, direction)
        assert np.abs(k1 - k2).max() <= 1e-4


def test_teacher_shifted_by_a_constant_per_row():
    """z_t = z_s + c_t with |c_t| up to 24 (an extra hidden unit on a column of
    ones): the distributions are equal, so KL and its gradient vanish; the
    log-ratio kept between the passes must not lose them to the shift."""
    rng = np.random.default_rng(11)
    T, d, V = 300, 64, 2000
    hs = synth.normal_bf16(rng, (T, d), 1.0)
    Ws = synth.normal_bf16(rng, (V, d), 0.3)
    c = torch.from_numpy(rng.uniform(-24, 24, size=(T, 8)).astype(np.float32)).to(torch.bfloat16)
    c[:, 1:] = 0
    ht = torch.cat([hs, c], 1)
    Wt = torch.cat([Ws, torch.zeros(V, 8, dtype=torch.bfloat16)], 1)
    Wt[:, d] = 1.0
    rows = np.arange(T, dtype=np.int32)
    gk = np.ones(T, dtype=np.float32)
    for direction in ("reverse", "forward"):
        kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction)
        assert np.abs(kl).max() <= 2e-5, direction
        assert np.abs(dhs).max() <= 1e-5, direction


@pytest.mark.parametrize("direction", ["reverse", "forward"])
def test_single_row_tile(direction):
    """T <= 128: one row tile, so all but one group of the gradient pass have
    no tile of their own."""
    hs, Ws, ht, Wt, rows, gk = _case(12, 100, 64, 64, 777)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction)
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows,
                                        1.0, direction, grad_kl=gk.astype(np.float64))
    assert_close_logp(kl, rkl, "kl")
    assert_close_grad(dhs, rdhs, "dH_s")


def test_forward_kl_with_a_collapsed_student():
    """The student puts a logit 100 above the rest on one token (an extra
    hidden unit), so inside that token's 256-column tile its other
    probabilities are below 2^-126 of the tile maximum, while the teacher
    spreads its mass.  Forward-KL gradients there are -p_t, which a p_s kept
    relative to the tile maximum in 8 exponent bits would lose."""
    rng = np.random.default_rng(13)
    T, d, V = 200, 64, 1000
    h = synth.normal_bf16(rng, (T, d), 1.0)
    W = synth.normal_bf16(rng, (V, d), 0.3)
    one = torch.zeros(T, 8, dtype=torch.bfloat16)
    one[:, 0] = 1.0
    hs = torch.cat([h, one], 1)
    Ws = torch.cat([W, torch.zeros(V, 8, dtype=torch.bfloat16)], 1)
    Ws[300, d] = 100.0
    rows = np.arange(T, dtype=np.int32)
    gk = np.ones(T, dtype=np.float32)
    kl, dhs = _gpu(hs, Ws, h, W, rows, gk, "forward")
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(h), to_f64(W), rows, 1.0,
                                        "forward", grad_kl=gk.astype(np.float64))
    assert_close_logp(kl, rkl, "kl")
    assert_close_grad(dhs, rdhs, "dH_s")


@pytest.mark.slow
def test_kl_medium_sampled_rows():
    """4096 rows, d_s = 1024, d_t = 1536, V = 65536 (W_s and W_t together
    larger than L2; ~2 GB on the device): KL and d/dh_s on sampled rows."""
    rng = np.random.default_rng(41)
    T, ds, dt, V = 4096, 1024, 1536, 65536
    hs = synth.rms_hidden_bf16(rng, (T, ds))
    Ws = synth.normal_bf16(rng, (V, ds), 0.02)
    ht = synth.rms_hidden_bf16(rng, (T, dt))
    Wt = synth.normal_bf16(rng, (V, dt), 0.02)
    rows = np.arange(T, dtype=np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, "reverse", grad_dtype=torch.bfloat16)
    pick = sample_rows(rows, 512, seed=4)
    rkl, rdhs = oracle.token_divergence(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick,
                                        grad_kl=gk.astype(np.float64))
    assert_close_logp(kl[pick], rkl[pick], "kl")
    assert rel_frob(dhs[pick], rdhs[pick]) <= 1e-2
    # the value-only sweep on the same rows
    kl0, none = _gpu(hs, Ws, ht, Wt, rows, None, "reverse")
    assert none is None
    assert np.abs(kl0 - kl).max() <= 1e-4


def test_empty_mask_with_gradient():
    """No masked rows: every launch has no tile to run, KL and d/dh_s are 0."""
    rng = np.random.default_rng(21)
    T, ds, dt, V = 200, 128, 64, 1000
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), 0.1)
    ht = synth.normal_bf16(rng, (T, dt), 1.0)
    Wt = synth.normal_bf16(rng, (V, dt), 0.1)
    rows = np.zeros(0, dtype=np.int32)
    gk = np.ones(T, dtype=np.float32)
    for direction in ("reverse", "forward"):
        r = torch.zeros(1, dtype=torch.int32, device="cuda")
        n = torch.zeros(1, dtype=torch.int32, device="cuda")
        st = B.new_status()
        kl, dhs = B.olive_token_divergence(hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda(), r, n, 1.0,
                                           direction, torch.from_numpy(gk).cuda(), torch.float32,
                                           dev_status=st)
        torch.cuda.synchronize()
        assert B.status_bits(st) == []
        assert not kl.any() and not dhs.any()


@pytest.mark.parametrize("direction", ["reverse", "forward"])
def test_wide_heads(direction):
    """Both heads 4096 wide: long Z jobs (K = 8192 over the two products),
    members' d_s chunks of 224 with a 64-wide last one, a partial last
    vocabulary tile and a phantom row tile."""
    rng = np.random.default_rng(33)
    T, ds, dt, V = 300, 4096, 4096, 3000
    hs = synth.rms_hidden_bf16(rng, (T, ds))
    Ws = synth.normal_bf16(rng, (V, ds), 0.02)
    ht = synth.rms_hidden_bf16(rng, (T, dt))
    Wt = synth.normal_bf16(rng, (V, dt), 0.02)
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False)).astype(np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    kl, dhs = _gpu(hs, Ws, ht, Wt, rows, gk, direction)
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, 1.0,
                                        direction, grad_kl=gk.astype(np.float64))
    assert_close_logp(kl, rkl, "kl")
    assert_close_grad(dhs, rdhs, "dH_s")
