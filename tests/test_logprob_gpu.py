"""olive_token_logprob_fwd (CUDA) against the oracle (Eq. (osd-ce))."""

import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_logp, assert_close_loss, gpu_pack, oracle_pack, to_f32, to_f64

pytestmark = pytest.mark.gpu


def _run(b, h, W, inv_tau=1.0, reduction="sum"):
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    logp, lse, loss = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"],
                                                inv_tau, reduction, dev_status=g["dev_status"])
    torch.cuda.synchronize()
    assert B.status_bits(g["dev_status"]) == []
    return g, logp.cpu().numpy(), lse.cpu().numpy(), float(loss.item())


def _full_check(b, h, W, inv_tau=1.0, reduction="sum"):
    g, logp, lse, loss = _run(b, h, W, inv_tau, reduction)
    o = oracle_pack(b)
    rl, rs, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"], inv_tau,
                                         reduction)
    assert_close_logp(logp, rl, "logp")
    assert_close_logp(lse, rs, "lse")
    assert_close_loss(loss, rloss)
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert np.all(logp[off] == 0) and np.all(lse[off] == 0)
    return logp


def test_tiny_workload_full():
    b = synth.make_batch("tiny")
    h = synth.make_hidden("tiny", b.T)
    W = synth.make_weight("tiny")
    _full_check(b, h, W)


@pytest.mark.parametrize("S,V,d,inv_tau,red", [
    (3, 4097, 64, 1.0, "sum"),     # one vocabulary column past a 256-tile
    (5, 300, 72, 0.7, "mean"),     # ragged K (72 = 64 + 8) and a 44-column tail tile
    (8, 1000, 128, 1.3, "sum"),    # several row tiles
    (2, 2, 64, 1.0, "sum"),        # two classes
    (12, 5000, 256, 1.0, "mean"),  # ~4 row tiles with a ragged last one
])
def test_random_shapes(S, V, d, inv_tau, red):
    b, h, W = synth.random_case(S * 31 + V, S, V, d, max_prefix=30, max_cont=80, std_h=1.0,
                                std_w=0.08)
    _full_check(b, h, W, inv_tau, red)


def test_sharp_logits_and_dominant_row():
    # large logits stress the online max; row 0 has one dominant vocabulary entry
    b, h, W = synth.random_case(5, 4, 3000, 64, std_h=3.0, std_w=0.5)
    W = W.clone()
    o = oracle_pack(b)
    t0 = int(o["rows"][0])
    y0 = int(o["targets"][t0])
    h = h.clone()
    h[t0] = 0
    h[t0, 0] = 1.0
    W[y0, 0] = 30.0
    logp = _full_check(b, h, W)
    assert abs(logp[t0]) < 1e-3


def test_uniform_logits_closed_form():
    b = synth.batch_from_lengths(np.random.default_rng(3), [5, 9], [40, 70], 4096)
    h = synth.normal_bf16(np.random.default_rng(4), (b.T, 128), 1.0)
    W = torch.zeros(4096, 128, dtype=torch.bfloat16)
    g, logp, lse, loss = _run(b, h, W)
    o = oracle_pack(b)
    assert np.allclose(logp[o["rows"]], -math.log(4096), atol=1e-5)
    assert abs(loss - 110 * math.log(4096)) <= 1e-4 * loss


def test_empty_and_single_row():
    # N_mask = 0: loss 0 and every output row 0
    b = synth.batch_from_lengths(np.random.default_rng(5), [7, 3], [0, 0], 500)
    h = synth.normal_bf16(np.random.default_rng(6), (b.T, 64), 1.0)
    W = synth.normal_bf16(np.random.default_rng(7), (500, 64), 0.1)
    for red in ("sum", "mean"):
        g, logp, lse, loss = _run(b, h, W, reduction=red)
        assert loss == 0.0 and not logp.any() and not lse.any()
    b1 = synth.batch_from_lengths(np.random.default_rng(8), [4], [1], 500)
    h1 = synth.normal_bf16(np.random.default_rng(9), (b1.T, 64), 1.0)
    _full_check(b1, h1, W)


def test_permuted_vocabulary_gives_same_logp():
    b, h, W = synth.random_case(11, 6, 2000, 128, std_w=0.1)
    g, base, _, _ = _run(b, h, W)
    perm = torch.from_numpy(np.random.default_rng(0).permutation(2000))
    inv = torch.argsort(perm)
    b2 = synth.Batch(inv[torch.from_numpy(b.prefix_ids.astype(np.int64))].numpy().astype(np.int32),
                     b.prefix_off,
                     inv[torch.from_numpy(b.cont_ids.astype(np.int64))].numpy().astype(np.int32),
                     b.cont_off, b.V)
    _, perm_logp, _, _ = _run(b2, h, W[perm].contiguous())
    assert np.allclose(base, perm_logp, atol=2e-5, rtol=1e-5)


def test_target_out_of_range_flagged():
    b = synth.batch_from_lengths(np.random.default_rng(12), [3], [5], 100)
    g = gpu_pack(b)
    tg = g["targets"].clone()
    rows = g["rows"][:1].long()
    tg[rows] = 150
    h = synth.normal_bf16(np.random.default_rng(13), (b.T, 64), 1.0).cuda()
    W = synth.normal_bf16(np.random.default_rng(14), (100, 64), 0.1).cuda()
    st = B.new_status()
    logp, _, _ = B.olive_token_logprob_fwd(h, W, tg, g["rows"], g["n_rows"], dev_status=st)
    assert "OLIVE_ERR_TOKEN_RANGE" in B.status_bits(st)
    assert math.isnan(float(logp[rows].item()))


@pytest.mark.slow
def test_scoring_workload_full():
    """2 x (4096 + 4096) tokens, d = 2048, V = 151936: the oracle recomputes
    every one of the 8192 masked rows, so log-probs, lse and the loss are
    compared in full (element by element, and the loss to 1e-3 relative)."""
    b = synth.make_batch("scoring")
    h = synth.make_hidden("scoring", b.T)
    W = synth.make_weight("scoring")
    g, logp, lse, loss = _run(b, h, W)
    o = oracle_pack(b)
    assert o["n_rows"] == 8192
    rl, rs, rloss = oracle.token_logprob(to_f32(h), to_f32(W), o["targets"], o["rows"])
    assert_close_logp(logp, rl, "logp")
    assert_close_logp(lse[o["rows"]], rs[o["rows"]], "lse")
    assert_close_loss(loss, rloss)
    # properties at full size: loss = -sum logp, logp <= 0, statistical band
    all_lp = logp[o["rows"]].astype(np.float64)
    assert np.all(all_lp <= 1e-6)
    assert abs(loss + all_lp.sum()) <= 1e-4 * abs(loss)
    sigma2 = 0.02 ** 2 * 2048
    assert abs(all_lp.mean() - (-math.log(151936) - sigma2 / 2)) < 0.05


def _integer_case(seed, S=6, V=3001, d=64):
    """bf16 inputs that are small integers (h in {-2..2}, W in {-1, 0, 1},
    mostly 0), so every logit is an integer of magnitude <= 2 d that fp32 and
    fp64 both hold exactly: only the exp / log / accumulation error is left."""
    rng = np.random.default_rng(seed)
    b = synth.batch_from_lengths(rng, rng.integers(1, 40, size=S), rng.integers(0, 120, size=S), V)
    h = torch.from_numpy(rng.integers(-2, 3, size=(b.T, d)).astype(np.float32)).to(torch.bfloat16)
    Wf = rng.integers(-1, 2, size=(V, d)).astype(np.float32)
    Wf *= rng.random(size=(V, d)) < 0.05
    W = torch.from_numpy(Wf).to(torch.bfloat16)
    return b, h, W


@pytest.mark.parametrize("seed", [0, 1])
def test_exact_integer_logits(seed):
    """With exact logits the GPU's log-probs carry only fp32 exp/log and
    accumulation error: 1e-5 + 1e-6 |logp|, 200x tighter than the general
    bound, for the forward and the single-pass forward + backward."""
    b, h, W = _integer_case(seed)
    z = to_f64(h) @ to_f64(W).T
    assert np.array_equal(z, np.round(z)) and np.abs(z).max() < 2 ** 24
    _, logp, lse, _ = _run(b, h, W)
    o = oracle_pack(b)
    rl, rs, _ = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"])
    r = o["rows"]
    assert np.abs(logp[r] - rl[r]).max() <= 1e-5 + 1e-6 * np.abs(rl[r]).max()
    assert np.abs(lse[r] - rs[r]).max() <= 1e-5 + 1e-6 * np.abs(rs[r]).max()
    g = gpu_pack(b)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    logp2, lse2, _, _, _ = B.olive_token_loss_fwd_bwd(h.cuda(), W.cuda(), g["targets"], g["rows"],
                                                      g["n_rows"], gl, dev_status=g["dev_status"])
    torch.cuda.synchronize()
    assert B.status_bits(g["dev_status"]) == []
    assert np.abs(logp2.cpu().numpy()[r] - rl[r]).max() <= 1e-5 + 1e-6 * np.abs(rl[r]).max()


def test_constant_column_shift_invariance():
    """A hidden unit fixed at 1 with W[:, j] = c adds c to every logit of the
    row: log-probs and the gradient with respect to the other units do not
    change (the softmax is shift invariant); lse moves by exactly c."""
    rng = np.random.default_rng(8)
    b = synth.batch_from_lengths(rng, rng.integers(1, 40, size=5), rng.integers(1, 150, size=5), 2000)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    h[:, 63] = 1.0
    W = synth.normal_bf16(rng, (2000, 64), 0.3)
    g = gpu_pack(b)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    res = []
    for c in (0.0, 24.0):
        Wc = W.clone()
        Wc[:, 63] = c
        out = B.olive_token_loss_fwd_bwd(h.cuda(), Wc.cuda(), g["targets"], g["rows"], g["n_rows"],
                                         gl, grad_dtype=torch.float32, dev_status=g["dev_status"])
        res.append([t.cpu().numpy() for t in out])
    torch.cuda.synchronize()
    assert B.status_bits(g["dev_status"]) == []
    o = oracle_pack(b)
    r = o["rows"]
    (l0, s0, _, dh0, dw0), (l1, s1, _, dh1, dw1) = res
    assert np.abs(l1[r] - l0[r]).max() <= 2e-5 * (1 + np.abs(l0[r]).max())
    assert np.abs((s1[r] - s0[r]) - 24.0).max() <= 1e-4
    assert np.linalg.norm(dh1[:, :63] - dh0[:, :63]) <= 2e-2 * np.linalg.norm(dh0[:, :63])
    assert np.linalg.norm(dw1[:, :63] - dw0[:, :63]) <= 2e-2 * np.linalg.norm(dw0[:, :63])
