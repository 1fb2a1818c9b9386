"""olive_token_loss_fwd_bwd (CUDA: forward and backward of Eq. (osd-ce), G
formed and consumed on chip) and olive_token_loss_fwd_bwd_slab (the same step
through an HBM slab of G) against the oracle's token_logprob and
token_loss_bwd."""


import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (FULL_SIZE_ROWS, assert_close_grad, assert_close_logp, assert_close_loss,
                          gpu_pack, oracle_pack, rel_frob, sample_rows, to_f32, to_f64)

pytestmark = pytest.mark.gpu


FORMS = ["onchip", "slab"]


def _gpu(b, h, W, inv_tau=1.0, reduction="sum", grad_loss=1.0, grad_dtype=torch.bfloat16,
         form="onchip", n_rows=None):
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    st = g["dev_status"]
    gl = torch.tensor([grad_loss], dtype=torch.float32, device="cuda")
    nr = g["n_rows"] if n_rows is None else torch.tensor([n_rows], dtype=torch.int32, device="cuda")
    logp, lse, loss, dh, dw = B.olive_token_loss_fwd_bwd(hc, Wc, g["targets"], g["rows"], nr,
                                                         gl, inv_tau, reduction, grad_dtype,
                                                         dev_status=st, slab=form == "slab")
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return (logp.cpu().numpy(), lse.cpu().numpy(), float(loss.item()), dh.float().cpu().numpy(),
            dw.float().cpu().numpy())


def _full_check(b, h, W, **kw):
    logp, lse, loss, dh, dw = _gpu(b, h, W, **kw)
    o = oracle_pack(b)
    tau, red = kw.get("inv_tau", 1.0), kw.get("reduction", "sum")
    rl, rlse, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"], tau, red)
    assert_close_logp(logp, rl)
    assert_close_logp(lse[o["rows"]], rlse[o["rows"]], "lse")
    assert_close_loss(loss, rloss)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"], tau, red,
                                     kw.get("grad_loss", 1.0))
    assert_close_grad(dh, rdh, "dH")
    assert_close_grad(dw, rdw, "dW")
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert not dh[off].any() and not logp[off].any()
    return logp, dh, dw


@pytest.mark.parametrize("form", FORMS)
def test_tiny_workload_full(form):
    b = synth.make_batch("tiny")
    _full_check(b, synth.make_hidden("tiny", b.T), synth.make_weight("tiny"), form=form)


@pytest.mark.parametrize("form", FORMS)
@pytest.mark.parametrize("S,V,d,kw", [
    (3, 4097, 64, dict()),
    (5, 300, 72, dict(inv_tau=0.7, reduction="mean", grad_loss=2.5)),
    (8, 1000, 128, dict(grad_dtype=torch.float32)),
    (12, 5000, 256, dict(reduction="mean", grad_dtype=torch.float32)),
    (4, 700, 320, dict(inv_tau=1.2)),  # d = 320: a partial 256-wide output tile
    (7, 13, 24, dict()),               # V below one 8-wide vector group
])
def test_random_shapes(S, V, d, kw, form):
    b, h, W = synth.random_case(S * 17 + V, S, V, d, max_prefix=30, max_cont=80, std_w=0.08)
    _full_check(b, h, W, form=form, **kw)


@pytest.mark.parametrize("form", FORMS)
def test_single_entry_vocabulary(form):
    rng = np.random.default_rng(4)
    b = synth.batch_from_lengths(rng, [3, 5], [7, 4], 1)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    W = synth.normal_bf16(rng, (1, 64), 0.3)
    logp, _, loss, dh, dw = _gpu(b, h, W, grad_dtype=torch.float32, form=form)
    # log p = 0 and G = p - 1 = 0 in real arithmetic; fp32 leaves a few ulp
    assert np.abs(logp).max() <= 1e-6 and abs(loss) <= 1e-5
    assert np.abs(dh).max() <= 1e-5 and np.abs(dw).max() <= 1e-5


@pytest.mark.parametrize("form", FORMS)
def test_matches_the_two_call_path(form):
    b, h, W = synth.random_case(77, 6, 3001, 128, max_prefix=40, max_cont=200, std_w=0.1)
    logp, dh, dw = _full_check(b, h, W, grad_dtype=torch.float32, form=form)
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    l2, lse2, _ = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"])
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    dh2, dw2 = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse2, gl,
                                      grad_dtype=torch.float32)
    assert np.abs(logp - l2.cpu().numpy()).max() <= 1e-4
    assert rel_frob(dh, dh2.cpu().numpy()) <= 5e-3
    assert rel_frob(dw, dw2.cpu().numpy()) <= 5e-3


@pytest.mark.parametrize("slab_rows,grad_dtype", [(256, torch.float32), (384, torch.bfloat16)])
def test_several_slabs(slab_rows, grad_dtype, monkeypatch):
    """The slab form with a lowered slab cap splits ~2.3k masked rows into many
    slabs: dW accumulates across them (fp32 accumulator for a bf16 output)."""
    monkeypatch.setenv("OLIVE_SLAB_ROWS", str(slab_rows))
    rng = np.random.default_rng(slab_rows)
    b = synth.batch_from_lengths(rng, [5, 40, 1], [900, 700, 750], 2000)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    W = synth.normal_bf16(rng, (2000, 64), 0.1)
    assert b.n_mask > 6 * slab_rows
    _full_check(b, h, W, reduction="mean", grad_dtype=grad_dtype, form="slab")


@pytest.mark.parametrize("grad_dtype", [torch.float32, torch.bfloat16])
def test_many_outer_tiles(grad_dtype):
    """~2.3k masked rows, d = 4096, V = 2000 on the on-chip form: groups of 16
    CTAs, 19 row tiles (pass A) and 16 vocabulary tiles (pass B) over 9
    groups, so groups run several outer tiles in both passes, the exchange
    ring wraps many times and the last vocabulary tile is partial."""
    rng = np.random.default_rng(991)
    b = synth.batch_from_lengths(rng, [5, 40, 1], [900, 700, 750], 2000)
    h = synth.rms_hidden_bf16(rng, (b.T, 4096))
    W = synth.normal_bf16(rng, (2000, 4096), 0.03)
    _full_check(b, h, W, reduction="mean", grad_dtype=grad_dtype)


def _two_sweep_width():
    """A width one 64-column tail past what one sweep of the on-chip form
    covers on this device (128 pairs of CTAs at most, 256 columns per member
    of a group spanning all of them)."""
    sms = min(torch.cuda.get_device_properties(0).multi_processor_count, 192)
    return sms // 2 * 256 + 64


def test_two_column_sweeps():
    """d wider than one sweep: the on-chip form runs passes A and B twice, the
    second sweep over the last 64 output columns with groups of one member,
    with the forward outputs written by the first sweep only."""
    rng = np.random.default_rng(19)
    d = _two_sweep_width()
    b = synth.batch_from_lengths(rng, [7, 30], [90, 120], 600)
    h = synth.rms_hidden_bf16(rng, (b.T, d))
    W = synth.normal_bf16(rng, (600, d), 0.01)
    _full_check(b, h, W, reduction="mean", grad_dtype=torch.float32)


@pytest.mark.parametrize("form", FORMS)
def test_empty_mask(form):
    rng = np.random.default_rng(22)
    b = synth.batch_from_lengths(rng, [9, 4], [0, 0], 300)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    W = synth.normal_bf16(rng, (300, 64), 0.1)
    logp, _, loss, dh, dw = _gpu(b, h, W, reduction="mean", form=form)
    assert loss == 0.0 and not logp.any() and not dh.any() and not dw.any()


@pytest.mark.parametrize("form", FORMS)
@pytest.mark.parametrize("spike", [0.2, 0.5])
def test_rows_far_above_their_first_tile(spike, form):
    """Each row's stored e' = 2^(x - R) is relative to the maximum R over the
    row's first 256 vocabulary entries.  Here one id far down the vocabulary
    (1000) has a logit 31-39 nats (spike 0.2: e' up to ~2^57, the scaled form)
    or 78-101 nats (spike 0.5: more than 2^100 above R, so its half tile keeps
    its own maximum and the row is rewritten relative to lse) above the first
    tile on half of the rows; the other rows stay unremarkable."""
    rng = np.random.default_rng(int(spike * 10))
    S, V, d = 6, 3000, 64
    b = synth.batch_from_lengths(rng, [20] * S, [60] * S, V)
    h = synth.normal_bf16(rng, (b.T, d), 1.0).float()
    h[::2] += 3.0                                   # sum over d ~ 192 on even rows
    h = h.to(torch.bfloat16)
    W = synth.normal_bf16(rng, (V, d), 0.05).float()
    W[1000] = spike
    W = W.to(torch.bfloat16)
    z = oracle.logits(to_f64(h), to_f64(W), 1.0)
    gap = (z.max(axis=1) - z[:, :256].max(axis=1))[::2]
    assert gap.min() > (25 if spike < 0.3 else 75)
    _full_check(b, h, W, grad_dtype=torch.float32, form=form)


@pytest.mark.parametrize("form", FORMS)
def test_confident_rows_keep_their_accuracy(form):
    """Targets equal to a dominant logit (p_y close to 1): G_y = g (p_y - 1) is
    small and formed from the fp32 target logit (a bf16-rounded p_y would be
    off by up to 2^-9 p_y), so each such row's dH keeps the gradient tolerance
    on its own.  Rows with 1 - p_y below ~1e-4 are left out: there fp32 itself
    (an ulp of the logit against 1 - p_y) bounds every implementation."""
    rng = np.random.default_rng(5)
    P, C, V, d = 40, 300, 1000, 64
    h = synth.normal_bf16(rng, (P + C, d), 1.0)
    W = synth.normal_bf16(rng, (V, d), 1.2)
    z = oracle.logits(to_f64(h), to_f64(W), 1.0)
    cont = np.argmax(z[P - 1:P + C - 1], axis=1)          # the target of row P-1+i is cont[i]
    b = synth.Batch(rng.integers(0, V, size=P).astype(np.int32), np.array([0, P], np.int32),
                    cont.astype(np.int32), np.array([0, C], np.int32), V)
    logp, dh, _ = _full_check(b, h, W, grad_dtype=torch.float32, form=form)
    o = oracle_pack(b)
    rdh, _ = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"])
    conf = [t for t in o["rows"] if -0.3 < logp[t] < -1e-2]
    assert len(conf) >= 30
    for t in conf:
        assert rel_frob(dh[t], rdh[t]) <= 2e-2, t


@pytest.mark.slow
def test_medium_vocab_sampled():
    """~8k masked rows, d = 4096, V = 32003: logp everywhere, dH on sampled
    rows and dW on sampled vocabulary rows."""
    rng = np.random.default_rng(31)
    b = synth.batch_from_lengths(rng, [1000, 777, 2048], [3000, 2500, 2700], 32003)
    h = synth.rms_hidden_bf16(rng, (b.T, 4096))
    W = synth.normal_bf16(rng, (32003, 4096), 0.02)
    logp, _, loss, dh, dw = _gpu(b, h, W, reduction="mean")
    o = oracle_pack(b)
    rows = sample_rows(o["rows"], 24, seed=3)
    rl, _, _ = oracle.token_logprob(to_f32(h), to_f32(W), o["targets"], rows)
    assert_close_logp(logp[rows], rl[rows])
    ref = oracle.token_loss_bwd_rows(to_f32(h), to_f32(W), o["targets"], rows, reduction="mean",
                                     n_mask=o["n_rows"])
    assert rel_frob(dh[rows], ref) <= 1e-2
    vocab = np.unique(np.concatenate([[int(o["targets"][o["rows"][0]]), 0, 32002],
                                      np.random.default_rng(4).integers(0, 32003, size=13)]))
    refw = oracle.token_loss_bwd_vocab(to_f32(h), to_f32(W), o["targets"], o["rows"], vocab,
                                       reduction="mean")
    assert rel_frob(dw[vocab], refw) <= 1e-2
    assert np.isclose(loss, -logp[o["rows"]].astype(np.float64).mean(), rtol=1e-5)


@pytest.mark.slow
def test_fwdbwd_workload_sampled():
    """8 x 4096 tokens, d = 4096, V = 151936 (the timed step's configuration):
    log-probs, lse and dH on 2048 sampled masked rows, dW on 40 vocabulary
    rows against the oracle and through the vocabulary-sum property, dH = 0
    off the mask, loss = -sum logp."""
    b = synth.make_batch("fwdbwd")
    h = synth.make_hidden("fwdbwd", b.T)
    W = synth.make_weight("fwdbwd")
    logp, lse, loss, dh, dw = _gpu(b, h, W)
    o = oracle_pack(b)
    rows = sample_rows(o["rows"], FULL_SIZE_ROWS, seed=1)
    hf, Wf = to_f32(h), to_f32(W)
    rl, rlse, _ = oracle.token_logprob(hf, Wf, o["targets"], rows)
    assert_close_logp(logp[rows], rl[rows])
    assert_close_logp(lse[rows], rlse[rows], "lse")
    ref = oracle.token_loss_bwd_rows(hf, Wf, o["targets"], rows)
    assert rel_frob(dh[rows], ref) <= 1e-2
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert not dh[off].any()
    # dW on 40 vocabulary rows (16 of them targets of sampled rows, the first
    # and the last id) against the oracle, which forms every masked row's
    # softmax for them (about 2e13 fp64 flops)
    V = W.shape[0]
    rng = np.random.default_rng(8)
    vocab = np.unique(np.concatenate([o["targets"][rows[:16]], [0, V - 1],
                                      rng.integers(0, V, size=22)]))
    refw = oracle.token_loss_bwd_vocab(hf, Wf, o["targets"], o["rows"], vocab)
    assert rel_frob(dw[vocab], refw) <= 1e-2
    # sum over the vocabulary of dW is sum_r G[r, :] . hc[r] with sum_v G[r, v] = 0
    assert np.abs(dw.astype(np.float64).sum(axis=0)).max() <= 2e-2 * np.abs(dw).sum(axis=0).max()
    assert np.isclose(loss, -logp[o["rows"]].astype(np.float64).sum(), rtol=1e-5)


@pytest.mark.slow
def test_varlen_rows_dw():
    """The variable-length batch (~528k packed tokens) with N_mask lowered to
    its first 4096 masked rows (spread over its first sequences): every
    output of the on-chip step against the oracle, dW on 40 vocabulary rows
    (targets among them) and dH, log-probs, lse on every one of those rows."""
    b = synth.make_batch("varlen")
    h = synth.make_hidden("varlen", b.T)
    W = synth.make_weight("varlen")
    n = 4096
    g = gpu_pack(b)
    st = g["dev_status"]
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    nr = torch.tensor([n], dtype=torch.int32, device="cuda")
    logp, lse, loss, dh, dw = B.olive_token_loss_fwd_bwd(h.cuda(), W.cuda(), g["targets"], g["rows"],
                                                         nr, gl, 1.0, "mean", dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    o = oracle_pack(b)
    rows = o["rows"][:n]
    sub = torch.from_numpy(rows).cuda()
    hs = to_f32(h[torch.from_numpy(rows)])
    ts = o["targets"][rows]
    local = np.arange(n)
    Wf = to_f32(W)
    rl, rs, rloss = oracle.token_logprob(hs, Wf, ts, local, reduction="mean")
    assert_close_logp(logp[sub].cpu().numpy(), rl)
    assert_close_logp(lse[sub].cpu().numpy(), rs, "lse")
    assert_close_loss(float(loss.item()), rloss)
    ref = oracle.token_loss_bwd_rows(hs, Wf, ts, local, reduction="mean")
    assert rel_frob(dh[sub].float().cpu().numpy(), ref) <= 1e-2
    V = W.shape[0]
    vocab = np.unique(np.concatenate([ts[:20], [0, V - 1], np.random.default_rng(9).integers(0, V, 18)]))
    refw = oracle.token_loss_bwd_vocab(hs, Wf, ts, local, vocab, reduction="mean")
    got = dw[torch.from_numpy(vocab).cuda()].float().cpu().numpy()
    assert rel_frob(got, refw) <= 1e-2
    rest = torch.from_numpy(o["rows"][n::101]).cuda()
    assert not dh[rest].any().item()


def test_runs_are_bitwise_reproducible():
    """Every reduction on these paths runs in a fixed order (per-row merges in
    tile order, the loss in one block, dW per slab): two runs agree bit for
    bit, for the single-pass call and for the two-call path."""
    b, h, W = synth.random_case(91, 8, 5000, 192, max_prefix=50, max_cont=400, std_w=0.1)
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    gl = torch.tensor([0.7], dtype=torch.float32, device="cuda")
    runs = []
    for _ in range(2):
        a = B.olive_token_loss_fwd_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], gl, 1.1, "mean")
        _, lse, loss = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], 1.1,
                                                 "mean")
        dh, dw = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl, 1.1,
                                        "mean")
        runs.append([t.clone() for t in (*a, lse, loss, dh, dw)])
    torch.cuda.synchronize()
    for x, y in zip(*runs):
        assert torch.equal(x, y)
