"""olive_token_loss_bwd (CUDA) against the oracle gradients of Eq. (osd-ce)."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (assert_close_grad, gpu_pack, oracle_pack, rel_frob, sample_rows, to_f32,
                          to_f64)

pytestmark = pytest.mark.gpu


def _gpu_grads(b, h, W, inv_tau=1.0, reduction="sum", grad_loss=1.0, grad_dtype=torch.bfloat16):
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    st = g["dev_status"]
    _, lse, _ = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], inv_tau,
                                          reduction, dev_status=st)
    gl = torch.tensor([grad_loss], dtype=torch.float32, device="cuda")
    dh, dw = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl, inv_tau,
                                    reduction, grad_dtype=grad_dtype, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return dh.float().cpu().numpy(), dw.float().cpu().numpy()


def _full_check(b, h, W, **kw):
    dh, dw = _gpu_grads(b, h, W, **kw)
    o = oracle_pack(b)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"],
                                     kw.get("inv_tau", 1.0), kw.get("reduction", "sum"),
                                     kw.get("grad_loss", 1.0))
    assert_close_grad(dh, rdh, "dH")
    assert_close_grad(dw, rdw, "dW")
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert not dh[off].any()
    return dh, dw


def test_tiny_workload_full():
    b = synth.make_batch("tiny")
    _full_check(b, synth.make_hidden("tiny", b.T), synth.make_weight("tiny"))


@pytest.mark.parametrize("S,V,d,kw", [
    (3, 4097, 64, dict()),
    (5, 300, 72, dict(inv_tau=0.7, reduction="mean", grad_loss=2.5)),
    (8, 1000, 128, dict(grad_dtype=torch.float32)),
    (12, 5000, 256, dict(reduction="mean", grad_dtype=torch.float32)),
    (4, 700, 320, dict(inv_tau=1.2)),  # d = 320: a partial 256-wide output tile
])
def test_random_shapes(S, V, d, kw):
    b, h, W = synth.random_case(S * 17 + V, S, V, d, max_prefix=30, max_cont=80, std_w=0.08)
    _full_check(b, h, W, **kw)


@pytest.mark.parametrize("slab_rows,grad_dtype", [(4096, torch.float32), (1024, torch.bfloat16)])
def test_several_slabs(slab_rows, grad_dtype, monkeypatch):
    """17000 masked rows with the slab cap lowered: G goes through several
    slabs, which wait on each other inside the one launch, and dW accumulates
    (fp32 accumulator for a bf16 output)."""
    monkeypatch.setenv("OLIVE_SLAB_ROWS", str(slab_rows))
    rng = np.random.default_rng(21)
    b = synth.batch_from_lengths(rng, [1] * 10, [1700] * 10, 600)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    W = synth.normal_bf16(rng, (600, 64), 0.1)
    assert b.n_mask > 4 * slab_rows
    _full_check(b, h, W, grad_dtype=grad_dtype)


def test_empty_mask_gives_zero_grads():
    b = synth.batch_from_lengths(np.random.default_rng(22), [9, 4], [0, 0], 300)
    h = synth.normal_bf16(np.random.default_rng(23), (b.T, 64), 1.0)
    W = synth.normal_bf16(np.random.default_rng(24), (300, 64), 0.1)
    dh, dw = _gpu_grads(b, h, W)
    assert not dh.any() and not dw.any()


def test_vocab_sum_of_dW_vanishes():
    b, h, W = synth.random_case(25, 6, 3000, 128, std_w=0.1)
    dh, dw = _gpu_grads(b, h, W, grad_dtype=torch.float32)
    col = np.abs(dw.sum(axis=0)).max()
    assert col <= 1e-3 * np.abs(dw).sum(axis=0).max()


@pytest.mark.slow
def test_medium_vocab_sampled_dh_and_dw():
    """~8k masked rows, d = 4096, V = 32003 (ragged last tile): dH on sampled
    rows and dW on sampled vocabulary rows, both against the oracle."""
    rng = np.random.default_rng(31)
    b = synth.batch_from_lengths(rng, [1000, 777, 2048], [3000, 2500, 2700], 32003)
    h = synth.rms_hidden_bf16(rng, (b.T, 4096))
    W = synth.normal_bf16(rng, (32003, 4096), 0.02)
    dh, dw = _gpu_grads(b, h, W, reduction="mean")
    o = oracle_pack(b)
    rows = sample_rows(o["rows"], 24, seed=3)
    ref = oracle.token_loss_bwd_rows(to_f32(h), to_f32(W), o["targets"], rows, reduction="mean",
                                     n_mask=o["n_rows"])
    assert rel_frob(dh[rows], ref) <= 1e-2
    # a target id, the last (ragged) tile and random ids
    vocab = np.unique(np.concatenate([[int(o["targets"][o["rows"][0]]), 0, 32002],
                                      np.random.default_rng(4).integers(0, 32003, size=13)]))
    refw = oracle.token_loss_bwd_vocab(to_f32(h), to_f32(W), o["targets"], o["rows"], vocab,
                                       reduction="mean")
    assert rel_frob(dw[vocab], refw) <= 1e-2


@pytest.mark.slow
def test_fwdbwd_workload_sampled():
    """8 x 4096 tokens, d = 4096, V = 151936: dH on sampled rows from the oracle;
    dW checked through its exact vocabulary-sum identity and magnitude."""
    b = synth.make_batch("fwdbwd")
    h = synth.make_hidden("fwdbwd", b.T)
    W = synth.make_weight("fwdbwd")
    dh, dw = _gpu_grads(b, h, W)
    o = oracle_pack(b)
    rows = sample_rows(o["rows"], 24, seed=1)
    ref = oracle.token_loss_bwd_rows(to_f32(h), to_f32(W), o["targets"], rows)
    assert rel_frob(dh[rows], ref) <= 1e-2
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert not dh[off].any()
    colsum = np.abs(dw.astype(np.float64).sum(axis=0)).max()
    assert colsum <= 1e-2 * np.abs(dw).sum(axis=0).max()


def test_two_column_sweeps():
    """d one 64-column tail wider than one sweep of the on-chip backward (the
    lse given): passes A and B run twice, the second time over the last 64
    columns with groups of one member."""
    rng = np.random.default_rng(23)
    sms = min(torch.cuda.get_device_properties(0).multi_processor_count, 192)
    d = sms // 2 * 256 + 64
    b = synth.batch_from_lengths(rng, [11, 25], [70, 140], 500)
    h = synth.rms_hidden_bf16(rng, (b.T, d))
    W = synth.normal_bf16(rng, (500, d), 0.01)
    _full_check(b, h, W, reduction="mean", grad_dtype=torch.float32)
