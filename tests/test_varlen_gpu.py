"""Variable-length packed batch end to end: 64 sequences, lengths U[1024,16384],
cut at U[10%,90%] of each length (~557k packed tokens, ~278k masked rows),
d = 4096, V = 151936: splice/pack -> forward -> backward on the GPU, with the
bf16 inputs drawn by synth; log-probs, lse and dH checked against the oracle
on 2048 sampled masked rows, the rest by properties that hold at any size
(test_fwd_bwd_gpu.py checks dW on this batch's first 4096 masked rows
against the oracle).  The one-call step (olive_token_loss_fwd_bwd, G on chip)
and the slab form (olive_token_loss_fwd_bwd_slab: 15 slabs of 18304 rows, dW
through the fp32 accumulator) run on the same batch and must agree with the
two calls."""

import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (FULL_SIZE_ROWS, assert_close_logp, gpu_pack, oracle_pack, rel_frob, sample_rows,
                          to_f32)

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def test_varlen_end_to_end():
    b = synth.make_batch("varlen")
    assert 400_000 < b.T < 700_000
    h = synth.make_hidden("varlen", b.T)
    W = synth.make_weight("varlen")
    g = gpu_pack(b)
    o = oracle_pack(b)
    n = int(g["n_rows"].item())
    assert n == o["n_rows"] and np.array_equal(g["rows"][:n].cpu().numpy(), o["rows"])
    hc, Wc = h.cuda(), W.cuda()
    st = g["dev_status"]
    logp, lse, loss = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"],
                                                reduction="mean", dev_status=st)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    dh, dw = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl,
                                    reduction="mean", dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    del hc
    logp = logp.cpu().numpy()
    # rows are independent: hand the oracle only the sampled rows
    rows = sample_rows(o["rows"], FULL_SIZE_ROWS, seed=5)
    hs = to_f32(h[torch.from_numpy(rows)])
    ts = o["targets"][rows]
    local = np.arange(len(rows))
    Wf = to_f32(W)
    rl, rs, _ = oracle.token_logprob(hs, Wf, ts, local)
    assert_close_logp(logp[rows], rl, "logp")
    assert_close_logp(lse.cpu().numpy()[rows], rs, "lse")
    ref = oracle.token_loss_bwd_rows(hs, Wf, ts, local, reduction="mean", n_mask=n)
    sub = torch.from_numpy(rows).cuda()
    assert rel_frob(dh[sub].float().cpu().numpy(), ref) <= 1e-2
    # properties at full size
    all_lp = logp[o["rows"]].astype(np.float64)
    assert abs(float(loss.item()) + all_lp.mean()) <= 1e-4 * abs(all_lp.mean())
    assert abs(all_lp.mean() - (-math.log(151936) - 0.02 ** 2 * 4096 / 2)) < 0.05
    col = dw.float().sum(dim=0).abs().max().item()
    assert col <= 1e-2 * dw.float().abs().sum(dim=0).max().item()
    off = np.ones(b.T, dtype=bool)
    off[o["rows"]] = False
    off_idx = torch.from_numpy(np.nonzero(off)[0][::97]).cuda()
    assert not dh[off_idx].any().item()
    # the one-call step and the slab form against the two calls above
    hd = h.cuda()
    for slab in (False, True):
        logp2, lse2, loss2, dh2, dw2 = B.olive_token_loss_fwd_bwd(hd, Wc, g["targets"], g["rows"],
                                                                  g["n_rows"], gl, reduction="mean",
                                                                  dev_status=st, slab=slab)
        torch.cuda.synchronize()
        assert B.status_bits(st) == []
        assert np.abs(logp2.cpu().numpy()[o["rows"]] - logp[o["rows"]]).max() <= 2e-4
        assert abs(float(loss2.item()) - float(loss.item())) <= 1e-5 * abs(float(loss.item()))
        assert rel_frob(dh2[sub].float().cpu().numpy(), ref) <= 1e-2
        assert (dh2.float() - dh.float()).norm().item() <= 5e-3 * dh.float().norm().item()
        assert (dw2.float() - dw.float()).norm().item() <= 5e-3 * dw.float().norm().item()
        del logp2, lse2, loss2, dh2, dw2
        torch.cuda.empty_cache()
