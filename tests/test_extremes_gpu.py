"""Extreme shapes against the oracle: the narrowest hidden widths (d < one
64-wide TMA box), a single-entry vocabulary, a long reduction (d = 8192) and
a vocabulary of 2^18 + 3 entries (ragged last tile, many segments)."""


import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (assert_close_grad, assert_close_logp, assert_close_loss, gpu_pack,
                          oracle_pack, to_f64)

pytestmark = pytest.mark.gpu


def _fwd_bwd(b, h, W, grad_dtype=torch.float32):
    g = gpu_pack(b)
    hc, Wc = h.cuda(), W.cuda()
    st = g["dev_status"]
    logp, lse, loss = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"],
                                                dev_status=st)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    dh, dw = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl,
                                    grad_dtype=grad_dtype, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return logp.cpu().numpy(), float(loss.item()), dh.float().cpu().numpy(), dw.float().cpu().numpy()


def _check(b, h, W, **kw):
    logp, loss, dh, dw = _fwd_bwd(b, h, W, **kw)
    o = oracle_pack(b)
    rl, _, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"])
    assert_close_logp(logp, rl)
    assert_close_loss(loss, rloss)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"])
    assert_close_grad(dh, rdh, "dH")
    assert_close_grad(dw, rdw, "dW")


@pytest.mark.parametrize("d", [8, 16, 24])
def test_narrow_hidden_width(d):
    b, h, W = synth.random_case(300 + d, 5, 700, d, max_prefix=30, max_cont=60, std_w=0.3)
    _check(b, h, W)


def test_single_entry_vocabulary():
    rng = np.random.default_rng(4)
    b = synth.batch_from_lengths(rng, [3, 5], [7, 4], 1)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0)
    W = synth.normal_bf16(rng, (1, 64), 0.3)
    logp, loss, dh, dw = _fwd_bwd(b, h, W)
    # log p = z - lse = 0 exactly in real arithmetic; fp32 leaves a few ulp
    assert np.abs(logp).max() <= 1e-6 and abs(loss) <= 1e-5
    # softmax - onehot = 0: the gradients vanish up to the same rounding
    assert np.abs(dh).max() <= 1e-5 and np.abs(dw).max() <= 1e-5


def test_long_reduction_d8192():
    b, h, W = synth.random_case(41, 4, 1000, 8192, max_prefix=40, max_cont=70, std_h=1.0,
                                std_w=0.01)
    _check(b, h, W)


@pytest.mark.slow
def test_vocab_2pow18_plus_3():
    V = (1 << 18) + 3
    b, h, W = synth.random_case(42, 3, V, 64, max_prefix=20, max_cont=70, std_w=0.2)
    _check(b, h, W, grad_dtype=torch.bfloat16)
    # the top-16 sweep over the same vocabulary
    o = oracle_pack(b)
    r = torch.from_numpy(o["rows"].astype(np.int32)).cuda()
    n = torch.tensor([o["n_rows"]], dtype=torch.int32, device="cuda")
    lse, ent, tv, ti = B.olive_token_topk_fwd(h.cuda(), W.cuda(), r, n, 16)
    rl, rH, rv, ri = oracle.token_topk(to_f64(h), to_f64(W), o["rows"], 16)
    assert_close_logp(lse.cpu().numpy(), rl)
    assert_close_logp(ent.cpu().numpy(), rH)
    assert_close_logp(tv.cpu().numpy(), rv)
