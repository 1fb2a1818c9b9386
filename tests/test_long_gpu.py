"""Full-size checks of every output of the timed training step (run with
--long): the bench's batch (8 x 4096 tokens, cut ~ U[256, 3840), d = 4096,
V = 151936, N_mask = 16711) through olive_token_loss_fwd_bwd, against the
oracle's token_logprob and token_loss_bwd over the whole batch (about
6e13 fp64 flops, several minutes on the host cores).  Every log-prob and lse
element by element, the loss to 1e-3 relative, dH and dW (bf16, as the bench
stores them) to 1e-2 relative Frobenius, as in the other parity tests."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import (assert_close_grad, assert_close_logp, assert_close_loss, gpu_pack, oracle_pack,
                          to_f32)

pytestmark = [pytest.mark.gpu, pytest.mark.slow, pytest.mark.long]


def test_fwdbwd_workload_every_output():
    b = synth.make_batch("fwdbwd")
    h = synth.make_hidden("fwdbwd", b.T)
    W = synth.make_weight("fwdbwd")
    g = gpu_pack(b)
    st = g["dev_status"]
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    logp, lse, loss, dh, dw = B.olive_token_loss_fwd_bwd(h.cuda(), W.cuda(), g["targets"], g["rows"],
                                                         g["n_rows"], gl, grad_dtype=torch.bfloat16,
                                                         dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    logp, lse, loss = logp.cpu().numpy(), lse.cpu().numpy(), float(loss.item())
    dh, dw = dh.float().cpu().numpy(), dw.float().cpu().numpy()
    torch.cuda.empty_cache()

    o = oracle_pack(b)
    assert o["n_rows"] == 16711
    hf, Wf = to_f32(h), to_f32(W)
    rl, rlse, rloss = oracle.token_logprob(hf, Wf, o["targets"], o["rows"])
    assert_close_logp(logp, rl, "logp")
    assert_close_logp(lse[o["rows"]], rlse[o["rows"]], "lse")
    assert_close_loss(loss, rloss)
    rdh, rdw = oracle.token_loss_bwd(hf, Wf, o["targets"], o["rows"])
    assert_close_grad(dh, rdh, "dH")
    assert_close_grad(dw, rdw, "dW")
    off = np.setdiff1d(np.arange(b.T), o["rows"])
    assert not dh[off].any() and not logp[off].any()
