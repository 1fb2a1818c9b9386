"""Failure detection without a GPU fault: every internal wait of the GEMM
kernels is bounded (OLIVE_WAIT_LIMIT_MS, read on each call).  With a limit of
0 ms the first wait that is not already satisfied gives up; the kernels must
then drain what they issued, free their tensor memory, return, and report
OLIVE_ERR_TIMEOUT in the device status word, leaving the CUDA context usable
for the next (normal) call."""

import os

import numpy as np
import pytest
import torch

from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import gpu_pack

pytestmark = pytest.mark.gpu


@pytest.fixture
def zero_wait_limit():
    old = os.environ.get("OLIVE_WAIT_LIMIT_MS")
    os.environ["OLIVE_WAIT_LIMIT_MS"] = "0"
    yield
    if old is None:
        del os.environ["OLIVE_WAIT_LIMIT_MS"]
    else:
        os.environ["OLIVE_WAIT_LIMIT_MS"] = old


def _case():
    b, h, W = synth.random_case(3, 6, 20000, 512, max_prefix=40, max_cont=200, std_w=0.05)
    return b, h.cuda(), W.cuda()


def _fwd_bwd(b, h, W, st):
    g = gpu_pack(b)
    _, lse, loss = B.olive_token_logprob_fwd(h, W, g["targets"], g["rows"], g["n_rows"], dev_status=st)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    dh, dw = B.olive_token_loss_bwd(h, W, g["targets"], g["rows"], g["n_rows"], lse, gl,
                                    dev_status=st)
    torch.cuda.synchronize()
    return loss, dh, dw


def test_zero_wait_limit_reports_timeout_and_context_survives(zero_wait_limit):
    b, h, W = _case()
    st = B.new_status()
    _fwd_bwd(b, h, W, st)
    assert "OLIVE_ERR_TIMEOUT" in B.status_bits(st)
    # the divergence kernels take the same path
    st2 = B.new_status()
    r = torch.arange(h.shape[0], dtype=torch.int32, device="cuda")
    n = torch.tensor([h.shape[0]], dtype=torch.int32, device="cuda")
    B.olive_token_divergence(h, W, h, W, r, n, grad_kl=torch.ones(h.shape[0], device="cuda"),
                             dev_status=st2)
    torch.cuda.synchronize()
    assert "OLIVE_ERR_TIMEOUT" in B.status_bits(st2)


def test_normal_limit_after_timeouts_is_clean():
    b, h, W = _case()
    st = B.new_status()
    loss, dh, dw = _fwd_bwd(b, h, W, st)
    assert B.status_bits(st) == []
    assert np.isfinite(float(loss.item()))
