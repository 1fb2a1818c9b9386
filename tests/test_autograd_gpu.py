"""fused_lmhead_ce (the Eq. (osd-ce) loss as a torch autograd op over the C
ABI) and olive_scale, against the oracle."""

import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_grad, assert_close_loss, gpu_pack, oracle_pack, to_f64

pytestmark = pytest.mark.gpu


def _case():
    b, h, W = synth.random_case(88, 6, 3001, 128, max_prefix=40, max_cont=200, std_w=0.1)
    return b, h, W


@pytest.mark.parametrize("single_pass", [True, False])
@pytest.mark.parametrize("reduction", ["sum", "mean"])
def test_autograd_matches_oracle(single_pass, reduction):
    b, h, W = _case()
    g = gpu_pack(b)
    hc = h.cuda().requires_grad_(True)
    Wc = W.cuda().requires_grad_(True)
    loss = B.fused_lmhead_ce(hc, Wc, g["targets"], g["rows"], g["n_rows"], 0.9, reduction,
                             single_pass=single_pass)
    (2.5 * loss).backward()
    torch.cuda.synchronize()
    o = oracle_pack(b)
    _, _, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"], 0.9, reduction)
    assert_close_loss(float(loss.item()), rloss)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"], 0.9, reduction,
                                     2.5)
    assert hc.grad.dtype == torch.bfloat16
    assert_close_grad(hc.grad.float().cpu().numpy(), rdh, "dH")
    assert_close_grad(Wc.grad.float().cpu().numpy(), rdw, "dW")


def test_backward_twice_accumulates():
    """retain_graph: the stored unit-gradient tensors are scaled out of place,
    so a second backward adds the same gradient again."""
    b, h, W = _case()
    g = gpu_pack(b)
    hc = h.cuda().float().requires_grad_(True)
    Wc = W.cuda().requires_grad_(True)
    loss = B.fused_lmhead_ce(hc.to(torch.bfloat16), Wc, g["targets"], g["rows"], g["n_rows"])
    loss.backward(retain_graph=True)
    first = Wc.grad.clone()
    loss.backward()
    torch.cuda.synchronize()
    assert torch.allclose(Wc.grad.float(), 2 * first.float(), rtol=1e-2, atol=1e-6)
    assert hc.grad is not None and hc.grad.dtype == torch.float32


def test_forward_only_without_grad():
    b, h, W = _case()
    g = gpu_pack(b)
    with torch.no_grad():
        loss = B.fused_lmhead_ce(h.cuda(), W.cuda(), g["targets"], g["rows"], g["n_rows"])
    o = oracle_pack(b)
    _, _, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"])
    assert_close_loss(float(loss.item()), rloss)


@pytest.mark.parametrize("dtype,n", [(torch.bfloat16, 1000003), (torch.float32, 77), (torch.bfloat16, 5)])
def test_scale(dtype, n):
    x = torch.randn(n, device="cuda").to(dtype)
    s = torch.tensor([-1.75], dtype=torch.float32, device="cuda")
    y = B.olive_scale(x, s)
    ref = (x.float() * -1.75).to(dtype)
    assert torch.equal(y, ref)
    B.olive_scale(x, s, out=x)  # in place
    assert torch.equal(x, ref)
