"""The library's calls inside a CUDA graph: one training step (splice/pack +
olive_token_loss_fwd_bwd) and a divergence value + gradient are captured
once and replayed; each replay must reproduce the eager results bit for bit
(every reduction in these paths runs in a fixed order) and must read the
inputs as they are at replay time."""

import numpy as np
import pytest
import torch

from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import batch_to_cuda

pytestmark = pytest.mark.gpu


def _step(ins, h, W, V, T, gl, ws, st):
    pk = B.olive_splice_pack(*ins, V, T, dev_status=st)
    return B.olive_token_loss_fwd_bwd(h, W, pk["targets"], pk["rows"], pk["n_rows"], gl, 1.0,
                                      "mean", torch.bfloat16, ws=ws, dev_status=st)


def test_training_step_replays_in_a_cuda_graph():
    b, h0, W0 = synth.random_case(5, 6, 3001, 128, max_prefix=60, max_cont=300, std_w=0.1)
    ins = batch_to_cuda(b)
    h, W = h0.cuda(), W0.cuda()
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    ws = B.workspace(B.olive_workspace_size("loss_fwd_bwd", b.T, 128, 3001))
    st = B.new_status()
    eager = [t.clone() for t in _step(ins, h, W, 3001, b.T, gl, ws, st)]
    # warm up on a side stream, as graph capture expects
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        _step(ins, h, W, 3001, b.T, gl, ws, st)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        outs = _step(ins, h, W, 3001, b.T, gl, ws, st)
    g.replay()
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    for got, ref in zip(outs, eager):
        assert torch.equal(got, ref)
    # new hidden values in the captured input buffer: the replay reads them
    h.copy_(synth.normal_bf16(np.random.default_rng(9), tuple(h.shape), 1.0).cuda())
    eager2 = [t.clone() for t in _step(ins, h, W, 3001, b.T, gl, ws, st)]
    g.replay()
    torch.cuda.synchronize()
    for got, ref in zip(outs, eager2):
        assert torch.equal(got, ref)
    assert not torch.equal(eager2[3], eager[3])


def test_divergence_with_gradient_replays_in_a_cuda_graph():
    rng = np.random.default_rng(3)
    T, ds, dt, V = 300, 64, 96, 2000
    hs, Ws = synth.normal_bf16(rng, (T, ds), 1.0).cuda(), synth.normal_bf16(rng, (V, ds), 0.2).cuda()
    ht, Wt = synth.normal_bf16(rng, (T, dt), 1.0).cuda(), synth.normal_bf16(rng, (V, dt), 0.2).cuda()
    rows = torch.arange(0, T, 2, dtype=torch.int32, device="cuda")
    n = torch.tensor([rows.numel()], dtype=torch.int32, device="cuda")
    gk = torch.ones(T, dtype=torch.float32, device="cuda")
    ws = B.workspace(B.olive_workspace_size("divergence", T, ds, V, d_t=dt, grad=True))
    st = B.new_status()
    run = lambda: B.olive_token_divergence(hs, Ws, ht, Wt, rows, n, 1.0, "reverse", gk,
                                           torch.float32, ws=ws, dev_status=st)
    eager = [t.clone() for t in run()]
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        outs = run()
    g.replay()
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    for got, ref in zip(outs, eager):
        assert torch.equal(got, ref)
