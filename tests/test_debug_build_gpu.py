"""The OLIVE_DEBUG build (build.build(debug=True) -> libolive_debug.so): its
kernels check copy coordinates and every index on the device and report a
failed check as OLIVE_ERR_BOUNDS instead of making the access.  On shapes that
reach every edge of the on-chip training step (partial row, vocabulary and
column tiles, groups with several outer tiles, a phantom outer tile on the odd
CTAs, the rows above their reference that are redone, an empty mask) no check
fires and the results match the oracle."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import build as _build
from paper_2609_36246_gb300 import synth
from tests.parity import (assert_close_grad, assert_close_logp, assert_close_loss, gpu_pack,
                          oracle_pack, to_f64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def debug_lib():
    path = _build.build(debug=True)
    B.use_library(path)
    try:
        yield path
    finally:
        B.use_library(B.LIB_PATH)


def _check(b, h, W, reduction="sum"):
    g = gpu_pack(b)
    st = g["dev_status"]
    gl = torch.tensor([1.3], dtype=torch.float32, device="cuda")
    hc, Wc = h.cuda(), W.cuda()
    logp, lse, loss, dh, dw = B.olive_token_loss_fwd_bwd(hc, Wc, g["targets"], g["rows"],
                                                         g["n_rows"], gl, 1.0, reduction,
                                                         torch.float32, dev_status=st)
    dh2, dw2 = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl, 1.0,
                                      reduction, torch.float32, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    o = oracle_pack(b)
    rl, _, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"], 1.0, reduction)
    assert_close_logp(logp.cpu().numpy(), rl)
    assert_close_loss(float(loss.item()), rloss)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"], 1.0, reduction,
                                     1.3)
    for got, ref, what in ((dh, rdh, "dH"), (dw, rdw, "dW"), (dh2, rdh, "dH bwd"), (dw2, rdw, "dW bwd")):
        assert_close_grad(got.cpu().numpy(), ref, what)


def test_debug_build_is_loaded(debug_lib):
    assert debug_lib.endswith("libolive_debug.so")
    assert B.lib()._name == debug_lib


@pytest.mark.parametrize("S,V,d", [(3, 4097, 64), (7, 13, 24), (4, 700, 4096), (9, 2000, 2056)])
def test_edges_pass_every_check(debug_lib, S, V, d):
    b, h, W = synth.random_case(S * 31 + V, S, V, d, max_prefix=40, max_cont=300, std_w=0.03)
    _check(b, h, W, reduction="mean")


def test_redo_rows_and_empty_mask(debug_lib):
    rng = np.random.default_rng(7)
    b = synth.batch_from_lengths(rng, [20] * 6, [60] * 6, 3000)
    h = synth.normal_bf16(rng, (b.T, 64), 1.0).float()
    h[::2] += 3.0
    W = synth.normal_bf16(rng, (3000, 64), 0.05).float()
    W[1000] = 0.5               # logits 78-101 nats above the first vocabulary tile
    _check(b, h.to(torch.bfloat16), W.to(torch.bfloat16))
    e = synth.batch_from_lengths(rng, [9, 4], [0, 0], 300)
    _check(e, synth.normal_bf16(rng, (e.T, 64), 1.0), synth.normal_bf16(rng, (300, 64), 0.1))


@pytest.mark.parametrize("direction", ["reverse", "forward"])
@pytest.mark.parametrize("T,ds,dt,V", [(300, 4096, 72, 700), (150, 2056, 64, 13)])
def test_divergence_gradient_edges(debug_lib, direction, T, ds, dt, V):
    """The divergence's on-chip gradient pass (both heads' logits per
    128-column tile, G formed in the epilogue): a partial last vocabulary tile,
    V below one tile, a member chunk cut short by d_s; no check fires and KL
    and d/dh_s match the oracle."""
    rng = np.random.default_rng(T + V)
    hs = synth.rms_hidden_bf16(rng, (T, ds))
    Ws = synth.normal_bf16(rng, (V, ds), 0.02)
    ht = synth.normal_bf16(rng, (T, dt), 1.0)
    Wt = synth.normal_bf16(rng, (V, dt), 0.2)
    rows = np.sort(rng.choice(T, size=T * 2 // 3, replace=False)).astype(np.int32)
    gk = rng.uniform(0.5, 1.5, size=T).astype(np.float32)
    st = B.new_status()
    kl, dhs = B.olive_token_divergence(hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda(),
                                       torch.from_numpy(rows).cuda(),
                                       torch.tensor([len(rows)], dtype=torch.int32, device="cuda"),
                                       1.0, direction, torch.from_numpy(gk).cuda(), torch.float32,
                                       dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    rkl, rdhs = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, 1.0,
                                        direction, grad_kl=gk.astype(np.float64))
    assert_close_logp(kl.cpu().numpy(), rkl, "kl")
    assert_close_grad(dhs.cpu().numpy(), rdhs, "dH_s")
