"""olive_splice_pack_masked (multi-turn OLIVE, Section 3.2) against the
oracle: bit-exact integers, then the forward and backward on the rows it
selects."""

import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_grad, assert_close_logp, assert_close_loss, batch_to_cuda, to_f64

pytestmark = pytest.mark.gpu

KEYS = ("ids", "targets", "loss_mask", "cu_seqlens", "cut_offsets")


def _gpu(b, flags, T_cap=None):
    pi, po, ci, co = batch_to_cuda(b)
    fl = torch.from_numpy(np.asarray(flags, dtype=np.uint8)).cuda()
    return B.olive_splice_pack_masked(pi, po, ci, co, fl, b.V, T_cap if T_cap else max(b.T, 1))


def _compare(b, flags, T_cap=None):
    g = _gpu(b, flags, T_cap)
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V, cont_loss=flags)
    n = int(g["n_rows"].item())
    assert n == o["n_rows"]
    for k in KEYS:
        gv = g[k].cpu().numpy().astype(np.int64)
        if k in ("ids", "targets", "loss_mask"):
            gv = gv[:b.T]
        if k == "cut_offsets":
            gv = gv[:b.S]
        assert np.array_equal(gv, o[k]), k
    assert np.array_equal(g["rows"][:n].cpu().numpy(), o["rows"])
    assert (g["rows"][n:] == -1).all()
    assert int(g["dev_status"].item()) == 0
    return g, o


def test_golden_turns_fixture():
    with open(os.path.join(os.path.dirname(__file__), "golden", "splice_pack_turns.json")) as f:
        gj = json.load(f)
    b = synth.Batch(np.array(gj["prefix_ids"], np.int32), np.array(gj["prefix_off"], np.int32),
                    np.array(gj["cont_ids"], np.int32), np.array(gj["cont_off"], np.int32), gj["V"])
    g, _ = _compare(b, gj["cont_loss"])
    assert g["rows"][:gj["expect"]["n_rows"]].tolist() == gj["expect"]["rows"]


@pytest.mark.parametrize("seed,S,maxlen", [(0, 5, 40), (1, 30, 300), (2, 12, 3000)])
def test_random_turn_flags(seed, S, maxlen):
    rng = np.random.default_rng(200 + seed)
    b = synth.batch_from_lengths(rng, rng.integers(1, maxlen, size=S), rng.integers(0, maxlen, size=S),
                                 5000)
    # teacher actions in runs, observations in between
    flags = (np.sin(np.arange(len(b.cont_ids)) / 7.0 + seed) > -0.2).astype(np.uint8)
    _compare(b, flags, T_cap=b.T + 100)


def _turn_runs(n, seed, action_len=200, obs_len=60):
    """Alternating runs over the continuation ids: teacher actions (flag 1) and
    observations (flag 0), each run's length geometric with the given mean."""
    rng = np.random.default_rng(seed)
    flags = np.empty(n, np.uint8)
    i, on = 0, True
    while i < n:
        L = int(rng.geometric(1.0 / (action_len if on else obs_len)))
        flags[i:i + L] = 1 if on else 0
        i += L
        on = not on
    return flags


def test_varlen_batch_with_turn_runs():
    """The largest packing input (64 sequences, 528k packed tokens) with teacher actions
    and observations alternating along every continuation: bit-exact against the oracle."""
    b = synth.make_batch("varlen")
    flags = _turn_runs(len(b.cont_ids), 310)
    g, o = _compare(b, flags)
    assert 0 < o["n_rows"] < b.n_mask


def test_all_ones_matches_plain_and_all_zero_is_empty():
    rng = np.random.default_rng(9)
    b = synth.batch_from_lengths(rng, rng.integers(1, 500, size=9), rng.integers(0, 900, size=9), 800)
    g, _ = _compare(b, np.ones(len(b.cont_ids), np.uint8))
    pi, po, ci, co = batch_to_cuda(b)
    plain = B.olive_splice_pack(pi, po, ci, co, b.V, b.T)
    for k in ("ids", "targets", "loss_mask", "rows", "n_rows"):
        assert torch.equal(g[k], plain[k]), k
    g0, _ = _compare(b, np.zeros(len(b.cont_ids), np.uint8))
    assert int(g0["n_rows"].item()) == 0 and not g0["loss_mask"].any()


def test_bad_offsets_flagged():
    b = synth.batch_from_lengths(np.random.default_rng(3), [4, 4], [5, 6], 50)
    g = _gpu(b, np.ones(11, np.uint8), T_cap=b.T - 2)
    assert "OLIVE_ERR_OFFSETS" in B.status_bits(g["dev_status"])
    assert int(g["n_rows"].item()) == 0 and not g["loss_mask"].any()


def test_multi_turn_forward_and_backward():
    rng = np.random.default_rng(77)
    b = synth.batch_from_lengths(rng, rng.integers(20, 200, size=6), rng.integers(50, 400, size=6), 3001)
    flags = (rng.random(len(b.cont_ids)) < 0.6).astype(np.uint8)
    h = synth.normal_bf16(rng, (b.T, 128), 1.0)
    W = synth.normal_bf16(rng, (3001, 128), 0.1)
    g, o = _compare(b, flags)
    hc, Wc = h.cuda(), W.cuda()
    st = g["dev_status"]
    logp, lse, loss = B.olive_token_logprob_fwd(hc, Wc, g["targets"], g["rows"], g["n_rows"],
                                                reduction="mean", dev_status=st)
    gl = torch.ones(1, dtype=torch.float32, device="cuda")
    dh, dw = B.olive_token_loss_bwd(hc, Wc, g["targets"], g["rows"], g["n_rows"], lse, gl,
                                    reduction="mean", grad_dtype=torch.float32, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    rl, _, rloss = oracle.token_logprob(to_f64(h), to_f64(W), o["targets"], o["rows"], reduction="mean")
    assert_close_logp(logp.cpu().numpy(), rl)
    assert_close_loss(float(loss.item()), rloss)
    rdh, rdw = oracle.token_loss_bwd(to_f64(h), to_f64(W), o["targets"], o["rows"], reduction="mean")
    assert_close_grad(dh.cpu().numpy(), rdh, "dH")
    assert_close_grad(dw.cpu().numpy(), rdw, "dW")
