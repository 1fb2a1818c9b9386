"""olive_topk_kl_fwd_bwd (CUDA: the student's top-K lists, the top-K KL and
its gradient from one sweep of the student's logits) against the oracle's
token_topk, token_topk_compare and token_topk_kl_bwd.

The student's set S_t is a selection: it is compared where the oracle's K-th
and (K+1)-th student log-probs differ by more than DECIDE (the candidates are
recomputed in fp32, so the decision is as sharp as olive_token_topk_fwd's).
Inside S_t the order of two log-probs closer than rounding is not unique, so
sets are compared as sets, the sorted values as values, and per-id outputs
after sorting each row by id.  The teacher's lse and ids come from
olive_token_topk_fwd on the teacher."""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import assert_close_grad, assert_close_logp, rel_frob, sample_rows, to_f32, to_f64

pytestmark = pytest.mark.gpu

DECIDE = 1e-3


def _gpu(hs, Ws, ht, Wt, rows, K, g, inv_tau=1.0, grad_dtype=torch.float32, with_ids=True):
    r = torch.from_numpy(np.asarray(rows, dtype=np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    hs, Ws, ht, Wt = hs.cuda(), Ws.cuda(), ht.cuda(), Wt.cuda()
    t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, r, n, K, inv_tau, dev_status=st)
    gk = torch.from_numpy(np.asarray(g, dtype=np.float32)).cuda()
    o = B.olive_topk_kl_fwd_bwd(hs, Ws, ht, Wt, r, n, K, t_lse, gk, t_id if with_ids else None,
                                inv_tau, grad_dtype=grad_dtype, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    return {k: (v.float().cpu().numpy() if v.dtype != torch.int32 else v.cpu().numpy())
            for k, v in o.items() if v is not None}


def _models(rng, T, ds, dt, V, std_w=0.4):
    hs = synth.normal_bf16(rng, (T, ds), 1.0)
    Ws = synth.normal_bf16(rng, (V, ds), std_w)
    # the teacher shares part of the student's structure, as in the overlap tests
    ht = torch.cat([hs, synth.normal_bf16(rng, (T, dt - ds), 1.0)], 1) if dt > ds else hs[:, :dt].contiguous()
    Wt = torch.cat([Ws, synth.normal_bf16(rng, (V, dt - ds), std_w)], 1) if dt > ds else Ws[:, :dt].contiguous()
    return hs, Ws, ht, Wt


def _by_id(ids, *vals):
    """Each row's ids in ascending order, with the values that go with them."""
    o = np.argsort(ids, axis=1, kind="stable")
    return [np.take_along_axis(ids, o, 1)] + [np.take_along_axis(v, o, 1) for v in vals]


def _decided_rows(hs, Ws, ht, Wt, cand, K, inv_tau):
    _, _, gs, _ = oracle.token_topk_compare(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), cand, K,
                                            inv_tau)
    rows = np.array([t for t in cand if gs[t] > DECIDE], dtype=np.int64)
    assert len(rows) >= 0.8 * len(cand)
    return rows


def _full_check(hs, Ws, ht, Wt, rows, K, g, inv_tau, **kw):
    o = _gpu(hs, Ws, ht, Wt, rows, K, g, inv_tau, **kw)
    H = lambda x: to_f64(x)
    lse, _, lp, ids = oracle.token_topk(H(hs), H(Ws), rows, K, inv_tau)
    ov, kl, _, gt = oracle.token_topk_compare(H(hs), H(Ws), H(ht), H(Wt), rows, K, inv_tau)
    assert_close_logp(o["s_lse"][rows], lse[rows], "s_lse")
    gi, = _by_id(o["s_ids"][rows])
    assert np.array_equal(gi, np.sort(ids[rows], axis=1))
    assert np.all(np.diff(o["s_logp"][rows], axis=1) <= 0)
    assert_close_logp(o["s_logp"][rows], lp[rows], "s_logp")
    assert_close_logp(o["kl_topk"][rows], kl[rows], "kl_topk")
    lpt, _ = oracle.log_softmax_rows(oracle.logits(H(ht)[rows], H(Wt), inv_tau))
    own = o["s_ids"][rows].astype(np.int64)
    assert_close_logp(o["t_logp_s"][rows], np.take_along_axis(lpt, own, 1), "t_logp_s")
    if "overlap" in o:
        sure = [k for k, t in enumerate(rows) if gt[t] > DECIDE]
        assert len(sure) >= 0.8 * len(rows)
        assert np.allclose(o["overlap"][rows][sure], ov[rows][sure], atol=1e-6)
    rdh, rdw = oracle.token_topk_kl_bwd(H(hs), H(Ws), H(ht), H(Wt), rows, K, inv_tau, grad=g)
    assert_close_grad(o["d_h_s"][rows], rdh[rows], "dH_s")
    assert_close_grad(o["d_W_s"], rdw, "dW_s")
    off = np.setdiff1d(np.arange(hs.shape[0]), rows)
    assert not o["d_h_s"][off].any() and not o["kl_topk"][off].any()
    assert (o["s_ids"][off] == -1).all() and not o["t_logp_s"][off].any()
    return o


@pytest.mark.parametrize("T,ds,dt,V,K,inv_tau,grad_dtype", [
    (200, 64, 96, 3000, 16, 1.0, torch.float32),
    (150, 128, 64, 800, 4, 0.8, torch.bfloat16),
    (300, 64, 64, 1000, 1, 1.0, torch.float32),
    (130, 72, 136, 4097, 9, 1.3, torch.float32),  # widths not a multiple of 64, a ragged tile
])
def test_small_shapes(T, ds, dt, V, K, inv_tau, grad_dtype):
    rng = np.random.default_rng(T + V + 31 * K)
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    cand = np.sort(rng.choice(T, size=T * 2 // 3, replace=False))
    rows = _decided_rows(hs, Ws, ht, Wt, cand, K, inv_tau)
    g = rng.uniform(0.5, 2.0, size=T)
    _full_check(hs, Ws, ht, Wt, rows, K, g, inv_tau, grad_dtype=grad_dtype)


def test_matches_the_multi_call_path():
    """Against olive_token_topk_fwd + olive_topk_compare + olive_topk_kl_bwd:
    the same lists and KL, and gradients that differ by the one extra bf16
    rounding of p_s in the single-pass G."""
    rng = np.random.default_rng(8)
    T, ds, dt, V, K = 260, 64, 96, 2500, 16
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(T), K, 1.0)
    g = rng.uniform(0.5, 2.0, size=T)
    o = _gpu(hs, Ws, ht, Wt, rows, K, g)
    r = torch.from_numpy(rows.astype(np.int32)).cuda()
    n = torch.tensor([len(rows)], dtype=torch.int32, device="cuda")
    st = B.new_status()
    c = [x.cuda() for x in (hs, Ws, ht, Wt)]
    s_lse, _, s_lp, s_id = B.olive_token_topk_fwd(c[0], c[1], r, n, K, dev_status=st)
    t_lse, _, _, t_id = B.olive_token_topk_fwd(c[2], c[3], r, n, K, dev_status=st)
    ov, kl, tlp = B.olive_topk_compare(c[2], c[3], r, n, s_id, s_lp, t_id, t_lse, dev_status=st,
                                       want_t_logp=True)
    gk = torch.from_numpy(g.astype(np.float32)).cuda()
    dh, dw = B.olive_topk_kl_bwd(c[0], c[1], r, n, s_lse, s_id, s_lp, tlp, kl, gk,
                                 grad_dtype=torch.float32, dev_status=st)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    a = _by_id(o["s_ids"], o["t_logp_s"])
    b = _by_id(s_id.cpu().numpy(), tlp.cpu().numpy())
    assert np.array_equal(a[0], b[0])
    assert np.abs(a[1] - b[1]).max() <= 1e-4
    assert np.array_equal(o["overlap"], ov.cpu().numpy())
    for k, ref in (("s_lse", s_lse), ("s_logp", s_lp), ("kl_topk", kl)):
        assert np.abs(o[k] - ref.cpu().numpy()).max() <= 1e-4, k
    assert rel_frob(o["d_h_s"], dh.cpu().numpy()) <= 5e-3
    assert rel_frob(o["d_W_s"], dw.cpu().numpy()) <= 5e-3


def test_full_set_equals_full_kl_gradient():
    """K = V: S_t is the whole vocabulary, P_S = 1, kl_topk is the full reverse
    KL and the gradient is olive_token_divergence's."""
    rng = np.random.default_rng(12)
    T, d, V = 140, 64, 16
    hs, Ws, ht, Wt = _models(rng, T, d, d + 32, V, std_w=0.5)
    rows = np.arange(0, T, 2)
    g = rng.uniform(0.5, 2.0, size=T)
    o = _gpu(hs, Ws, ht, Wt, rows, V, g)
    rkl, rfull = oracle.token_divergence(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, 1.0,
                                         "reverse", grad_kl=g)
    assert_close_logp(o["kl_topk"][rows], rkl[rows], "kl")
    assert_close_grad(o["d_h_s"][rows], rfull[rows], "dH_s")
    assert np.all(o["overlap"][rows] == 1.0)
    assert np.all(np.sort(o["s_ids"][rows], axis=1) == np.arange(V))


def test_identical_models():
    """Student = teacher: every truncated KL is 0, the overlap is 1 and the
    gradient is g p_s(u) (1 - P_S) on S_t and -g P_S p_s(u) elsewhere: it is
    the gradient of sum_t g_t kl_topk[t] at a point where kl_topk = 0 but P_S
    still moves, so it does not vanish; the oracle's is compared."""
    rng = np.random.default_rng(5)
    T, d, V = 130, 64, 2000
    h = synth.normal_bf16(rng, (T, d), 1.0)
    W = synth.normal_bf16(rng, (V, d), 0.4)
    rows = _decided_rows(h, W, h, W, np.arange(T), 16, 1.0)
    g = np.ones(T)
    o = _gpu(h, W, h, W, rows, 16, g)
    assert np.all(o["overlap"][rows] == 1.0)
    assert np.abs(o["kl_topk"][rows]).max() <= 1e-5
    rdh, _ = oracle.token_topk_kl_bwd(to_f64(h), to_f64(W), to_f64(h), to_f64(W), rows, 16, grad=g,
                                      with_dW=False)
    assert_close_grad(o["d_h_s"][rows], rdh[rows], "dH_s")


def test_without_teacher_ids():
    rng = np.random.default_rng(21)
    hs, Ws, ht, Wt = _models(rng, 90, 64, 64, 700)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(90), 8, 1.0)
    g = rng.uniform(0.5, 2.0, size=90)
    o = _full_check(hs, Ws, ht, Wt, rows, 8, g, 1.0, with_ids=False)
    assert "overlap" not in o


def test_several_slabs(monkeypatch):
    """The slab cap lowered to 128 rows: the per-row selection, the G pass and
    dW's fp32 accumulation run across many slabs."""
    monkeypatch.setenv("OLIVE_SLAB_ROWS", "128")
    rng = np.random.default_rng(61)
    T, ds, dt, V, K = 700, 64, 96, 1500, 8
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(T), K, 1.0)
    assert len(rows) > 4 * 128
    g = rng.uniform(0.5, 2.0, size=T)
    _full_check(hs, Ws, ht, Wt, rows, K, g, 1.0, grad_dtype=torch.bfloat16)


@pytest.mark.parametrize("spike", [0.2, 0.5])
def test_rows_far_above_their_first_tile(spike):
    """One student id far down the vocabulary (1000) sits 31-39 nats (spike
    0.2: the scaled form, e' up to ~2^57) or 78-101 nats (spike 0.5: beyond
    the reference window, the row is rewritten as G) above the row's first
    256 logits on half of the rows."""
    rng = np.random.default_rng(int(spike * 10) + 40)
    T, d, V, K = 160, 64, 3000, 8
    hs = synth.normal_bf16(rng, (T, d), 1.0).float()
    hs[::2] += 3.0
    hs = hs.to(torch.bfloat16)
    Ws = synth.normal_bf16(rng, (V, d), 0.05).float()
    Ws[1000] = spike
    Ws = Ws.to(torch.bfloat16)
    ht = synth.normal_bf16(rng, (T, d), 1.0)
    Wt = synth.normal_bf16(rng, (V, d), 0.3)
    z = oracle.logits(to_f64(hs), to_f64(Ws), 1.0)
    gap = (z.max(axis=1) - z[:, :256].max(axis=1))[::2]
    assert gap.min() > (25 if spike < 0.3 else 75)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(T), K, 1.0)
    g = rng.uniform(0.5, 2.0, size=T)
    _full_check(hs, Ws, ht, Wt, rows, K, g, 1.0)


def test_tiny_weights_take_the_rewritten_form():
    """Rows with g_t = 1e-30 put the row scale below 2^-96, so their G is
    written out in full; each such row still matches on its own."""
    rng = np.random.default_rng(77)
    T, ds, dt, V, K = 120, 64, 96, 2000, 16
    hs, Ws, ht, Wt = _models(rng, T, ds, dt, V)
    rows = _decided_rows(hs, Ws, ht, Wt, np.arange(T), K, 1.0)
    g = np.where(np.arange(T) % 3 == 0, 1e-30, rng.uniform(0.5, 2.0, size=T))
    o = _full_check(hs, Ws, ht, Wt, rows, K, g, 1.0)
    rdh, _ = oracle.token_topk_kl_bwd(to_f64(hs), to_f64(Ws), to_f64(ht), to_f64(Wt), rows, K, grad=g,
                                      with_dW=False)
    tiny = [t for t in rows if t % 3 == 0][:8]
    assert len(tiny) >= 4
    for t in tiny:
        assert rel_frob(o["d_h_s"][t], rdh[t]) <= 2e-2, t


def test_empty_mask():
    rng = np.random.default_rng(3)
    hs, Ws, ht, Wt = _models(rng, 40, 64, 64, 300)
    r = torch.zeros(1, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = B.new_status()
    c = [x.cuda() for x in (hs, Ws, ht, Wt)]
    t_lse = torch.zeros(40, dtype=torch.float32, device="cuda")
    g = torch.ones(40, dtype=torch.float32, device="cuda")
    o = B.olive_topk_kl_fwd_bwd(*c, r, n, 4, t_lse, g, dev_status=st, grad_dtype=torch.float32)
    torch.cuda.synchronize()
    assert B.status_bits(st) == []
    assert not o["d_h_s"].any() and not o["d_W_s"].any() and not o["kl_topk"].any()
    assert (o["s_ids"] == -1).all()


@pytest.mark.slow
def test_kl_workload_sampled():
    """Student d = 4096 / teacher d = 5120, V = 151936, K = 16; lists, KL and
    dH_s on sampled decided rows (each depends on its own row alone)."""
    T = 2048
    hs = synth.make_hidden("kl", T)
    Ws = synth.make_weight("kl")
    ht, Wt = synth.make_teacher("kl", T)
    rng = np.random.default_rng(3)
    g = rng.uniform(0.5, 2.0, size=T)
    o = _gpu(hs, Ws, ht, Wt, np.arange(T), 16, g, grad_dtype=torch.bfloat16)
    assert np.isfinite(o["d_W_s"]).all()
    pick = sample_rows(np.arange(T), 256, seed=5)
    _, _, gs, _ = oracle.token_topk_compare(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick, 16)
    pick = np.array([t for t in pick if gs[t] > DECIDE])
    assert len(pick) >= 128
    _, _, lp, ids = oracle.token_topk(to_f32(hs), to_f32(Ws), pick, 16)
    assert np.array_equal(np.sort(o["s_ids"][pick], axis=1), np.sort(ids[pick], axis=1))
    assert_close_logp(o["s_logp"][pick], lp[pick], "s_logp")
    rdh, _ = oracle.token_topk_kl_bwd(to_f32(hs), to_f32(Ws), to_f32(ht), to_f32(Wt), pick, 16, grad=g,
                                      with_dW=False)
    for t in pick:
        assert_close_grad(o["d_h_s"][t], rdh[t], f"dH_s[{t}]")
