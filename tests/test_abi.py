"""Host-side checks of libolive.so that need no GPU.

The library is (re)built with nvcc for sm_103a, loaded, and every entry point
declared in include/olive.h must be exported.  Argument validation happens
before any CUDA call, so bad pointers, shapes, alignment and workspace sizes
are rejected here with the documented status codes; a call that passes
validation on a machine without a usable device ends in OLIVE_ERR_CUDA (or
OLIVE_ERR_UNSUPPORTED_DEVICE) without launching anything.
"""

import ctypes

import pytest
import torch

from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import build


@pytest.fixture(scope="module")
def L():
    build.build()
    return B.lib()


def test_exports_every_declared_symbol(L):
    names = B.declared_symbols()
    assert set(names) >= {"olive_splice_pack", "olive_token_logprob_fwd", "olive_token_loss_bwd",
                          "olive_token_divergence", "olive_workspace_size", "olive_status_string",
                          "olive_abi_version"}
    for n in names:
        assert hasattr(L, n), n


def test_abi_version_and_status_strings(L):
    assert B.olive_abi_version() == 1
    for code in range(10):
        s = B.olive_status_string(code)
        assert s and s != "unknown status"
    assert B.olive_status_string(42) == "unknown status"


def test_workspace_sizes(L):
    T, d, V = 32768, 4096, 151936
    fwd = B.olive_workspace_size("logprob_fwd", T, d, V)
    bwd16 = B.olive_workspace_size("loss_bwd", T, d, V, grad_dtype=torch.bfloat16)
    bwd32 = B.olive_workspace_size("loss_bwd", T, d, V, grad_dtype=torch.float32)
    kl = B.olive_workspace_size("divergence", 16384, 4096, V, d_t=5120, grad=True)
    assert fwd >= 2 * T * d and fwd % 256 == 0
    # the on-chip backward stores no [rows, V] array and no [V, d]
    # accumulator: its workspace does not grow with V or the gradient dtype
    assert bwd16 == bwd32
    assert bwd16 == B.olive_workspace_size("loss_bwd", T, d, 8192)
    fb = B.olive_workspace_size("loss_fwd_bwd", T, d, V)
    assert fb == bwd16 and fb < 2 * T * d + 256 * 2**20
    # the slab variant holds G for up to 32768 rows (~5.6 GB at this V)
    slab = B.olive_workspace_size("loss_fwd_bwd_slab", T, d, V)
    assert slab >= 2 * 18304 * V
    assert kl > B.olive_workspace_size("divergence", 16384, 4096, V, d_t=5120, grad=False)
    # invalid requests give 0
    assert B.olive_workspace_size("logprob_fwd", 0, d, V) == 0
    assert B.olive_workspace_size("logprob_fwd", T, 12, V) == 0
    assert L.olive_workspace_size(7, T, d, 0, V, 1, 0) == 0


def test_slab_rows_rule(L, monkeypatch):
    """The slab forms' row rule through the ABI: ~5.6 GB of bf16 G in whole
    128-row tiles, at most 32768 rows and T rounded up to 128, lowered (never
    raised) by OLIVE_SLAB_ROWS."""
    V = 151936
    tc = B.olive_slab_rows(32768, V)
    assert tc % 128 == 0 and 2 * tc * V <= 5.6e9 < 2 * (tc + 128) * V
    assert B.olive_slab_rows(100, V) == 128 and B.olive_slab_rows(300, 4096) == 384
    assert B.olive_slab_rows(10**6, 100) == 32768
    assert B.olive_slab_rows(0, V) == 0 and B.olive_slab_rows(5, 0) == 0
    monkeypatch.setenv("OLIVE_SLAB_ROWS", "256")
    assert B.olive_slab_rows(32768, V) == 256
    monkeypatch.setenv("OLIVE_SLAB_ROWS", "1000000")
    assert B.olive_slab_rows(32768, V) == tc


def _fake(n=1 << 20):
    # host buffer used only for its (16-byte aligned) address: validation
    # never dereferences it
    buf = ctypes.create_string_buffer(n + 256)
    base = (ctypes.addressof(buf) + 255) // 256 * 256
    return buf, base


def test_fwd_argument_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    args = dict(hidden=P(p), W=P(p), targets=P(p), rows=P(p), n_rows=P(p), T=64, d=64, V=100,
                inv_tau=1.0, red=0, logp=P(p), lse=P(p), loss=P(p), ws=P(p), ws_bytes=1 << 20,
                st=P(p), stream=None)

    def call(**kw):
        a = dict(args, **kw)
        return L.olive_token_logprob_fwd(a["hidden"], a["W"], a["targets"], a["rows"], a["n_rows"],
                                         a["T"], a["d"], a["V"], a["inv_tau"], a["red"], a["logp"],
                                         a["lse"], a["loss"], a["ws"], a["ws_bytes"], a["st"],
                                         a["stream"])

    assert call(hidden=None) == 1
    assert call(red=5) == 1
    assert call(inv_tau=0.0) == 1
    assert call(inv_tau=float("nan")) == 1
    assert call(T=0) == 2
    assert call(V=0) == 2
    assert call(d=60) == 3
    assert call(hidden=P(p + 2)) == 3
    assert call(ws_bytes=16) == 9
    assert call(ws=P(p + 8)) == 9
    assert call(ws=None) == 1 or call(ws=None) == 9
    # valid arguments: without a usable sm_103 device nothing launches
    if not torch.cuda.is_available():
        assert call() in (7, 8)


def test_bwd_and_divergence_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    # bwd: bad grad dtype, misaligned d_W
    st = L.olive_token_loss_bwd(P(p), P(p), P(p), P(p), P(p), 64, 64, 100, 1.0, 0, P(p), P(p),
                                P(p), P(p), 3, P(p), 1 << 20, P(p), None)
    assert st == 1
    st = L.olive_token_loss_bwd(P(p), P(p), P(p), P(p), P(p), 64, 64, 100, 1.0, 0, P(p), P(p),
                                P(p), P(p + 4), 0, P(p), 1 << 20, P(p), None)
    assert st == 3
    # divergence: grad_kl without d_h_s
    st = L.olive_token_divergence(P(p), P(p), 64, P(p), P(p), 64, P(p), P(p), 64, 100, 1.0, 0,
                                  P(p), P(p), None, 0, P(p), 1 << 20, P(p), None)
    assert st == 1
    st = L.olive_token_divergence(P(p), P(p), 64, P(p), P(p), 64, P(p), P(p), 64, 100, 1.0, 9,
                                  P(p), None, None, 0, P(p), 1 << 20, P(p), None)
    assert st == 1
    # splice/pack: empty batch, null output
    st = L.olive_splice_pack(P(p), P(p), P(p), P(p), 0, 10, 10, P(p), P(p), P(p), P(p), P(p), P(p),
                             P(p), P(p), None)
    assert st == 2
    st = L.olive_splice_pack(P(p), P(p), P(p), P(p), 1, 10, 10, None, P(p), P(p), P(p), P(p), P(p),
                             P(p), P(p), None)
    assert st == 1


def test_new_entry_points_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    # top-K: K outside [1, 16] or above V, misaligned width
    for K, V, want in ((0, 100, 2), (17, 100, 2), (8, 4, 2)):
        st = L.olive_token_topk_fwd(P(p), P(p), P(p), P(p), 64, 64, V, 1.0, K, P(p), P(p), P(p),
                                    P(p), P(p), 1 << 20, P(p), None)
        assert st == want, (K, V)
    st = L.olive_token_topk_fwd(P(p), P(p), P(p), P(p), 64, 60, 100, 1.0, 4, P(p), P(p), P(p),
                                P(p), P(p), 1 << 20, P(p), None)
    assert st == 3
    st = L.olive_token_topk_fwd(P(p), P(p), P(p), P(p), 64, 64, 100, 1.0, 4, None, P(p), P(p),
                                P(p), P(p), 1 << 20, P(p), None)
    assert st == 1
    # top-K compare: null list, bad K
    st = L.olive_topk_compare(P(p), P(p), 64, P(p), P(p), 64, 100, 1.0, 4, None, P(p), P(p), P(p),
                              P(p), P(p), None, P(p), None)
    assert st == 1
    st = L.olive_topk_compare(P(p), P(p), 64, P(p), P(p), 64, 100, 1.0, 20, P(p), P(p), P(p), P(p),
                              P(p), P(p), None, P(p), None)
    assert st == 2
    # top-K KL backward: missing t_logp_s, bad K, bad dtype, misaligned d_W_s, workspace
    ws = B.olive_workspace_size("topk_kl_bwd", 64, 64, 100, grad_dtype=torch.float32)
    assert ws > 2 * 64 * 100  # its G slab

    def kl_bwd(**kw):
        a = dict(tlp=P(p), K=4, dt=1, dw=P(p), ws_bytes=1 << 20)
        a.update(kw)
        return L.olive_topk_kl_bwd(P(p), P(p), P(p), P(p), 64, 64, 100, 1.0, a["K"], P(p), P(p),
                                   P(p), a["tlp"], P(p), P(p), P(p), a["dw"], a["dt"], P(p),
                                   a["ws_bytes"], P(p), None)
    assert kl_bwd(tlp=None) == 1
    assert kl_bwd(K=0) == 2 and kl_bwd(K=17) == 2
    assert kl_bwd(dt=4) == 1
    assert kl_bwd(dw=P(p + 4)) == 3
    assert kl_bwd(ws_bytes=ws - 1) == 9
    if not torch.cuda.is_available():
        assert kl_bwd(ws_bytes=ws) in (7, 8)
    # multi-turn splice: null flags, workspace too small
    st = L.olive_splice_pack_masked(P(p), P(p), P(p), P(p), None, 1, 10, 10, P(p), P(p), P(p), P(p),
                                    P(p), P(p), P(p), P(p), 1 << 20, P(p), None)
    assert st == 1
    st = L.olive_splice_pack_masked(P(p), P(p), P(p), P(p), P(p), 1, 10, 100000, P(p), P(p), P(p),
                                    P(p), P(p), P(p), P(p), P(p), 8, P(p), None)
    assert st == 9
    assert B.olive_workspace_size("splice_masked", 100000, 8, 1) >= 4 * 49
    assert B.olive_workspace_size("topk_fwd", 4096, 4096, 151936) > B.olive_workspace_size(
        "logprob_fwd", 4096, 4096, 151936)


def test_opd_stats_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    ws = B.olive_workspace_size("opd_stats", 64, 64, 100, d_t=96)
    assert ws > 0 and B.olive_workspace_size("opd_stats", 64, 64, 100, d_t=90) == 0

    def call(outs=None, **kw):
        a = dict(K=16, dirn=0, dt=96, ws_bytes=ws)
        a.update(kw)
        o = outs if outs is not None else [P(p)] * 9
        return L.olive_opd_token_stats(P(p), P(p), 64, P(p), P(p), a["dt"], P(p), P(p), 64, 100, 1.0,
                                       a["dirn"], a["K"], *o, P(p), a["ws_bytes"], P(p), None)
    assert call(outs=[None] * 9) == 1
    assert call(dirn=2) == 1
    assert call(K=0) == 2 and call(K=17) == 2
    assert call(dt=90) == 3
    assert call(ws_bytes=ws - 1) == 9
    if not torch.cuda.is_available():
        assert call(outs=[None] * 8 + [P(p)]) in (7, 8)


def test_topk_kl_fwd_bwd_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    ws = B.olive_workspace_size("topk_kl_fwd_bwd", 64, 64, 100, grad_dtype=torch.bfloat16)
    assert ws >= B.olive_workspace_size("loss_fwd_bwd_slab", 64, 64, 100, grad_dtype=torch.bfloat16)
    assert L.olive_workspace_size(8, 64, 64, 0, 100, 1, 2) == 0  # no fp16 gradients

    def call(**kw):
        a = dict(ds=64, dt=96, K=8, tids=P(p), ov=P(p), dt_=0, dh=P(p), ws_bytes=ws, tlse=P(p))
        a.update(kw)
        return L.olive_topk_kl_fwd_bwd(P(p), P(p), a["ds"], P(p), P(p), a["dt"], P(p), P(p), 64,
                                       100, 1.0, a["K"], a["tlse"], a["tids"], P(p), P(p), P(p),
                                       P(p), P(p), P(p), a["ov"], a["dh"], P(p), a["dt_"], P(p),
                                       a["ws_bytes"], P(p), None)
    assert call(tlse=None) == 1
    assert call(ov=None) == 1          # teacher ids without an overlap output
    assert call(dt_=2) == 1
    assert call(K=0) == 2 and call(K=17) == 2 and call(K=16, dt=64) != 2
    assert call(ds=60) == 3 and call(dt=90) == 3 and call(dh=P(p + 4)) == 3
    assert call(ws_bytes=ws - 1) == 9
    if not torch.cuda.is_available():
        assert call() in (7, 8)
        assert call(tids=None, ov=None) in (7, 8)


def test_scale_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    assert L.olive_scale(None, P(p), 8, 0, P(p), None) == 1
    assert L.olive_scale(P(p), P(p), 8, 3, P(p), None) == 1
    assert L.olive_scale(P(p), P(p), 0, 0, P(p), None) == 2
    assert L.olive_scale(P(p + 2), P(p), 8, 0, P(p), None) == 3
    if not torch.cuda.is_available():
        assert L.olive_scale(P(p), P(p), 8, 1, P(p), None) in (7, 8)


def test_fwd_bwd_validation(L):
    keep, p = _fake()
    P = ctypes.c_void_p
    ws = B.olive_workspace_size("loss_fwd_bwd", 64, 64, 100, grad_dtype=torch.bfloat16)
    assert ws >= B.olive_workspace_size("loss_bwd", 64, 64, 100, grad_dtype=torch.bfloat16) - 4096

    def call(**kw):
        a = dict(gl=P(p), red=0, dt=0, dh=P(p), d=64, ws_bytes=ws)
        a.update(kw)
        return L.olive_token_loss_fwd_bwd(P(p), P(p), P(p), P(p), P(p), 64, a["d"], 100, 1.0,
                                          a["red"], a["gl"], P(p), P(p), P(p), a["dh"], P(p),
                                          a["dt"], P(p), a["ws_bytes"], P(p), None)
    assert call(gl=None) == 1
    assert call(red=3) == 1 and call(dt=2) == 1
    assert call(d=60) == 3 and call(dh=P(p + 2)) == 3
    assert call(ws_bytes=ws - 1) == 9
    if not torch.cuda.is_available():
        assert call() in (7, 8)


def test_binding_rejects_cpu_tensors(L):
    h = torch.zeros(8, 64, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        B.olive_token_logprob_fwd(h, h, torch.zeros(8, dtype=torch.int32),
                                  torch.zeros(8, dtype=torch.int32), torch.zeros(1, dtype=torch.int32))
