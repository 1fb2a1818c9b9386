"""Thin ctypes binding over libolive.so (include/olive.h), same entry names.

Every function here only marshals torch tensors into pointers and sizes and
calls the C ABI on the current torch CUDA stream; all computation happens in
the library's CUDA kernels.  There is no fallback: if libolive.so is missing
or fails to load, every call raises.
"""

from __future__ import annotations

import ctypes
import os
import re

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libolive.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "olive.h")

OLIVE_OK = 0
STATUS_NAMES = {
    0: "OLIVE_OK", 1: "OLIVE_ERR_INVALID_ARG", 2: "OLIVE_ERR_SHAPE", 3: "OLIVE_ERR_ALIGNMENT",
    4: "OLIVE_ERR_TOKEN_RANGE", 5: "OLIVE_ERR_OFFSETS", 6: "OLIVE_ERR_TIMEOUT",
    7: "OLIVE_ERR_UNSUPPORTED_DEVICE", 8: "OLIVE_ERR_CUDA", 9: "OLIVE_ERR_WORKSPACE",
    10: "OLIVE_ERR_BOUNDS",
}
REDUCE = {"sum": 0, "mean": 1}
DIRECTION = {"reverse": 0, "forward": 1}
DTYPE = {torch.bfloat16: 0, torch.float32: 1}
OP = {"logprob_fwd": 0, "loss_bwd": 1, "divergence": 2, "topk_fwd": 3, "splice_masked": 4,
      "topk_kl_bwd": 5, "loss_fwd_bwd": 6, "opd_stats": 7, "topk_kl_fwd_bwd": 8,
      "loss_fwd_bwd_slab": 9}


class OliveError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int32
_F = ctypes.c_float
_S = ctypes.c_size_t


def lib() -> ctypes.CDLL:
    """Loads libolive.so (raises if it is not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise OliveError(8, f"libolive.so not found at {LIB_PATH}; build it with "
                            "paper_2609_36246_gb300.build.build()")
    _lib = _configure(ctypes.CDLL(LIB_PATH))
    return _lib


def use_library(path: str) -> ctypes.CDLL:
    """Makes every call of this module go through the library at `path`
    (e.g. the OLIVE_DEBUG build, paper_2609_36246_gb300.build.build(debug=True))
    and returns it; use_library(LIB_PATH) goes back to the release build."""
    global _lib
    _lib = _configure(ctypes.CDLL(path))
    return _lib


def _configure(L: ctypes.CDLL) -> ctypes.CDLL:
    L.olive_abi_version.restype = ctypes.c_int
    L.olive_abi_version.argtypes = []
    L.olive_slab_rows.restype = _I
    L.olive_slab_rows.argtypes = [_I, _I]
    L.olive_status_string.restype = ctypes.c_char_p
    L.olive_status_string.argtypes = [ctypes.c_int]
    L.olive_workspace_size.restype = _S
    L.olive_workspace_size.argtypes = [ctypes.c_int, _I, _I, _I, _I, ctypes.c_int, ctypes.c_int]
    L.olive_splice_pack.restype = ctypes.c_int
    L.olive_splice_pack.argtypes = [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P]
    L.olive_token_logprob_fwd.restype = ctypes.c_int
    L.olive_token_logprob_fwd.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I, _F, ctypes.c_int,
                                          _P, _P, _P, _P, _S, _P, _P]
    L.olive_token_loss_bwd.restype = ctypes.c_int
    L.olive_token_loss_bwd.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I, _F, ctypes.c_int, _P, _P,
                                       _P, _P, ctypes.c_int, _P, _S, _P, _P]
    L.olive_token_divergence.restype = ctypes.c_int
    L.olive_token_divergence.argtypes = [_P, _P, _I, _P, _P, _I, _P, _P, _I, _I, _F, ctypes.c_int,
                                         _P, _P, _P, ctypes.c_int, _P, _S, _P, _P]
    L.olive_splice_pack_masked.restype = ctypes.c_int
    L.olive_splice_pack_masked.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P,
                                           _P, _P, _S, _P, _P]
    L.olive_topk_compare.restype = ctypes.c_int
    L.olive_topk_compare.argtypes = [_P, _P, _I, _P, _P, _I, _I, _F, _I, _P, _P, _P, _P, _P, _P, _P,
                                     _P, _P]
    L.olive_scale.restype = ctypes.c_int
    L.olive_scale.argtypes = [_P, _P, _S, ctypes.c_int, _P, _P]
    L.olive_opd_token_stats.restype = ctypes.c_int
    L.olive_opd_token_stats.argtypes = [_P, _P, _I, _P, _P, _I, _P, _P, _I, _I, _F, ctypes.c_int, _I,
                                        _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _S, _P, _P]
    L.olive_token_loss_fwd_bwd.restype = ctypes.c_int
    L.olive_token_loss_fwd_bwd.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I, _F, ctypes.c_int, _P, _P,
                                           _P, _P, _P, _P, ctypes.c_int, _P, _S, _P, _P]
    L.olive_token_loss_fwd_bwd_slab.restype = ctypes.c_int
    L.olive_token_loss_fwd_bwd_slab.argtypes = L.olive_token_loss_fwd_bwd.argtypes
    L.olive_topk_kl_fwd_bwd.restype = ctypes.c_int
    L.olive_topk_kl_fwd_bwd.argtypes = [_P, _P, _I, _P, _P, _I, _P, _P, _I, _I, _F, _I, _P, _P, _P,
                                        _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_int, _P, _S, _P,
                                        _P]
    L.olive_topk_kl_bwd.restype = ctypes.c_int
    L.olive_topk_kl_bwd.argtypes = [_P, _P, _P, _P, _I, _I, _I, _F, _I, _P, _P, _P, _P, _P, _P, _P,
                                    _P, ctypes.c_int, _P, _S, _P, _P]
    L.olive_token_topk_fwd.restype = ctypes.c_int
    L.olive_token_topk_fwd.argtypes = [_P, _P, _P, _P, _I, _I, _I, _F, _I, _P, _P, _P, _P, _P, _S,
                                       _P, _P]
    L.olive_token_logprob_fwd_noalloc.restype = ctypes.c_int
    L.olive_token_logprob_fwd_noalloc.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I, _F, ctypes.c_int,
                                                  _P, _P, _P, _P, _P]
    return L


def declared_symbols() -> list[str]:
    """Entry points declared with OLIVE_API in include/olive.h."""
    with open(HEADER) as f:
        text = f.read()
    return re.findall(r"OLIVE_API\s+[\w\s\*]*?\b(olive_\w+)\s*\(", text)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _check(st: int, where: str):
    if st != OLIVE_OK:
        raise OliveError(st, where)


def _need(t, dtype, name):
    if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise TypeError(f"{name} must be a contiguous CUDA {dtype} tensor")


def new_status(device=None) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


def status_bits(dev_status: torch.Tensor) -> list[str]:
    """Names of the error bits set in a device status word (synchronises)."""
    v = int(dev_status.item())
    return [STATUS_NAMES[c] for c in range(1, 11) if v & (1 << c)]


def olive_abi_version() -> int:
    return lib().olive_abi_version()


def olive_status_string(status: int) -> str:
    return lib().olive_status_string(status).decode()


def olive_workspace_size(op: str, T: int, d: int, V: int, d_t: int = 0, grad: bool = True,
                         grad_dtype=torch.bfloat16) -> int:
    return int(lib().olive_workspace_size(OP[op], T, d, d_t, V, int(grad), DTYPE[grad_dtype]))


def olive_slab_rows(T: int, V: int) -> int:
    """Rows of one G slab of the slab forms for T packed rows and V vocabulary
    entries (the library's rule, OLIVE_SLAB_ROWS included)."""
    return int(lib().olive_slab_rows(T, V))


def workspace(nbytes: int, device=None) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device or "cuda")


def _pack_outputs(S: int, T_cap: int, dev, dev_status):
    out = {
        "ids": torch.empty(T_cap, dtype=torch.int32, device=dev),
        "targets": torch.empty(T_cap, dtype=torch.int32, device=dev),
        "loss_mask": torch.empty(T_cap, dtype=torch.uint8, device=dev),
        "cu_seqlens": torch.empty(S + 1, dtype=torch.int32, device=dev),
        "cut_offsets": torch.empty(max(S, 1), dtype=torch.int32, device=dev),
        "rows": torch.empty(T_cap, dtype=torch.int32, device=dev),
        "n_rows": torch.empty(1, dtype=torch.int32, device=dev),
    }
    out["dev_status"] = dev_status if dev_status is not None else new_status(dev)
    return out


def olive_splice_pack(prefix_ids, prefix_off, cont_ids, cont_off, V: int, T_cap: int,
                      dev_status=None) -> dict:
    """Packs the spliced sequences; returns the device outputs of olive.h."""
    for t, n in ((prefix_ids, "prefix_ids"), (prefix_off, "prefix_off"), (cont_ids, "cont_ids"),
                 (cont_off, "cont_off")):
        _need(t, torch.int32, n)
    S = prefix_off.numel() - 1
    dev = prefix_off.device
    out = _pack_outputs(S, T_cap, dev, dev_status)
    # empty id arrays still need a valid device address
    pid = prefix_ids if prefix_ids.numel() else torch.zeros(1, dtype=torch.int32, device=dev)
    cid = cont_ids if cont_ids.numel() else torch.zeros(1, dtype=torch.int32, device=dev)
    st = lib().olive_splice_pack(_ptr(pid), _ptr(prefix_off), _ptr(cid), _ptr(cont_off), S, V, T_cap,
                                 _ptr(out["ids"]), _ptr(out["targets"]), _ptr(out["loss_mask"]),
                                 _ptr(out["cu_seqlens"]), _ptr(out["cut_offsets"]),
                                 _ptr(out["rows"]), _ptr(out["n_rows"]), _ptr(out["dev_status"]),
                                 _stream())
    _check(st, "olive_splice_pack")
    return out


def olive_splice_pack_masked(prefix_ids, prefix_off, cont_ids, cont_off, cont_loss, V: int,
                             T_cap: int, dev_status=None) -> dict:
    """Multi-turn packing: cont_loss (uint8, one flag per continuation id)
    selects the teacher-action tokens that carry the loss."""
    for t, n in ((prefix_ids, "prefix_ids"), (prefix_off, "prefix_off"), (cont_ids, "cont_ids"),
                 (cont_off, "cont_off")):
        _need(t, torch.int32, n)
    _need(cont_loss, torch.uint8, "cont_loss")
    S = prefix_off.numel() - 1
    dev = prefix_off.device
    out = _pack_outputs(S, T_cap, dev, dev_status)
    pid = prefix_ids if prefix_ids.numel() else torch.zeros(1, dtype=torch.int32, device=dev)
    cid = cont_ids if cont_ids.numel() else torch.zeros(1, dtype=torch.int32, device=dev)
    cfl = cont_loss if cont_loss.numel() else torch.zeros(1, dtype=torch.uint8, device=dev)
    ws = workspace(olive_workspace_size("splice_masked", T_cap, 8, 1), dev)
    st = lib().olive_splice_pack_masked(_ptr(pid), _ptr(prefix_off), _ptr(cid), _ptr(cont_off),
                                        _ptr(cfl), S, V, T_cap, _ptr(out["ids"]),
                                        _ptr(out["targets"]), _ptr(out["loss_mask"]),
                                        _ptr(out["cu_seqlens"]), _ptr(out["cut_offsets"]),
                                        _ptr(out["rows"]), _ptr(out["n_rows"]), _ptr(ws), ws.numel(),
                                        _ptr(out["dev_status"]), _stream())
    _check(st, "olive_splice_pack_masked")
    return out


def olive_token_logprob_fwd(hidden, W, targets, rows, n_rows, inv_tau: float = 1.0,
                            reduction: str = "sum", ws=None, dev_status=None, out=None):
    """Per-token log-probs, lse and the Eq. (osd-ce) loss. Returns (logp, lse, loss)."""
    _need(hidden, torch.bfloat16, "hidden")
    _need(W, torch.bfloat16, "W")
    _need(targets, torch.int32, "targets")
    _need(rows, torch.int32, "rows")
    _need(n_rows, torch.int32, "n_rows")
    T, d = hidden.shape
    V = W.shape[0]
    if W.shape[1] != d:
        raise ValueError("hidden and W widths differ")
    dev = hidden.device
    if out is None:
        out = (torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(1, dtype=torch.float32, device=dev))
    logp, lse, loss = out
    need = olive_workspace_size("logprob_fwd", T, d, V)
    if ws is None:
        ws = workspace(need, dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_token_logprob_fwd(_ptr(hidden), _ptr(W), _ptr(targets), _ptr(rows), _ptr(n_rows),
                                       T, d, V, float(inv_tau), REDUCE[reduction], _ptr(logp),
                                       _ptr(lse), _ptr(loss), _ptr(ws), ws.numel(), _ptr(ds),
                                       _stream())
    _check(st, "olive_token_logprob_fwd")
    return logp, lse, loss


def olive_token_topk_fwd(hidden, W, rows, n_rows, K: int = 16, inv_tau: float = 1.0, ws=None,
                         dev_status=None):
    """Per-token lse, entropy and the K largest log-probs with their ids.

    Returns (lse [T], entropy [T], topk_logp [T, K], topk_ids [T, K])."""
    _need(hidden, torch.bfloat16, "hidden")
    _need(W, torch.bfloat16, "W")
    _need(rows, torch.int32, "rows")
    _need(n_rows, torch.int32, "n_rows")
    T, d = hidden.shape
    V = W.shape[0]
    dev = hidden.device
    lse = torch.empty(T, dtype=torch.float32, device=dev)
    ent = torch.empty(T, dtype=torch.float32, device=dev)
    tv = torch.empty(T, K, dtype=torch.float32, device=dev)
    ti = torch.empty(T, K, dtype=torch.int32, device=dev)
    if ws is None:
        ws = workspace(olive_workspace_size("topk_fwd", T, d, V), dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_token_topk_fwd(_ptr(hidden), _ptr(W), _ptr(rows), _ptr(n_rows), T, d, V,
                                    float(inv_tau), int(K), _ptr(lse), _ptr(ent), _ptr(tv), _ptr(ti),
                                    _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_token_topk_fwd")
    return lse, ent, tv, ti


def olive_topk_compare(h_t, W_t, rows, n_rows, s_ids, s_logp, t_ids, t_lse, inv_tau: float = 1.0,
                       dev_status=None, want_t_logp=False):
    """Top-K overlap ratio and top-K truncated reverse KL per masked row.

    Returns (overlap [T], kl_topk [T]), plus the teacher's log-probs at the
    student's top-K ids [T, K] when want_t_logp."""
    _need(h_t, torch.bfloat16, "h_t")
    _need(W_t, torch.bfloat16, "W_t")
    _need(s_ids, torch.int32, "s_ids")
    _need(t_ids, torch.int32, "t_ids")
    _need(s_logp, torch.float32, "s_logp")
    _need(t_lse, torch.float32, "t_lse")
    T, d_t = h_t.shape
    V = W_t.shape[0]
    K = s_ids.shape[1]
    dev = h_t.device
    ov = torch.empty(T, dtype=torch.float32, device=dev)
    kl = torch.empty(T, dtype=torch.float32, device=dev)
    tlp = torch.empty(T, K, dtype=torch.float32, device=dev) if want_t_logp else None
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_topk_compare(_ptr(h_t), _ptr(W_t), d_t, _ptr(rows), _ptr(n_rows), T, V,
                                  float(inv_tau), K, _ptr(s_ids), _ptr(s_logp), _ptr(t_ids),
                                  _ptr(t_lse), _ptr(ov), _ptr(kl), _ptr(tlp), _ptr(ds), _stream())
    _check(st, "olive_topk_compare")
    return (ov, kl, tlp) if want_t_logp else (ov, kl)


OPD_STATS_KEYS = ("kl", "s_lse", "t_lse", "s_entropy", "s_topk_logp", "s_topk_ids", "t_logp_s",
                  "overlap", "kl_topk")


def olive_opd_token_stats(h_s, W_s, h_t, W_t, rows, n_rows, K: int = 16, inv_tau: float = 1.0,
                          direction: str = "reverse", want=OPD_STATS_KEYS, ws=None,
                          dev_status=None) -> dict:
    """OPD's per-token KL, lse of both heads, student entropy and top-K lists,
    teacher log-probs at the student's top-K ids, top-K overlap and top-K KL
    from one sweep.  Returns a dict with the requested keys of OPD_STATS_KEYS."""
    for t, n in ((h_s, "h_s"), (W_s, "W_s"), (h_t, "h_t"), (W_t, "W_t")):
        _need(t, torch.bfloat16, n)
    _need(rows, torch.int32, "rows")
    _need(n_rows, torch.int32, "n_rows")
    T, d_s = h_s.shape
    d_t = h_t.shape[1]
    V = W_s.shape[0]
    if W_t.shape[0] != V or h_t.shape[0] != T:
        raise ValueError("student and teacher shapes disagree")
    dev = h_s.device
    shapes = {"s_topk_logp": (T, K), "s_topk_ids": (T, K), "t_logp_s": (T, K)}
    out = {}
    for k in OPD_STATS_KEYS:
        if k in want:
            dt = torch.int32 if k == "s_topk_ids" else torch.float32
            out[k] = torch.empty(shapes.get(k, (T,)), dtype=dt, device=dev)
    if ws is None:
        ws = workspace(olive_workspace_size("opd_stats", T, d_s, V, d_t=d_t), dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_opd_token_stats(_ptr(h_s), _ptr(W_s), d_s, _ptr(h_t), _ptr(W_t), d_t,
                                     _ptr(rows), _ptr(n_rows), T, V, float(inv_tau),
                                     DIRECTION[direction], int(K),
                                     *[_ptr(out.get(k)) for k in OPD_STATS_KEYS],
                                     _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_opd_token_stats")
    return out


def olive_topk_kl_bwd(h_s, W_s, rows, n_rows, s_lse, s_ids, s_logp, t_logp_s, kl_topk, grad_kl,
                      inv_tau: float = 1.0, grad_dtype=torch.bfloat16, ws=None, dev_status=None,
                      out=None):
    """Gradient of sum_t grad_kl[t] kl_topk[t] with respect to h_s and W_s,
    the student's top-K set held fixed.  Returns (d_h_s [T, d], d_W_s [V, d])."""
    _need(h_s, torch.bfloat16, "h_s")
    _need(W_s, torch.bfloat16, "W_s")
    _need(s_ids, torch.int32, "s_ids")
    for t, n in ((s_lse, "s_lse"), (s_logp, "s_logp"), (t_logp_s, "t_logp_s"), (kl_topk, "kl_topk"),
                 (grad_kl, "grad_kl")):
        _need(t, torch.float32, n)
    T, d = h_s.shape
    V = W_s.shape[0]
    K = s_ids.shape[1]
    dev = h_s.device
    if out is None:
        out = (torch.empty(T, d, dtype=grad_dtype, device=dev),
               torch.empty(V, d, dtype=grad_dtype, device=dev))
    dh, dw = out
    if ws is None:
        ws = workspace(olive_workspace_size("topk_kl_bwd", T, d, V, grad_dtype=grad_dtype), dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_topk_kl_bwd(_ptr(h_s), _ptr(W_s), _ptr(rows), _ptr(n_rows), T, d, V,
                                 float(inv_tau), K, _ptr(s_lse), _ptr(s_ids), _ptr(s_logp),
                                 _ptr(t_logp_s), _ptr(kl_topk), _ptr(grad_kl), _ptr(dh), _ptr(dw),
                                 DTYPE[grad_dtype], _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_topk_kl_bwd")
    return dh, dw


def olive_topk_kl_fwd_bwd(h_s, W_s, h_t, W_t, rows, n_rows, K, t_lse, grad_kl, t_ids=None,
                          inv_tau: float = 1.0, grad_dtype=torch.bfloat16, ws=None,
                          dev_status=None, out=None):
    """The student's top-K lists, the top-K KL against the teacher and its
    gradient in one sweep of the student's logits.  t_lse (and t_ids, for the
    overlap) come from olive_token_topk_fwd on the teacher.  Returns a dict
    with s_lse, s_ids, s_logp, t_logp_s, kl_topk, overlap (None without
    t_ids), d_h_s and d_W_s."""
    _need(h_s, torch.bfloat16, "h_s")
    _need(W_s, torch.bfloat16, "W_s")
    _need(h_t, torch.bfloat16, "h_t")
    _need(W_t, torch.bfloat16, "W_t")
    _need(t_lse, torch.float32, "t_lse")
    _need(grad_kl, torch.float32, "grad_kl")
    if t_ids is not None:
        _need(t_ids, torch.int32, "t_ids")
    T, ds = h_s.shape
    V = W_s.shape[0]
    dt = h_t.shape[1]
    dev = h_s.device
    if out is None:
        f = lambda *shape: torch.empty(*shape, dtype=torch.float32, device=dev)
        out = dict(s_lse=f(T), s_ids=torch.empty(T, K, dtype=torch.int32, device=dev),
                   s_logp=f(T, K), t_logp_s=f(T, K), kl_topk=f(T),
                   overlap=f(T) if t_ids is not None else None,
                   d_h_s=torch.empty(T, ds, dtype=grad_dtype, device=dev),
                   d_W_s=torch.empty(V, ds, dtype=grad_dtype, device=dev))
    if ws is None:
        ws = workspace(olive_workspace_size("topk_kl_fwd_bwd", T, ds, V, grad_dtype=grad_dtype), dev)
    st_buf = dev_status if dev_status is not None else new_status(dev)
    o = out
    st = lib().olive_topk_kl_fwd_bwd(
        _ptr(h_s), _ptr(W_s), ds, _ptr(h_t), _ptr(W_t), dt, _ptr(rows), _ptr(n_rows), T, V,
        float(inv_tau), K, _ptr(t_lse), _ptr(t_ids) if t_ids is not None else None, _ptr(grad_kl),
        _ptr(o["s_lse"]), _ptr(o["s_ids"]), _ptr(o["s_logp"]), _ptr(o["t_logp_s"]),
        _ptr(o["kl_topk"]), _ptr(o["overlap"]) if o["overlap"] is not None else None,
        _ptr(o["d_h_s"]), _ptr(o["d_W_s"]), DTYPE[grad_dtype], _ptr(ws), ws.numel(),
        _ptr(st_buf), _stream())
    _check(st, "olive_topk_kl_fwd_bwd")
    return out


def olive_token_loss_bwd(hidden, W, targets, rows, n_rows, lse, grad_loss, inv_tau: float = 1.0,
                         reduction: str = "sum", grad_dtype=torch.bfloat16, ws=None,
                         dev_status=None, out=None):
    """d loss/d hidden and d loss/d W. grad_loss is a 1-element fp32 CUDA tensor."""
    _need(hidden, torch.bfloat16, "hidden")
    _need(W, torch.bfloat16, "W")
    _need(lse, torch.float32, "lse")
    _need(grad_loss, torch.float32, "grad_loss")
    T, d = hidden.shape
    V = W.shape[0]
    dev = hidden.device
    if out is None:
        out = (torch.empty(T, d, dtype=grad_dtype, device=dev),
               torch.empty(V, d, dtype=grad_dtype, device=dev))
    dh, dw = out
    need = olive_workspace_size("loss_bwd", T, d, V, grad_dtype=grad_dtype)
    if ws is None:
        ws = workspace(need, dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_token_loss_bwd(_ptr(hidden), _ptr(W), _ptr(targets), _ptr(rows), _ptr(n_rows),
                                    T, d, V, float(inv_tau), REDUCE[reduction], _ptr(lse),
                                    _ptr(grad_loss), _ptr(dh), _ptr(dw), DTYPE[grad_dtype],
                                    _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_token_loss_bwd")
    return dh, dw


def olive_token_loss_fwd_bwd(hidden, W, targets, rows, n_rows, grad_loss, inv_tau: float = 1.0,
                             reduction: str = "sum", grad_dtype=torch.bfloat16, ws=None,
                             dev_status=None, out=None, slab: bool = False):
    """Forward and backward of one training step in one call (G on chip;
    slab=True: olive_token_loss_fwd_bwd_slab, G through an HBM slab).

    grad_loss is a 1-element fp32 CUDA tensor (the loss gradient, known before
    the call).  Returns (logp [T], lse [T], loss [1], d_hidden [T, d], d_W [V, d])."""
    _need(hidden, torch.bfloat16, "hidden")
    _need(W, torch.bfloat16, "W")
    _need(grad_loss, torch.float32, "grad_loss")
    T, d = hidden.shape
    V = W.shape[0]
    dev = hidden.device
    if out is None:
        out = (torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(1, dtype=torch.float32, device=dev),
               torch.empty(T, d, dtype=grad_dtype, device=dev),
               torch.empty(V, d, dtype=grad_dtype, device=dev))
    logp, lse, loss, dh, dw = out
    if ws is None:
        op = "loss_fwd_bwd_slab" if slab else "loss_fwd_bwd"
        ws = workspace(olive_workspace_size(op, T, d, V, grad_dtype=grad_dtype), dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    fn = lib().olive_token_loss_fwd_bwd_slab if slab else lib().olive_token_loss_fwd_bwd
    st = fn(_ptr(hidden), _ptr(W), _ptr(targets), _ptr(rows), _ptr(n_rows), T, d, V,
            float(inv_tau), REDUCE[reduction], _ptr(grad_loss), _ptr(logp), _ptr(lse), _ptr(loss),
            _ptr(dh), _ptr(dw), DTYPE[grad_dtype], _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_token_loss_fwd_bwd_slab" if slab else "olive_token_loss_fwd_bwd")
    return logp, lse, loss, dh, dw


def olive_token_divergence(h_s, W_s, h_t, W_t, rows, n_rows, inv_tau: float = 1.0,
                           direction: str = "reverse", grad_kl=None, grad_dtype=torch.bfloat16,
                           ws=None, dev_status=None):
    """Per-token full-vocabulary KL; with grad_kl also d(sum g_t KL_t)/d h_s.

    Returns (kl [T] fp32, d_h_s or None)."""
    for t, n in ((h_s, "h_s"), (W_s, "W_s"), (h_t, "h_t"), (W_t, "W_t")):
        _need(t, torch.bfloat16, n)
    T, d_s = h_s.shape
    d_t = h_t.shape[1]
    V = W_s.shape[0]
    if W_t.shape[0] != V or h_t.shape[0] != T:
        raise ValueError("student and teacher shapes disagree")
    dev = h_s.device
    kl = torch.empty(T, dtype=torch.float32, device=dev)
    dhs = None
    if grad_kl is not None:
        _need(grad_kl, torch.float32, "grad_kl")
        dhs = torch.empty(T, d_s, dtype=grad_dtype, device=dev)
    need = olive_workspace_size("divergence", T, d_s, V, d_t=d_t, grad=grad_kl is not None)
    if ws is None:
        ws = workspace(need, dev)
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_token_divergence(_ptr(h_s), _ptr(W_s), d_s, _ptr(h_t), _ptr(W_t), d_t,
                                      _ptr(rows), _ptr(n_rows), T, V, float(inv_tau),
                                      DIRECTION[direction], _ptr(kl), _ptr(grad_kl), _ptr(dhs),
                                      DTYPE[grad_dtype], _ptr(ws), ws.numel(), _ptr(ds), _stream())
    _check(st, "olive_token_divergence")
    return kl, dhs


def olive_token_logprob_fwd_noalloc(hidden, W, targets, rows, n_rows, inv_tau: float = 1.0,
                                    reduction: str = "sum", dev_status=None, out=None):
    """olive_token_logprob_fwd without a workspace: scratch comes from the
    library's fixed device array (see include/olive.h for the size limit and
    the rule that overlapping calls must be serialised)."""
    _need(hidden, torch.bfloat16, "hidden")
    _need(W, torch.bfloat16, "W")
    T, d = hidden.shape
    V = W.shape[0]
    dev = hidden.device
    if out is None:
        out = (torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(T, dtype=torch.float32, device=dev),
               torch.empty(1, dtype=torch.float32, device=dev))
    logp, lse, loss = out
    ds = dev_status if dev_status is not None else new_status(dev)
    st = lib().olive_token_logprob_fwd_noalloc(_ptr(hidden), _ptr(W), _ptr(targets), _ptr(rows),
                                               _ptr(n_rows), T, d, V, float(inv_tau),
                                               REDUCE[reduction], _ptr(logp), _ptr(lse), _ptr(loss),
                                               _ptr(ds), _stream())
    _check(st, "olive_token_logprob_fwd_noalloc")
    return logp, lse, loss


def olive_scale(x, scale, out=None):
    """out = x * scale (scale: 1-element fp32 CUDA tensor); bf16 or fp32, in
    place when out is x."""
    if x.dtype not in DTYPE:
        raise TypeError("x must be bf16 or fp32")
    _need(x, x.dtype, "x")
    _need(scale, torch.float32, "scale")
    out = torch.empty_like(x) if out is None else out
    st = lib().olive_scale(_ptr(x), _ptr(out), x.numel(), DTYPE[x.dtype], _ptr(scale), _stream())
    _check(st, "olive_scale")
    return out


class FusedLMHeadCE(torch.autograd.Function):
    """Eq. (osd-ce) loss over the masked rows as an autograd op (gradients in
    the dtype of hidden).

    With a gradient needed, the forward runs olive_token_loss_fwd_bwd with a
    unit loss gradient (each logit tile computed once) and the backward scales
    the stored gradients by the incoming one (olive_scale); otherwise, or with
    single_pass=False, it runs olive_token_logprob_fwd and the backward
    recomputes the logits (olive_token_loss_bwd)."""

    @staticmethod
    def forward(ctx, hidden, W, targets, rows, n_rows, inv_tau=1.0, reduction="sum",
                single_pass=True):
        ctx.inv_tau, ctx.reduction = inv_tau, reduction
        ctx.single = bool(single_pass and (hidden.requires_grad or W.requires_grad))
        if ctx.single:
            one = torch.ones(1, dtype=torch.float32, device=hidden.device)
            _, _, loss, dh, dw = olive_token_loss_fwd_bwd(hidden, W, targets, rows, n_rows, one,
                                                          inv_tau, reduction, grad_dtype=hidden.dtype)
            ctx.save_for_backward(dh, dw)
        else:
            _, lse, loss = olive_token_logprob_fwd(hidden, W, targets, rows, n_rows, inv_tau,
                                                   reduction)
            ctx.save_for_backward(hidden, W, targets, rows, n_rows, lse)
        return loss[0]

    @staticmethod
    def backward(ctx, g):
        gl = g.reshape(1).to(torch.float32).contiguous()
        if ctx.single:
            dh1, dw1 = ctx.saved_tensors
            return (olive_scale(dh1, gl), olive_scale(dw1, gl), None, None, None, None, None, None)
        hidden, W, targets, rows, n_rows, lse = ctx.saved_tensors
        dh, dw = olive_token_loss_bwd(hidden, W, targets, rows, n_rows, lse, gl, ctx.inv_tau,
                                      ctx.reduction, grad_dtype=hidden.dtype)
        return dh, dw, None, None, None, None, None, None


def fused_lmhead_ce(hidden, W, targets, rows, n_rows, inv_tau=1.0, reduction="sum",
                    single_pass=True):
    return FusedLMHeadCE.apply(hidden, W, targets, rows, n_rows, inv_tau, reduction, single_pass)
