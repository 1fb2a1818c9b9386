"""Shared helpers for the GPU parity tests (CUDA path vs the fp64 oracle).

Tolerances (floating point):
  log-probs, lse, KL : |gpu - ref| <= 2e-3 + 2e-3 |ref|   (element by element)
  loss               : |gpu - ref| <= 1e-3 |ref|  (absolute 1e-6 when ref = 0)
  gradients          : ||gpu - ref||_F <= 1e-2 ||ref||_F
Integer outputs of splice/pack are compared bit for bit.
"""

from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth

LOGP_ATOL = 2e-3
LOGP_RTOL = 2e-3
LOSS_RTOL = 1e-3
GRAD_RTOL = 1e-2

# Rows the oracle recomputes one by one at the full workload sizes (d = 4096,
# V = 151936): log-probs / lse / KL and the hidden-state gradient are compared
# element by element on this many seeded masked rows of the GPU's full run.
FULL_SIZE_ROWS = 2048


def assert_close_logp(gpu, ref, what="logp"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(gpu - ref)
    bound = LOGP_ATOL + LOGP_RTOL * np.abs(ref)
    bad = ~(err <= bound)
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside tolerance; "
                           f"worst err {np.nanmax(err):.3e} at {int(np.nanargmax(err))}")


def assert_close_loss(gpu, ref):
    gpu, ref = float(gpu), float(ref)
    if ref == 0.0:
        assert abs(gpu) <= 1e-6, (gpu, ref)
    else:
        assert abs(gpu - ref) <= LOSS_RTOL * abs(ref), (gpu, ref, abs(gpu - ref) / abs(ref))


def rel_frob(gpu, ref) -> float:
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    num = np.linalg.norm(gpu - ref)
    den = np.linalg.norm(ref)
    return float(num / den) if den > 0 else float(num)


def assert_close_grad(gpu, ref, what="grad"):
    r = rel_frob(gpu, ref)
    ref_norm = np.linalg.norm(np.asarray(ref, dtype=np.float64))
    if ref_norm == 0:
        assert r <= 1e-6, f"{what}: expected zeros, |gpu| = {r:.3e}"
    else:
        assert r <= GRAD_RTOL, f"{what}: relative Frobenius error {r:.3e}"


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact widening of a (bf16 / fp32) tensor to float64 numpy."""
    return t.detach().to("cpu").double().numpy()


def to_f32(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> float32 numpy (exact), for the oracle's big inputs."""
    return t.detach().to("cpu").float().numpy()


def batch_to_cuda(b: synth.Batch):
    dev = "cuda"
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)
    return f(b.prefix_ids), f(b.prefix_off), f(b.cont_ids), f(b.cont_off)


def gpu_pack(b: synth.Batch, T_cap: int | None = None):
    pi, po, ci, co = batch_to_cuda(b)
    return B.olive_splice_pack(pi, po, ci, co, b.V, T_cap if T_cap is not None else max(b.T, 1))


def oracle_pack(b: synth.Batch):
    return oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)


def sample_rows(rows: np.ndarray, k: int, seed: int) -> np.ndarray:
    """k masked rows spread over the list (first, last and random ones)."""
    rows = np.asarray(rows)
    if len(rows) <= k:
        return rows
    rng = np.random.default_rng(seed)
    pick = rng.choice(len(rows), size=k - 2, replace=False)
    idx = np.unique(np.concatenate([[0, len(rows) - 1], pick]))
    return rows[idx]
