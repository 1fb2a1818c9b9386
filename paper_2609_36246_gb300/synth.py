"""Seeded synthetic inputs shaped like the OLIVE reasoning workload.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic, so both the CUDA path and the fp64 oracle consume what it
produces.  Every workload is generated from a numpy PCG64 stream (platform
independent) and rounded fp32 -> bf16 by round-to-nearest-even (torch).

Workloads (the paper's RLVE setting: prefix cut at student token 4096 with a
1024-token teacher continuation, 64 prompts x 4 rollouts per step; Section 4.1
and Appendix A, Table rose-config).  The paper prints neither the hidden width
nor the vocabulary size; the widths below are those of the measured workloads:
student d=4096 (2048 in the scoring case), teacher d=5120, V=151936.

  tiny     4 x 128 tokens, cut ~ U[16,112), ids ~ U[0,4096), d=256, V=4096,
           hidden and W ~ N(0, 0.02)
  scoring  2 sequences, prefix 4096 + continuation 4096, d=2048, V=151936,
           hidden = RMS-normalised N(0,1), W ~ N(0, 0.02)
  kl       16384 scored rows; student d=4096, teacher d=5120, V=151936,
           independent hidden/W drawn as in "scoring"
  fwdbwd   8 x 4096 tokens, cut ~ U[256,3840), d=4096, V=151936
  varlen   64 sequences, length ~ U[1024,16384], cut = floor(u*len) with
           u ~ U[0.1,0.9], d=4096, V=151936
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

RMS_EPS = 1e-6  # RMS-normalisation epsilon for the synthetic hidden states


@dataclass
class Batch:
    """A packed batch in the CSR form the splice/pack step takes."""

    prefix_ids: np.ndarray  # int32, all prefixes back to back
    prefix_off: np.ndarray  # int32 [S+1]
    cont_ids: np.ndarray    # int32, all continuations back to back
    cont_off: np.ndarray    # int32 [S+1]
    V: int

    @property
    def S(self) -> int:
        return len(self.prefix_off) - 1

    @property
    def T(self) -> int:
        return int(self.prefix_off[-1] + self.cont_off[-1])

    @property
    def n_mask(self) -> int:
        return int(self.cont_off[-1])


WORKLOADS = {
    "tiny": dict(seed=0, d=256, V=4096, hidden="normal002"),
    "scoring": dict(seed=1, d=2048, V=151936, hidden="rms"),
    "kl": dict(seed=2, d=4096, d_t=5120, V=151936, hidden="rms", T=16384),
    "fwdbwd": dict(seed=3, d=4096, V=151936, hidden="rms"),
    "varlen": dict(seed=4, d=4096, V=151936, hidden="rms"),
}


def _csr(parts):
    off = np.zeros(len(parts) + 1, dtype=np.int32)
    off[1:] = np.cumsum([len(p) for p in parts])
    ids = np.concatenate(parts).astype(np.int32) if parts else np.zeros(0, np.int32)
    return ids, off


def batch_from_lengths(rng: np.random.Generator, prefix_lens, cont_lens, V: int) -> Batch:
    """Uniform ids in [0, V) for the given per-sequence prefix/continuation lengths."""
    pre = [rng.integers(0, V, size=int(p), dtype=np.int64) for p in prefix_lens]
    con = [rng.integers(0, V, size=int(c), dtype=np.int64) for c in cont_lens]
    pi, po = _csr(pre)
    ci, co = _csr(con)
    return Batch(pi, po, ci, co, V)


def make_batch(name: str) -> Batch:
    """Token-id batch of a named workload (see the module docstring)."""
    w = WORKLOADS[name]
    rng = np.random.default_rng([w["seed"], 1])
    V = w["V"]
    if name == "tiny":
        cut = rng.integers(16, 112, size=4)
        return batch_from_lengths(rng, cut, 128 - cut, V)
    if name == "scoring":
        return batch_from_lengths(rng, [4096, 4096], [4096, 4096], V)
    if name == "kl":
        # one context row followed by 16384 scored rows
        return batch_from_lengths(rng, [1], [w["T"]], V)
    if name == "fwdbwd":
        cut = rng.integers(256, 3840, size=8)
        return batch_from_lengths(rng, cut, 4096 - cut, V)
    if name == "varlen":
        L = rng.integers(1024, 16384, size=64, endpoint=True)
        u = rng.uniform(0.1, 0.9, size=64)
        cut = np.floor(u * L).astype(np.int64)
        return batch_from_lengths(rng, cut, L - cut, V)
    raise KeyError(name)


def to_bf16(x: np.ndarray) -> torch.Tensor:
    """fp32 numpy -> bf16 torch (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def normal_bf16(rng: np.random.Generator, shape, std: float) -> torch.Tensor:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    x *= np.float32(std)
    return to_bf16(x)


def rms_hidden_bf16(rng: np.random.Generator, shape) -> torch.Tensor:
    """N(0,1) rows scaled to unit RMS in fp32, then rounded to bf16."""
    x = rng.standard_normal(size=shape, dtype=np.float32)
    ms = np.mean(np.square(x, dtype=np.float32), axis=1, keepdims=True, dtype=np.float32)
    x /= np.sqrt(ms + np.float32(RMS_EPS))
    return to_bf16(x)


def make_hidden(name: str, T: int, d: int | None = None, stream: int = 2) -> torch.Tensor:
    """bf16 hidden states [T, d] for a workload (CPU tensor)."""
    w = WORKLOADS[name]
    d = w["d"] if d is None else d
    rng = np.random.default_rng([w["seed"], stream])
    if w["hidden"] == "normal002":
        return normal_bf16(rng, (T, d), 0.02)
    return rms_hidden_bf16(rng, (T, d))


def make_weight(name: str, V: int | None = None, d: int | None = None, stream: int = 3) -> torch.Tensor:
    """bf16 LM-head weight [V, d] ~ N(0, 0.02) for a workload (CPU tensor)."""
    w = WORKLOADS[name]
    V = w["V"] if V is None else V
    d = w["d"] if d is None else d
    rng = np.random.default_rng([w["seed"], stream])
    return normal_bf16(rng, (V, d), 0.02)


def make_teacher(name: str, T: int) -> tuple[torch.Tensor, torch.Tensor]:
    """Teacher hidden [T, d_t] and weight [V, d_t] for the KL workload."""
    w = WORKLOADS[name]
    d_t = w.get("d_t", w["d"])
    h = make_hidden(name, T, d=d_t, stream=4)
    W = make_weight(name, d=d_t, stream=5)
    return h, W


def random_case(seed: int, S: int, V: int, d: int, min_prefix=1, max_prefix=40,
                max_cont=40, std_h=1.0, std_w=0.05):
    """Small random batch + bf16 hidden/W for parity tests of any shape."""
    rng = np.random.default_rng([seed, 7])
    P = rng.integers(min_prefix, max_prefix + 1, size=S)
    C = rng.integers(0, max_cont + 1, size=S)
    b = batch_from_lengths(rng, P, C, V)
    h = normal_bf16(rng, (b.T, d), std_h)
    W = normal_bf16(rng, (V, d), std_w)
    return b, h, W
