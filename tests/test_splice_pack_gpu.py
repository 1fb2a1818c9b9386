"""olive_splice_pack (CUDA) against the oracle: bit-exact integers."""

import json
import os

import numpy as np
import pytest

from paper_2609_36246_gb300 import binding as B
from paper_2609_36246_gb300 import synth
from tests.parity import gpu_pack, oracle_pack

pytestmark = pytest.mark.gpu

KEYS = ("ids", "targets", "loss_mask", "cu_seqlens", "cut_offsets")


def _compare(b, T_cap=None):
    g = gpu_pack(b, T_cap)
    o = oracle_pack(b)
    T = b.T
    n = int(g["n_rows"].item())
    assert n == o["n_rows"]
    for k in KEYS:
        gv = g[k].cpu().numpy().astype(np.int64)
        if k in ("ids", "targets", "loss_mask"):
            gv = gv[:T]
        if k == "cut_offsets":
            gv = gv[:b.S]
        assert np.array_equal(gv, o[k]), k
    assert np.array_equal(g["rows"][:n].cpu().numpy(), o["rows"])
    assert int(g["dev_status"].item()) == 0
    return g


def test_golden_fixture():
    with open(os.path.join(os.path.dirname(__file__), "golden", "splice_pack_small.json")) as f:
        gj = json.load(f)
    b = synth.Batch(np.array(gj["prefix_ids"], np.int32), np.array(gj["prefix_off"], np.int32),
                    np.array(gj["cont_ids"], np.int32), np.array(gj["cont_off"], np.int32), gj["V"])
    g = _compare(b)
    assert g["rows"][:5].tolist() == gj["expect"]["rows"]


@pytest.mark.parametrize("name", ["tiny", "scoring", "kl", "fwdbwd", "varlen"])
def test_workload_batches(name):
    b = synth.make_batch(name)
    g = _compare(b)
    if name == "varlen":
        assert b.T > 200_000


@pytest.mark.parametrize("seed", range(4))
def test_random_batches_with_empty_continuations(seed):
    rng = np.random.default_rng(100 + seed)
    S = int(rng.integers(1, 40))
    P = rng.integers(1, 60, size=S)
    C = rng.integers(0, 60, size=S)
    C[rng.random(S) < 0.3] = 0
    _compare(synth.batch_from_lengths(rng, P, C, 5000))


def test_many_sequences_multi_chunk_scan():
    rng = np.random.default_rng(7)
    S = 3000  # > one 1024-thread scan chunk
    P = rng.integers(1, 5, size=S)
    C = rng.integers(0, 5, size=S)
    _compare(synth.batch_from_lengths(rng, P, C, 100))


def test_capacity_tail_is_cleared():
    b = synth.batch_from_lengths(np.random.default_rng(1), [3, 2], [4, 0], 50)
    g = _compare(b, T_cap=b.T + 37)
    assert (g["ids"][b.T:] == 0).all() and (g["targets"][b.T:] == -1).all()
    assert (g["loss_mask"][b.T:] == 0).all()
    assert (g["rows"][int(g["n_rows"].item()):] == -1).all()


def test_capacity_overflow_and_empty_prefix_flag_offsets():
    b = synth.batch_from_lengths(np.random.default_rng(2), [5, 6], [3, 3], 50)
    g = gpu_pack(b, T_cap=b.T - 1)
    assert "OLIVE_ERR_OFFSETS" in B.status_bits(g["dev_status"])
    assert int(g["n_rows"].item()) == 0
    assert (g["loss_mask"] == 0).all()
    bad = synth.Batch(np.array([1, 2], np.int32), np.array([0, 2, 2], np.int32),
                      np.array([3], np.int32), np.array([0, 1, 1], np.int32), 10)
    g = gpu_pack(bad, T_cap=16)
    assert "OLIVE_ERR_OFFSETS" in B.status_bits(g["dev_status"])


def test_token_out_of_range_is_flagged_and_copied():
    b = synth.Batch(np.array([1, 2, 99], np.int32), np.array([0, 3], np.int32),
                    np.array([-4, 5], np.int32), np.array([0, 2], np.int32), 10)
    g = gpu_pack(b)
    assert B.status_bits(g["dev_status"]) == ["OLIVE_ERR_TOKEN_RANGE"]
    assert g["ids"].tolist() == [1, 2, 99, -4, 5]
