"""include/olive.h is a C header and libolive.so a C library: a C11 program
(tests/c_abi/olive_c_check.c) is compiled with gcc against the header alone,
linked to the library, and run.  On the CPU it exercises the host-side entry
points; on a GPU it runs olive_splice_pack, and splice/pack followed by the
on-chip training step, whose outputs are compared with the oracle."""

import os
import shutil
import subprocess

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36246_gb300 import build
from paper_2609_36246_gb300 import synth

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


@pytest.fixture(scope="module")
def exe(tmp_path_factory):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    lib = build.build()
    libdir = os.path.dirname(lib)
    out = str(tmp_path_factory.mktemp("c_abi") / "olive_c_check")
    cmd = ["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(CUDA, "include"), os.path.join(HERE, "c_abi", "olive_c_check.c"),
           "-o", out, "-L", libdir, "-l:libolive.so", f"-Wl,-rpath,{libdir}",
           "-L", os.path.join(CUDA, "lib64"), "-lcudart", f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}",
           "-Wl,--allow-shlib-undefined"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return out


def test_host_entry_points_from_c(exe):
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "ok"


@pytest.mark.gpu
def test_splice_pack_from_c(exe):
    rng = np.random.default_rng(12)
    b = synth.batch_from_lengths(rng, [3, 1, 7], [4, 0, 5], 50)
    lines = [f"{len(b.prefix_off) - 1} {b.V} {b.T + 3}",
             " ".join(map(str, b.prefix_off)), " ".join(map(str, b.prefix_ids)),
             " ".join(map(str, b.cont_off)), " ".join(map(str, b.cont_ids))]
    r = subprocess.run([exe, "splice"], input="\n".join(lines) + "\n", capture_output=True,
                       text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    got = {ln.split()[0]: list(map(int, ln.split()[1:])) for ln in r.stdout.strip().splitlines()}
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)
    assert got["status"] == [0]
    assert got["n_rows"] == [o["n_rows"]]
    assert got["rows"] == o["rows"].tolist()
    assert got["targets"] == o["targets"].tolist()
    assert got["mask"] == o["loss_mask"].astype(int).tolist()


@pytest.mark.gpu
def test_training_step_from_c(exe, tmp_path):
    """splice/pack and the on-chip training step (olive_token_loss_fwd_bwd),
    called from C with a workspace sized through the header: log-probs, lse,
    loss, d_hidden and d_W against the oracle."""
    from tests.parity import assert_close_grad, assert_close_logp, assert_close_loss
    rng = np.random.default_rng(31)
    b = synth.batch_from_lengths(rng, [9, 3, 20], [40, 7, 70], 900)
    d = 192
    h = synth.normal_bf16(rng, (b.T, d), 1.0)
    W = synth.normal_bf16(rng, (b.V, d), 0.1)
    S = len(b.prefix_off) - 1
    path_in, path_out = tmp_path / "step.in", tmp_path / "step.out"
    with open(path_in, "wb") as f:
        f.write(np.array([S, b.V, b.T, d], dtype=np.int32).tobytes())
        for a in (b.prefix_off, b.cont_off, b.prefix_ids, b.cont_ids):
            f.write(np.asarray(a, dtype=np.int32).tobytes())
        for t in (h, W):
            f.write(t.contiguous().view(torch.int16).numpy().tobytes())
    r = subprocess.run([exe, "step", str(path_in), str(path_out)], capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr
    raw = np.fromfile(path_out, dtype=np.float32)
    T, V = b.T, b.V
    assert raw[:1].view(np.int32)[0] == 0
    logp, lse = raw[1:1 + T], raw[1 + T:1 + 2 * T]
    loss = float(raw[1 + 2 * T])
    dh = raw[2 + 2 * T:2 + 2 * T + T * d].reshape(T, d)
    dw = raw[2 + 2 * T + T * d:].reshape(V, d)
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)
    h64, W64 = h.double().numpy(), W.double().numpy()
    rl, rlse, rloss = oracle.token_logprob(h64, W64, o["targets"], o["rows"])
    assert_close_logp(logp, rl)
    assert_close_logp(lse[o["rows"]], rlse[o["rows"]], "lse")
    assert_close_loss(loss, rloss)
    rdh, rdw = oracle.token_loss_bwd(h64, W64, o["targets"], o["rows"])
    assert_close_grad(dh, rdh, "dH")
    assert_close_grad(dw, rdw, "dW")
