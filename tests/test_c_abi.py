"""include/olive.h is a C header and libolive.so a C library: a C11 program
(tests/c_abi/olive_c_check.c) is compiled with gcc against the header alone,
linked to the library, and run.  On the CPU it exercises the host-side entry
points; on a GPU it runs olive_splice_pack, whose output is compared with the
oracle."""

import os
import shutil
import subprocess

import numpy as np
import pytest

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
