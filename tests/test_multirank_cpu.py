"""bench.py's multi-rank host logic on CPU with two gloo ranks.

Under torchrun every rank runs its own replica (no collective on the data
path); the timing is the maximum over ranks and rank 0 alone prints the JSON
line.  The reference arm runs on rank 0 only.  This drives those pieces with
world_size 2 over gloo (127.0.0.1), substituting the tiny workload for the
inputs so the test stays short.
"""

import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    from paper_2609_36246_gb300 import synth

    def tiny_inputs(_rank):
        b = synth.make_batch("tiny")
        return b, synth.make_hidden("tiny", b.T), synth.make_weight("tiny")

    bench.make_inputs = tiny_inputs
    w, r, _ = bench.dist_setup()
    assert dist.get_backend() == "gloo"
    m = bench.max_over_ranks(10.0 * (r + 1), w)

    class Args:
        steps, warmup, cpu_rows = 2, 1, 8

    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(Args, w, r)
    bench.barrier(w)
    dist.destroy_process_group()
    q.put((r, m, buf.getvalue()))


@pytest.mark.timeout(300)
def test_two_gloo_ranks_max_timing_and_rank0_output():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = {}
    for _ in procs:
        r, m, text = q.get(timeout=240)
        out[r] = (m, text)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # the timing reduction is the maximum over ranks on every rank
    assert out[0][0] == out[1][0] == 20.0
    # rank 0 prints exactly one JSON line, the other rank nothing
    assert out[1][1] == ""
    lines = [l for l in out[0][1].splitlines() if l.strip()]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == 2 and rec["value"] > 0
    assert rec["cpu_baseline"]["kind"] == "oracle"
    assert rec["e2e"]["h2d_bytes_per_step"] == 0
