"""Throughput of the OLIVE per-token training path on GB300.

One step = the whole hot path over one packed batch: splice/pack of the
spliced sequences (student prefix || teacher continuation), then one
olive_token_loss_fwd_bwd call: the LM-head forward with online log-sum-exp
and the masked continuation loss of Eq. (osd-ce) (log-probs, lse, loss) and
its backward (d hidden, d W in bf16), the logit gradient formed and consumed
on chip (no [rows, V] array is stored; the logits are computed twice, once
per pass).  Workload: 8 sequences of 4096 tokens, cut ~ U[256, 3840),
d = 4096, V = 151936, bf16, synthetic seeded data (the "fwdbwd" workload of
paper_2609_36246_gb300.synth).

Metric: masked continuation tokens per second, i.e. N_mask * steps / time,
and the fraction of bf16 dense tensor peak of the counted work
6 * N_mask * d * V FLOPs per step (forward product, dH and dW products).
Secondary lines on the same batch: the slab form
(olive_token_loss_fwd_bwd_slab, which keeps e' = exp(z - R) for every masked
row in HBM and computes each logit once) and the two-call path
(olive_token_logprob_fwd + olive_token_loss_bwd).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun (N > 1) every rank runs its own batch of the same shape with
no collective on the data path (weak scaling); rank 0 prints the line.
"""

from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "masked continuation tokens/sec (fwd+bwd, fused LM-head loss) and % bf16 tensor peak"
WORKLOAD = "fwdbwd"
CONFIG = {"workload": "fused fwd+bwd LM-head loss: 8 x 4096 packed tokens, cut ~ U[256,3840), "
                      "d=4096, V=151936, bf16",
          "S": 8, "seq_len": 4096, "d": 4096, "V": 151936, "grad_dtype": "bf16",
          "l2": "inputs larger than L2 (hidden 268 MB, W 1.24 GB)"}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("bf16_tflops", 1900.0), d.get("bf16_tflops_sustained", 1700.0), "measured"
    return 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out = ""

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def make_inputs(rank: int):
    from paper_2609_36246_gb300 import synth
    b = synth.make_batch(WORKLOAD)
    h = synth.make_hidden(WORKLOAD, b.T)
    W = synth.make_weight(WORKLOAD)
    return b, h, W


# --------------------------------------------------------------------------- oracle legs
def oracle_sample_rate(b, h, W, n_rows: int, seed: int = 0, warm: bool = True):
    """fp64 oracle on samples of masked rows: forward log-probs, dH of those
    rows and their dW contribution (the same per-row work as one step).  Each
    oracle call also pays a fixed cost (W widened to fp64, the [V, d] fp64 dW
    zeroed and written: seconds at V = 151936, d = 4096), so the rate is
    differential: after one untimed call (first-touch costs), the same
    computation on n and on 5n rows, rate = 4n / (t(5n) - t(n)),
    fixed = t(n) - n / rate (if t(5n) <= t(n), the plain 5n / t(5n)).
    Returns (masked tokens per second, fixed seconds, seconds timed, rows)."""
    import oracle
    o = oracle.splice_pack(b.prefix_ids, b.prefix_off, b.cont_ids, b.cont_off, b.V)
    rng = np.random.default_rng(seed)
    hf = h.float().numpy()
    Wf = W.float().numpy()

    def run(k):
        rows = np.sort(rng.choice(o["rows"], size=min(k, len(o["rows"])), replace=False))
        t0 = time.perf_counter()
        oracle.token_logprob(hf, Wf, o["targets"], rows)
        oracle.token_loss_bwd(hf, Wf, o["targets"], rows)
        return time.perf_counter() - t0

    if warm:
        run(n_rows)
    t1, t5 = run(n_rows), run(5 * n_rows)
    if t5 > t1:
        rate = 4 * n_rows / (t5 - t1)
        fixed = max(t1 - n_rows / rate, 0.0)
    else:
        rate, fixed = 5 * n_rows / t5, 0.0
    return rate, fixed, t1 + t5, 6 * n_rows


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


# --------------------------------------------------------------------------- GPU arm
def run_ours(args, world, rank, local):
    from paper_2609_36246_gb300 import binding as B
    from paper_2609_36246_gb300 import build as _build

    _build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    b, h_cpu, W_cpu = make_inputs(rank)
    N_mask, T, d, V = b.n_mask, b.T, 4096, 151936
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32))
    pre_h, poff_h, con_h, coff_h = (i32(b.prefix_ids).pin_memory(), i32(b.prefix_off).pin_memory(),
                                    i32(b.cont_ids).pin_memory(), i32(b.cont_off).pin_memory())
    hid_h = h_cpu.pin_memory()
    pre, poff, con, coff = (x.to(dev) for x in (pre_h, poff_h, con_h, coff_h))
    hidden = hid_h.to(dev)
    W = W_cpu.to(dev)
    st = B.new_status(dev)
    ws_fb = B.workspace(B.olive_workspace_size("loss_fwd_bwd", T, d, V, grad_dtype=torch.bfloat16),
                        dev)
    logp = torch.empty(T, dtype=torch.float32, device=dev)
    lse = torch.empty_like(logp)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    dh = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
    dw = torch.empty(V, d, dtype=torch.bfloat16, device=dev)
    gl = torch.ones(1, dtype=torch.float32, device=dev)
    loss_h = torch.empty(1, dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream()

    ev = {k: [] for k in ("splice", "fwd_bwd")}

    def step(timed: bool):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)] if timed else None
        if e: e[0].record(stream)
        pk = B.olive_splice_pack(pre, poff, con, coff, V, T, dev_status=st)
        if e: e[1].record(stream)
        B.olive_token_loss_fwd_bwd(hidden, W, pk["targets"], pk["rows"], pk["n_rows"], gl, 1.0,
                                   "sum", torch.bfloat16, ws=ws_fb, dev_status=st,
                                   out=(logp, lse, loss, dh, dw))
        if e:
            e[2].record(stream)
            ev["splice"].append((e[0], e[1]))
            ev["fwd_bwd"].append((e[1], e[2]))

    for _ in range(args.warmup):
        step(False)
    torch.cuda.synchronize()
    if int(st.item()) != 0:
        raise RuntimeError(f"device status {B.status_bits(st)}")

    # ---- device-resident timed region ----
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(args.steps):
            step(True)
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms_local = t0.elapsed_time(t1)
    ms = max_over_ranks(ms_local, world)
    ms_per_step = ms / args.steps
    total_tokens = N_mask * args.steps * world
    value = total_tokens / (ms / 1e3)

    # ---- end to end through the public API with host buffers ----
    # every step copies its inputs from pinned host memory and reads its loss
    # back; the copy of step i+1 runs on a second stream while step i
    # computes (two device input sets), as a training loop would overlap them
    barrier(world)
    torch.cuda.synchronize()
    e_steps = max(1, args.steps)
    host_in = (pre_h, poff_h, con_h, coff_h, hid_h)
    dev_in = [(pre, poff, con, coff, hidden), tuple(torch.empty_like(x) for x in (pre, poff, con, coff, hidden))]
    copy_stream = torch.cuda.Stream()
    ready = [torch.cuda.Event(), torch.cuda.Event()]
    free = [torch.cuda.Event(), torch.cuda.Event()]

    def copy_in(k):
        copy_stream.wait_event(free[k])  # the step that last read this set is done
        with torch.cuda.stream(copy_stream):
            for dst, src in zip(dev_in[k], host_in):
                dst.copy_(src, non_blocking=True)
        ready[k].record(copy_stream)

    def e2e_steps(n):
        for k in (0, 1):
            free[k].record(stream)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        copy_stream.wait_event(e0)
        copy_in(0)
        for i in range(n):
            k = i % 2
            if i + 1 < n:
                copy_in(1 - k)
            stream.wait_event(ready[k])
            p_, po_, c_, co_, h_ = dev_in[k]
            pk_e = B.olive_splice_pack(p_, po_, c_, co_, V, T, dev_status=st)
            B.olive_token_loss_fwd_bwd(h_, W, pk_e["targets"], pk_e["rows"], pk_e["n_rows"], gl,
                                       1.0, "sum", torch.bfloat16, ws=ws_fb, dev_status=st,
                                       out=(logp, lse, loss, dh, dw))
            free[k].record(stream)
            loss_h.copy_(loss, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0, e1

    # untimed warm-up of this loop (the first use of the copy stream and of the
    # second input set costs ~14 ms once), then the timed steps
    e2e_steps(2)
    barrier(world)
    e0, e1 = e2e_steps(e_steps)
    e_ms = max_over_ranks(e0.elapsed_time(e1), world)
    h2d = sum(x.numel() * x.element_size() for x in host_in)
    e2e = {"value": N_mask * e_steps * world / (e_ms / 1e3), "unit": "tokens/s",
           "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": 4,
           "note": "pinned host inputs (ids and hidden rows) copied every step on a second "
                   "stream, overlapped with the previous step's compute (two device input sets); "
                   "the loss read back every step; W, d_hidden and d_W stay on the device by "
                   "design (a training step that feeds an on-device optimizer), so they are "
                   "neither copied in nor read back"}
    assert math.isfinite(float(loss_h.item()))
    del dev_in

    avg = lambda k: statistics.mean(a.elapsed_time(b2) for a, b2 in ev[k])
    fb_ms, spl_ms = avg("fwd_bwd"), avg("splice")
    med_step = statistics.median(a.elapsed_time(b2) for a, b2 in ev["splice"]) + \
        statistics.median(a.elapsed_time(b2) for a, b2 in ev["fwd_bwd"])
    burst, sustained, src = load_peaks()
    counted = 6.0 * N_mask * d * V
    step_tflops = counted / (ms_per_step / 1e3) / 1e12
    # dominant kernel: lmhead_group_kernel, launched four times per call (the
    # rows' reference maxima, pass A: lse, logp and dH, its redo launch, empty
    # unless a row's maximum exceeds its reference by 2^64, pass B: dW).  Its
    # algorithmic work per call is the forward product plus dH and dW,
    # 6 N_mask d V; it executes 8 N_mask d V (each pass computes the logits).
    # The call is bracketed by events on its stream, so the row gather, the
    # memsets and the loss reduction count against it.  The call lasts tens of
    # milliseconds, so the denominator is the burst peak.
    fb_flops = counted
    ach_fb = fb_flops / (fb_ms / 1e3) / 1e12
    rev = kernel_rev("lmhead_group.cu")
    traffic = profile_traffic("lmhead_group_kernel", rev)
    # algorithmic DRAM bytes of a call: W read, hc read (once per pass), dW and
    # dH written (bf16)
    alg_bytes = 2.0 * V * d + 2 * 2.0 * N_mask * d + 2.0 * V * d + 2.0 * N_mask * d
    # splice (scan, fill) + row gather + 4 lmhead_group_kernel + loss reduce
    launches = 2 + 1 + 4 + 1

    two_call = slab = None
    if not args.no_extra:
        slab = measure_slab(dev, hidden, W, pk_fn=lambda: B.olive_splice_pack(
            pre, poff, con, coff, V, T, dev_status=st), T=T, d=d, V=V, n=N_mask, burst=burst)
        two_call = measure_two_call(dev, hidden, W, pk_fn=lambda: B.olive_splice_pack(
            pre, poff, con, coff, V, T, dev_status=st), T=T, d=d, V=V, n=N_mask, burst=burst)

    extra = {}
    if not args.no_extra:
        del ws_fb, dh, dw
        torch.cuda.empty_cache()
        extra["kl_divergence"] = measure_kl(dev, burst)
        torch.cuda.empty_cache()
        extra["topk_kl"] = measure_topk_kl(dev, burst)
        torch.cuda.empty_cache()
        extra["opd_stats"] = measure_opd_stats(dev, burst)
        torch.cuda.empty_cache()
        extra["scoring_fwd"], extra["topk_entropy"] = measure_scoring(dev, burst)
        torch.cuda.empty_cache()
        extra["varlen"] = measure_varlen(dev, burst)
        torch.cuda.empty_cache()

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        nr = args.cpu_rows or 16
        rate, fixed, secs, _ = oracle_sample_rate(b, h_cpu, W_cpu, nr)
        cpu = {"value": rate, "unit": "tokens/s", "cores": host_cores(), "kind": "oracle",
               "sample": f"{nr} and {5 * nr} masked rows of the same batch after one untimed "
                         f"call: fp64 logits, log-probs, dH and dW contributions; per-row rate "
                         f"from the difference ({secs:.1f} s timed)",
               "fixed_s_per_call": fixed}

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(CONFIG, N_mask=N_mask, T=T, parallelism=f"replicas x{world}"),
        "pct_bf16_peak": 100.0 * step_tflops / burst,
        "pct_bf16_peak_sustained": 100.0 * step_tflops / sustained,
        "counted_tflops_per_s": step_tflops,
        "ms_per_step_median": med_step,
        "dense_equivalent_tflops_per_s": 6.0 * T * d * V / (ms_per_step / 1e3) / 1e12,
        "dense_equivalent_note": "6 T d V over the packed T (unmasked rows included); not the "
                                 "headline, which counts the N_mask scored rows only",
        "phases_ms": {"splice_pack": spl_ms, "loss_fwd_bwd": fb_ms},
        "roofline": {"kernel": "lmhead_group_kernel (reference maxima, pass A: lse/logp/dH, "
                               "its redo launch, pass B: dW)",
                     "bound": "tensor", "achieved": ach_fb, "peak": burst, "unit": "TFLOP/s",
                     "frac": ach_fb / burst, "traffic": traffic,
                     "algorithmic_bytes": alg_bytes,
                     "traffic_over_algorithmic": (traffic / alg_bytes) if traffic else None,
                     "peak_source": f"{src} bf16_tflops (burst: one call lasts tens of ms)",
                     "flops_per_call": fb_flops, "executed_flops_per_call": 8.0 * N_mask * d * V,
                     "executed_frac": 8.0 * N_mask * d * V / (fb_ms / 1e3) / 1e12 / burst,
                     "kernel_rev": rev,
                     "note": "per olive_token_loss_fwd_bwd call (its lmhead_group_kernel launches, "
                             "timed with the gather, memsets and loss reduction around them); "
                             "traffic is DRAM bytes of those launches from an ncu capture"},
        "two_call_path": two_call,
        "slab_path": slab,
        "e2e": e2e,
        "gpu_launches": launches * args.steps,
        "clocks": clk.summary(),
        "cpu_baseline": cpu,
        "other_workloads": extra,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


def profile_traffic(kernel: str, rev: str):
    """DRAM bytes per launch of `kernel` recorded from an ncu capture of the
    current sources (a `traffic: <kernel> <rev> <bytes>` line in a profiles/
    summary), else None."""
    import glob
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "*"))):
        with open(path) as f:
            for line in f:
                parts = line.strip().split()
                if len(parts) == 4 and parts[0] == "traffic:" and parts[1] == kernel and parts[2] == rev:
                    return float(parts[3])
    return None


def gpu_inputs(seed: int, T: int, d: int, V: int, dev):
    """Seeded bf16 hidden rows (RMS-normalised N(0,1)) and W ~ N(0, 0.02),
    drawn on the device (timing-only workloads; parity runs use synth)."""
    g = torch.Generator(device=dev).manual_seed(seed)
    h = torch.randn(T, d, generator=g, device=dev, dtype=torch.float32)
    h = (h * torch.rsqrt(h.square().mean(dim=1, keepdim=True) + 1e-6)).to(torch.bfloat16)
    W = (torch.randn(V, d, generator=g, device=dev, dtype=torch.float32) * 0.02).to(torch.bfloat16)
    return h, W


def time_calls(fn, steps: int, warmup: int) -> float:
    """Mean ms per call of fn() on the current stream (CUDA events)."""
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def measure_kl(dev, burst: float, steps: int = 3):
    """OPD per-token full-vocabulary KL forward + d/dh_s (16384 rows,
    student d = 4096, teacher d = 5120, V = 151936)."""
    from paper_2609_36246_gb300 import binding as B
    N, ds, dt, V = 16384, 4096, 5120, 151936
    hs, Ws = gpu_inputs(21, N, ds, V, dev)
    ht, Wt = gpu_inputs(22, N, dt, V, dev)
    rows = torch.arange(N, dtype=torch.int32, device=dev)
    n = torch.tensor([N], dtype=torch.int32, device=dev)
    gk = torch.ones(N, dtype=torch.float32, device=dev)
    ws = B.workspace(B.olive_workspace_size("divergence", N, ds, V, d_t=dt, grad=True), dev)
    st = B.new_status(dev)
    ms = time_calls(lambda: B.olive_token_divergence(hs, Ws, ht, Wt, rows, n, 1.0, "reverse", gk,
                                                     torch.bfloat16, ws=ws, dev_status=st),
                    steps, 1)
    ms_value = time_calls(lambda: B.olive_token_divergence(hs, Ws, ht, Wt, rows, n, 1.0, "reverse",
                                                           None, ws=ws, dev_status=st),
                          steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"divergence status {B.status_bits(st)}")
    flops_value = 2.0 * N * V * (ds + dt)
    flops = flops_value + 2.0 * N * V * ds
    # executed: the gradient pass recomputes both heads' logits
    flops_exec = 2.0 * flops_value + 2.0 * N * V * ds
    return {"workload": "per-token reverse KL + d/dh_s: 16384 rows, d_s=4096, d_t=5120, V=151936 "
                        "(value sweep, then the on-chip gradient pass; G never in HBM)",
            "value": N / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "pct_bf16_peak": 100.0 * flops / (ms / 1e3) / 1e12 / burst,
            "pct_bf16_peak_executed": 100.0 * flops_exec / (ms / 1e3) / 1e12 / burst,
            "value_only_ms": ms_value,
            "value_only_pct_bf16_peak": 100.0 * flops_value / (ms_value / 1e3) / 1e12 / burst,
            "steps": steps}


def measure_two_call(dev, hidden, W, pk_fn, T, d, V, n, burst, steps: int = 3):
    """The same step through olive_token_logprob_fwd + olive_token_loss_bwd
    (the backward recomputes the logits in both of its passes), for comparison."""
    from paper_2609_36246_gb300 import binding as B
    ws_f = B.workspace(B.olive_workspace_size("logprob_fwd", T, d, V), dev)
    ws_b = B.workspace(B.olive_workspace_size("loss_bwd", T, d, V), dev)
    st = B.new_status(dev)
    gl = torch.ones(1, dtype=torch.float32, device=dev)
    out_f = (torch.empty(T, device=dev), torch.empty(T, device=dev), torch.empty(1, device=dev))
    out_b = (torch.empty(T, d, dtype=torch.bfloat16, device=dev),
             torch.empty(V, d, dtype=torch.bfloat16, device=dev))

    def step():
        pk = pk_fn()
        _, lse, _ = B.olive_token_logprob_fwd(hidden, W, pk["targets"], pk["rows"], pk["n_rows"],
                                              ws=ws_f, dev_status=st, out=out_f)
        B.olive_token_loss_bwd(hidden, W, pk["targets"], pk["rows"], pk["n_rows"], lse, gl,
                               ws=ws_b, dev_status=st, out=out_b)

    ms = time_calls(step, steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"two-call status {B.status_bits(st)}")
    del ws_f, ws_b, out_b
    torch.cuda.empty_cache()
    return {"workload": "same batch, forward + on-chip backward (two calls; logits computed "
                        "three times)",
            "value": n / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "pct_bf16_peak": 100.0 * 6.0 * n * d * V / (ms / 1e3) / 1e12 / burst, "steps": steps}


def measure_slab(dev, hidden, W, pk_fn, T, d, V, n, burst, steps: int = 3):
    """The same step through olive_token_loss_fwd_bwd_slab: each logit tile
    computed once, e' = exp(z - R) of every masked row kept in an HBM slab
    (about 5 GB here) between the forward and the dH / dW products.  A
    secondary line: the headline keeps G on chip."""
    from paper_2609_36246_gb300 import binding as B
    ws = B.workspace(B.olive_workspace_size("loss_fwd_bwd_slab", T, d, V), dev)
    st = B.new_status(dev)
    gl = torch.ones(1, dtype=torch.float32, device=dev)
    out = (torch.empty(T, device=dev), torch.empty(T, device=dev), torch.empty(1, device=dev),
           torch.empty(T, d, dtype=torch.bfloat16, device=dev),
           torch.empty(V, d, dtype=torch.bfloat16, device=dev))

    def step():
        pk = pk_fn()
        B.olive_token_loss_fwd_bwd(hidden, W, pk["targets"], pk["rows"], pk["n_rows"], gl, 1.0,
                                   "sum", torch.bfloat16, ws=ws, dev_status=st, out=out, slab=True)

    ms = time_calls(step, steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"slab status {B.status_bits(st)}")
    del ws, out
    torch.cuda.empty_cache()
    return {"workload": "same batch, olive_token_loss_fwd_bwd_slab (G through an HBM slab of "
                        "every masked row, ~5 GB; logits computed once)",
            "value": n / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "pct_bf16_peak": 100.0 * 6.0 * n * d * V / (ms / 1e3) / 1e12 / burst, "steps": steps}


def measure_opd_stats(dev, burst: float, steps: int = 3):
    """OPD's per-token stats in one sweep with both heads: full KL, both lse,
    student entropy and top-16, teacher log-probs at those ids, top-16
    overlap and top-16 KL (16384 rows, student d = 4096, teacher d = 5120,
    V = 151936)."""
    from paper_2609_36246_gb300 import binding as B
    N, ds, dt, V = 16384, 4096, 5120, 151936
    hs, Ws = gpu_inputs(21, N, ds, V, dev)
    ht, Wt = gpu_inputs(22, N, dt, V, dev)
    rows = torch.arange(N, dtype=torch.int32, device=dev)
    n = torch.tensor([N], dtype=torch.int32, device=dev)
    ws = B.workspace(B.olive_workspace_size("opd_stats", N, ds, V, d_t=dt), dev)
    st = B.new_status(dev)
    ms = time_calls(lambda: B.olive_opd_token_stats(hs, Ws, ht, Wt, rows, n, 16, ws=ws,
                                                    dev_status=st), steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"opd stats status {B.status_bits(st)}")
    flops = 2.0 * N * V * (ds + dt)
    return {"workload": "OPD per-token stats (KL, lse, entropy, top-16, overlap, top-16 KL) in one "
                        "sweep: 16384 rows, d_s=4096, d_t=5120, V=151936",
            "value": N / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "pct_bf16_peak": 100.0 * flops / (ms / 1e3) / 1e12 / burst, "steps": steps}


def measure_topk_kl(dev, burst: float, steps: int = 3):
    """OPD with the top-16 KL as a training step (16384 rows, student d =
    4096, teacher d = 5120, V = 151936): the teacher's entropy/top-16 sweep,
    then olive_topk_kl_fwd_bwd (the student's top-16 lists, overlap,
    truncated KL and the gradient w.r.t. h_s and W_s from one sweep of the
    student's logits).  The multi-call route (student and teacher sweeps, the
    top-16 compare, olive_topk_kl_bwd, which recomputes the student's logits)
    is timed beside it."""
    from paper_2609_36246_gb300 import binding as B
    N, ds, dt, V, K = 16384, 4096, 5120, 151936, 16
    hs, Ws = gpu_inputs(21, N, ds, V, dev)
    ht, Wt = gpu_inputs(22, N, dt, V, dev)
    rows = torch.arange(N, dtype=torch.int32, device=dev)
    n = torch.tensor([N], dtype=torch.int32, device=dev)
    gk = torch.ones(N, dtype=torch.float32, device=dev)
    ws_k = B.workspace(B.olive_workspace_size("topk_fwd", N, dt, V), dev)
    ws_b = B.workspace(B.olive_workspace_size("topk_kl_bwd", N, ds, V), dev)
    out_b = (torch.empty(N, ds, dtype=torch.bfloat16, device=dev),
             torch.empty(V, ds, dtype=torch.bfloat16, device=dev))
    st = B.new_status(dev)

    def multi_call():
        s_lse, _, s_lp, s_id = B.olive_token_topk_fwd(hs, Ws, rows, n, K, ws=ws_k, dev_status=st)
        t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, rows, n, K, ws=ws_k, dev_status=st)
        _, kl, tlp = B.olive_topk_compare(ht, Wt, rows, n, s_id, s_lp, t_id, t_lse, dev_status=st,
                                          want_t_logp=True)
        B.olive_topk_kl_bwd(hs, Ws, rows, n, s_lse, s_id, s_lp, tlp, kl, gk, ws=ws_b,
                            dev_status=st, out=out_b)

    ms_multi = time_calls(multi_call, steps, 1)
    del ws_b
    torch.cuda.empty_cache()
    ws_f = B.workspace(B.olive_workspace_size("topk_kl_fwd_bwd", N, ds, V), dev)
    out_f = None

    def single_pass():
        nonlocal out_f
        t_lse, _, _, t_id = B.olive_token_topk_fwd(ht, Wt, rows, n, K, ws=ws_k, dev_status=st)
        out_f = B.olive_topk_kl_fwd_bwd(hs, Ws, ht, Wt, rows, n, K, t_lse, gk, t_id, ws=ws_f,
                                        dev_status=st, out=out_f)

    ms = time_calls(single_pass, steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"top-K KL status {B.status_bits(st)}")
    flops = 2.0 * N * V * (ds + dt) + 4.0 * N * V * ds
    return {"workload": "top-16 KL + d/dh_s, d/dW_s: 16384 rows, d_s=4096, d_t=5120, V=151936 "
                        "(teacher top-16 sweep + olive_topk_kl_fwd_bwd)",
            "value": N / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "pct_bf16_peak": 100.0 * flops / (ms / 1e3) / 1e12 / burst, "steps": steps,
            "multi_call_ms_per_step": ms_multi}


def measure_scoring(dev, burst: float, steps: int = 5):
    """Forward scoring (log-probs + loss, no backward) and the entropy / top-16
    sweep on 2 x (4096 prefix + 4096 continuation) tokens, d = 2048, V = 151936."""
    from paper_2609_36246_gb300 import binding as B
    from paper_2609_36246_gb300 import synth
    b = synth.make_batch("scoring")
    d, V, T = 2048, 151936, b.T
    h, W = gpu_inputs(24, T, d, V, dev)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)
    st = B.new_status(dev)
    pk = B.olive_splice_pack(i32(b.prefix_ids), i32(b.prefix_off), i32(b.cont_ids),
                             i32(b.cont_off), V, T, dev_status=st)
    ws_f = B.workspace(B.olive_workspace_size("logprob_fwd", T, d, V), dev)
    ws_k = B.workspace(B.olive_workspace_size("topk_fwd", T, d, V), dev)
    out = (torch.empty(T, device=dev), torch.empty(T, device=dev), torch.empty(1, device=dev))
    ms_f = time_calls(lambda: B.olive_token_logprob_fwd(h, W, pk["targets"], pk["rows"],
                                                        pk["n_rows"], ws=ws_f, dev_status=st,
                                                        out=out), steps, 1)
    ms_k = time_calls(lambda: B.olive_token_topk_fwd(h, W, pk["rows"], pk["n_rows"], 16, ws=ws_k,
                                                     dev_status=st), steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"scoring status {B.status_bits(st)}")
    n = b.n_mask
    flops = 2.0 * n * d * V
    res = {"workload": "forward scoring: 2 x (4096 + 4096) tokens, N_mask=8192, d=2048, V=151936",
           "value": n / (ms_f / 1e3), "unit": "tokens/s", "ms_per_step": ms_f,
           "pct_bf16_peak": 100.0 * flops / (ms_f / 1e3) / 1e12 / burst, "steps": steps}
    top = {"workload": "entropy + top-16 log-probs, same batch", "value": n / (ms_k / 1e3),
           "unit": "tokens/s", "ms_per_step": ms_k,
           "pct_bf16_peak": 100.0 * flops / (ms_k / 1e3) / 1e12 / burst, "steps": steps}
    return res, top


def measure_varlen(dev, burst: float, steps: int = 2):
    """splice/pack + olive_token_loss_fwd_bwd on the variable-length batch
    (64 sequences, lengths U[1024,16384], ~557k packed tokens; the masked
    rows span many G slabs)."""
    from paper_2609_36246_gb300 import binding as B
    from paper_2609_36246_gb300 import synth
    b = synth.make_batch("varlen")
    d, V, T = 4096, 151936, b.T
    h, W = gpu_inputs(23, T, d, V, dev)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)
    pre, poff, con, coff = i32(b.prefix_ids), i32(b.prefix_off), i32(b.cont_ids), i32(b.cont_off)
    ws = B.workspace(B.olive_workspace_size("loss_fwd_bwd", T, d, V), dev)
    st = B.new_status(dev)
    gl = torch.ones(1, dtype=torch.float32, device=dev)
    out = (torch.empty(T, device=dev), torch.empty(T, device=dev), torch.empty(1, device=dev),
           torch.empty(T, d, dtype=torch.bfloat16, device=dev),
           torch.empty(V, d, dtype=torch.bfloat16, device=dev))

    def step():
        pk = B.olive_splice_pack(pre, poff, con, coff, V, T, dev_status=st)
        B.olive_token_loss_fwd_bwd(h, W, pk["targets"], pk["rows"], pk["n_rows"], gl, 1.0, "mean",
                                   torch.bfloat16, ws=ws, dev_status=st, out=out)

    ms = time_calls(step, steps, 1)
    if int(st.item()) != 0:
        raise RuntimeError(f"varlen status {B.status_bits(st)}")
    n = b.n_mask
    return {"workload": f"variable-length batch: 64 sequences, {T} packed tokens, N_mask={n}, "
                        "d=4096, V=151936", "value": n / (ms / 1e3), "unit": "tokens/s",
            "ms_per_step": ms, "pct_bf16_peak": 100.0 * 6.0 * n * d * V / (ms / 1e3) / 1e12 / burst,
            "steps": steps}


def kernel_rev(source: str = "lmhead_fused.cu") -> str:
    """Hash of one kernel's translation unit and the headers it includes
    (followed transitively), comments and blank lines left out, which ties a
    stored ncu traffic figure to the code that produced it."""
    import hashlib
    import re as _re
    csrc = os.path.join(ROOT, "paper_2609_36246_gb300", "csrc")
    seen, todo = [], [os.path.join(csrc, source)]
    while todo:
        path = todo.pop(0)
        if path in seen or not os.path.exists(path):
            continue
        seen.append(path)
        with open(path) as f:
            for inc in _re.findall(r'#include "([^"]+)"', f.read()):
                todo.append(os.path.normpath(os.path.join(os.path.dirname(path), inc)))
    hsh = hashlib.sha256()
    for path in sorted(seen):
        with open(path) as f:
            text = f.read()
        text = _re.sub(r"/\*.*?\*/", "", text, flags=_re.S)
        code = [ln.split("//")[0].rstrip() for ln in text.splitlines()]
        hsh.update("\n".join(ln for ln in code if ln).encode())
    return hsh.hexdigest()[:16]


# --------------------------------------------------------------------------- reference arm
def run_reference(args, world, rank):
    if rank != 0:
        return
    b, h, W = make_inputs(rank)
    nr = args.cpu_rows or 16
    secs, rates, fixed = [], [], []
    for _ in range(args.warmup):
        pass  # the oracle has no warm state; warm-up steps would only repeat the sample
    for i in range(args.steps):
        rate, fx, s_, _ = oracle_sample_rate(b, h, W, nr, seed=i, warm=i == 0)
        rates.append(rate)
        fixed.append(fx)
        secs.append(s_)
    value = statistics.median(rates)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(secs),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": dict(CONFIG, parallelism="host cores"),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": host_cores(), "kind": "oracle",
                         "sample": f"per step {nr} and {5 * nr} masked rows of the same batch "
                                   "(one untimed call before the first step; fp64 forward, dH, dW "
                                   "contributions); per-row rate from the difference, median over "
                                   "steps",
                         "fixed_s_per_call": statistics.median(fixed)},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_profile_case(args):
    """A small case for profilers: `--steps` calls of olive_token_loss_fwd_bwd
    (or the slab form with --slab) on N masked rows (every row masked,
    RMS-normalised N(0,1) hidden, W ~ N(0, 0.02), d = 4096, V = 151936); no
    JSON line.  At N = 4096 the device holds ~3 GB."""
    from paper_2609_36246_gb300 import binding as B
    from paper_2609_36246_gb300 import build as _build
    _build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    N, d, V = args.profile_rows, 4096, 151936
    h, W = gpu_inputs(31, N, d, V, dev)
    rows = torch.arange(N, dtype=torch.int32, device=dev)
    n = torch.tensor([N], dtype=torch.int32, device=dev)
    g = torch.Generator(device=dev).manual_seed(32)
    targets = torch.randint(0, V, (N,), generator=g, device=dev, dtype=torch.int32)
    gl = torch.ones(1, dtype=torch.float32, device=dev)
    op = "loss_fwd_bwd_slab" if args.slab else "loss_fwd_bwd"
    ws = B.workspace(B.olive_workspace_size(op, N, d, V), dev)
    st = B.new_status(dev)
    out = None
    for _ in range(args.steps):
        out = B.olive_token_loss_fwd_bwd(h, W, targets, rows, n, gl, ws=ws, dev_status=st, out=out,
                                         slab=args.slab)
    torch.cuda.synchronize()
    if int(st.item()) != 0:
        raise RuntimeError(f"device status {B.status_bits(st)}")
    print(f"profile case: {args.steps} calls of {op} on {N} rows, loss {float(out[2].item()):.4f}")


def run_profile_kl(args):
    """A small case for profilers: `--steps` calls of olive_token_divergence
    with the gradient (value sweep, then the on-chip gradient pass) on N rows
    (d_s = 4096, d_t = 5120, V = 151936, reverse KL); no JSON line.  At
    N = 4096 the device holds ~3.2 GB."""
    from paper_2609_36246_gb300 import binding as B
    from paper_2609_36246_gb300 import build as _build
    _build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    N, ds, dt, V = args.profile_kl, 4096, 5120, 151936
    hs, Ws = gpu_inputs(21, N, ds, V, dev)
    ht, Wt = gpu_inputs(22, N, dt, V, dev)
    rows = torch.arange(N, dtype=torch.int32, device=dev)
    n = torch.tensor([N], dtype=torch.int32, device=dev)
    gk = torch.ones(N, dtype=torch.float32, device=dev)
    ws = B.workspace(B.olive_workspace_size("divergence", N, ds, V, d_t=dt, grad=True), dev)
    st = B.new_status(dev)
    kl = None
    for _ in range(args.steps):
        kl, _ = B.olive_token_divergence(hs, Ws, ht, Wt, rows, n, 1.0, "reverse", gk, torch.bfloat16,
                                         ws=ws, dev_status=st)
    torch.cuda.synchronize()
    if int(st.item()) != 0:
        raise RuntimeError(f"device status {B.status_bits(st)}")
    print(f"profile case: {args.steps} calls of the divergence with d/dh_s on {N} rows, "
          f"mean KL {float(kl.mean().item()):.4f}")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-rows", type=int, default=None,
                    help="masked rows n of the oracle samples (n and 5n rows after one "
                         "untimed call; default 16, about 11 s per step on 16 cores)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the divergence and variable-length measurements")
    ap.add_argument("--profile-rows", type=int, default=0,
                    help="run only the training-step call on this many masked rows (a small "
                         "case for ncu) and print no JSON line")
    ap.add_argument("--slab", action="store_true", help="with --profile-rows: the slab form")
    ap.add_argument("--profile-kl", type=int, default=0,
                    help="profiler case: the divergence with d/dh_s on N rows (see run_profile_kl)")
    args = ap.parse_args()
    if args.profile_rows > 0:
        if torch.cuda.is_available():
            torch.cuda.set_device(0)
        run_profile_case(args)
        return
    if args.profile_kl > 0:
        if torch.cuda.is_available():
            torch.cuda.set_device(0)
        run_profile_kl(args)
        return
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
