#!/usr/bin/env python
"""Forward throughput of random-Fourier-feature linear attention on GB300.

Default workload: nonstationary (Flexformer_n) causal forward, bf16 storage,
B=4, H=16, N=16384, d=64, M=128 (d'=256), seeded synthetic inputs.  A step is one call
of flex_linattn_fwd over the whole batch.  Prints one JSON line (rank 0).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME]

`--impl reference` times the fp64 CPU oracle on the host cores instead (each step a
bounded sample of whole sequences of the same workload).  Under torchrun each rank runs
its own full replica of the workload (the (b, h) sequences are independent; no
collective on the data path), so the value is weak-scaled.
"""
from __future__ import annotations

import argparse
import dataclasses
import glob
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2606_27748_gb300 import workloads  # noqa: E402

METRIC = "RFF linear-attn fwd tokens/s (N=16K causal) & % of bf16 tensor/HBM roofline"
METRIC_TRAIN = "RFF linear-attn fwd+bwd training-step tokens/s & % of roofline"
METRIC_DECODE = ("RFF linear-attn recurrent decode tokens/s (one new token per sequence, fp32 "
                 "running state) & % of HBM roofline")
METRIC_AWD = ("RFF attention-weight distillation loss tokens/s (softmax teacher vs kernel "
              "weights, blockwise N x N) & % of roofline")
METRIC_AWD_TRAIN = ("RFF attention-weight distillation training-step tokens/s (loss and its "
                    "gradient w.r.t. the frequencies, blockwise N x N) & % of roofline")
L2_BYTES = 129e6
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
PREFACTOR = "exp(|x|^2 / exp(tau)), tau per head (workloads.draw_tau)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=workloads.HEADLINE.name,
                    choices=list(workloads.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--sweep-n", default=None,
                    help="comma-separated sequence lengths: time the workload's forward at "
                         "each N (same B, H, d, M) and print one JSON line per N with the "
                         "time and the device memory held (the linear-scaling curve)")
    ap.add_argument("--prefactor", action="store_true",
                    help="with the norm prefactor exp(|x|^2 / exp(tau)) of the paper's "
                         "Flexformer_n, tau per head from the workload generator (both arms)")
    ap.add_argument("--batch", type=int, default=None,
                    help="run the workload with this batch B instead of its own (a smaller "
                         "case for profiling; the line's config names the changed workload)")
    return ap.parse_args()


# ---------------------------------------------------------------------------------------
# Work accounting (algorithmic, per token-head): q, k, v read + out written; flops of the
# two projections and of the state read and update (Eq. linear att, Eq. phi_n/phi_non).
# ---------------------------------------------------------------------------------------
def elem_bytes(w):
    return 2 if w.dtype == "bf16" else 4


def algorithmic_bytes(w):
    return w.token_heads * 4 * w.d * elem_bytes(w)


def algorithmic_flops(w):
    """Forward: the two projections and the state read and update; a training step counts
    the backward as twice the forward."""
    mc = 2 * w.M if w.variant == "n" else w.M
    per = 2 * (2 * w.d * mc) + 2 * (2 * (2 * w.M) * w.d)
    return w.token_heads * per * (3 if w.backward else 1)


def sincos_count(w):
    """sin/cos evaluations on the path: per feature vector 2M (s: cos a, sin a) or 3M (n:
    cos u, sin u, cos w); the forward builds phi(q) and phi(k); the backward rebuilds both
    and, for n, also needs sin w (4M per vector)."""
    fwd = (3 if w.variant == "n" else 2) * w.M
    bwd = (4 if w.variant == "n" else 2) * w.M
    per = 2 * fwd + (2 * bwd if w.backward else 0)
    return w.token_heads * per


SFU_PER_CLK_PER_SM = 16  # sin/cos results per clock per SM (measured 15.9 by a probe)


def roofline(w, kernel_ms, peaks, sms, traffic):
    """The three roofs of the path; `bound` is the unit with the longest time at peak."""
    sec = kernel_ms * 1e-3
    nbytes = algorithmic_bytes(w)
    if w.backward:  # + backward: read q, k, v, out, dO; write dq, dk, dv
        nbytes += w.token_heads * 8 * w.d * elem_bytes(w)
    flops, ops = algorithmic_flops(w), sincos_count(w)
    sfu_peak = SFU_PER_CLK_PER_SM * sms * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e9  # G/s
    roofs = {
        "hbm": (nbytes / sec / 1e9, peaks["hbm_gbs"], "GB/s", nbytes / (peaks["hbm_gbs"] * 1e9)),
        "tensor": (flops / sec / 1e12, peaks["bf16_tflops"], "TFLOP/s",
                   flops / (peaks["bf16_tflops"] * 1e12)),
        "alu": (ops / sec / 1e9, sfu_peak, "Gsincos/s", ops / (sfu_peak * 1e9)),
    }
    bound = max(roofs, key=lambda k: roofs[k][3])
    a, pk, unit, _ = roofs[bound]
    return {"bound": bound, "achieved": a, "peak": pk, "unit": unit, "frac": a / pk,
            "traffic": traffic,
            "algorithmic_bytes_per_launch": nbytes, "algorithmic_flops_per_launch": flops,
            "sincos_per_launch": ops,
            "time_at_peak_us": {k: v[3] * 1e6 for k, v in roofs.items()},
            "fracs": {k: v[0] / v[1] for k, v in roofs.items()},
            "alu_peak_note": f"{SFU_PER_CLK_PER_SM} sin/cos per clock per SM x {sms} SMs x "
                             f"{peaks.get('sm_max_mhz', 2070.0):.0f} MHz",
            "kernel_ms": kernel_ms}


def source_digest(files=None):
    """sha256 over the given kernel sources (paths relative to the repository root), or
    over every file of csrc/."""
    if files is None:
        files = sorted(os.path.relpath(f, ROOT) for f in
                       glob.glob(os.path.join(ROOT, "paper_2606_27748_gb300", "csrc", "*")))
    h = hashlib.sha256()
    for f in files:
        h.update(open(os.path.join(ROOT, f), "rb").read())
    return h.hexdigest()


def load_peaks():
    if os.path.exists(PEAKS_FILE):
        return json.load(open(PEAKS_FILE)), "measured"
    return FALLBACK_PEAKS, "fallback"


def recorded_traffic(w):
    """DRAM bytes per launch from the committed ncu summary, if the kernel sources it was
    taken from are unchanged."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    try:
        t = json.load(open(TRAFFIC_FILE)).get(w.name)
        if not t or t.get("source_sha256") != source_digest(t.get("sources")):
            return None
    except (ValueError, OSError):
        return None
    return t.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------------------
# Clock sampling during the timed region.
# ---------------------------------------------------------------------------------------
class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.2)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[5:9]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        smax = max(r[1] for r in rows)
        loaded = [r for r in rows if r[2] > 200.0] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": smax,
                "reasons": reasons, "samples": len(rows), "samples_under_load": len(loaded)}


# ---------------------------------------------------------------------------------------
# CPU oracle timing (the reported baseline and the reference arm).
# ---------------------------------------------------------------------------------------
def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_sample(w, nseq, cores, prefactor=False):
    """Time the oracle over the first `nseq` whole sequences of `w`: the forward, and for a
    training workload (w.backward) the backward after it."""
    import oracle
    nb = -(-nseq // w.H)
    ins = workloads.make_inputs(w, bs=range(nb))
    # the first nseq (b, h) sequences in order, laid out as one batch row of nseq "heads",
    # each with its own head's frequencies
    q, k, v = (ins[n].reshape(nb * w.H, w.N, w.d)[None, :nseq] for n in "qkv")
    heads = [s % w.H for s in range(nseq)]
    W1 = ins["W1"][heads]
    W2 = None if ins["W2"] is None else ins["W2"][heads]
    tau = workloads.draw_tau(w)[heads] if prefactor else None
    dO = ins["dO"].reshape(nb * w.H, w.N, w.d)[None, :nseq] if w.backward else None
    t0 = time.perf_counter()
    oracle.fwd(q, k, v, W1, W2, w.causal, nthreads=cores, tau=tau)
    if w.backward:
        oracle.bwd(q, k, v, W1, W2, w.causal, dO, nthreads=cores, tau=tau)
    return time.perf_counter() - t0


def cpu_baseline(w, cores, target_s=12.0, prefactor=False):
    bh = w.B * w.H
    n1 = min(bh, cores)
    t1 = oracle_sample(w, n1, cores, prefactor)
    nseq, t = n1, t1
    if t1 < target_s / 2 and n1 < bh:
        nseq = min(bh, n1 * max(1, int(target_s / max(t1, 1e-3))))
        if nseq > n1:
            t = oracle_sample(w, nseq, cores, prefactor)
    tokens = nseq * w.N / w.H
    return {"value": tokens / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{nseq} of {bh} whole (b,h) sequences of N={w.N} (fp64 C oracle, "
                      f"{cores} threads), {t:.2f} s; tokens = sequences*N/H"}


def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    if w.decode:
        for _ in range(args.warmup):
            oracle_decode_sample(w, 1, args.prefactor)
        step = sum(oracle_decode_sample(w, 1, args.prefactor)
                   for _ in range(args.steps)) / args.steps
        value = w.B / step
        print(json.dumps({
            "metric": METRIC_DECODE, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "d": w.d, "M": w.M,
                       "variant": w.variant, "causal": True},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                             "sample": f"one decode step of all {w.B}x{w.H} sequences per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}), flush=True)
        return
    if w.awd:
        nseq = 8
        for _ in range(args.warmup):
            oracle_awd_sample(w, nseq, args.prefactor)
        step = sum(oracle_awd_sample(w, nseq, args.prefactor)
                   for _ in range(args.steps)) / args.steps
        value = nseq * w.N / w.H / step
        print(json.dumps({
            "metric": METRIC_AWD_TRAIN if w.backward else METRIC_AWD, "value": value,
            "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "d": w.d, "M": w.M,
                       "variant": w.variant, "causal": w.causal},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                             "sample": f"{nseq} sequences of N={w.N} per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}), flush=True)
        return
    cores = cpu_cores()
    nseq = min(w.B * w.H, cores)
    for _ in range(args.warmup):
        oracle_sample(w, nseq, cores, args.prefactor)
    times = [oracle_sample(w, nseq, cores, args.prefactor) for _ in range(args.steps)]
    step = sum(times) / len(times)
    value = nseq * w.N / w.H / step
    line = {
        "metric": METRIC_TRAIN if w.backward else METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "impl": "reference",
        "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "d": w.d, "M": w.M,
                   "variant": w.variant, "causal": w.causal},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"{nseq} whole (b,h) sequences of N={w.N} per step"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------------------
# Multi-rank bookkeeping: every rank runs a full replica; the step time of the job is the
# maximum over ranks and the value counts the work of all ranks.
# ---------------------------------------------------------------------------------------
def max_over_ranks(values, world, device="cpu"):
    """Element-wise maximum of a list of floats over all ranks (identity when world = 1)."""
    if world <= 1:
        return list(values)
    import torch
    import torch.distributed as dist
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_value(world, tokens_per_rank, ms_per_step):
    """Whole-job tokens/s: the tokens all ranks processed over the slowest rank's time."""
    return world * tokens_per_rank / (ms_per_step * 1e-3)


# ---------------------------------------------------------------------------------------
# Our arm.
# ---------------------------------------------------------------------------------------
def run_ours(args, w):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2606_27748_gb300 import build, flexattn

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0 or not os.path.exists(flexattn.LIBRARY):
        build.build()
    if world > 1:
        dist.barrier()
    flexattn.load()

    def barrier():
        if world > 1:
            dist.barrier()

    ins = workloads.make_inputs(w)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    host = {n: torch.from_numpy(ins[n]).to(tdt).pin_memory() for n in "qkv"}
    W1 = torch.from_numpy(ins["W1"]).to(dev)
    W2 = None if ins["W2"] is None else torch.from_numpy(ins["W2"]).to(dev)
    del ins
    q, k, v = (host[n].to(dev) for n in "qkv")
    out = torch.empty_like(q)
    den = torch.empty(q.shape[:3], dtype=torch.float32, device=dev)
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.workspace(shape, w.causal, False, dev)
    stream = torch.cuda.current_stream()
    tau = torch.from_numpy(workloads.draw_tau(w)).to(dev) if args.prefactor else None
    dtau = torch.empty_like(tau) if args.prefactor else None

    if w.backward:  # a training step: forward, then backward of sum(dO * out)
        host["dO"] = torch.from_numpy(workloads.draw_activation(w, workloads.DO)).to(tdt).pin_memory()
        dO = host["dO"].to(dev)
        grads = [torch.empty_like(q), torch.empty_like(k), torch.empty_like(v),
                 torch.empty_like(W1), None if W2 is None else torch.empty_like(W2)]
        ws_b = flexattn.workspace(shape, w.causal, True, dev)

    def step():
        flexattn.linattn_fwd(q, k, v, W1, W2, w.causal, out=out, den=den, ws=ws, tau=tau)
        if w.backward:
            flexattn.linattn_bwd(q, k, v, W1, W2, w.causal, out, den, dO, *grads, ws=ws_b,
                                 tau=tau, dtau=dtau)

    for _ in range(max(3, args.warmup)):
        step()
    flexattn.check_status(ws)

    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
    barrier()
    torch.cuda.synchronize()
    launches0 = flexattn.kernel_launches()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(K):
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = flexattn.kernel_launches() - launches0
    clk = clocks.stop() if clocks else None
    flexattn.check_status(ws)
    total_ms = t_start.elapsed_time(t_end)
    kernel_ms = sum(a.elapsed_time(b) for a, b in ev) / K
    total_ms, kernel_ms = max_over_ranks([total_ms, kernel_ms], world, dev)
    ms_per_step = total_ms / K
    value = job_value(world, w.tokens, ms_per_step)

    # End to end through the same C-ABI call with host buffers: H2D of q, k, v from pinned
    # memory, the forward, D2H of out, every step.
    e2e = None
    if not args.no_e2e:
        # inference: the output comes back; training: the frequency gradient (dq, dk, dv
        # feed the layers below on the device)
        result = grads[3] if w.backward else out
        host_out = torch.empty(result.shape, dtype=result.dtype).pin_memory()
        inputs = (("q", q), ("k", k), ("v", v)) + ((("dO", dO),) if w.backward else ())

        def e2e_step():
            for n, t in inputs:
                t.copy_(host[n], non_blocking=True)
            step()
            host_out.copy_(result, non_blocking=True)

        for _ in range(max(3, args.warmup)):
            e2e_step()
        barrier()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(K):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = a.elapsed_time(b) / K
        e2e_ms = max_over_ranks([e2e_ms], world, dev)[0]
        h2d = sum(host[n].numel() * host[n].element_size() for n, _ in inputs)
        e2e = {"value": job_value(world, w.tokens, e2e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": host_out.numel() * host_out.element_size()}

    peaks, peaks_src = load_peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    # the recorded DRAM traffic is that of the kernel without the prefactor
    roof = roofline(w, kernel_ms, peaks, sms, None if args.prefactor else recorded_traffic(w))
    roof["peak_source"] = peaks_src

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, cpu_cores(), prefactor=args.prefactor)

    if rank == 0:
        line = {
            "metric": METRIC_TRAIN if w.backward else METRIC, "value": value,
            "unit": "tokens/s", "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "d": w.d, "M": w.M,
                       "variant": w.variant, "causal": w.causal,
                       "l2": f"inputs {3 * w.token_heads * w.d * elem_bytes(w) / 1e6:.0f} MB "
                             f"> L2 {L2_BYTES / 1e6:.0f} MB, no flush",
                       "parallelism": f"replicas x{world}",
                       "prefactor": PREFACTOR if args.prefactor else None},
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ---------------------------------------------------------------------------------------
# Recurrent decode workload: a step gives every sequence one new token (its q, k, v), which
# updates the fp32 running state (S, z) and yields its output.
# ---------------------------------------------------------------------------------------
def decode_work(w):
    """(bytes, flops, sin/cos) per decode step: the state read and written once, the new
    tokens' q, k, v read and out written, the frequencies read once."""
    F, bh = 2 * w.M, w.B * w.H
    mc = 2 * w.M if w.variant == "n" else w.M
    nbytes = (bh * (F * w.d + F) * 4 * 2 + bh * 4 * w.d * elem_bytes(w)
              + w.H * w.M * w.d * 4 * (2 if w.variant == "n" else 1))
    flops = bh * (2 * (2 * w.d * mc) + 3 * (2 * F * w.d))
    ops = bh * 2 * (3 if w.variant == "n" else 2) * w.M
    return nbytes, flops, ops


def oracle_decode_sample(w, steps, prefactor=False):
    """Seconds per oracle decode step of all B x H sequences (the first token)."""
    import numpy as np
    import oracle
    ins = workloads.make_inputs(w, N=1)
    q, k, v = (ins[n][:, :, 0] for n in "qkv")
    W1, W2 = ins["W1"], ins["W2"]
    S = np.zeros((w.B, w.H, 2 * w.M, w.d))
    z = np.zeros((w.B, w.H, 2 * w.M))
    tau = workloads.draw_tau(w) if prefactor else None
    t0 = time.perf_counter()
    for _ in range(steps):
        _, _, S, z = oracle.decode(q, k, v, W1, W2, S, z, tau=tau)
    return (time.perf_counter() - t0) / steps


def run_decode(args, w):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2606_27748_gb300 import build, flexattn

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0 or not os.path.exists(flexattn.LIBRARY):
        build.build()
    if world > 1:
        dist.barrier()
    flexattn.load()
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    ins = workloads.make_inputs(w)
    toks = [[torch.from_numpy(np.ascontiguousarray(ins[n][:, :, i])).to(tdt).to(dev)
             for n in "qkv"] for i in range(w.N)]
    host = [[t.cpu().pin_memory() for t in tk] for tk in toks]
    W1 = torch.from_numpy(ins["W1"]).to(dev)
    W2 = None if ins["W2"] is None else torch.from_numpy(ins["W2"]).to(dev)
    del ins
    S, z = flexattn.decode_state(w.B, w.H, w.M, w.d, dev)
    ws = flexattn.decode_workspace(w.B, w.H, w.M, w.d, dev)
    tau = torch.from_numpy(workloads.draw_tau(w)).to(dev) if args.prefactor else None
    out = torch.empty_like(toks[0][0])
    den = torch.empty(w.B, w.H, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    it = [0]

    def step(tk=None):
        q, k, v = tk if tk is not None else toks[it[0] % w.N]
        it[0] += 1
        flexattn.linattn_decode(q, k, v, W1, W2, S, z, out=out, den=den, ws=ws, tau=tau)

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(max(3, args.warmup)):
        step()
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
    barrier()
    torch.cuda.synchronize()
    launches0 = flexattn.kernel_launches()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(K):
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = flexattn.kernel_launches() - launches0
    clk = clocks.stop() if clocks else None
    total_ms = t_start.elapsed_time(t_end)
    kernel_ms = sum(a.elapsed_time(b) for a, b in ev) / K
    total_ms, kernel_ms = max_over_ranks([total_ms, kernel_ms], world, dev)
    ms_per_step = total_ms / K
    value = job_value(world, w.B, ms_per_step)

    e2e = None
    if not args.no_e2e:  # the new tokens from pinned host memory, the outputs back
        host_out = torch.empty(out.shape, dtype=out.dtype).pin_memory()
        dev_tok = [torch.empty_like(t) for t in toks[0]]

        def e2e_step():
            for t, hsrc in zip(dev_tok, host[it[0] % w.N]):
                t.copy_(hsrc, non_blocking=True)
            step(dev_tok)
            host_out.copy_(out, non_blocking=True)

        for _ in range(max(3, args.warmup)):
            e2e_step()
        barrier()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(K):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = max_over_ranks([a.elapsed_time(b) / K], world, dev)[0]
        e2e = {"value": job_value(world, w.B, e2e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in host[0]),
               "d2h_bytes_per_step": host_out.numel() * host_out.element_size()}

    peaks, peaks_src = load_peaks()
    nbytes, flops, ops = decode_work(w)
    sec = kernel_ms * 1e-3
    roof = {"bound": "hbm", "achieved": nbytes / sec / 1e9, "peak": peaks["hbm_gbs"],
            "unit": "GB/s", "frac": nbytes / sec / 1e9 / peaks["hbm_gbs"],
            "traffic": None if args.prefactor else recorded_traffic(w),
            "peak_source": peaks_src, "algorithmic_bytes_per_launch": nbytes,
            "fracs": {"hbm": nbytes / sec / 1e9 / peaks["hbm_gbs"],
                      "tensor": flops / sec / 1e12 / peaks["bf16_tflops"]},
            "kernel_ms": kernel_ms}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t = oracle_decode_sample(w, 3, args.prefactor)
        cpu = {"value": w.B / t, "unit": "tokens/s", "cores": 1, "kind": "oracle",
               "sample": f"3 decode steps of all {w.B}x{w.H} sequences (fp64 C oracle, "
                         f"one thread), {t:.3f} s per step"}

    if rank == 0:
        line = {
            "metric": METRIC_DECODE, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "d": w.d, "M": w.M,
                       "variant": w.variant, "causal": True,
                       "l2": f"state {w.B * w.H * 2 * w.M * (w.d + 1) * 4 / 1e6:.0f} MB > L2 "
                             f"{L2_BYTES / 1e6:.0f} MB, no flush",
                       "parallelism": f"replicas x{world}",
                       "prefactor": PREFACTOR if args.prefactor else None},
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ---------------------------------------------------------------------------------------
# Attention-weight distillation loss: a step is the loss of every sequence of the batch.
# ---------------------------------------------------------------------------------------
def awd_work(w):
    """(bytes, flops, sin/cos+exp/log/reciprocal) per step: q, k read, the loss written; the
    score and kernel contractions over the (masked) pairs plus the feature projections; per
    pair one exp and one log, per token and frequency 2 (s) or 3 (n) sin/cos for q and for
    k.  A training step (w.backward) adds the gradient: W read and dW written; per pair and
    side the score and kernel contractions again and G phi (2M features), one exp and one
    reciprocal; per token and side the projection and dW' = da^T x (2 P d each, P = M (s)
    or 2M (n)) and the sin/cos of the chain rule."""
    bh, N = w.B * w.H, w.N
    pairs = bh * (N * (N + 1) // 2 if w.causal else N * N)
    c = 2 if w.variant == "n" else 1
    nbytes = bh * N * w.d * elem_bytes(w) * 2 + bh * 4
    flops = 2 * pairs * (w.d + 2 * w.M) + 2 * bh * N * 2 * w.d * w.M * c
    ops = 2 * pairs + bh * N * 2 * w.M * (3 if w.variant == "n" else 2)
    if w.backward:
        nbytes += 2 * c * w.H * w.M * w.d * 4
        flops += 2 * (2 * pairs * (w.d + 4 * w.M)) + 2 * (2 * bh * N * 2 * c * w.M * w.d)
        ops += 2 * (2 * pairs) + 2 * bh * N * w.M * (4 if w.variant == "n" else 2)
    return nbytes, flops, ops


def oracle_awd_sample(w, nseq, prefactor=False):
    """Seconds of the oracle loss (and, for a training step, its gradient) over the first
    `nseq` sequences (one thread)."""
    import oracle
    nb = -(-nseq // w.H)
    ins = workloads.make_inputs(w, bs=range(nb))
    q, k = (ins[n].reshape(nb * w.H, w.N, w.d)[None, :nseq] for n in "qk")
    heads = [s_ % w.H for s_ in range(nseq)]
    W1 = ins["W1"][heads]
    W2 = None if ins["W2"] is None else ins["W2"][heads]
    tau = workloads.draw_tau(w)[heads] if prefactor else None
    t0 = time.perf_counter()
    oracle.awd(q, k, W1, W2, w.causal, tau=tau)
    if w.backward:
        oracle.awd_bwd(q, k, W1, W2, w.causal, tau=tau)
    return time.perf_counter() - t0


def run_awd(args, w):
    import torch
    import torch.distributed as dist

    from paper_2606_27748_gb300 import build, flexattn

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0 or not os.path.exists(flexattn.LIBRARY):
        build.build()
    if world > 1:
        dist.barrier()
    flexattn.load()
    tdt = torch.bfloat16
    ins = workloads.make_inputs(w)
    host = {n: torch.from_numpy(ins[n]).to(tdt).pin_memory() for n in "qk"}
    q, k = host["q"].to(dev), host["k"].to(dev)
    W1 = torch.from_numpy(ins["W1"]).to(dev)
    W2 = None if ins["W2"] is None else torch.from_numpy(ins["W2"]).to(dev)
    del ins
    tau = torch.from_numpy(workloads.draw_tau(w)).to(dev) if args.prefactor else None
    shape = flexattn.shape_of(q, W1)
    train = w.backward  # loss and its gradient (mean over the sequences) per step
    ws = (flexattn.awd_bwd_workspace if train else flexattn.awd_workspace)(shape, dev)
    loss = torch.empty(w.B, w.H, dtype=torch.float32, device=dev)
    dloss = torch.full((w.B, w.H), 1.0 / (w.B * w.H), dtype=torch.float32, device=dev)
    grads = [torch.empty_like(W1)] + ([torch.empty_like(W2)] if W2 is not None else [])
    dtau = torch.empty_like(tau) if tau is not None else None
    if dtau is not None:
        grads.append(dtau)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # > L2: a cold step
    stream = torch.cuda.current_stream()

    def step():
        if train:
            flexattn.awd_loss_bwd(q, k, W1, W2, w.causal, tau=tau, dloss=dloss, loss=loss,
                                  dW1=grads[0], dW2=grads[1] if W2 is not None else None,
                                  dtau=dtau, ws=ws)
        else:
            flexattn.awd_loss(q, k, W1, W2, w.causal, tau=tau, loss=loss, ws=ws)

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(max(3, args.warmup)):
        step()
    flexattn.check_status(ws)
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
    barrier()
    torch.cuda.synchronize()
    launches0 = flexattn.kernel_launches()
    for i in range(K):
        flush.zero_()  # outside the step's events
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = flexattn.kernel_launches() - launches0
    clk = clocks.stop() if clocks else None
    flexattn.check_status(ws)
    kernel_ms = sum(a.elapsed_time(b) for a, b in ev) / K
    kernel_ms = max_over_ranks([kernel_ms], world, dev)[0]
    value = job_value(world, w.tokens, kernel_ms)

    e2e = None
    if not args.no_e2e:  # q, k from pinned host memory, the losses (and gradients) back
        results = [loss] + (grads if train else [])
        host_outs = [torch.empty(r.shape, dtype=r.dtype).pin_memory() for r in results]

        def e2e_step():
            q.copy_(host["q"], non_blocking=True)
            k.copy_(host["k"], non_blocking=True)
            step()
            for ho, r in zip(host_outs, results):
                ho.copy_(r, non_blocking=True)

        for _ in range(max(3, args.warmup)):
            e2e_step()
        barrier()
        torch.cuda.synchronize()
        tot = 0.0
        for _ in range(K):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            e2e_step()
            b.record(stream)
            torch.cuda.synchronize()
            tot += a.elapsed_time(b)
        barrier()
        e2e_ms = max_over_ranks([tot / K], world, dev)[0]
        e2e = {"value": job_value(world, w.tokens, e2e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in host.values()),
               "d2h_bytes_per_step": sum(t.numel() * t.element_size() for t in host_outs)}

    peaks, peaks_src = load_peaks()
    nbytes, flops, ops = awd_work(w)
    sec = kernel_ms * 1e-3
    sms = 152
    sfu_peak = SFU_PER_CLK_PER_SM * sms * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e9
    roofs = {"hbm": (nbytes / sec / 1e9, peaks["hbm_gbs"], "GB/s", nbytes / (peaks["hbm_gbs"] * 1e9)),
             "tensor": (flops / sec / 1e12, peaks["bf16_tflops"], "TFLOP/s",
                        flops / (peaks["bf16_tflops"] * 1e12)),
             "alu": (ops / sec / 1e9, sfu_peak, "Gops/s", ops / (sfu_peak * 1e9))}
    bound = max(roofs, key=lambda r: roofs[r][3])
    ach, pk, unit, _ = roofs[bound]
    roof = {"bound": bound, "achieved": ach, "peak": pk, "unit": unit, "frac": ach / pk,
            "traffic": None, "peak_source": peaks_src, "algorithmic_bytes_per_launch": nbytes,
            "algorithmic_flops_per_launch": flops, "sfu_ops_per_launch": ops,
            "time_at_peak_us": {r: v[3] * 1e6 for r, v in roofs.items()},
            "fracs": {r: v[0] / v[1] for r, v in roofs.items()},
            "alu_peak_note": f"{SFU_PER_CLK_PER_SM} MUFU results (ex2, lg2, rcp, sin, cos) per clock "
                             f"per SM x {sms} SMs x {peaks.get('sm_max_mhz', 2070.0):.0f} MHz",
            "kernel_ms": kernel_ms}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        nseq = w.B * w.H // (4 if train else 1)  # ~10 s of one core
        t = oracle_awd_sample(w, nseq, args.prefactor)
        cpu = {"value": nseq * w.N / w.H / t, "unit": "tokens/s", "cores": 1, "kind": "oracle",
               "sample": f"{nseq} of {w.B * w.H} sequences of N={w.N} (fp64 C oracle, one "
                         f"thread), {t:.2f} s; tokens = sequences*N/H"}

    if rank == 0:
        line = {
            "metric": METRIC_AWD_TRAIN if train else METRIC_AWD, "value": value,
            "unit": "tokens/s", "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": kernel_ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "H": w.H, "N": w.N, "d": w.d, "M": w.M,
                       "variant": w.variant, "causal": w.causal,
                       "l2": "flushed (256 MB write) before each timed step",
                       "parallelism": f"replicas x{world}",
                       "prefactor": PREFACTOR if args.prefactor else None},
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_sweep(args, w):
    """Forward time and device memory against N for one workload family (the paper's
    time-and-memory-versus-length comparison, our own curve only).  Per N: inputs from the
    workload's generator at that N, warm-up, then `steps` forwards each timed with CUDA
    events on the launching stream, L2 flushed (a 256 MB write) before each; memory is
    the peak held by this program's device allocations (inputs, out, den, workspace)."""
    import statistics as st

    import torch

    from paper_2606_27748_gb300 import build, flexattn
    build.build()
    flexattn.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    for n in (int(x) for x in args.sweep_n.split(",")):
        wn = w.replace(N=n, name=f"{w.name}@N{n}")
        ins = workloads.make_inputs(wn)
        torch.cuda.synchronize()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        q, k, v = (torch.from_numpy(ins[x]).to(tdt).to(dev) for x in "qkv")
        W1 = torch.from_numpy(ins["W1"]).to(dev)
        W2 = None if ins["W2"] is None else torch.from_numpy(ins["W2"]).to(dev)
        del ins
        out = torch.empty_like(q)
        den = torch.empty(q.shape[:3], dtype=torch.float32, device=dev)
        shape = flexattn.shape_of(q, W1)
        ws = flexattn.workspace(shape, w.causal, False, dev)
        for _ in range(max(3, args.warmup)):
            flexattn.linattn_fwd(q, k, v, W1, W2, w.causal, out=out, den=den, ws=ws)
        flexattn.check_status(ws)
        times = []
        for _ in range(args.steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            flexattn.linattn_fwd(q, k, v, W1, W2, w.causal, out=out, den=den, ws=ws)
            b.record(stream)
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b))
        flexattn.check_status(ws)
        ms = st.median(times)
        peak = torch.cuda.max_memory_allocated(dev) - base
        print(json.dumps({
            "sweep": "N", "workload": wn.name, "N": n, "B": w.B, "H": w.H, "d": w.d,
            "M": w.M, "variant": w.variant, "causal": w.causal, "dtype": w.dtype,
            "ms_per_forward": ms, "tokens_per_s": w.B * n / (ms * 1e-3),
            "ns_per_token_head": ms * 1e6 / (w.B * w.H * n),
            "device_bytes": peak, "workspace_bytes": ws.numel(),
            "bytes_per_token_head": peak / (w.B * w.H * n), "steps": args.steps,
            "l2": "flushed before each timed forward"}), flush=True)
        del q, k, v, W1, W2, out, den, ws


def main():
    args = parse_args()
    w = workloads.WORKLOADS[args.workload]
    if args.batch is not None and args.batch != w.B:
        w = dataclasses.replace(w, B=args.batch, name=f"{w.name}@B{args.batch}")
    if args.sweep_n:
        if w.decode or w.backward:
            raise SystemExit("--sweep-n times the forward of a forward workload")
        run_sweep(args, w)
    elif args.impl == "reference":
        run_reference(args, w)
    elif w.decode:
        run_decode(args, w)
    elif w.awd:
        run_awd(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
