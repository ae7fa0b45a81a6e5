"""Benchmark: back-propagation training throughput in connections per second.

Workload (default): 203-120-26 sigmoid MLP (NETtalk-shaped), float32,
65,536 synthetic patterns, minibatch 512, lr 0.05, momentum 0.9.  One bench
step = one epoch = 128 training updates of 512 patterns, run as one persistent
launch of the library's training kernel through the C ABI.

Connections per second follow the paper's definition (Section 7.1): the number
of connections, bias connections included, times the patterns presented,
divided by the time.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU: the path runs on one GPU; with N > 1 every rank trains its own
replica (no collective on the data path) and `value` adds up all ranks.
`--impl reference` times the float64 CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "connections/sec (fwd+bwd per connection per pattern) and % of roofline, 1 GB300"
UNIT = "connections/s"
WORKLOAD = "nettalk120"
FP32_LANES_PER_SM = 128            # FP32 FFMA lanes per Blackwell SM
SM_MAX_MHZ_NOMINAL = 2070.0
L2_FLUSH_BYTES = 512 << 20         # > 129 MB of L2


def env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def workload_desc(w):
    return (f"{'-'.join(map(str, w['sizes']))} sigmoid MLP, {w['dtype']}, {w['patterns']:,} "
            f"synthetic NETtalk-shaped patterns, minibatch {w['minibatch']}, lr {w['lr']}, "
            f"momentum {w['momentum']}; one step = one epoch "
            f"({w['patterns'] // w['minibatch']} updates)")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.t is not None:
            self.t.join(timeout=5)
        mhz, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                mhz.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(mhz)}


# ------------------------------------------------------------------ distributed
def dist_setup():
    world = env_int("WORLD_SIZE", 1)
    rank = env_int("RANK", 0)
    local = env_int("LOCAL_RANK", 0)
    if world > 1:
        import torch.distributed as dist
        backend = "nccl"
        try:
            import torch
            if not torch.cuda.is_available():
                backend = "gloo"
        except Exception:
            backend = "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def allreduce_max(x, world, device):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ oracle timing
def _oracle_child(patterns_cap, budget_s, steps=1, warmup=0, min_s=0.0, max_epochs=1,
                  workload=WORKLOAD):
    """Runs in a fresh interpreter with one BLAS thread: times the oracle on the
    leading `patterns_cap` patterns of the workload (one update per minibatch),
    `warmup` untimed then `steps` timed times, each bounded by `budget_s`."""
    from oracle import bp_oracle as O
    from paper_1801_01554_gb300 import synth
    w = synth.WORKLOADS[workload]
    sizes, X, T, theta = synth.make_workload(workload, patterns=patterns_cap)
    st = O.State(sizes, theta, lr=w["lr"], momentum=w["momentum"])
    mb = w["minibatch"]
    out = []
    for k in range(warmup + steps):
        done = 0
        t0 = time.perf_counter()
        # cycle through the patterns in index order (epoch after epoch) until at
        # least min_s seconds have passed, at most max_epochs epochs
        while True:
            p0 = done % len(X)
            O.train_batch(st, X[p0:p0 + mb], T[p0:p0 + mb])
            done += min(mb, len(X) - p0)
            el = time.perf_counter() - t0
            if el > budget_s or done >= max_epochs * len(X) or (el >= min_s and done % len(X) == 0):
                break
        if k >= warmup:
            out.append({"patterns": done, "seconds": time.perf_counter() - t0})
    return out


def time_oracle(patterns_cap, budget_s, steps=1, warmup=0, min_s=0.0, max_epochs=1,
                workload=WORKLOAD):
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = "1"
    code = ("import json,sys; sys.path.insert(0, %r); import bench; "
            "print(json.dumps(bench._oracle_child(%d, %f, %d, %d, %f, %d, %r)))"
            % (ROOT, patterns_cap, budget_s, steps, warmup, min_s, max_epochs, workload))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       cwd=ROOT, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError("oracle timing failed: " + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


# DRAM bytes per pattern of the float32 training kernel on the 203-120-26
# workload: 15,513,856 bytes (15,293,952 read + 219,904 written) in one ncu
# capture of the timed k_train launch of `bench.py --patterns 16384` (16,384
# patterns after an L2 flush; profiles/k_train_nettalk120_launches.md).  The
# inputs and targets are read once (916 bytes per pattern); everything else
# stays in L2.  Re-measure after any change to the kernel.
K_TRAIN_DRAM_BYTES_PER_PATTERN = 15_513_856 / 16_384


def connections(sizes):
    return sum((sizes[l - 1] + 1) * sizes[l] for l in range(1, len(sizes)))


def algorithmic_flops_per_pattern(sizes):
    # forward 2W, backward 2W_i + 4(W - W_i) (Section 6.1 cycle counts)
    W = connections(sizes)
    Wi = (sizes[0] + 1) * sizes[1]
    return 2 * W + 2 * Wi + 4 * (W - Wi)


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except (OSError, ValueError):
        return {}


# ------------------------------------------------------------------ reference arm
def run_reference(args, world, rank):
    if rank != 0:
        return 0
    from paper_1801_01554_gb300 import synth
    w = synth.WORKLOADS[WORKLOAD]
    sizes = w["sizes"]
    W = connections(sizes)
    sample = 4096                      # 8 updates of 512 patterns per step
    runs = time_oracle(sample, 60.0, steps=args.steps, warmup=args.warmup)
    tot_p = sum(r["patterns"] for r in runs)
    tot_s = sum(r["seconds"] for r in runs)
    cps = W * tot_p / tot_s
    line = {
        "impl": "reference", "metric": METRIC, "value": cps, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot_s / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(w), "global_batch": w["minibatch"],
                   "patterns_per_step": sample, "parallelism": "none (host oracle)"},
        "cpu_baseline": {"value": cps, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{sample} patterns (8 updates of 512) of the workload per "
                                   "step, float64 numpy oracle, one BLAS thread"},
        "e2e": {"value": cps, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ our arm
def run_ours(args, world, rank, local):
    import torch
    from paper_1801_01554_gb300 import bp, synth

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    w = synth.WORKLOADS[args.workload]
    sizes, X, T, theta = synth.make_workload(args.workload, patterns=args.patterns)
    n, mb = len(X), w["minibatch"]
    updates = (n + mb - 1) // mb
    W = connections(sizes)

    # CPU baseline first (before any GPU work in this process is irrelevant: it
    # runs in its own interpreter), on rank 0 only, single-GPU runs only.
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # whole epochs until at least --cpu-seconds of CPU work (60 s cap)
        r = time_oracle(n, 60.0, min_s=args.cpu_seconds, max_epochs=10 ** 6,
                        workload=args.workload)[0]
        cpu = {"value": W * r["patterns"] / r["seconds"], "unit": UNIT, "cores": 1,
               "kind": "oracle",
               "sample": f"{r['patterns']} patterns ({r['patterns'] / n:.2f} epochs of the "
                         f"workload, {(r['patterns'] + mb - 1) // mb} updates of {mb}), float64 "
                         f"numpy oracle, one BLAS thread, {r['seconds']:.1f} s"}

    Xd = torch.tensor(X, dtype=torch.float32, device=device)
    Td = torch.tensor(T, dtype=torch.float32, device=device)
    sse = torch.zeros(updates, dtype=torch.float32, device=device)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    stream = torch.cuda.current_stream(device)

    net = bp.Net(sizes, w["lr"], w["momentum"], bp.BP_F32, max_batch=mb)
    net.set_weights(theta)
    for _ in range(args.warmup):
        net.train_epoch(Xd, Td, n, mb, sse, stream)
    net.check(stream)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize(device)
    clocks.start()
    time.sleep(0.3)   # let the sampler start before the timed region
    t_wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.fill_(float(k))                  # evict the previous epoch from L2
        starts[k].record(stream)
        net.train_epoch(Xd, Td, n, mb, sse, stream)
        ends[k].record(stream)
    torch.cuda.synchronize(device)
    t_wall = time.perf_counter() - t_wall0
    clk = clocks.stop()
    barrier(world)
    net.check(stream)
    per_step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    dev_s = sum(per_step_ms) / 1e3
    dev_s_max = allreduce_max(dev_s, world, device)
    patterns_all = n * args.steps * world
    value = W * patterns_all / dev_s_max

    # end to end: host buffers through bp_train_epoch_host, copies inside the timed region
    Xh = torch.tensor(X, dtype=torch.float32).pin_memory()
    Th = torch.tensor(T, dtype=torch.float32).pin_memory()
    sse_h = np.zeros(updates, dtype=np.float32)
    e2e_steps = max(1, min(args.steps, 20))
    net.train_epoch_host(Xh, Th, n, mb, sse_h, stream)     # staging allocation, untimed
    barrier(world)
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        net.train_epoch_host(Xh, Th, n, mb, sse_h, stream)
    e2e_s = allreduce_max(time.perf_counter() - t0, world, device)
    e2e_value = W * n * e2e_steps * world / e2e_s
    net.close()

    # roofline of the training kernel: algorithmic flops / FFMA peak
    flops_launch = algorithmic_flops_per_pattern(sizes) * n
    kernel_s = dev_s / args.steps
    achieved = flops_launch / kernel_s / 1e12
    peaks = measured_peaks()
    sm_max = float(peaks.get("sm_max_mhz", SM_MAX_MHZ_NOMINAL))
    num_sms = torch.cuda.get_device_properties(device).multi_processor_count
    peak = num_sms * FP32_LANES_PER_SM * 2 * sm_max * 1e6 / 1e12

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dev_s_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": workload_desc(w), "global_batch": mb,
                   "patterns_per_step": n, "updates_per_step": updates,
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": f"flushed ({L2_FLUSH_BYTES >> 20} MB write) before every timed epoch; "
                         "an epoch reads each pattern once"},
        "roofline": {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak,
                     "traffic": K_TRAIN_DRAM_BYTES_PER_PATTERN * n if args.workload == WORKLOAD
                     else None,
                     "traffic_basis": "ncu dram__bytes_read.sum + dram__bytes_write.sum of the "
                                      "timed k_train launch of bench.py --patterns 16384 (after "
                                      "an L2 flush), scaled to the launch's patterns",
                     "kernel": "k_train (persistent cooperative training kernel)",
                     "peak_basis": f"{num_sms} SMs x {FP32_LANES_PER_SM} FP32 lanes x 2 flop x "
                                   f"{sm_max:.0f} MHz"},
        "e2e": {"value": e2e_value, "unit": UNIT,
                "h2d_bytes_per_step": int(Xh.numel() * 4 + Th.numel() * 4),
                "d2h_bytes_per_step": int(sse_h.nbytes)},
        "gpu_launches": args.steps,
        "clocks": clk,
        "wall_s_timed": t_wall,
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def run_wide(args, world, rank, local):
    """BF16 tensor-core workloads: one step = one training update on the full batch."""
    import torch
    from paper_1801_01554_gb300 import bp, synth

    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    name = args.workload
    w = synth.WORKLOADS[name]
    sizes, X, T, theta = synth.make_workload(name)
    B = w["minibatch"]
    W = connections(sizes)
    Xd = torch.tensor(X, dtype=torch.float32, device=device).to(torch.bfloat16)
    Td = torch.tensor(T, dtype=torch.float32, device=device).to(torch.bfloat16)
    del X, T
    sse = torch.zeros(1, dtype=torch.float32, device=device)
    stream = torch.cuda.current_stream(device)
    net = bp.Net(sizes, w["lr"], w["momentum"], bp.BP_BF16, max_batch=B)
    net.set_weights(theta)
    for _ in range(args.warmup):
        net.train_batch(Xd, Td, B, sse, stream)
    net.check(stream)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize(device)
    clocks.start()
    time.sleep(0.3)
    for k in range(args.steps):
        starts[k].record(stream)
        net.train_batch(Xd, Td, B, sse, stream)
        ends[k].record(stream)
    torch.cuda.synchronize(device)
    clk = clocks.stop()
    net.check(stream)
    dev_s = sum(s_.elapsed_time(e_) for s_, e_ in zip(starts, ends)) / 1e3
    dev_s_max = allreduce_max(dev_s, world, device)
    value = W * B * args.steps * world / dev_s_max
    flops = algorithmic_flops_per_pattern(sizes) * B
    achieved = flops / (dev_s / args.steps) / 1e12
    peaks = measured_peaks()
    peak = float(peaks.get("bf16_tflops_sustained", 1700.0))
    net.close()
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dev_s_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": f"{'-'.join(map(str, sizes))} sigmoid MLP, bf16 activations and "
                               f"weight copies, fp32 accumulate and master weights, batch {B}, "
                               f"lr {w['lr']}, momentum {w['momentum']}; one step = one update",
                   "global_batch": B, "parallelism": "single GPU",
                   "l2": "activations of one step exceed the 129 MB L2"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None,
                     "kernel": "whole training step (k_gemm forward, hidden-delta and pooled-change "
                               "GEMMs, transposes, update); flops = (6W - 2W_i) per pattern",
                     "peak_basis": "measured bf16 cuBLAS, sustained"},
        "clocks": clk,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ group-size sweep
def run_sweep(args, world, rank, local):
    """CPS against the group size B on the 203-120-26 net (the paper's group-size
    question, Section 5): one JSON line per B, from CUDA events around whole
    epochs with the L2 flushed before each.  B <= 4 runs on the one-CTA kernel,
    larger groups on the persistent kernel."""
    import torch
    from paper_1801_01554_gb300 import bp, perf_model, synth

    if rank != 0:
        return 0
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    sizes = synth.WORKLOADS[WORKLOAD]["sizes"]
    X, T = synth.nettalk_patterns(65536, seed=0)
    theta = synth.round_to(synth.init_uniform(sizes, -0.3, 0.3, 0), "f32")
    Xd = torch.tensor(X, dtype=torch.float32, device=device)
    Td = torch.tensor(T, dtype=torch.float32, device=device)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    W = connections(sizes)
    for B in (1, 2, 4) + tuple(synth.SWEEP_BATCHES[1:]):
        n = 65536 if B >= 512 else B * 512          # at least 128 updates per epoch
        updates = (n + B - 1) // B
        net = bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B)
        net.set_weights(theta)
        for _ in range(3):
            net.train_epoch(Xd, Td, n, B)
        ms = []
        for k in range(5):
            flush.fill_(float(k))
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            net.train_epoch(Xd, Td, n, B)
            e1.record()
            torch.cuda.synchronize(device)
            ms.append(e0.elapsed_time(e1))
        net.check()
        net.close()
        t = sorted(ms)[len(ms) // 2] / 1e3
        print(json.dumps({"sweep": "group size", "B": B, "patterns": n, "updates": updates,
                          "us_per_update": 1e6 * t / updates,
                          "model_us_per_update": perf_model.gb300_update_us(B),
                          "value": W * n / t, "unit": UNIT,
                          "kernel": "one-CTA" if B <= 4 else "persistent cooperative",
                          "dtype": "f32", "data": "synthetic"}), flush=True)
    return 0


# ------------------------------------------------------------------ width crossover
def run_crossover(args, world, rank, local):
    """fp32 kernels (CUDA cores, weights resident or streamed from L2) against
    the bf16 GEMM chain (tcgen05 tensor cores) as the hidden layer widens: a
    208-H-32 net (the NETtalk sizes rounded up to the bf16 path's multiple of
    8), groups of 512 patterns, one JSON line per H with both times per update."""
    import torch
    from paper_1801_01554_gb300 import bp, synth

    if rank != 0:
        return 0
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    B, n = 512, 512 * 32
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    for H in (64, 128, 256, 512, 1024, 2048, 4096):
        sizes = (208, H, 32)
        X, T = synth.gaussian_patterns(n, sizes[0], sizes[-1], 0.1, seed=H)
        theta = synth.init_normal_fanin(sizes, seed=H)
        out = {"crossover": "hidden width", "sizes": list(sizes), "B": B, "patterns": n,
               "connections": connections(sizes)}
        for name, dt in (("f32", bp.BP_F32), ("bf16", bp.BP_BF16)):
            Xd = torch.tensor(X, dtype=torch.float32 if dt == bp.BP_F32 else torch.bfloat16,
                              device=device)
            Td = torch.tensor(T, dtype=Xd.dtype, device=device)
            net = bp.Net(sizes, 0.01, 0.9, dt, max_batch=B)
            net.set_weights(theta)
            for _ in range(2):
                net.train_epoch(Xd, Td, n, B)
            ms = []
            for k in range(5):
                flush.fill_(float(k))
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                net.train_epoch(Xd, Td, n, B)
                e1.record()
                torch.cuda.synchronize(device)
                ms.append(e0.elapsed_time(e1))
            net.check()
            net.close()
            t = sorted(ms)[len(ms) // 2] / 1e3
            out[name + "_us_per_update"] = 1e6 * t / (n // B)
            out[name + "_cps"] = connections(sizes) * n / t
        out["faster"] = "bf16" if out["bf16_us_per_update"] < out["f32_us_per_update"] else "f32"
        print(json.dumps(out), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=("nettalk60", "nettalk120", "wide3", "wide4096"),
                    help="workload to time (default: the 203-120-26 NETtalk-shaped net)")
    ap.add_argument("--patterns", type=int, default=None,
                    help="patterns per epoch (default: the workload's; a smaller epoch of the "
                         "same net and group size is for profiler captures, not a bench line)")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the bench line: CPS against the group size (203-120-26)")
    ap.add_argument("--crossover", action="store_true",
                    help="instead of the bench line: fp32 against bf16 as the hidden layer widens")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    world, rank, local = dist_setup()
    if args.impl == "reference":
        rc = run_reference(args, world, rank)
    elif args.sweep:
        rc = run_sweep(args, world, rank, local)
    elif args.crossover:
        rc = run_crossover(args, world, rank, local)
    elif args.workload in ("wide3", "wide4096"):
        rc = run_wide(args, world, rank, local)
    else:
        rc = run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
