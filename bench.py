"""Benchmark: back-propagation training throughput in connections per second.

Headline workload: 203-120-26 sigmoid MLP (NETtalk-shaped), float32, 65,536
synthetic patterns, minibatch 512, lr 0.05, momentum 0.9, 5 epochs.  One bench
step = the workload's 5 epochs = 640 training updates, run as 5 persistent
launches (one per epoch) of the library's training kernel through the C ABI.
The same JSON line carries a `configs` object with the other workloads:
203-60-26 (one step = its 10 full-batch epochs), the group-size sweep on
203-120-26, and the bf16 nets 1024-2048-2048-512 and 4096^5 (one step = one
update of the full batch), each with its roofline, CPU baseline and end-to-end
figure through the host-buffer entry point.

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
                 "--format=csv,noheader,nounits", "-lms", "20"],
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
THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def _cpu_child(spec):
    """Runs in a fresh interpreter: times the CPU oracle on a bounded sample of a
    workload and returns {"patterns", "seconds", "cores"}.

    spec["mode"]: "serial" (the oracle as it stands, one BLAS thread),
    "case_parallel" (Section 4.1's scheme: oracle/case_parallel.py with
    spec["workers"] processes of one thread each) or "blas" (the oracle with
    numpy's BLAS on every host core).  Groups of spec["minibatch"] patterns of
    the workload's first spec["patterns"] are taken in index order, epoch after
    epoch, until at least spec["min_s"] seconds have passed at an epoch's end
    (or spec["max_s"] at a group's end); spec["groups"] > 0 times exactly that
    many groups instead.  The all-core modes first run one untimed group (worker
    start-up, BLAS thread pools)."""
    from oracle import bp_oracle as O
    from paper_1801_01554_gb300 import synth
    w = synth.WORKLOADS[spec["workload"]]
    sizes, X, T, theta = synth.make_workload(spec["workload"], patterns=spec["patterns"])
    mb = spec["minibatch"]
    n = len(X)
    st = O.State(sizes, theta, lr=w["lr"], momentum=w["momentum"])
    cp = None
    if spec["mode"] == "case_parallel":
        from oracle.case_parallel import CaseParallel
        cp = CaseParallel(sizes, X, T, workers=spec["workers"])
        step = lambda p0, nb: cp.train_batch(st, p0, nb)  # noqa: E731
        cores = spec["workers"]
    else:
        step = lambda p0, nb: O.train_batch(st, X[p0:p0 + nb], T[p0:p0 + nb])  # noqa: E731
        cores = 1 if spec["mode"] == "serial" else (os.cpu_count() or 1)
    try:
        if spec["mode"] != "serial":
            step(0, min(mb, n))                  # warm-up: worker start, BLAS threads
        done, g = 0, 0
        groups_per_epoch = -(-n // mb)
        t0 = time.perf_counter()
        while True:
            p0 = (g % groups_per_epoch) * mb
            nb = min(mb, n - p0)
            step(p0, nb)
            done += nb
            g += 1
            el = time.perf_counter() - t0
            if spec.get("groups", 0) > 0:
                if g >= spec["groups"]:
                    break
            elif el >= spec["max_s"] or (el >= spec["min_s"] and p0 + nb == n):
                break
        return {"patterns": done, "seconds": time.perf_counter() - t0, "cores": cores}
    finally:
        if cp is not None:
            cp.close()


def time_cpu(spec):
    env = dict(os.environ)
    if spec["mode"] == "blas":
        for k in THREAD_VARS:
            env.pop(k, None)
    else:
        env.update({k: "1" for k in THREAD_VARS})
    code = ("import json,sys; sys.path.insert(0, %r); import bench; "
            "print(json.dumps(bench._cpu_child(json.loads(sys.argv[1]))))" % ROOT)
    r = subprocess.run([sys.executable, "-c", code, json.dumps(spec)], env=env, capture_output=True,
                       text=True, cwd=ROOT, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError("oracle timing failed: " + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_baselines(name, minibatch, patterns, one_core, all_cores, label):
    """{value, unit, cores, kind, sample, one_core} for a workload: the serial
    oracle on one core (one_core) and the all-core schemes given; value and
    cores are those of the fastest."""
    W = connections(synth_sizes(name))
    r1 = time_cpu(dict(one_core, workload=name, minibatch=minibatch, patterns=patterns))
    out = {"value": None, "unit": UNIT, "cores": None, "kind": "oracle",
           "one_core": W * r1["patterns"] / r1["seconds"]}
    best = None
    for spec in all_cores:
        r = time_cpu(dict(spec, workload=name, minibatch=minibatch, patterns=patterns))
        v = W * r["patterns"] / r["seconds"]
        if best is None or v > best[0]:
            best = (v, r, spec["mode"])
    if best is None or best[0] < out["one_core"]:
        # the exchange per group costs more than it saves at this group size
        out.update(value=out["one_core"], cores=1,
                   sample=f"{label}; serial on one core, {r1['patterns']} patterns in "
                          f"{r1['seconds']:.1f} s" + ("" if best is None else
                                                      f"; {best[2]} on {best[1]['cores']} "
                                                      f"cores slower ({best[0]:.3g})"))
    else:
        out.update(value=best[0], cores=best[1]["cores"],
                   sample=f"{label}; {best[2]} on {best[1]['cores']} cores, "
                          f"{best[1]['patterns']} patterns in {best[1]['seconds']:.1f} s")
    return out


def synth_sizes(name):
    from paper_1801_01554_gb300 import synth
    return synth.WORKLOADS[name]["sizes"]


# DRAM bytes (read + write) per pattern of each workload's roofline unit, from
# single-pass ncu captures (dram__bytes_read.sum + dram__bytes_write.sum; the
# commands are in profiles/dram_traffic_all_workloads.md): one k_train launch
# for the float32 nets (one epoch; 203-120-26 captured on a 16,384-pattern epoch
# and scaled by patterns, as its traffic is the inputs read once), the whole
# training step (all launches) for the bf16 nets.  Re-measure after any change
# to these kernels; a workload whose kernels changed since its capture has none
# (the bf16 nets: the update kernel's bias part changed after their capture).
TRAFFIC_PER_PATTERN = {
    "nettalk60": 1_116_416 / 1024,          # 1.12 MB per launch (one update of 1,024)
    "nettalk120": 15_408_128 / 16384,       # 61.6 MB per 65,536-pattern launch
}
# sweep groups of 203-120-26 with a capture of their own (bytes per pattern of one launch);
# at B = 65,536 the group's scratch rows no longer fit the L2 and make a DRAM round trip
SWEEP_TRAFFIC_PER_PATTERN = {512: TRAFFIC_PER_PATTERN["nettalk120"], 65536: 676_348_928 / 65536}


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


def alu_peak_tflops(num_sms):
    sm_max = float(measured_peaks().get("sm_max_mhz", SM_MAX_MHZ_NOMINAL))
    return num_sms * FP32_LANES_PER_SM * 2 * sm_max * 1e6 / 1e12, sm_max


def bf16_peak_tflops():
    p = measured_peaks().get("bf16_tflops")
    return (float(p), "measured bf16 cuBLAS, burst") if p else (1900.0, "fallback bf16 burst")


# ------------------------------------------------------------------ reference arm
def run_reference(args, world, rank):
    if rank != 0:
        return 0
    from paper_1801_01554_gb300 import synth
    w = synth.WORKLOADS[WORKLOAD]
    sizes = w["sizes"]
    W = connections(sizes)
    sample = 4096                      # 8 updates of 512 patterns per step
    tot_p = tot_s = 0.0
    for k in range(args.warmup + args.steps):
        r = time_cpu({"mode": "serial", "workload": WORKLOAD, "minibatch": w["minibatch"],
                      "patterns": sample, "min_s": 0.0, "max_s": 60.0})
        if k >= args.warmup:
            tot_p += r["patterns"]
            tot_s += r["seconds"]
    cps = W * tot_p / tot_s
    line = {
        "impl": "reference", "metric": METRIC, "value": cps, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot_s / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(w), "global_batch": w["minibatch"],
                   "patterns_per_step": sample, "parallelism": "none (host oracle)"},
        "cpu_baseline": {"value": cps, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{sample} patterns (8 updates of 512) per step, float64 numpy "
                                   "oracle, one BLAS thread"},
        "e2e": {"value": cps, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ our arm: pieces
def _events(n):
    import torch
    return [torch.cuda.Event(enable_timing=True) for _ in range(n)]


def time_f32_launches(net, Xd, Td, n, mb, launches, steps, warmup, flush, stream, sse):
    """`steps` timed steps of `launches` epoch launches each (L2 flushed before
    every step).  Returns (per-step ms, per-launch ms)."""
    import torch
    for _ in range(warmup):
        for _ in range(launches):
            net.train_epoch(Xd, Td, n, mb, sse, stream)
    net.check(stream)
    ev = [_events(launches + 1) for _ in range(steps)]
    torch.cuda.synchronize()
    for k in range(steps):
        flush.fill_(float(k))
        ev[k][0].record(stream)
        for e in range(launches):
            net.train_epoch(Xd, Td, n, mb, sse, stream)
            ev[k][e + 1].record(stream)
    torch.cuda.synchronize()
    net.check(stream)
    step_ms = [ev[k][0].elapsed_time(ev[k][-1]) for k in range(steps)]
    launch_ms = [ev[k][e].elapsed_time(ev[k][e + 1]) for k in range(steps) for e in range(launches)]
    return step_ms, launch_ms


def time_f32_e2e(net, X, T, n, mb, launches, steps, stream, world, device):
    """The same steps through bp_train_epoch_host on pinned host buffers: the
    copies in and the error sums out are inside the timed region."""
    import torch
    Xh = torch.tensor(X, dtype=torch.float32).pin_memory()
    Th = torch.tensor(T, dtype=torch.float32).pin_memory()
    sse_h = np.zeros(-(-n // mb), dtype=np.float32)
    net.train_epoch_host(Xh, Th, n, mb, sse_h, stream)      # staging allocation, untimed
    barrier(world)
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    for _ in range(steps):
        for _ in range(launches):
            net.train_epoch_host(Xh, Th, n, mb, sse_h, stream)
    t = allreduce_max(time.perf_counter() - t0, world, device)
    return t, launches * int(Xh.numel() * 4 + Th.numel() * 4), launches * int(sse_h.nbytes)


def f32_entry(name, sizes, n, mb, launches, step_ms, launch_ms, e2e, num_sms, cpu, label):
    """Compact config entry of a float32 workload."""
    W = connections(sizes)
    step_s = sum(step_ms) / len(step_ms) / 1e3
    launch_s = sum(launch_ms) / len(launch_ms) / 1e3
    peak, _ = alu_peak_tflops(num_sms)
    achieved = algorithmic_flops_per_pattern(sizes) * n / launch_s / 1e12
    tr = TRAFFIC_PER_PATTERN.get(name)
    ent = {"workload": label, "value": W * n * launches / step_s, "ms_per_step": 1e3 * step_s,
           "roofline": {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                        "frac": achieved / peak, "traffic": tr * n if tr else None}}
    if e2e is not None:
        t, bi, bo = e2e[0], e2e[1], e2e[2]
        ent["e2e"] = {"value": W * n * launches * e2e[3] / t, "unit": UNIT,
                      "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo}
    if cpu is not None:
        ent["cpu_baseline"] = cpu
    return ent


def bf16_entry(name, sizes, B, step_ms, e2e, cpu, label):
    W = connections(sizes)
    step_s = sum(step_ms) / len(step_ms) / 1e3
    peak, basis = bf16_peak_tflops()
    achieved = algorithmic_flops_per_pattern(sizes) * B / step_s / 1e12
    tr = TRAFFIC_PER_PATTERN.get(name)
    ent = {"workload": label, "value": W * B / step_s, "ms_per_step": 1e3 * step_s,
           "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                        "frac": achieved / peak, "traffic": tr * B if tr else None,
                        "peak_basis": basis}}
    if e2e is not None:
        t, bi, bo, steps = e2e
        ent["e2e"] = {"value": W * B * steps / t, "unit": UNIT, "h2d_bytes_per_step": bi,
                      "d2h_bytes_per_step": bo}
    if cpu is not None:
        ent["cpu_baseline"] = cpu
    return ent


def measure_bf16(name, steps, warmup, stream, device, world, with_e2e=True):
    """One bench step = one training update of the full batch (bp_train_batch);
    `steps` updates back to back, each timed with CUDA events."""
    import torch
    from paper_1801_01554_gb300 import bp, synth
    w = synth.WORKLOADS[name]
    sizes, X, T, theta = synth.make_workload(name)
    B = w["minibatch"]
    Xh = torch.tensor(X, dtype=torch.float32).to(torch.bfloat16)
    Th = torch.tensor(T, dtype=torch.float32).to(torch.bfloat16)
    del X, T
    Xd, Td = Xh.to(device), Th.to(device)
    sse = torch.zeros(1, dtype=torch.float32, device=device)
    with bp.Net(sizes, w["lr"], w["momentum"], bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        for _ in range(warmup):
            net.train_batch(Xd, Td, B, sse, stream)
        net.check(stream)
        ev = _events(steps + 1)
        torch.cuda.synchronize(device)
        ev[0].record(stream)
        for k in range(steps):
            net.train_batch(Xd, Td, B, sse, stream)
            ev[k + 1].record(stream)
        torch.cuda.synchronize(device)
        net.check(stream)
        step_ms = [ev[k].elapsed_time(ev[k + 1]) for k in range(steps)]
        e2e = None
        if with_e2e:
            Xp, Tp = Xh.pin_memory(), Th.pin_memory()
            sse_h = np.zeros(1, dtype=np.float32)
            net.train_epoch_host(Xp, Tp, B, B, sse_h, stream)       # staging allocation
            e2e_steps = max(1, min(steps, 10))
            barrier(world)
            torch.cuda.synchronize(device)
            t0 = time.perf_counter()
            for _ in range(e2e_steps):
                net.train_epoch_host(Xp, Tp, B, B, sse_h, stream)
            t = allreduce_max(time.perf_counter() - t0, world, device)
            e2e = (t, int(Xp.numel() * 2 + Tp.numel() * 2), int(sse_h.nbytes), e2e_steps)
    return sizes, B, step_ms, e2e


WIDE_LABEL = {"wide3": "1024-2048-2048-512 bf16, batch 8,192, lr 0.01, m 0.9; step = 1 update",
              "wide4096": "4096^5 bf16, batch 16,384, lr 0.01, m 0.9; step = 1 update"}
F32_LABEL = {"nettalk60": "203-60-26 f32, 1,024 patterns, full batch, lr 0.1; step = 10 epochs",
             "nettalk120": "203-120-26 f32, 65,536 patterns, mb 512, lr 0.05; step = 5 epochs"}


def cpu_for(name, mb=None, patterns=None, quick=False, seconds=10.0):
    """CPU baselines of a workload (bounded samples; see _cpu_child)."""
    from paper_1801_01554_gb300 import synth
    w = synth.WORKLOADS[name]
    ncpu = os.cpu_count() or 1
    if name in ("wide3", "wide4096"):
        # one full group of the 1024-2048-2048-512 net; one group of 1,024 of the
        # 4096^5 net (its 16,384 would take minutes on one core); CPS per pattern
        B = w["minibatch"] if name == "wide3" else 1024
        return cpu_baselines(name, B, B, {"mode": "serial", "groups": 1},
                             [{"mode": "blas", "groups": 1}],
                             f"one update of {B} patterns, numpy float64 oracle")
    mb = mb or w["minibatch"]
    n = patterns or w["patterns"]
    s1 = 2.0 if quick else seconds
    specs = []
    if mb >= 64:
        specs.append({"mode": "case_parallel", "workers": ncpu, "min_s": s1 / 2, "max_s": 2 * s1})
    return cpu_baselines(name, mb, n, {"mode": "serial", "min_s": s1, "max_s": 6 * s1}, specs,
                         f"groups of {mb} of {n} patterns, numpy float64 oracle")


def run_ours(args, world, rank, local):
    """Headline: the 203-120-26 workload, one step = its 5 epochs (5 persistent
    launches); `configs`: the other workloads, each with its own roofline,
    CPU baseline and end-to-end figure."""
    import torch
    from paper_1801_01554_gb300 import bp, synth

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    stream = torch.cuda.current_stream(device)
    num_sms = torch.cuda.get_device_properties(device).multi_processor_count
    lead = rank == 0 and world == 1 and not args.no_cpu_baseline

    # CPU baselines first, each in its own interpreter (no GPU work running)
    cpu = {}
    if lead:
        cpu["nettalk120"] = cpu_for("nettalk120", patterns=args.patterns, seconds=args.cpu_seconds)
        if not args.headline_only:
            cpu["nettalk60"] = cpu_for("nettalk60", quick=True)
            for B in synth.SWEEP_BATCHES:
                n = 65536 if B >= 512 else B * 512
                cpu[("sweep", B)] = cpu_for("nettalk120", mb=B, patterns=n, quick=True)
            cpu["wide3"] = cpu_for("wide3")
            cpu["wide4096"] = cpu_for("wide4096")

    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    w = synth.WORKLOADS[WORKLOAD]
    sizes, X, T, theta = synth.make_workload(WORKLOAD, patterns=args.patterns)
    n, mb = len(X), args.minibatch or w["minibatch"]
    epochs = w["epochs"]
    updates = -(-n // mb)
    W = connections(sizes)
    Xd = torch.tensor(X, dtype=torch.float32, device=device)
    Td = torch.tensor(T, dtype=torch.float32, device=device)
    sse = torch.zeros(updates, dtype=torch.float32, device=device)
    net = bp.Net(sizes, w["lr"], w["momentum"], bp.BP_F32, max_batch=mb)
    net.set_weights(theta)
    for _ in range(args.warmup):
        for _ in range(epochs):
            net.train_epoch(Xd, Td, n, mb, sse, stream)
    net.check(stream)
    ev = [_events(epochs + 1) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize(device)
    clocks.start()
    time.sleep(0.3)   # let the sampler start before the timed region
    t_wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.fill_(float(k))                  # evict the previous step from L2
        ev[k][0].record(stream)
        for e in range(epochs):
            net.train_epoch(Xd, Td, n, mb, sse, stream)
            ev[k][e + 1].record(stream)
    torch.cuda.synchronize(device)
    t_wall = time.perf_counter() - t_wall0
    clk = clocks.stop()
    barrier(world)
    net.check(stream)
    step_ms = [ev[k][0].elapsed_time(ev[k][-1]) for k in range(args.steps)]
    launch_ms = [ev[k][e].elapsed_time(ev[k][e + 1]) for k in range(args.steps) for e in range(epochs)]
    dev_s = sum(step_ms) / 1e3
    dev_s_max = allreduce_max(dev_s, world, device)
    value = W * n * epochs * args.steps * world / dev_s_max
    e2e_steps = max(1, min(args.steps, 10))
    t_e2e, bi, bo = time_f32_e2e(net, X, T, n, mb, epochs, e2e_steps, stream, world, device)
    net.close()

    launch_s = sum(launch_ms) / len(launch_ms) / 1e3
    peak, sm_max = alu_peak_tflops(num_sms)
    achieved = algorithmic_flops_per_pattern(sizes) * n / launch_s / 1e12
    tr = TRAFFIC_PER_PATTERN[WORKLOAD] if args.patterns is None and args.minibatch is None else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dev_s_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": F32_LABEL[WORKLOAD] if args.minibatch is None
                   else F32_LABEL[WORKLOAD] + f"; minibatch {mb} for a profiler capture",
                   "global_batch": mb,
                   "patterns_per_step": n * epochs, "updates_per_step": updates * epochs,
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": "flushed (512 MB write) before every timed step"},
        "roofline": {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": tr * n if tr else None,
                     "kernel": "k_train, one launch per epoch (CUDA events per launch)",
                     "peak_basis": f"{num_sms} SMs x {FP32_LANES_PER_SM} FFMA lanes x 2 x "
                                   f"{sm_max:.0f} MHz"},
        "e2e": {"value": W * n * epochs * e2e_steps * world / t_e2e, "unit": UNIT,
                "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo},
        "gpu_launches": args.steps * epochs,
        "clocks": clk,
        "wall_s_timed": t_wall,
    }
    if "nettalk120" in cpu:
        line["cpu_baseline"] = cpu["nettalk120"]

    if not args.headline_only:
        configs = {}
        # 203-60-26: one step = its 10 epochs of one full-batch update each
        w0 = synth.WORKLOADS["nettalk60"]
        s0, X0, T0, th0 = synth.make_workload("nettalk60")
        n0 = len(X0)
        with bp.Net(s0, w0["lr"], w0["momentum"], bp.BP_F32, max_batch=n0) as net0:
            net0.set_weights(th0)
            X0d = torch.tensor(X0, dtype=torch.float32, device=device)
            T0d = torch.tensor(T0, dtype=torch.float32, device=device)
            sse0 = torch.zeros(1, device=device)
            sm, lm = time_f32_launches(net0, X0d, T0d, n0, n0, w0["epochs"], 20, args.warmup, flush,
                                       stream, sse0)
            e = time_f32_e2e(net0, X0, T0, n0, n0, w0["epochs"], 10, stream, world, device)
        configs["nettalk60"] = f32_entry("nettalk60", s0, n0, n0, w0["epochs"], sm, lm,
                                         (e[0], e[1], e[2], 10), num_sms, cpu.get("nettalk60"),
                                         F32_LABEL["nettalk60"])
        # group-size sweep on 203-120-26: one step = one epoch
        sweep = []
        for B in synth.SWEEP_BATCHES:
            nb = 65536 if B >= 512 else B * 512
            with bp.Net(sizes, w["lr"], w["momentum"], bp.BP_F32, max_batch=B) as netb:
                netb.set_weights(theta)
                sseb = torch.zeros(-(-nb // B), device=device)
                sm, lm = time_f32_launches(netb, Xd, Td, nb, B, 1, 5, 3, flush, stream, sseb)
                e = time_f32_e2e(netb, X[:nb], T[:nb], nb, B, 1, 3, stream, world, device)
            ent = f32_entry("sweep", sizes, nb, B, 1, sm, lm, (e[0], e[1], e[2], 3), num_sms,
                            None, "")
            c = cpu.get(("sweep", B))
            sweep.append({"B": B, "patterns": nb, "value": ent["value"],
                          "us_per_update": 1e3 * ent["ms_per_step"] / -(-nb // B),
                          "frac": ent["roofline"]["frac"],
                          "traffic": (SWEEP_TRAFFIC_PER_PATTERN[B] * nb if B in SWEEP_TRAFFIC_PER_PATTERN
                                      else None),
                          "e2e": ent["e2e"]["value"],
                          "cpu_one_core": c["one_core"] if c else None,
                          "cpu_all_cores": c["value"] if c else None,
                          "cpu_cores": c["cores"] if c else None})
        configs["sweep_nettalk120"] = sweep
        for name in ("wide3", "wide4096"):
            steps = synth.WORKLOADS[name]["steps"]
            sz, B, sm, e = measure_bf16(name, steps, args.warmup, stream, device, world)
            configs[name] = bf16_entry(name, sz, B, sm, e, cpu.get(name), WIDE_LABEL[name])
        line["configs"] = configs
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def run_nettalk60(args, world, rank, local):
    """The 203-60-26 workload alone (for profiler captures): its compact entry;
    one step = its 10 full-batch epochs, one launch each."""
    import torch
    from paper_1801_01554_gb300 import bp, synth
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    stream = torch.cuda.current_stream(device)
    num_sms = torch.cuda.get_device_properties(device).multi_processor_count
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    w0 = synth.WORKLOADS["nettalk60"]
    s0, X0, T0, th0 = synth.make_workload("nettalk60")
    n0 = len(X0)
    with bp.Net(s0, w0["lr"], w0["momentum"], bp.BP_F32, max_batch=n0) as net0:
        net0.set_weights(th0)
        X0d = torch.tensor(X0, dtype=torch.float32, device=device)
        T0d = torch.tensor(T0, dtype=torch.float32, device=device)
        sse0 = torch.zeros(1, device=device)
        sm, lm = time_f32_launches(net0, X0d, T0d, n0, n0, w0["epochs"], args.steps, args.warmup,
                                   flush, stream, sse0)
    if rank == 0:
        print(json.dumps({"nettalk60": f32_entry("nettalk60", s0, n0, n0, w0["epochs"], sm, lm, None,
                                                 num_sms, None, F32_LABEL["nettalk60"])}), flush=True)
    return 0


def run_wide(args, world, rank, local):
    """One bf16 workload alone (for profiler captures): its compact entry."""
    import torch
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    stream = torch.cuda.current_stream(device)
    sz, B, sm, e = measure_bf16(args.workload, args.steps, args.warmup, stream, device, world,
                                with_e2e=False)
    if rank == 0:
        print(json.dumps({args.workload: bf16_entry(args.workload, sz, B, sm, e, None,
                                                    WIDE_LABEL[args.workload])}), flush=True)
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
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="one-core oracle seconds for the headline workload's CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=("nettalk120", "nettalk60", "wide3", "wide4096"),
                    help="nettalk120 (default): the headline and every config; nettalk60, wide3, "
                         "wide4096: that workload alone, for profiler captures")
    ap.add_argument("--headline-only", action="store_true",
                    help="the 203-120-26 headline alone (no configs object)")
    ap.add_argument("--patterns", type=int, default=None,
                    help="patterns per epoch (default: the workload's; a smaller epoch of the "
                         "same net and group size is for profiler captures, not a bench line)")
    ap.add_argument("--minibatch", type=int, default=None,
                    help="group size of the headline net (default: the workload's 512; another "
                         "size is for profiler captures, not a bench line)")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the bench line: CPS against the group size (203-120-26)")
    ap.add_argument("--crossover", action="store_true",
                    help="instead of the bench line: fp32 against bf16 as the hidden layer widens")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.patterns is not None or args.minibatch is not None:
        args.headline_only = True      # a shortened epoch or another group size: profiler captures only
    world, rank, local = dist_setup()
    if args.impl == "reference":
        rc = run_reference(args, world, rank)
    elif args.sweep:
        rc = run_sweep(args, world, rank, local)
    elif args.crossover:
        rc = run_crossover(args, world, rank, local)
    elif args.workload in ("wide3", "wide4096"):
        rc = run_wide(args, world, rank, local)
    elif args.workload == "nettalk60":
        rc = run_nettalk60(args, world, rank, local)
    else:
        rc = run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
