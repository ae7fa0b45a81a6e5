"""Run by tests/test_gpu_checked.py in a fresh process against the checked
build named on the command line (argv: library, "barrier" or "chunk", case
name): makes a wait of a training launch run out of time with a 1 ms limit,
either its first grid barrier (a count that no CTA will reach) or the first
chunk of each CTA's weight phase (a copy that never comes: the barrier is armed,
no copy is issued), then trains the same epoch normally, and prints what
happened as JSON.

No GPU fault is involved: every wait is bounded, the kernel latches the
timeout and every CTA returns with every copy it issued landed."""
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_1801_01554_gb300 import bp, synth  # noqa: E402

bp.load(sys.argv[1])
MODE = sys.argv[2] if len(sys.argv) > 2 else "barrier"
CASES = {"nettalk120_512": ((203, 120, 26), 2048, 512),      # whole-tile weight phase
         "nettalk60_12288": ((203, 60, 26), 24576, 12288)}   # balanced weight phase
sizes, n, mb = CASES[sys.argv[3] if len(sys.argv) > 3 else "nettalk120_512"]
X, T = synth.nettalk_patterns(n, seed=71)
theta = synth.round_to(synth.init_uniform(sizes, -0.3, 0.3, 71), "f32")
Xd = torch.tensor(X, dtype=torch.float32, device="cuda")
Td = torch.tensor(T, dtype=torch.float32, device="cuda")
out = {}
with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
    net.set_weights(theta)
    sse = torch.zeros(n // mb, device="cuda")
    bp.bp_debug_wait_test(net.h, 1_000_000, 1 if MODE == "barrier" else 2)   # 1 ms limit
    t0 = time.perf_counter()
    net.train_epoch(Xd, Td, n, mb, sse)
    try:
        net.check()
        out["status"] = bp.BP_OK
    except bp.BPError as e:
        out["status"] = e.status
    out["seconds"] = time.perf_counter() - t0
    out["weights_unchanged"] = bool(np.array_equal(net.get_weights(), theta.astype(np.float32)))
    net.check()                                          # the latch was cleared
    bp.bp_debug_wait_test(net.h, 0, 0)                   # default limit, nothing planted
    net.train_epoch(Xd, Td, n, mb, sse)
    net.check()
    out["w"] = net.get_weights().tolist()
    out["v"] = net.get_velocity().tolist()
    out["sse"] = sse.cpu().numpy().tolist()
print(json.dumps(out))
