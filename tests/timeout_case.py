"""Run by tests/test_gpu_checked.py in a fresh process against the checked
build named on the command line: makes the first grid barrier of a training
launch run out of time (a count that no CTA will reach, a 1 ms limit), then
trains the same epoch normally, and prints what happened as JSON.

No GPU fault is involved: the wait is bounded, the kernel latches the timeout
and every CTA returns at that barrier, where no copy is in flight."""
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
sizes, n, mb = (203, 120, 26), 2048, 512
X, T = synth.nettalk_patterns(n, seed=71)
theta = synth.round_to(synth.init_uniform(sizes, -0.3, 0.3, 71), "f32")
Xd = torch.tensor(X, dtype=torch.float32, device="cuda")
Td = torch.tensor(T, dtype=torch.float32, device="cuda")
out = {}
with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
    net.set_weights(theta)
    sse = torch.zeros(n // mb, device="cuda")
    bp.bp_debug_wait_test(net.h, 1_000_000, True)       # 1 ms, unreachable first barrier
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
    bp.bp_debug_wait_test(net.h, 0, False)               # default limit, reachable barrier
    net.train_epoch(Xd, Td, n, mb, sse)
    net.check()
    out["w"] = net.get_weights().tolist()
    out["v"] = net.get_velocity().tolist()
    out["sse"] = sse.cpu().numpy().tolist()
print(json.dumps(out))
