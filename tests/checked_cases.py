"""Run by tests/test_gpu_checked.py in a fresh process: loads the library named
on the command line and prints, as JSON, the results of a few training runs
that go through every float32 kernel (persistent training with whole-tile and
balanced weight phases, one-CTA groups, forward/backward/update, the
allocation-free entry point, diagnostic mode)."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_1801_01554_gb300 import bp, synth  # noqa: E402

bp.load(sys.argv[1])


def dev(a):
    return torch.tensor(np.asarray(a), dtype=torch.float32, device="cuda")


out = {}
# the last case runs two groups of 24 chunks (the balanced weight phase) and a ragged third
for sizes, n, mb in (((203, 120, 26), 1100, 512), ((203, 60, 26), 40, 2), ((64, 33, 17, 9), 300, 300),
                     ((7, 9, 5, 11, 6, 8, 4, 10, 3), 66, 33), ((203, 60, 26), 26000, 12288)):
    X, T = synth.gaussian_patterns(n, sizes[0], sizes[-1], 0.3, seed=3)
    theta = synth.round_to(synth.init_uniform(sizes, -0.5, 0.5, 3), "f32")
    key = "-".join(map(str, sizes)) + f"/{mb}"
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=max(mb, n)) as net:
        net.set_weights(theta)
        Xd, Td = dev(X), dev(T)
        sse = torch.zeros(-(-n // mb), device="cuda")
        net.train_epoch(Xd, Td, n, mb, sse)
        net.check()
        net.forward(Xd, n)
        net.backward(Td, n)
        net.update()
        net.check()
        d_sse, _, agree = net.diagnose(Xd, Td, min(n, 64))
        out[key] = {"w": net.get_weights().tolist(), "sse": sse.cpu().numpy().tolist(),
                    "diag": float(d_sse[0]), "agree": agree}
    if len(sizes) == 3 and mb <= 2048:   # (larger groups do not fit the entry point's static scratch)
        th, V = dev(theta), torch.zeros(theta.size, device="cuda")
        bp.bp_train_epoch_noalloc(sizes, 0.05, 0.9, 1.0, th, V, Xd, Td, n, mb)
        torch.cuda.synchronize()
        out[key]["noalloc"] = th.cpu().numpy().tolist()
print(json.dumps(out))
