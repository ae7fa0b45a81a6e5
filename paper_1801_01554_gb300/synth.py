"""Seeded synthetic inputs for the back-propagation step.

This module holds no part of the method's arithmetic: it only draws patterns,
targets and initial weights, in float64 on the host, so that the CPU oracle and
the CUDA path can be fed the very same buffers.

The paper's NETtalk corpus (Section 6.3: 203 input units in 7 letter windows of
29 symbols, 26 output features, 12,022 patterns) is not available; the
generators below reproduce its shapes and structure instead:

* ``nettalk_patterns`` -- each input is 7 one-hot blocks of 29 (one uniformly
  drawn letter per block), each target is a 26-dim binary vector with exactly 3
  ones at distinct, uniformly drawn positions.
* ``gaussian_patterns`` -- inputs N(0, 1), targets Bernoulli(p) in {0, 1}; the
  stand-in for wide layers that the paper does not measure.

Parameters are one flat vector in layer order, for l = 1..L: the weight matrix
W_l (n_l rows of n_{l-1} inputs, row-major) followed by the n_l bias weights
b_l (the connections from the paper's always-on "true" unit, Section 6.3).
"""
from __future__ import annotations

import numpy as np

NETTALK_BLOCKS = 7
NETTALK_LETTERS = 29
NETTALK_OUTPUTS = 26
NETTALK_ONES = 3


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), int(stream)])


def param_layout(sizes):
    """(offset of W_l, offset of b_l) for each layer, and the total length."""
    off = []
    pos = 0
    for l in range(1, len(sizes)):
        w_off = pos
        pos += sizes[l] * sizes[l - 1]
        b_off = pos
        pos += sizes[l]
        off.append((w_off, b_off))
    return off, pos


def nettalk_patterns(n: int, seed: int = 0, n_in: int = 203, n_out: int = 26):
    """NETtalk-shaped patterns: X [n, 203] one-hot blocks, T [n, 26] 3-hot."""
    if n_in != NETTALK_BLOCKS * NETTALK_LETTERS or n_out != NETTALK_OUTPUTS:
        raise ValueError("NETtalk-shaped patterns are 203 inputs and 26 outputs")
    rng = _rng(seed, 0)
    letters = rng.integers(0, NETTALK_LETTERS, size=(n, NETTALK_BLOCKS))
    X = np.zeros((n, n_in), dtype=np.float64)
    cols = letters + NETTALK_LETTERS * np.arange(NETTALK_BLOCKS)[None, :]
    X[np.arange(n)[:, None], cols] = 1.0
    # 3 distinct positions per pattern: the first 3 of a random permutation.
    keys = rng.random((n, n_out))
    ones = np.argsort(keys, axis=1, kind="stable")[:, :NETTALK_ONES]
    T = np.zeros((n, n_out), dtype=np.float64)
    T[np.arange(n)[:, None], ones] = 1.0
    return X, T


def gaussian_patterns(n: int, n_in: int, n_out: int, p_one: float, seed: int = 0):
    """Inputs N(0, 1) [n, n_in]; targets Bernoulli(p_one) [n, n_out] in {0, 1}."""
    rng = _rng(seed, 0)
    X = rng.standard_normal((n, n_in))
    T = (rng.random((n, n_out)) < p_one).astype(np.float64)
    return X, T


def init_uniform(sizes, lo: float, hi: float, seed: int = 0) -> np.ndarray:
    """Every weight, bias weights included, drawn from U(lo, hi)."""
    _, total = param_layout(sizes)
    return _rng(seed, 1).uniform(lo, hi, size=total)


def init_normal_fanin(sizes, seed: int = 0) -> np.ndarray:
    """W_l entries N(0, 1/n_{l-1}); bias weights zero."""
    offs, total = param_layout(sizes)
    rng = _rng(seed, 1)
    theta = np.zeros(total, dtype=np.float64)
    for l, (w_off, b_off) in enumerate(offs, start=1):
        nw = sizes[l] * sizes[l - 1]
        theta[w_off:w_off + nw] = rng.standard_normal(nw) / np.sqrt(sizes[l - 1])
    return theta


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values once to the path dtype and return them as float64."""
    if dtype == "f32":
        return np.asarray(x, dtype=np.float32).astype(np.float64)
    if dtype == "bf16":
        return bf16_round(x)
    raise ValueError(dtype)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even to bfloat16 (via float32), returned as float64."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


# The five workloads of the benchmark suite, named by what they are.
WORKLOADS = {
    "nettalk60": dict(
        sizes=(203, 60, 26), dtype="f32", patterns=1024, minibatch=1024,
        lr=0.1, momentum=0.9, epochs=10, seed=0, data="nettalk",
        init=("uniform", -0.3, 0.3)),
    "nettalk120": dict(
        sizes=(203, 120, 26), dtype="f32", patterns=65536, minibatch=512,
        lr=0.05, momentum=0.9, epochs=5, seed=0, data="nettalk",
        init=("uniform", -0.3, 0.3)),
    "wide3": dict(
        sizes=(1024, 2048, 2048, 512), dtype="bf16", patterns=8192, minibatch=8192,
        lr=0.01, momentum=0.9, steps=100, seed=0, data=("gaussian", 0.1),
        init=("normal_fanin",)),
    "wide4096": dict(
        sizes=(4096, 4096, 4096, 4096, 4096), dtype="bf16", patterns=16384,
        minibatch=16384, lr=0.01, momentum=0.9, steps=50, seed=0,
        data=("gaussian", 0.5), init=("normal_fanin",)),
}
# Batch sizes of the 203-120-26 batch sweep.
SWEEP_BATCHES = (1, 8, 64, 512, 4096, 65536)


def make_workload(name: str, patterns: int | None = None, seed: int | None = None):
    """(sizes, X, T, theta0) in float64 for a named workload, rounded to its dtype."""
    w = WORKLOADS[name]
    sizes = w["sizes"]
    n = w["patterns"] if patterns is None else patterns
    s = w["seed"] if seed is None else seed
    if w["data"] == "nettalk":
        X, T = nettalk_patterns(n, s, sizes[0], sizes[-1])
    else:
        X, T = gaussian_patterns(n, sizes[0], sizes[-1], w["data"][1], s)
    if w["init"][0] == "uniform":
        theta = init_uniform(sizes, w["init"][1], w["init"][2], s)
    else:
        theta = init_normal_fanin(sizes, s)
    dt = w["dtype"]
    # fp32 master weights on both paths; activations in the path dtype.
    return sizes, round_to(X, dt), round_to(T, dt), round_to(theta, "f32")
