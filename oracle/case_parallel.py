"""Case-parallel driver for the CPU oracle (Section 4.1 on the host's cores).

TEST INFRASTRUCTURE ONLY: used by ``bench.py``'s ``cpu_baseline`` leg and by
``tests/``; nothing on the product path imports it.

Section 4.1 trains with case parallelism: every processor holds the whole net,
runs the forward and backward passes of its own share of a group's patterns,
and the changes are summed over all processors before one update.  This module
does the same with P worker processes over the oracle as it stands: worker k
takes patterns [p0 + k*nb/P, p0 + (k+1)*nb/P) of each group, computes their
pooled change and error with ``bp_oracle.step_quantities``, and writes them to
its slot of a shared-memory array; the parent sums the slots in worker order
and applies ``bp_oracle.apply_update``.  Workers start with the 'spawn' method
(never forked from a process that may hold a CUDA context) and each uses one
BLAS thread.  The result equals the serial oracle's up to the order of the
float64 sums.
"""
from __future__ import annotations

import multiprocessing as mp
import os
from multiprocessing import shared_memory

import numpy as np

from oracle import bp_oracle as O


def _attach(name, shape):
    shm = shared_memory.SharedMemory(name=name)
    return shm, np.ndarray(shape, dtype=np.float64, buffer=shm.buf)


_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def _worker(k, P, sizes, names, shapes, squash, conn):
    shms = {}
    arr = {}
    for key in ("X", "T", "theta", "G"):
        shms[key], arr[key] = _attach(names[key], shapes[key])
    st = O.State(sizes, np.zeros(shapes["theta"]), lr=0.0, momentum=0.0, squash=squash)
    while True:
        msg = conn.recv()
        if msg is None:
            break
        p0, nb = msg
        a = p0 + (nb * k) // P
        b = p0 + (nb * (k + 1)) // P
        st.theta = arr["theta"]
        if b > a:
            _, _, G, e = O.step_quantities(st, arr["X"][a:b], arr["T"][a:b])
            arr["G"][k, :-1] = G
            arr["G"][k, -1] = e
        else:
            arr["G"][k, :] = 0.0
        conn.send(True)
    for s in shms.values():
        s.close()


class CaseParallel:
    """P spawned workers over the patterns X, T (float64, [n, n_0] / [n, n_L])."""

    def __init__(self, sizes, X, T, workers, squash="logistic"):
        self.sizes = tuple(int(s) for s in sizes)
        self.P = int(workers)
        n_par = O.connections(self.sizes)
        shapes = {"X": np.shape(X), "T": np.shape(T), "theta": (n_par,), "G": (self.P, n_par + 1)}
        self._shm = {}
        self._arr = {}
        for key, shape in shapes.items():
            nbytes = max(8, int(np.prod(shape)) * 8)
            self._shm[key] = shared_memory.SharedMemory(create=True, size=nbytes)
            self._arr[key] = np.ndarray(shape, dtype=np.float64, buffer=self._shm[key].buf)
        self._arr["X"][...] = X
        self._arr["T"][...] = T
        names = {k: s.name for k, s in self._shm.items()}
        ctx = mp.get_context("spawn")
        self._conns = []
        self._procs = []
        # one BLAS thread per worker, set before the children import numpy
        saved = {v: os.environ.get(v) for v in _THREAD_VARS}
        os.environ.update({v: "1" for v in _THREAD_VARS})
        try:
            for k in range(self.P):
                a, b = ctx.Pipe()
                p = ctx.Process(target=_worker, args=(k, self.P, self.sizes, names, shapes, squash, b),
                                daemon=True)
                p.start()
                self._conns.append(a)
                self._procs.append(p)
        finally:
            for v, val in saved.items():
                if val is None:
                    os.environ.pop(v, None)
                else:
                    os.environ[v] = val

    def train_batch(self, state: O.State, p0: int, nb: int) -> float:
        """One group (patterns [p0, p0 + nb)): pooled change summed over the
        workers in order, then the oracle's update of `state`.  Returns the SSE."""
        self._arr["theta"][...] = state.theta
        for c in self._conns:
            c.send((p0, nb))
        for c in self._conns:
            c.recv()
        acc = np.zeros(self._arr["G"].shape[1])
        for k in range(self.P):
            acc += self._arr["G"][k]
        state.G = state.G + acc[:-1]
        O.apply_update(state)
        return float(acc[-1])

    def train_epoch(self, state: O.State, n: int, minibatch: int):
        return [self.train_batch(state, p0, min(minibatch, n - p0)) for p0 in range(0, n, minibatch)]

    def close(self):
        for c in self._conns:
            try:
                c.send(None)
            except (BrokenPipeError, OSError):
                pass
        for p in self._procs:
            p.join(timeout=10)
            if p.is_alive():
                p.terminate()
        for s in self._shm.values():
            s.close()
            s.unlink()
        self._procs = []
        self._conns = []
        self._shm = {}

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
