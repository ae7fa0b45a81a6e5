"""ctypes binding of libbp.so (the C ABI declared in include/bp.h).

Argument marshalling only: every step of the back-propagation path runs in the
library's CUDA kernels.  Functions keep the C names; device buffers are passed
as torch CUDA tensors (or raw integer addresses), host buffers as numpy arrays
or CPU tensors.  A missing library raises at first use: there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libbp.so")
_lib = None

BP_OK, BP_EINVAL, BP_ENOMEM, BP_ECUDA, BP_ESHAPE, BP_ETIMEOUT, BP_ENONFINITE, BP_ESTATE = range(8)
STATUS_NAMES = ["BP_OK", "BP_EINVAL", "BP_ENOMEM", "BP_ECUDA", "BP_ESHAPE", "BP_ETIMEOUT",
                "BP_ENONFINITE", "BP_ESTATE"]
BP_F32, BP_BF16 = 0, 1
BP_SIGMOID_LOGISTIC, BP_SIGMOID_TABLE = 0, 1
BP_MAX_SIZES = 9

# name -> (restype, argtypes); every symbol declared in include/bp.h
_VP = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_FP = ctypes.POINTER(ctypes.c_float)
SIGNATURES = {
    "bp_create": (_I, [ctypes.POINTER(_I), _I, _F, _F, _I, _I, ctypes.POINTER(_VP)]),
    "bp_destroy": (None, [_VP]),
    "bp_set_hparams": (_I, [_VP, _F, _F, _F]),
    "bp_set_sigmoid": (_I, [_VP, _I]),
    "bp_set_guard": (_I, [_VP, _F]),
    "bp_get_faults": (_I, [_VP, ctypes.POINTER(ctypes.c_int64), _I]),
    "bp_diagnose": (_I, [_VP, _VP, _VP, _I, _FP, ctypes.POINTER(_I), _I, ctypes.POINTER(_I),
                         ctypes.POINTER(_I)]),
    "bp_vote": (_I, [_FP, _I, _FP, ctypes.POINTER(_I)]),
    "bp_num_params": (ctypes.c_int64, [_VP]),
    "bp_set_weights": (_I, [_VP, _FP]),
    "bp_get_weights": (_I, [_VP, _FP]),
    "bp_set_velocity": (_I, [_VP, _FP]),
    "bp_get_velocity": (_I, [_VP, _FP]),
    "bp_get_grads": (_I, [_VP, _FP]),
    "bp_forward": (_I, [_VP, _VP, _I, _VP, _VP]),
    "bp_backward": (_I, [_VP, _VP, _I, _VP, _VP]),
    "bp_update": (_I, [_VP, _VP]),
    "bp_train_batch": (_I, [_VP, _VP, _VP, _I, _VP, _VP]),
    "bp_train_epoch": (_I, [_VP, _VP, _VP, _I, _I, _VP, _VP]),
    "bp_train_epoch_host": (_I, [_VP, _VP, _VP, _I, _I, _FP, _VP]),
    "bp_check": (_I, [_VP, _VP]),
    "bp_train_epoch_noalloc": (_I, [ctypes.POINTER(_I), _I, _F, _F, _F, _VP, _VP, _VP, _VP, _I, _I,
                                    _VP, _VP, _VP]),
    "bp_debug_wait_test": (_I, [_VP, ctypes.c_ulonglong, _I]),
    "bp_last_error": (ctypes.c_char_p, []),
}


class BPError(RuntimeError):
    def __init__(self, status: int, message: str):
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"{name}: {message}")
        self.status = status


def lib_path() -> str:
    return _LIB_PATH


def load(path: str | None = None):
    """Load libbp.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or _LIB_PATH
    if not os.path.exists(p):
        raise ImportError(f"{p} is missing: build it first (python -c 'import __graft_entry__ as g; "
                          "g.build()')")
    lib = ctypes.CDLL(p)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status: int):
    if status != BP_OK:
        raise BPError(status, load().bp_last_error().decode())


def _dptr(x):
    """Device address of a CUDA tensor (or an int address, or None -> NULL)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not x.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return x.data_ptr()


def _hptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("expected a C-contiguous array")
        return x.ctypes.data
    if x.is_cuda or not x.is_contiguous():
        raise ValueError("expected a contiguous CPU tensor")
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _f32_host(arr, n):
    a = np.ascontiguousarray(arr, dtype=np.float32)
    if a.size != n:
        raise ValueError(f"expected {n} parameters, got {a.size}")
    return a


# ------------------------------------------------------------------ C names
def bp_create(sizes, lr, momentum, dtype=BP_F32, max_batch=1024):
    sizes = [int(s) for s in sizes]
    arr = (ctypes.c_int * len(sizes))(*sizes)
    out = ctypes.c_void_p()
    _check(load().bp_create(arr, len(sizes), float(lr), float(momentum), int(dtype),
                            int(max_batch), ctypes.byref(out)))
    return out.value


def bp_destroy(h):
    load().bp_destroy(h)


def bp_set_hparams(h, lr, momentum, grad_scale=1.0):
    _check(load().bp_set_hparams(h, float(lr), float(momentum), float(grad_scale)))


def bp_set_sigmoid(h, mode):
    _check(load().bp_set_sigmoid(h, int(mode)))


def bp_set_guard(h, threshold):
    _check(load().bp_set_guard(h, float(threshold)))


def bp_get_faults(h, reset=False) -> int:
    c = ctypes.c_int64(0)
    _check(load().bp_get_faults(h, ctypes.byref(c), 1 if reset else 0))
    return int(c.value)


def bp_diagnose(h, X, T, batch, capacity=1024):
    """Diagnostic mode: (per-CTA error sums, SM ids, number agreeing with the vote)."""
    sse = np.zeros(capacity, dtype=np.float32)
    sm = np.zeros(capacity, dtype=np.int32)
    n = ctypes.c_int(0)
    agree = ctypes.c_int(0)
    _check(load().bp_diagnose(h, _dptr(X), _dptr(T), int(batch), sse.ctypes.data_as(_FP),
                              sm.ctypes.data_as(ctypes.POINTER(_I)), capacity, ctypes.byref(n),
                              ctypes.byref(agree)))
    return sse[:n.value], sm[:n.value], agree.value


def bp_vote(values):
    """(the value most entries equal bit for bit, how many equal it)."""
    a = np.ascontiguousarray(values, dtype=np.float32)
    mode = ctypes.c_float(0.0)
    agree = ctypes.c_int(0)
    _check(load().bp_vote(a.ctypes.data_as(_FP), int(a.size), ctypes.byref(mode), ctypes.byref(agree)))
    return float(mode.value), agree.value


def bp_num_params(h) -> int:
    return int(load().bp_num_params(h))


def bp_set_weights(h, theta):
    a = _f32_host(theta, bp_num_params(h))
    _check(load().bp_set_weights(h, a.ctypes.data_as(_FP)))


def bp_get_weights(h) -> np.ndarray:
    a = np.empty(bp_num_params(h), dtype=np.float32)
    _check(load().bp_get_weights(h, a.ctypes.data_as(_FP)))
    return a


def bp_set_velocity(h, v):
    a = _f32_host(v, bp_num_params(h))
    _check(load().bp_set_velocity(h, a.ctypes.data_as(_FP)))


def bp_get_velocity(h) -> np.ndarray:
    a = np.empty(bp_num_params(h), dtype=np.float32)
    _check(load().bp_get_velocity(h, a.ctypes.data_as(_FP)))
    return a


def bp_get_grads(h) -> np.ndarray:
    a = np.empty(bp_num_params(h), dtype=np.float32)
    _check(load().bp_get_grads(h, a.ctypes.data_as(_FP)))
    return a


def bp_forward(h, X, batch, Y=None, stream=None):
    _check(load().bp_forward(h, _dptr(X), int(batch), _dptr(Y), _stream(stream)))


def bp_backward(h, T, batch, sse=None, stream=None):
    _check(load().bp_backward(h, _dptr(T), int(batch), _dptr(sse), _stream(stream)))


def bp_update(h, stream=None):
    _check(load().bp_update(h, _stream(stream)))


def bp_train_batch(h, X, T, batch, sse=None, stream=None):
    _check(load().bp_train_batch(h, _dptr(X), _dptr(T), int(batch), _dptr(sse), _stream(stream)))


def bp_train_epoch(h, X, T, n_patterns, minibatch, sse=None, stream=None):
    _check(load().bp_train_epoch(h, _dptr(X), _dptr(T), int(n_patterns), int(minibatch),
                                 _dptr(sse), _stream(stream)))


def bp_train_epoch_host(h, X, T, n_patterns, minibatch, sse=None, stream=None):
    sp = None
    if sse is not None:
        if isinstance(sse, np.ndarray):
            if sse.dtype != np.float32 or not sse.flags["C_CONTIGUOUS"]:
                raise ValueError("sse must be a C-contiguous float32 array")
            sp = sse.ctypes.data_as(_FP)
        else:
            sp = ctypes.cast(_hptr(sse), _FP)
    _check(load().bp_train_epoch_host(h, _hptr(X), _hptr(T), int(n_patterns), int(minibatch), sp,
                                      _stream(stream)))


def bp_check(h, stream=None):
    _check(load().bp_check(h, _stream(stream)))


def bp_train_epoch_noalloc(sizes, lr, momentum, grad_scale, theta, V, X, T, n_patterns, minibatch,
                           sse=None, status=None, stream=None):
    """Training epoch that allocates nothing: every buffer is the caller's
    (float32 CUDA tensors theta and V are updated in place)."""
    sizes = [int(s) for s in sizes]
    arr = (ctypes.c_int * len(sizes))(*sizes)
    _check(load().bp_train_epoch_noalloc(arr, len(sizes), float(lr), float(momentum),
                                         float(grad_scale), _dptr(theta), _dptr(V), _dptr(X),
                                         _dptr(T), int(n_patterns), int(minibatch), _dptr(sse),
                                         _dptr(status), _stream(stream)))


def bp_debug_wait_test(h, wait_ns, unreachable):
    """Checked builds only: grid-barrier and weight-phase wait limit (0 =
    default); unreachable = 1: a first grid barrier that the next training
    launch cannot pass; 2: a first weight-phase chunk copy that never comes."""
    _check(load().bp_debug_wait_test(h, int(wait_ns), int(unreachable)))


def bp_last_error() -> str:
    return load().bp_last_error().decode()


# ------------------------------------------------------------------ convenience
class Net:
    """Owns one bp_net handle; methods forward to the C names above."""

    def __init__(self, sizes, lr, momentum, dtype=BP_F32, max_batch=1024, grad_scale=1.0):
        self.sizes = tuple(int(s) for s in sizes)
        self.dtype = dtype
        self.h = bp_create(self.sizes, lr, momentum, dtype, max_batch)
        if grad_scale != 1.0:
            bp_set_hparams(self.h, lr, momentum, grad_scale)

    def close(self):
        if self.h:
            bp_destroy(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def num_params(self):
        return bp_num_params(self.h)

    def set_hparams(self, lr, momentum, grad_scale=1.0):
        bp_set_hparams(self.h, lr, momentum, grad_scale)

    def set_sigmoid(self, mode):
        bp_set_sigmoid(self.h, mode)

    def set_guard(self, threshold):
        bp_set_guard(self.h, threshold)

    def get_faults(self, reset=False):
        return bp_get_faults(self.h, reset)

    def diagnose(self, X, T, batch):
        return bp_diagnose(self.h, X, T, batch)

    def set_weights(self, theta):
        bp_set_weights(self.h, theta)

    def get_weights(self):
        return bp_get_weights(self.h)

    def set_velocity(self, v):
        bp_set_velocity(self.h, v)

    def get_velocity(self):
        return bp_get_velocity(self.h)

    def get_grads(self):
        return bp_get_grads(self.h)

    def forward(self, X, batch, Y=None, stream=None):
        bp_forward(self.h, X, batch, Y, stream)

    def backward(self, T, batch, sse=None, stream=None):
        bp_backward(self.h, T, batch, sse, stream)

    def update(self, stream=None):
        bp_update(self.h, stream)

    def train_batch(self, X, T, batch, sse=None, stream=None):
        bp_train_batch(self.h, X, T, batch, sse, stream)

    def train_epoch(self, X, T, n_patterns, minibatch, sse=None, stream=None):
        bp_train_epoch(self.h, X, T, n_patterns, minibatch, sse, stream)

    def train_epoch_host(self, X, T, n_patterns, minibatch, sse=None, stream=None):
        bp_train_epoch_host(self.h, X, T, n_patterns, minibatch, sse, stream)

    def check(self, stream=None):
        bp_check(self.h, stream)


def connections(sizes) -> int:
    """Connections counted as the paper counts them, bias connections included."""
    return sum((sizes[l - 1] + 1) * sizes[l] for l in range(1, len(sizes)))
