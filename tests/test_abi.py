"""The C ABI library loads and exports every symbol include/bp.h declares;
argument errors are reported before any device work.  CPU only."""
import ctypes
import os
import re

import pytest

from paper_1801_01554_gb300 import bp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include")))
           if f.endswith(".h")]


def declared_functions():
    names = []
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(bp_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(bp.lib_path()):
        from paper_1801_01554_gb300 import build
        build.build()
    return bp.load()


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("bp_create", "bp_forward", "bp_backward", "bp_update", "bp_train_batch",
                     "bp_destroy"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert names
    for n in names:
        assert hasattr(lib, n), n
        assert n in bp.SIGNATURES, f"binding lacks {n}"


def test_binding_covers_only_declared_symbols():
    assert set(bp.SIGNATURES) <= set(declared_functions())


@pytest.mark.parametrize("sizes,n_layers,batch,dtype", [
    ((203, 60, 26), 1, 10, 0),      # one layer is not a net
    ((203, 0, 26), 3, 10, 0),       # empty layer
    ((203, 60, 26), 3, 0, 0),       # no batch capacity
    ((203, 60, 26), 3, 10, 7),      # unknown dtype
    ((4,) * 10, 10, 10, 0),         # more than BP_MAX_SIZES sizes
])
def test_create_rejects_bad_arguments_before_device_work(lib, sizes, n_layers, batch, dtype):
    arr = (ctypes.c_int * len(sizes))(*sizes)
    out = ctypes.c_void_p()
    st = lib.bp_create(arr, n_layers, 0.1, 0.9, dtype, batch, ctypes.byref(out))
    assert st == bp.BP_EINVAL
    assert out.value is None
    assert lib.bp_last_error()


def test_null_handles_are_rejected(lib):
    assert lib.bp_update(None, None) == bp.BP_EINVAL
    assert lib.bp_forward(None, None, 1, None, None) == bp.BP_EINVAL
    assert lib.bp_check(None, None) == bp.BP_EINVAL
    assert lib.bp_num_params(None) == 0
    assert lib.bp_set_sigmoid(None, bp.BP_SIGMOID_TABLE) == bp.BP_EINVAL
    assert lib.bp_set_guard(None, 1.0) == bp.BP_EINVAL
    assert lib.bp_get_faults(None, None, 0) == bp.BP_EINVAL
    lib.bp_destroy(None)   # NULL-safe


@pytest.mark.parametrize("bad", ["d_theta", "d_V", "d_X", "d_T", "d_sse", "d_status"])
def test_noalloc_rejects_misaligned_pointers_before_any_cuda_call(lib, bad):
    """The allocation-free entry point reads its buffers as float32 words: a
    pointer off a 4-byte boundary is refused with BP_EINVAL before the call
    touches the device (this runs without a GPU, so any CUDA call would fail
    with BP_ECUDA instead).  The addresses are never dereferenced."""
    sizes = (203, 120, 26)
    arr = (ctypes.c_int * 3)(*sizes)
    ptrs = {k: 0x10000 * (i + 1) for i, k in enumerate(["d_theta", "d_V", "d_X", "d_T", "d_sse",
                                                        "d_status"])}
    ptrs[bad] += 2
    st = lib.bp_train_epoch_noalloc(arr, 3, 0.05, 0.9, 1.0, ptrs["d_theta"], ptrs["d_V"],
                                    ptrs["d_X"], ptrs["d_T"], 512, 512, ptrs["d_sse"],
                                    ptrs["d_status"], None)
    assert st == bp.BP_EINVAL
    msg = lib.bp_last_error().decode()
    assert bad in msg and "aligned" in msg
