"""The allocation-free training entry point, for callers that cannot call
cudaMalloc (a host framework that owns the allocator, a fixed memory budget, a
plug-in limited to the buffers it is given).  It must give the same result as
the ordinary entry point, call after call, although its scratch is a static
device array that every call reuses.

This file is collected last so that a failure here never hides another test."""
import numpy as np
import pytest

from paper_1801_01554_gb300 import bp, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-5   # the float32 parity tolerance used by the other tests


def normwise(x, y):
    x = np.asarray(x, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    return float(np.max(np.abs(x - y)) / max(np.max(np.abs(y)), 1e-30))


def test_noalloc_epoch_matches_bp_train_epoch_twice_in_a_row():
    sizes, n, mb, lr, m = (203, 120, 26), 3000, 512, 0.05, 0.9
    X, T = synth.nettalk_patterns(n, seed=21)
    theta = synth.round_to(synth.init_uniform(sizes, -0.3, 0.3, 21), "f32")
    Xd = torch.tensor(X, dtype=torch.float32, device="cuda")
    Td = torch.tensor(T, dtype=torch.float32, device="cuda")
    steps = (n + mb - 1) // mb

    ref_w, ref_sse = [], []
    with bp.Net(sizes, lr, m, bp.BP_F32, max_batch=mb) as net:
        net.set_weights(theta)
        for _ in range(2):
            sse = torch.zeros(steps, device="cuda")
            net.train_epoch(Xd, Td, n, mb, sse)
            net.check()
            ref_w.append(net.get_weights())
            ref_sse.append(sse.cpu().numpy())

    th = torch.tensor(theta, dtype=torch.float32, device="cuda")
    V = torch.zeros_like(th)
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    for k in range(2):
        sse = torch.zeros(steps, device="cuda")
        bp.bp_train_epoch_noalloc(sizes, lr, m, 1.0, th, V, Xd, Td, n, mb, sse, status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert normwise(th.cpu().numpy() - theta, ref_w[k] - theta) <= TOL
        np.testing.assert_allclose(sse.cpu().numpy(), ref_sse[k], rtol=TOL)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    sizes = (203, 120, 26)
    th = torch.zeros(bp.connections(sizes), device="cuda")
    X = torch.zeros((16, 203), device="cuda")
    T = torch.zeros((16, 26), device="cuda")
    with pytest.raises(bp.BPError) as e:
        bp.bp_train_epoch_noalloc(sizes, 0.1, 0.9, 1.0, th, th.clone(), X, T, 16, 100000)
    assert e.value.status == bp.BP_EINVAL
    assert "scratch" in bp.bp_last_error()


def test_noalloc_smaller_call_after_a_larger_one():
    """The static scratch keeps the previous call's activations, deltas and
    padded weights.  A call on a larger net and minibatch, then one on a
    smaller, deeper net: the second must match bp_train_epoch on a fresh net
    within the float32 bar, per layer, so nothing stale from the first call
    reaches it (stale rows would change the pooled change by far more)."""
    big, n1, mb1 = (203, 120, 26), 4096, 2048
    X1, T1 = synth.nettalk_patterns(n1, seed=31)
    th1 = torch.tensor(synth.round_to(synth.init_uniform(big, -0.3, 0.3, 31), "f32"),
                       dtype=torch.float32, device="cuda")
    bp.bp_train_epoch_noalloc(big, 0.05, 0.9, 1.0, th1, torch.zeros_like(th1),
                              torch.tensor(X1, dtype=torch.float32, device="cuda"),
                              torch.tensor(T1, dtype=torch.float32, device="cuda"), n1, mb1)
    torch.cuda.synchronize()

    small, n, mb = (64, 33, 17, 9), 300, 100
    X, T = synth.gaussian_patterns(n, small[0], small[-1], 0.3, seed=32)
    X = synth.round_to(X, "f32")
    theta = synth.round_to(synth.init_uniform(small, -0.5, 0.5, 32), "f32")
    Xd = torch.tensor(X, dtype=torch.float32, device="cuda")
    Td = torch.tensor(T, dtype=torch.float32, device="cuda")
    steps = -(-n // mb)
    with bp.Net(small, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
        net.set_weights(theta)
        sse_ref = torch.zeros(steps, device="cuda")
        net.train_epoch(Xd, Td, n, mb, sse_ref)
        net.check()
        w_ref, v_ref = net.get_weights(), net.get_velocity()
    th = torch.tensor(theta, dtype=torch.float32, device="cuda")
    V = torch.zeros_like(th)
    sse = torch.zeros(steps, device="cuda")
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    bp.bp_train_epoch_noalloc(small, 0.05, 0.9, 1.0, th, V, Xd, Td, n, mb, sse, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    offs, _ = synth.param_layout(small)
    w, v = th.cpu().numpy().astype(np.float64), V.cpu().numpy().astype(np.float64)
    for l, (wo, bo) in enumerate(offs, start=1):
        for a, b in ((wo, wo + small[l] * small[l - 1]), (bo, bo + small[l])):
            assert normwise(v[a:b], v_ref[a:b]) <= TOL, l
            assert normwise(w[a:b] - theta[a:b], w_ref[a:b] - theta[a:b]) <= TOL, l
    np.testing.assert_allclose(sse.cpu().numpy(), sse_ref.cpu().numpy(), rtol=TOL)
