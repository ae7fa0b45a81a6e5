"""bfloat16 tensor-core path against the float64 oracle, through the C ABI.

Tolerance (bf16 tensor-core path): normwise relative error <= 2e-2 on outputs
and on weights after 10 updates; the pooled change is held to the same 2e-2
(inputs, weight copies, activations and deltas are each rounded to bfloat16,
unit roundoff 2^-9, and the products accumulate in fp32).
"""
import numpy as np
import pytest

from oracle import bp_oracle as O
from paper_1801_01554_gb300 import bp, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 2e-2


def normwise(x, y):
    x = np.asarray(x, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    return float(np.max(np.abs(x - y)) / max(np.max(np.abs(y)), 1e-30))


def dev_bf16(a):
    return torch.tensor(np.asarray(a), dtype=torch.float32, device="cuda").to(torch.bfloat16)


def problem(sizes, B, seed=0, p_one=0.3):
    X, T = synth.gaussian_patterns(B, sizes[0], sizes[-1], p_one, seed=seed)
    X = synth.round_to(X, "bf16")
    theta = synth.round_to(synth.init_normal_fanin(sizes, seed), "f32")
    # small random biases so that the bias path is exercised from the first step
    off, _ = synth.param_layout(sizes)
    rng = np.random.default_rng(seed + 100)
    for (w_off, b_off), n in zip(off, sizes[1:]):
        theta[b_off:b_off + n] = synth.round_to(rng.uniform(-0.2, 0.2, n), "f32")
    return X, T, theta


SHAPES = [((64, 128, 32), 200), ((128, 256, 64), 300), ((8, 16, 8), 8), ((200, 136, 72, 24), 1000),
          ((256, 512, 256), 128), ((1024, 2048, 2048, 512), 1024)]


@pytest.mark.parametrize("sizes,B", SHAPES)
def test_forward_backward_match_oracle(sizes, B):
    X, T, theta = problem(sizes, B, seed=B)
    st = O.State(sizes, theta, lr=0.01, momentum=0.9)
    As, Ds, G_ref, e_ref = O.step_quantities(st, X, T)
    Xd, Td = dev_bf16(X), dev_bf16(T)
    Yd = torch.empty((B, sizes[-1]), dtype=torch.bfloat16, device="cuda")
    sse = torch.zeros(1, device="cuda")
    with bp.Net(sizes, 0.01, 0.9, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        net.forward(Xd, B, Yd)
        net.backward(Td, B, sse)
        net.check()
        G = net.get_grads()
    y = Yd.float().cpu().numpy()
    assert normwise(y, As[-1]) <= TOL
    assert abs(sse.item() - e_ref) <= TOL * e_ref
    offs, _ = synth.param_layout(sizes)
    for l, (w_off, b_off) in enumerate(offs, start=1):
        n_w = sizes[l] * sizes[l - 1]
        err_w = normwise(G[w_off:w_off + n_w], G_ref[w_off:w_off + n_w])
        err_b = normwise(G[b_off:b_off + sizes[l]], G_ref[b_off:b_off + sizes[l]])
        assert err_w <= TOL, (l, err_w)
        assert err_b <= TOL, (l, err_b)


@pytest.mark.parametrize("sizes,B", [((64, 128, 32), 256), ((200, 136, 72, 24), 520),
                                     ((1024, 2048, 2048, 512), 1024)])
def test_ten_updates_match_oracle(sizes, B):
    X, T, theta = problem(sizes, B, seed=5, p_one=0.1)
    lr, m = 0.01, 0.9
    st = O.State(sizes, theta, lr=lr, momentum=m)
    Xd, Td = dev_bf16(X), dev_bf16(T)
    with bp.Net(sizes, lr, m, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        sse = torch.zeros(10, device="cuda")
        for k in range(10):
            net.train_batch(Xd, Td, B, sse[k:k + 1])
        net.check()
        th = net.get_weights()
    e_ref = [O.train_batch(st, X, T) for _ in range(10)]
    print("W:", normwise(th, st.theta), "W10-W0:", normwise(th - theta, st.theta - theta))
    assert normwise(th, st.theta) <= TOL
    assert normwise(th - theta, st.theta - theta) <= 5 * TOL
    np.testing.assert_allclose(sse.cpu().numpy(), e_ref, rtol=TOL)


def test_separate_calls_equal_train_batch():
    sizes, B = (128, 256, 64), 256
    X, T, theta = problem(sizes, B, seed=7)
    Xd, Td = dev_bf16(X), dev_bf16(T)
    out = []
    for fused in (True, False):
        with bp.Net(sizes, 0.05, 0.9, bp.BP_BF16, max_batch=B) as net:
            net.set_weights(theta)
            for _ in range(3):
                if fused:
                    net.train_batch(Xd, Td, B)
                else:
                    net.forward(Xd, B)
                    net.backward(Td, B)
                    net.update()
            net.check()
            out.append(net.get_weights())
    assert normwise(out[1] - theta, out[0] - theta) <= 1e-3


def test_epoch_of_minibatches_matches_oracle():
    sizes, n, mb = (64, 128, 32), 1000, 256
    X, T, theta = problem(sizes, n, seed=8)
    st = O.State(sizes, theta, lr=0.01, momentum=0.9)
    e_ref = O.train_epoch(st, X, T, mb)
    with bp.Net(sizes, 0.01, 0.9, bp.BP_BF16, max_batch=mb) as net:
        net.set_weights(theta)
        sse = torch.zeros(len(e_ref), device="cuda")
        net.train_epoch(dev_bf16(X), dev_bf16(T), n, mb, sse)
        net.check()
        th = net.get_weights()
    np.testing.assert_allclose(sse.cpu().numpy(), e_ref, rtol=TOL)
    assert normwise(th - theta, st.theta - theta) <= 5 * TOL


def test_pooled_change_adds_over_groups():
    # Section 4.1: the change over a group is the sum of the changes of its parts
    sizes, B = (256, 512, 256), 512
    X, T, theta = problem(sizes, B, seed=9)
    Gs = []
    with bp.Net(sizes, 0.0, 0.0, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        for sl in (slice(0, B), slice(0, 256), slice(256, B)):
            Xs, Ts = dev_bf16(X[sl]), dev_bf16(T[sl])
            nb = sl.stop - sl.start
            net.forward(Xs, nb)
            net.backward(Ts, nb)
            Gs.append(net.get_grads())
            net.update()       # lr = 0, momentum = 0: only zeroes G
    assert normwise(Gs[1] + Gs[2], Gs[0]) <= 1e-5


def test_shape_rules():
    with pytest.raises(bp.BPError) as e:
        bp.Net((203, 120, 26), 0.1, 0.9, bp.BP_BF16, max_batch=64)
    assert e.value.status == bp.BP_ESHAPE
    with pytest.raises(bp.BPError) as e:
        bp.Net((64, 124, 32), 0.1, 0.9, bp.BP_BF16, max_batch=100)
    assert e.value.status == bp.BP_ESHAPE


def test_runs_are_bitwise_reproducible():
    sizes, B = (256, 512, 256), 384
    X, T, theta = problem(sizes, B, seed=10)
    Xd, Td = dev_bf16(X), dev_bf16(T)
    out = []
    for _ in range(2):
        with bp.Net(sizes, 0.01, 0.9, bp.BP_BF16, max_batch=B) as net:
            net.set_weights(theta)
            for _ in range(3):
                net.train_batch(Xd, Td, B)
            out.append(net.get_weights())
    np.testing.assert_array_equal(out[0], out[1])


@pytest.mark.slow
@pytest.mark.parametrize("name", ["wide3", "wide4096"])
def test_full_size_workload_sampled(name):
    """Full batch size, launched as the training step is: outputs of sampled
    patterns against the oracle's forward pass of those patterns; the error sum
    of the step against the sum over the path's own outputs."""
    sizes, X, T, theta = synth.make_workload(name)
    w = synth.WORKLOADS[name]
    B = w["minibatch"]
    Xd, Td = dev_bf16(X), dev_bf16(T)
    Yd = torch.empty((B, sizes[-1]), dtype=torch.bfloat16, device="cuda")
    rows = np.random.default_rng(0).choice(B, 16, replace=False)
    Ws, bs = O.unpack(sizes, theta)
    y_ref = O.forward(Ws, bs, X[rows])[-1]
    with bp.Net(sizes, w["lr"], w["momentum"], bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        net.forward(Xd, B, Yd)
        net.check()
        y = Yd.float().cpu().numpy()
        assert normwise(y[rows], y_ref) <= TOL
        sse = torch.zeros(2, device="cuda")
        net.train_batch(Xd, Td, B, sse[0:1])
        net.train_batch(Xd, Td, B, sse[1:2])
        net.check()
        th = net.get_weights()
    assert np.all(np.isfinite(th))
    assert np.any(th != theta.astype(np.float32))
    e_own = float(np.sum((T - y) ** 2))
    assert abs(sse[0].item() - e_own) <= 1e-3 * e_own


def test_fault_guard_zeroes_and_counts_on_the_bf16_update():
    """Section 8's guard on the bf16 update kernel: a threshold below every
    change zeroes them all (the weights keep their momentum-free values and
    every nonzero change is counted); a threshold above them all changes nothing."""
    sizes, B = (64, 128, 32), 256
    X, T, theta = problem(sizes, B, seed=7)
    Xd, Td = dev_bf16(X), dev_bf16(T)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        net.set_guard(1e-30)
        net.train_batch(Xd, Td, B)
        net.check()
        n = net.get_faults(reset=True)
        assert 0.99 * theta.size <= n <= theta.size
        np.testing.assert_array_equal(net.get_weights(), theta.astype(np.float32))
        net.set_guard(1e30)
        net.train_batch(Xd, Td, B)
        net.check()
        assert net.get_faults() == 0
        st = O.State(sizes, theta, lr=0.05, momentum=0.9)
        O.train_batch(st, X, T)
        assert normwise(net.get_weights() - theta, st.theta - theta) <= TOL


def test_deepest_net_the_boundary_allows():
    """BP_MAX_SIZES layer sizes (8 weight layers): outputs and one update's
    weight change, held to the same 2e-2 as every bf16 step."""
    sizes = (8, 16, 8, 24, 8, 16, 8, 16, 8)
    assert len(sizes) == bp.BP_MAX_SIZES
    B = 40
    X, T, theta = problem(sizes, B, seed=9)
    st = O.State(sizes, theta, lr=0.1, momentum=0.9)
    Y_ref = O.predict(st, X)
    O.train_batch(st, X, T)
    with bp.Net(sizes, 0.1, 0.9, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        Xd, Td = dev_bf16(X), dev_bf16(T)
        Y = torch.zeros(B, sizes[-1], dtype=torch.bfloat16, device="cuda")
        net.forward(Xd, B, Y)
        net.train_batch(Xd, Td, B)
        net.check()
        assert normwise(Y.float().cpu().numpy(), Y_ref) <= TOL
        assert normwise(net.get_weights() - theta, st.theta - theta) <= TOL


def test_misaligned_pattern_buffers_are_rejected_before_any_launch():
    """bf16 rows move in 16-byte pieces: X, T and Y must start on a 16-byte
    boundary.  A buffer offset by one element is refused with BP_EINVAL and
    the net stays usable."""
    sizes, B = (64, 128, 32), 64
    X, T, theta = problem(sizes, B, seed=3)
    Xd = dev_bf16(np.vstack([X, X[:1]])).flatten()
    Td = dev_bf16(np.vstack([T, T[:1]])).flatten()
    with bp.Net(sizes, 0.05, 0.9, bp.BP_BF16, max_batch=B) as net:
        net.set_weights(theta)
        for args in ((Xd[1:], Td[:B * sizes[-1]]), (Xd[:B * sizes[0]], Td[1:])):
            with pytest.raises(bp.BPError) as e:
                net.train_batch(args[0], args[1], B)
            assert e.value.status == bp.BP_EINVAL
        Y = torch.empty(B * sizes[-1] + 8, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(bp.BPError) as e:
            net.forward(Xd[:B * sizes[0]], B, Y[1:])
        assert e.value.status == bp.BP_EINVAL
        net.train_batch(Xd[:B * sizes[0]], Td[:B * sizes[-1]], B)
        net.check()
        st = O.State(sizes, theta, lr=0.05, momentum=0.9)
        O.train_batch(st, X, T)
        assert normwise(net.get_weights() - theta, st.theta - theta) <= TOL
