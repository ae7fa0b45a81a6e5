"""bfloat16 tensor-core path against the float64 oracle, through the C ABI.

Tolerance (bf16 tensor-core path): normwise relative error <= 2e-2 on outputs,
on the error sums, on the pooled change of a step and, per layer, on the weights
and on the weight change W10 - W0 after 10 updates (inputs, weight copies,
activations and deltas are each rounded to bfloat16, unit roundoff 2^-9, and
the products accumulate in fp32).  Errors are taken per layer, separately for
W_l and b_l (tests/parity.py).

The 10-update runs at the 4096-wide layers use the mean (grad_scale = 1/B):
with the pooled sum, the first update of a net that wide drives its units into
saturation, and the float64 oracle's own 10-update weight change then moves by
more than 100% under a perturbation of the size of one bf16 rounding (pinned on
the CPU by tests/test_oracle.py), so no rounded path can be held to it there.
The sum-mode step at those widths is held to the bar on its first update, at
B = 1024 and at the full batch.
"""
import numpy as np
import pytest

from oracle import bp_oracle as O
from paper_1801_01554_gb300 import bp, synth
from parity import assert_layers, normwise

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 2e-2


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


SHAPES = [((64, 128, 32), 200, 0.3), ((128, 256, 64), 300, 0.3), ((8, 16, 8), 8, 0.3),
          ((200, 136, 72, 24), 1000, 0.3), ((256, 512, 256), 128, 0.3),
          ((1024, 2048, 2048, 512), 1024, 0.1), ((4096,) * 5, 1024, 0.5)]


@pytest.mark.parametrize("sizes,B,p_one", SHAPES)
def test_forward_backward_update_match_oracle(sizes, B, p_one):
    """One step in sum mode: outputs, error sum, the pooled change of every
    layer, and the update it makes (W1 - W0 and V1 per layer)."""
    X, T, theta = problem(sizes, B, seed=B, p_one=p_one)
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
        net.update()
        net.check()
        W1, V1 = net.get_weights(), net.get_velocity()
    y = Yd.float().cpu().numpy()
    assert normwise(y, As[-1]) <= TOL
    assert abs(sse.item() - e_ref) <= TOL * e_ref
    assert_layers(sizes, G, G_ref, TOL, None, "G")
    st.G = G_ref
    O.apply_update(st)
    assert_layers(sizes, W1 - theta, st.theta - theta, TOL, None, "W1-W0")
    assert_layers(sizes, V1, st.V, TOL, None, "V1")


TEN = [((64, 128, 32), 256, 0.1, "sum"), ((200, 136, 72, 24), 520, 0.1, "sum"),
       ((1024, 2048, 2048, 512), 1024, 0.1, "sum"), ((1024, 2048, 2048, 512), 1024, 0.1, "mean"),
       ((4096,) * 5, 1024, 0.5, "mean")]


@pytest.mark.parametrize("sizes,B,p_one,mode", TEN)
def test_ten_updates_match_oracle(sizes, B, p_one, mode):
    """Ten updates on one group: the pooled change of the first step per layer,
    the weights and the weight change W10 - W0 per layer, and every update's
    error sum."""
    X, T, theta = problem(sizes, B, seed=5, p_one=p_one)
    lr, m = 0.01, 0.9
    gs = 1.0 if mode == "sum" else 1.0 / B
    st = O.State(sizes, theta, lr=lr, momentum=m, grad_scale=gs)
    G_ref = O.step_quantities(st, X, T)[2]
    Xd, Td = dev_bf16(X), dev_bf16(T)
    with bp.Net(sizes, lr, m, bp.BP_BF16, max_batch=B, grad_scale=gs) as net:
        net.set_weights(theta)
        net.forward(Xd, B)
        net.backward(Td, B)
        net.check()
        G1 = net.get_grads()
    with bp.Net(sizes, lr, m, bp.BP_BF16, max_batch=B, grad_scale=gs) as net:
        net.set_weights(theta)
        sse = torch.zeros(10, device="cuda")
        for k in range(10):
            net.train_batch(Xd, Td, B, sse[k:k + 1])
        net.check()
        th = net.get_weights()
    e_ref = [O.train_batch(st, X, T) for _ in range(10)]
    assert_layers(sizes, G1, G_ref, TOL, None, "G1")
    errs = assert_layers(sizes, th - theta, st.theta - theta, TOL, None, "W10-W0")
    print("W10-W0 per part:", {k: f"{v:.2e}" for k, v in errs.items()})
    assert_layers(sizes, th, st.theta, TOL, None, "W10")
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
    assert_layers(sizes, out[1] - theta, out[0] - theta, 1e-3, None, "separate vs fused")


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
    assert_layers(sizes, th - theta, st.theta - theta, TOL, None, "epoch W-W0")


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
def test_full_size_step_matches_oracle(name):
    """The benchmark's workload at its full batch, launched as bench.py times
    it (bp_train_batch on the whole group, sum mode): outputs of sampled
    patterns against the oracle's forward pass of those patterns, then one
    training step -- its error sum and the weight change of every layer --
    against the oracle's full step (6.6 TFLOP in float64 for 4096^5)."""
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
        sse = torch.zeros(1, device="cuda")
        net.train_batch(Xd, Td, B, sse)
        net.check()
        th = net.get_weights()
    del Xd, Td, Yd
    torch.cuda.empty_cache()
    st = O.State(sizes, theta, lr=w["lr"], momentum=w["momentum"])
    e_ref = O.train_batch(st, X, T)
    assert abs(sse.item() - e_ref) <= TOL * e_ref
    errs = assert_layers(sizes, th - theta, st.theta - theta, TOL, None, "W1-W0")
    print(name, "W1-W0 per part:", {k: f"{v:.2e}" for k, v in errs.items()})


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
        assert_layers(sizes, net.get_weights() - theta, st.theta - theta, TOL, None, "W-W0")


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
        assert_layers(sizes, net.get_weights() - theta, st.theta - theta, TOL, None, "W1-W0")


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
        assert_layers(sizes, net.get_weights() - theta, st.theta - theta, TOL, None, "W1-W0")
