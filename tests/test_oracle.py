"""Pins for the CPU oracle: what the paper and the mathematics fix, not the
oracle's own code.  CPU only."""
import math
import os

import numpy as np
import pytest
from scipy.special import expit

from oracle import bp_oracle as O
from paper_1801_01554_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                k, *v = line.split()
                out[k] = [float(x) for x in v]
    return out


# ------------------------------------------------------------------ counting
def test_connection_count_matches_paper():
    g = _golden("nettalk_counts.txt")
    sizes = tuple(int(x) for x in g["sizes"])
    assert O.connections(sizes) == int(g["connections"][0])


def test_flop_factor_matches_paper():
    g = _golden("nettalk_counts.txt")
    sizes = tuple(int(x) for x in g["sizes"])
    f = O.flops_per_connection(sizes)
    assert round(f, 2) == g["flop_factor"][0]
    # 901 MCPS x 4.23 = 3.8 GFLOPS (Section 7.2)
    assert round(g["mcps"][0] * f / 1000.0, 1) == g["gflops"][0]
    # the per-pattern cycle counts of Section 6.1 give the same factor
    assert O.flops_per_pattern(sizes) == pytest.approx(f * O.connections(sizes), rel=1e-12)


# ------------------------------------------------------------------ sigmoid
def test_sigmoid_against_library_and_symmetry():
    x = np.linspace(-40, 40, 2001)
    np.testing.assert_allclose(O.sigmoid(x), expit(x), rtol=1e-14, atol=1e-300)
    assert O.sigmoid(0.0) == 0.5
    np.testing.assert_allclose(O.sigmoid(-x), 1.0 - O.sigmoid(x), atol=1e-15)


def test_sigmoid_derivative_identity():
    # sigma'(x) = sigma(x)(1 - sigma(x)), against central differences of sigma
    x = np.linspace(-8, 8, 161)
    h = 1e-5
    fd = (O.sigmoid(x + h) - O.sigmoid(x - h)) / (2 * h)
    s = O.sigmoid(x)
    np.testing.assert_allclose(s * (1 - s), fd, rtol=1e-7, atol=1e-10)


# ------------------------------------------------------------------ gradients
def _half_sse(sizes, theta, X, T):
    Ws, bs = O.unpack(sizes, theta)
    return 0.5 * O.sse(O.forward(Ws, bs, X)[-1], T)


def fd_relative_error(sizes, n_pat=5, seed=0, h=1e-6):
    """max |G + dE/dtheta| / max |dE/dtheta| over every weight and bias, with
    E = SSE/2 and dE/dtheta from central differences."""
    rng = np.random.default_rng(seed)
    theta = rng.uniform(-1.0, 1.0, O.connections(sizes))
    X = rng.standard_normal((n_pat, sizes[0]))
    T = (rng.random((n_pat, sizes[-1])) < 0.5).astype(float)
    st = O.State(sizes, theta, lr=0.0, momentum=0.0)
    _, _, G, _ = O.step_quantities(st, X, T)
    fd = np.empty_like(theta)
    for k in range(theta.size):
        tp = theta.copy(); tp[k] += h
        tm = theta.copy(); tm[k] -= h
        fd[k] = (_half_sse(sizes, tp, X, T) - _half_sse(sizes, tm, X, T)) / (2 * h)
    # G is the pooled delta*activation, i.e. minus the gradient of E/2
    return np.max(np.abs(G + fd)) / np.max(np.abs(fd))


@pytest.mark.parametrize("sizes", [(2, 3, 2), (4, 5, 3, 2), (3, 1), (3, 4, 4, 4, 2)])
def test_gradient_matches_finite_differences(sizes):
    assert fd_relative_error(sizes) < 1e-6


@pytest.mark.parametrize("mistake", ["sign", "no_derivative", "no_bias_grad", "transposed"])
def test_planted_mistakes_fail_the_finite_difference_pin(monkeypatch, mistake):
    """A plausible mistake anywhere in the backward pass must break the pin."""
    if mistake == "sign":
        monkeypatch.setattr(O, "output_delta", lambda Oo, T: (Oo - T) * Oo * (1 - Oo))
    elif mistake == "no_derivative":
        monkeypatch.setattr(O, "hidden_delta", lambda Wn, Dn, A: Dn @ Wn)
    elif mistake == "no_bias_grad":
        real = O.gradients
        monkeypatch.setattr(O, "gradients",
                            lambda As, Ds: (real(As, Ds)[0], [0 * D.sum(0) for D in Ds]))
    elif mistake == "transposed":
        # square hidden layers so that the transposed product still has the right shape
        monkeypatch.setattr(O, "hidden_delta", lambda Wn, Dn, A: (Dn @ Wn.T) * A * (1 - A))
    sizes = (3, 4, 4, 4) if mistake == "transposed" else (2, 3, 2)
    assert fd_relative_error(sizes) > 1e-2


def test_pooled_change_is_sum_of_single_pattern_changes():
    # Section 4.1: the pooled change is the sum of the per-pattern changes
    sizes = (7, 6, 3)
    X, T = synth.gaussian_patterns(9, 7, 3, 0.5, seed=3)
    st = O.State(sizes, synth.init_uniform(sizes, -0.5, 0.5, 3), 0.1, 0.9)
    _, _, G, e = O.step_quantities(st, X, T)
    parts = [O.step_quantities(st, X[p:p + 1], T[p:p + 1]) for p in range(9)]
    np.testing.assert_allclose(G, sum(q[2] for q in parts), rtol=1e-12, atol=1e-15)
    assert e == pytest.approx(sum(q[3] for q in parts), rel=1e-12)


def test_pooled_change_is_order_independent():
    # Section 4.1: changes may be applied in any order with the same result
    sizes = (7, 6, 3)
    X, T = synth.gaussian_patterns(33, 7, 3, 0.3, seed=4)
    st = O.State(sizes, synth.init_uniform(sizes, -0.5, 0.5, 4), 0.1, 0.9)
    perm = np.random.default_rng(1).permutation(33)
    G1 = O.step_quantities(st, X, T)[2]
    G2 = O.step_quantities(st, X[perm], T[perm])[2]
    np.testing.assert_allclose(G1, G2, rtol=1e-12, atol=1e-14)


def test_sse_is_plain_sum_of_squares():
    Oo = np.full((5, 4), 0.5)
    T = np.ones((5, 4))
    assert O.sse(Oo, T) == 5 * 4 * 0.25


# ------------------------------------------------------------------ update
def test_zero_learning_rate_leaves_weights_unchanged():
    sizes = (4, 3, 2)
    X, T = synth.gaussian_patterns(6, 4, 2, 0.5, seed=5)
    th = synth.init_uniform(sizes, -0.5, 0.5, 5)
    for m in (0.0, 0.9):
        st = O.State(sizes, th, lr=0.0, momentum=m)
        for _ in range(3):
            O.train_batch(st, X, T)
        np.testing.assert_array_equal(st.theta, th)
        assert not st.G.any()


def test_momentum_closed_form_under_constant_change():
    # with the same pooled change g every time, V_k = lr g (1 - m^k)/(1 - m)
    # and W_k = W_0 + lr g sum_{j=1..k} (1 - m^j)/(1 - m)
    rng = np.random.default_rng(7)
    w0 = rng.standard_normal(10)
    g = rng.standard_normal(10)
    lr, m = 0.3, 0.7
    w, v = w0.copy(), np.zeros(10)
    for k in range(1, 8):
        w, v = O.momentum_update(w, v, g, lr, m)
        np.testing.assert_allclose(v, lr * g * (1 - m ** k) / (1 - m), rtol=1e-13)
        geo = sum((1 - m ** j) / (1 - m) for j in range(1, k + 1))
        np.testing.assert_allclose(w, w0 + lr * g * geo, rtol=1e-12, atol=1e-13)


def test_one_weight_net_two_steps_by_hand():
    # 1-1 net: o = sigma(w x + b); delta = (t - o) o (1 - o);
    # G_w = delta x, G_b = delta; v <- lr G + m v; w <- w + v
    w, b, x, t, lr, m = 0.4, -0.2, 1.5, 1.0, 0.5, 0.9
    st = O.State((1, 1), np.array([w, b]), lr=lr, momentum=m)
    vw = vb = 0.0
    for _ in range(2):
        o = 1.0 / (1.0 + math.exp(-(w * x + b)))
        d = (t - o) * o * (1 - o)
        e = O.train_batch(st, np.array([[x]]), np.array([[t]]))
        assert e == pytest.approx((t - o) ** 2, rel=1e-14)
        vw, vb = lr * d * x + m * vw, lr * d + m * vb
        w, b = w + vw, b + vb
        np.testing.assert_allclose(st.theta, [w, b], rtol=1e-14)
        np.testing.assert_allclose(st.V, [vw, vb], rtol=1e-14)


def test_xor_converges():
    # a 2-2-1 net trained with pooled updates learns XOR
    X = np.array([[0, 0], [0, 1], [1, 0], [1, 1]], float)
    T = np.array([[0], [1], [1], [0]], float)
    st = O.State((2, 2, 1), synth.init_uniform((2, 2, 1), -1, 1, 2), lr=0.5, momentum=0.9)
    for _ in range(3000):
        e = O.train_batch(st, X, T)
    assert e < 0.04
    assert np.all(np.abs(O.predict(st, X) - T) < 0.2)


def test_mean_scaling_equals_scaled_learning_rate():
    sizes = (5, 4, 3)
    X, T = synth.gaussian_patterns(8, 5, 3, 0.5, seed=8)
    th = synth.init_uniform(sizes, -0.5, 0.5, 8)
    a = O.State(sizes, th, lr=0.2, momentum=0.5, grad_scale=1.0 / 8)
    b = O.State(sizes, th, lr=0.2 / 8, momentum=0.5)
    for _ in range(3):
        O.train_batch(a, X, T)
        O.train_batch(b, X, T)
    np.testing.assert_allclose(a.theta, b.theta, rtol=1e-12)


def test_epoch_takes_minibatches_in_index_order():
    sizes = (5, 4, 3)
    X, T = synth.gaussian_patterns(10, 5, 3, 0.5, seed=9)
    th = synth.init_uniform(sizes, -0.5, 0.5, 9)
    a = O.State(sizes, th, 0.1, 0.9)
    errs = O.train_epoch(a, X, T, minibatch=4)
    assert len(errs) == 3            # 4 + 4 + ragged 2
    b = O.State(sizes, th, 0.1, 0.9)
    for sl in (slice(0, 4), slice(4, 8), slice(8, 10)):
        O.train_batch(b, X[sl], T[sl])
    np.testing.assert_array_equal(a.theta, b.theta)
    c = O.State(sizes, th, 0.1, 0.9)
    assert O.train_epoch(c, X, T, minibatch=10)[0] == pytest.approx(
        O.sse(O.forward(*O.unpack(sizes, th), X)[-1], T))


def test_pack_unpack_round_trip():
    sizes = (3, 4, 2)
    th = np.arange(O.connections(sizes), dtype=float)
    Ws, bs = O.unpack(sizes, th)
    assert Ws[0].shape == (4, 3) and bs[0].shape == (4,)
    assert Ws[0][1, 0] == 3.0 and bs[0][0] == 12.0   # W_1 row-major, then b_1
    np.testing.assert_array_equal(O.pack(Ws, bs), th)


# ------------------------------------------------------------------ inputs
def test_nettalk_patterns_structure():
    X, T = synth.nettalk_patterns(257, seed=0)
    assert X.shape == (257, 203) and T.shape == (257, 26)
    blocks = X.reshape(257, 7, 29)
    assert np.all(blocks.sum(axis=2) == 1)
    assert np.all(T.sum(axis=1) == 3)
    assert set(np.unique(X)) <= {0.0, 1.0}


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(0).standard_normal(10000) * 10
    ref = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(synth.bf16_round(x), ref)


# ---------------------------------------------------------------- table sigmoid (Section 4.3)
def _table_nodes():
    # 256 points spread evenly over [-15, 15] (Section 4.3, Figure 3)
    return np.linspace(-15.0, 15.0, 256)


def test_sigmoid_table_is_exact_at_its_points():
    x = _table_nodes()
    np.testing.assert_allclose(O.sigmoid_table(x), expit(x), rtol=0, atol=1e-15)


def test_sigmoid_table_interpolates_linearly_between_points():
    x = _table_nodes()
    for k in (0, 17, 127, 128, 200, 254):
        for t in (0.25, 0.5, 0.9):
            xm = x[k] + t * (x[k + 1] - x[k])
            want = expit(x[k]) + t * (expit(x[k + 1]) - expit(x[k]))
            assert abs(O.sigmoid_table(xm) - want) <= 1e-13


def test_sigmoid_table_error_bound():
    # linear interpolation error <= h^2/8 max|s''| with h = 30/255 and
    # max|s''| = 1/(6 sqrt 3) (at s = 1/2 -/+ 1/(2 sqrt 3)); outside [-15, 15]
    # the error is at most s(-15).  The bound is nearly reached near the
    # inflections of s', so the grid's worst case sits just below it.
    h = 30.0 / 255.0
    bound = h * h / 8.0 / (6.0 * math.sqrt(3.0))
    x = np.linspace(-25.0, 25.0, 2_000_001)
    err = np.abs(O.sigmoid_table(x) - expit(x))
    assert err.max() <= bound
    assert err.max() >= 0.97 * bound
    assert 1.6e-4 < bound < 1.7e-4


def test_sigmoid_table_clamps_to_its_end_values():
    for x, end in ((40.0, 15.0), (-40.0, -15.0), (15.0, 15.0), (-15.0, -15.0)):
        assert O.sigmoid_table(x) == pytest.approx(expit(end), abs=1e-16)


def test_sigmoid_table_is_odd_about_one_half_and_monotone():
    x = np.random.default_rng(5).uniform(-20, 20, 10_000)
    np.testing.assert_allclose(O.sigmoid_table(-x) + O.sigmoid_table(x), 1.0, rtol=0, atol=1e-15)
    g = np.linspace(-16, 16, 100_001)
    assert np.all(np.diff(O.sigmoid_table(g)) >= 0)


def test_table_squash_changes_a_step_by_at_most_its_error():
    # one training step with the table logistic against the exact one: the
    # outputs differ by no more than the table's error bound propagated through
    # a 2-layer net of small weights (a loose, order-of-magnitude pin)
    sizes = (203, 60, 26)
    X, T = synth.nettalk_patterns(64, seed=3)
    theta = synth.init_uniform(sizes, -0.3, 0.3, 3)
    a = O.State(sizes, theta, lr=0.05, momentum=0.9)
    b = O.State(sizes, theta, lr=0.05, momentum=0.9, squash="table")
    ya, yb = O.predict(a, X), O.predict(b, X)
    assert 0 < np.abs(ya - yb).max() < 1e-3
    O.train_batch(a, X, T)
    O.train_batch(b, X, T)
    assert np.abs(a.theta - b.theta).max() < 1e-3


# ---------------------------------------------------------------- fault guard (Section 8)
def test_guard_zeroes_and_counts_out_of_range_changes():
    g = np.array([0.5, -3.0, 2.0, -1.0, np.nan, np.inf, 0.0])
    out, n = O.guard_changes(g, 1.0)
    np.testing.assert_array_equal(out, [0.5, 0.0, 0.0, -1.0, 0.0, 0.0, 0.0])
    assert n == 4
    same, n0 = O.guard_changes(g[:4], 0.0)          # off
    np.testing.assert_array_equal(same, g[:4])
    assert n0 == 0


def test_guarded_update_skips_only_the_zeroed_weights():
    sizes = (4, 3, 2)
    theta = np.linspace(-0.5, 0.5, O.connections(sizes))
    X = np.array([[1.0, 0.0, 1.0, 0.0], [0.0, 1.0, 0.0, 1.0]])
    T = np.array([[1.0, 0.0], [0.0, 1.0]])
    free = O.State(sizes, theta, lr=0.5, momentum=0.0)
    O.backward_accumulate(free, X, T)
    G = free.G.copy()
    guard = float(np.median(np.abs(G)))
    st = O.State(sizes, theta, lr=0.5, momentum=0.0, guard=guard)
    O.train_batch(st, X, T)
    big = np.abs(G) > guard
    assert st.faults == int(big.sum()) > 0
    np.testing.assert_array_equal(st.theta[big], theta[big])
    np.testing.assert_allclose(st.theta[~big], theta[~big] + 0.5 * G[~big], rtol=0, atol=1e-15)


def _trajectory_sensitivity(width, B, grad_scale):
    """Relative change, per part, of the oracle's 10-update weight change on a
    width^5 net (bf16 inputs, Bernoulli(0.5) targets, N(0, 1/fan_in) weights,
    lr 0.01, momentum 0.9) when the initial weights move by one bf16 rounding."""
    import sys
    sys.path.insert(0, os.path.dirname(__file__))
    from parity import layer_errors
    sizes = (width,) * 5
    X, T = synth.gaussian_patterns(B, width, width, 0.5, seed=5)
    X = synth.round_to(X, "bf16")
    theta = synth.round_to(synth.init_normal_fanin(sizes, 5), "f32")
    thp = theta * (1 + np.random.default_rng(7).uniform(-2.0 ** -9, 2.0 ** -9, theta.size))
    dws = []
    for th in (theta, thp):
        st = O.State(sizes, th, lr=0.01, momentum=0.9, grad_scale=grad_scale)
        for _ in range(10):
            O.train_batch(st, X, T)
        dws.append(st.theta - th)
    return layer_errors(sizes, dws[1], dws[0])


def test_wide_sum_mode_trajectory_is_ill_conditioned_and_mean_mode_is_not():
    """The reading behind the bf16 10-update parity runs: with the pooled sum,
    the first update of a wide net drives its units into saturation, and the
    exact 10-update weight change of the output layer then moves by more than
    50% when the initial weights move by one bf16 rounding (2^-9), so a
    bf16 path cannot be held to it; with the mean the same perturbation moves
    every layer's change by under 1%."""
    s = _trajectory_sensitivity(512, 1024, 1.0)
    assert s["W4"] > 0.5
    m = _trajectory_sensitivity(512, 1024, 1.0 / 1024)
    assert max(m.values()) < 1e-2


def test_case_parallel_driver_equals_the_serial_oracle():
    """Section 4.1's case parallelism: the changes of the workers' shares of
    each group, summed, give the serial oracle's update (up to the order of
    the float64 sums), ragged last group included."""
    from oracle.case_parallel import CaseParallel
    sizes, n, mb = (203, 30, 26), 700, 128
    X, T = synth.nettalk_patterns(n, seed=3)
    theta = synth.init_uniform(sizes, -0.3, 0.3, 3)
    a = O.State(sizes, theta, lr=0.05, momentum=0.9)
    e_ref = O.train_epoch(a, X, T, mb)
    b = O.State(sizes, theta, lr=0.05, momentum=0.9)
    with CaseParallel(sizes, X, T, workers=3) as cp:
        e = cp.train_epoch(b, n, mb)
    np.testing.assert_allclose(e, e_ref, rtol=1e-12)
    np.testing.assert_allclose(b.theta, a.theta, rtol=0, atol=1e-12)
    np.testing.assert_allclose(b.V, a.V, rtol=0, atol=1e-12)
