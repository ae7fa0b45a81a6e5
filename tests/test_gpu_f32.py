"""float32 CUDA path against the float64 oracle, through the C ABI.

Tolerance (fp32 SIMT path): normwise relative error
    max|x_gpu - x_ref| / max|x_ref| <= 1e-5
per layer, separately for each W_l and b_l (tests/parity.py), on outputs,
pooled changes, error sums, weight changes and momentum terms; elementwise
relative error is ill-posed where a sigmoid saturates.  For pooled changes
whose sums cancel, the bar applies to the magnitude of the sum's terms
(1e-5 times the layer's cancellation factor kappa >= 1, parity.kappa).

Multi-update runs are held to the bar at every update: runs of a few large
groups are compared at their end state (their rounding does not compound
measurably), and the long per-pattern and small-group trajectories step by
step -- each update from the GPU's own previous state against the oracle's
update from that state -- together with a check that one launch over the whole
epoch gives the same bits as one launch per group.  Inputs are seeded and
synthetic (NETtalk-shaped or Gaussian).
"""
import numpy as np
import pytest

from oracle import bp_oracle as O
from paper_1801_01554_gb300 import bp, synth
from parity import assert_layers, kappa, layer_errors, layer_parts, normwise

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-5


def dev(a):
    return torch.tensor(np.asarray(a), dtype=torch.float32, device="cuda")


def problem(sizes, B, seed=0, lo=-0.3, hi=0.3):
    if sizes[0] == 203 and sizes[-1] == 26:
        X, T = synth.nettalk_patterns(B, seed=seed)
    else:
        X, T = synth.gaussian_patterns(B, sizes[0], sizes[-1], 0.3, seed=seed)
        X = synth.round_to(X, "f32")
    theta = synth.round_to(synth.init_uniform(sizes, lo, hi, seed), "f32")
    return X, T, theta


U32 = 2.0 ** -24   # float32 unit roundoff


def check_state(sizes, theta0, W, V, st, kap, what, n_upd=1):
    """End state of a run of n_upd updates against the oracle's: W - W0 and V
    per layer.  W - W0 carries the rounding of the stored float32 weights after
    every update (half an ulp of |W| each), which sets its floor when the
    change is small next to the weights.  The floor of the reference's size is
    the one normwise() divides by, so that a part whose reference change is
    exactly zero gets the absolute bar n_upd * u * max|W| (in float64)."""
    kap = kap or [1.0] * (2 * (len(sizes) - 1))
    floor = []
    for k, (lab, sl) in zip(kap, layer_parts(sizes)):
        dref = max(float(np.max(np.abs(st.theta[sl] - theta0[sl]))), 1e-30)
        floor.append(k + n_upd * U32 * float(np.max(np.abs(st.theta[sl]))) / (TOL * dref))
    e = assert_layers(sizes, W - theta0, st.theta - theta0, TOL, floor, what + " W-W0")
    assert_layers(sizes, V, st.V, TOL, kap, what + " V")
    return e


def change_bar(sizes, kap, V_k, dv_ref):
    """Bar factors for a step's change lr*G read back as V_k - m*V_prev: the
    stored float32 V_k rounds it (two roundings of |V_k|), which dominates when
    the momentum term is much larger than the change (a net whose changes have
    died out in saturation).  A part whose reference change is exactly zero (a
    saturated layer) gets the absolute bar 2 u max|V_k|: the floor of the
    reference's size is the one normwise() divides by, and the arithmetic is
    float64 (a float32 quotient would round the bar to infinity)."""
    out = []
    for k, (lab, sl) in zip(kap, layer_parts(sizes)):
        dref = max(float(np.max(np.abs(dv_ref[sl]))), 1e-30)
        out.append(k + 2 * U32 * float(np.max(np.abs(V_k[sl]))) / (TOL * dref))
    return out


def stepwise(sizes, X, T, theta, V0, mb, lr, m, squash="logistic", kap_every=1, epochs=1):
    """`epochs` epochs as one launch each (as the benchmark launches them),
    then as one launch per group: every update of the second run is compared
    with the oracle's update from the GPU's own previous state, and the two
    runs must give the same bits.  Returns (GPU weights, GPU velocity) at the end."""
    n = len(X)
    steps = -(-n // mb)
    Xd, Td = dev(X), dev(T)
    with bp.Net(sizes, lr, m, bp.BP_F32, max_batch=mb) as a:
        a.set_weights(theta)
        a.set_velocity(V0)
        if squash == "table":
            a.set_sigmoid(bp.BP_SIGMOID_TABLE)
        sse_a = torch.zeros(epochs * steps, device="cuda")
        for ep in range(epochs):
            a.train_epoch(Xd, Td, n, mb, sse_a[ep * steps:(ep + 1) * steps])
        a.check()
        W_a, V_a, e_a = a.get_weights(), a.get_velocity(), sse_a.cpu().numpy()
    worst = {}
    with bp.Net(sizes, lr, m, bp.BP_F32, max_batch=mb) as b:
        b.set_weights(theta)
        b.set_velocity(V0)
        if squash == "table":
            b.set_sigmoid(bp.BP_SIGMOID_TABLE)
        W_prev = theta.astype(np.float32)
        V_prev = np.asarray(V0, dtype=np.float32)
        e_b = np.zeros(epochs * steps, dtype=np.float32)
        kap = None
        for k in range(epochs * steps):
            p0 = (k % steps) * mb
            nb = min(mb, n - p0)
            sse = torch.zeros(1, device="cuda")
            b.train_epoch(Xd[p0:p0 + nb], Td[p0:p0 + nb], nb, mb, sse)
            b.check()
            W_k, V_k = b.get_weights(), b.get_velocity()
            e_b[k] = sse.item()
            st = O.State(sizes, W_prev, lr=lr, momentum=m, V=V_prev.astype(np.float64), squash=squash)
            e_ref = O.train_batch(st, X[p0:p0 + nb], T[p0:p0 + nb])
            assert abs(e_b[k] - e_ref) <= TOL * e_ref, (k, e_b[k], e_ref)
            if kap is None or k % kap_every == 0:
                kap = kappa(sizes, W_prev, X[p0:p0 + nb], T[p0:p0 + nb], squash)
            # the update of this step: V_k = lr*G + m*V_prev, W_k = W_prev + V_k
            dv_gpu = V_k.astype(np.float64) - m * V_prev.astype(np.float64)
            dv_ref = st.V - m * V_prev.astype(np.float64)
            dv = assert_layers(sizes, dv_gpu, dv_ref, TOL, change_bar(sizes, kap, V_k, dv_ref),
                               f"step {k} lr*G")
            assert_layers(sizes, W_k, st.theta, TOL, None, f"step {k} W")
            for lab, e in dv.items():
                worst[lab] = max(worst.get(lab, 0.0), e)
            W_prev, V_prev = W_k, V_k
    np.testing.assert_array_equal(W_prev, W_a)
    np.testing.assert_array_equal(V_prev, V_a)
    np.testing.assert_array_equal(e_b, e_a)
    print("worst per-step lr*G error per part:", {k: f"{v:.2e}" for k, v in worst.items()})
    return W_a, V_a


SHAPES = [((203, 60, 26), 1), ((203, 60, 26), 37), ((203, 60, 26), 1024),
          ((203, 120, 26), 512), ((203, 120, 26), 1000), ((5, 3, 2), 7),
          ((64, 33, 17, 9), 300), ((40, 300, 200, 1), 257)]


@pytest.mark.parametrize("sizes,B", SHAPES)
def test_forward_backward_update_match_oracle(sizes, B):
    X, T, theta = problem(sizes, B, seed=B)
    st = O.State(sizes, theta, lr=0.1, momentum=0.9)
    As, Ds, G_ref, e_ref = O.step_quantities(st, X, T)
    kap = kappa(sizes, theta, X, T)
    Xd, Td = dev(X), dev(T)
    Yd = torch.empty((B, sizes[-1]), device="cuda")
    sse = torch.zeros(1, device="cuda")
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        net.forward(Xd, B, Yd)
        net.backward(Td, B, sse)
        net.check()
        G = net.get_grads()
        assert normwise(Yd.cpu().numpy(), As[-1]) <= TOL
        assert_layers(sizes, G, G_ref, TOL, kap, "G")
        assert abs(sse.item() - e_ref) <= TOL * e_ref
        net.update()
        net.check()
        st.G = G_ref
        O.apply_update(st)
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, kap, "update")
        assert not net.get_grads().any()          # the update zeroes G


@pytest.mark.parametrize("sizes,B", [((203, 60, 26), 1024), ((203, 120, 26), 512),
                                     ((203, 120, 26), 77), ((64, 33, 17, 9), 300)])
def test_train_batch_matches_oracle(sizes, B):
    X, T, theta = problem(sizes, B, seed=3)
    st = O.State(sizes, theta, lr=0.05, momentum=0.9)
    kap = kappa(sizes, theta, X, T)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        sse = torch.zeros(3, device="cuda")
        for k in range(3):
            net.train_batch(dev(X), dev(T), B, sse[k:k + 1])
        net.check()
        e_ref = [O.train_batch(st, X, T) for _ in range(3)]
        np.testing.assert_allclose(sse.cpu().numpy(), e_ref, rtol=TOL)
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, kap, "3 updates", 3)


@pytest.mark.parametrize("B,lr", [(200, 0.1), (12288, 0.01)])
def test_pending_change_is_folded_into_train_batch(B, lr):
    """bp_backward's pending G is added into the next training update; at
    B = 12,288 (24 chunks) the update runs in the balanced weight phase."""
    sizes = (203, 60, 26)
    X, T, theta = problem(sizes, B, seed=4)
    X2, T2, _ = problem(sizes, B, seed=5)
    kap = [max(a, b) for a, b in zip(kappa(sizes, theta, X, T), kappa(sizes, theta, X2, T2))]
    st = O.State(sizes, theta, lr=lr, momentum=0.5)
    with bp.Net(sizes, lr, 0.5, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        Xd = dev(X)                      # must outlive the matching bp_backward
        net.forward(Xd, B)
        net.backward(dev(T), B)
        net.train_batch(dev(X2), dev(T2), B)
        net.check()
        O.backward_accumulate(st, X, T)
        O.train_batch(st, X2, T2)
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, kap, "folded")
        assert not net.get_grads().any()


def test_backward_accumulates_across_groups():
    sizes, B = (203, 60, 26), 100
    X, T, theta = problem(sizes, B, seed=6)
    st = O.State(sizes, theta, lr=0.1, momentum=0.9)
    G_ref = O.step_quantities(st, X, T)[2]
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        Xd, Td = dev(X), dev(T)
        for _ in range(2):
            net.forward(Xd, B)
            net.backward(Td, B)
        net.check()
        assert_layers(sizes, net.get_grads(), 2 * G_ref, TOL, kappa(sizes, theta, X, T), "2G")


@pytest.mark.parametrize("n,mb", [(4096, 512), (1000, 300)])
def test_train_epoch_matches_oracle(n, mb):
    """A few large groups in one persistent launch, compared at the end state."""
    sizes = (203, 120, 26)
    X, T, theta = problem(sizes, n, seed=7)
    st = O.State(sizes, theta, lr=0.05, momentum=0.9)
    e_ref = O.train_epoch(st, X, T, mb)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
        net.set_weights(theta)
        sse = torch.zeros(len(e_ref), device="cuda")
        net.train_epoch(dev(X), dev(T), n, mb, sse)
        net.check()
        np.testing.assert_allclose(sse.cpu().numpy(), e_ref, rtol=TOL)
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, None, "epoch",
                    len(e_ref))


def test_weights_beyond_shared_memory_at_large_groups_step_by_step():
    """203-512-26 in groups of 4,096: 460 KB of padded weights do not fit in
    shared memory, so the pattern passes (of 8: passes of 32 need the weights
    in shared memory) read them from global memory, and its 516 weight tiles
    are more than the CTAs (each CTA takes several in turn)."""
    sizes = (203, 512, 26)
    X, T, theta = problem(sizes, 8192, seed=81, lo=-0.3, hi=0.3)
    stepwise(sizes, X, T, theta, np.zeros_like(theta), 4096, 0.01, 0.9)


# Groups of at least 24 chunks of 512 patterns, on nets with fewer weight tiles
# than SMs, run the balanced weight phase: each CTA takes an equal run of the
# tiles' chunk sequence and the pieces are added in CTA order after a grid
# barrier.  Cases: two balanced groups then a ragged one of 12 chunks in the
# same launch; a 2-tile net (fewer chunks than CTAs, so some runs are empty);
# exactly 24 chunks.
@pytest.mark.parametrize("sizes,n,mb", [((203, 120, 26), 30000, 12288), ((20, 8, 3), 25500, 12500),
                                        ((203, 60, 26), 24576, 12288)])
def test_balanced_weight_phase_matches_oracle_step_by_step(sizes, n, mb):
    X, T, theta = problem(sizes, n, seed=71)
    stepwise(sizes, X, T, theta, np.zeros_like(theta), mb, 0.02, 0.9)


@pytest.mark.parametrize("sizes,n,mb,lr", [((203, 120, 26), 777, 1, 0.05), ((203, 120, 26), 300, 1, 0.05),
                                            ((203, 120, 26), 301, 2, 0.05), ((203, 60, 26), 259, 3, 0.05),
                                            ((203, 60, 26), 256, 4, 0.05), ((5, 3, 2), 50, 1, 0.05),
                                            ((64, 33, 17, 9), 130, 4, 0.05),
                                            ((40, 300, 200, 1), 64, 2, 0.02)])
def test_small_group_epoch_matches_oracle_step_by_step(sizes, n, mb, lr):
    """Groups of 1-4 patterns (the per-pattern update of Section 3 at mb = 1),
    ragged last groups, a deep net, and a net too large for one CTA: every
    update against the oracle's from the same state, and the one-launch epoch
    bit for bit against the launch-per-group run.  (The single-output net runs
    at lr 0.02: at 0.05 its output comes within 6e-6 of 1, where float32 holds
    1 - o, and so the whole step's change, to about 1% only.)"""
    X, T, theta = problem(sizes, n, seed=21)
    V0 = synth.round_to(np.random.default_rng(3).uniform(-1e-3, 1e-3, theta.size), "f32")
    stepwise(sizes, X, T, theta, V0, mb, lr, 0.9)


def test_one_launch_epoch_is_reproducible():
    sizes, n, mb = (203, 120, 26), 301, 2
    X, T, theta = problem(sizes, n, seed=22)
    runs = []
    for _ in range(2):
        with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
            net.set_weights(theta)
            sse = torch.zeros(-(-n // mb), device="cuda")
            net.train_epoch(dev(X), dev(T), n, mb, sse)
            net.check()
            runs.append((net.get_weights(), sse.cpu().numpy()))
    assert np.array_equal(runs[0][0], runs[1][0]) and np.array_equal(runs[0][1], runs[1][1])


@pytest.mark.parametrize("sizes,n,mb", [((203, 120, 26), 1024, 512), ((64, 33, 17, 9), 257, 256),
                                        ((203, 120, 26), 8192, 4096)])   # passes of 32
def test_table_sigmoid_matches_oracle(sizes, n, mb):
    """The table-lookup logistic of Section 4.3 on the persistent kernel: the
    outputs of a forward pass and an epoch of updates against the oracle's
    table mode; the mode is per net and switches back to the logistic."""
    X, T, theta = problem(sizes, n, seed=31, lo=-1.0, hi=1.0)
    st = O.State(sizes, theta, lr=0.05, momentum=0.9, squash="table")
    Y_ref = O.predict(st, X)
    kap = kappa(sizes, theta, X[:mb], T[:mb], "table")
    e_ref = O.train_epoch(st, X, T, mb)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=max(mb, n)) as net:
        net.set_weights(theta)
        net.set_sigmoid(bp.BP_SIGMOID_TABLE)
        Y = torch.zeros(n, sizes[-1], device="cuda")
        Xd, Td = dev(X), dev(T)
        net.forward(Xd, n, Y)
        net.check()
        assert normwise(Y.cpu().numpy(), Y_ref) <= TOL
        sse = torch.zeros(len(e_ref), device="cuda")
        net.train_epoch(Xd, Td, n, mb, sse)
        net.check()
        np.testing.assert_allclose(sse.cpu().numpy(), e_ref, rtol=TOL)
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, kap, "table epoch",
                    n_upd=len(e_ref))
        # back to the logistic: outputs follow the exact logistic again (the
        # oracle's forward pass with the GPU's weights)
        net.set_sigmoid(bp.BP_SIGMOID_LOGISTIC)
        net.forward(Xd, n, Y)
        net.check()
        exact = O.State(sizes, net.get_weights(), lr=0.05, momentum=0.9)
        assert normwise(Y.cpu().numpy(), O.predict(exact, X)) <= TOL


@pytest.mark.parametrize("sizes,n,mb", [((203, 60, 26), 300, 1), ((203, 60, 26), 301, 4)])
def test_table_sigmoid_on_small_groups_step_by_step(sizes, n, mb):
    """The table-lookup logistic on the one-CTA kernel, update by update."""
    X, T, theta = problem(sizes, n, seed=31, lo=-1.0, hi=1.0)
    stepwise(sizes, X, T, theta, np.zeros_like(theta), mb, 0.05, 0.9, squash="table")

def test_table_sigmoid_mode_errors():
    with bp.Net((4, 3, 2), 0.1, 0.9, bp.BP_F32, max_batch=8) as net:
        with pytest.raises(bp.BPError) as e:
            net.set_sigmoid(7)
        assert e.value.status == bp.BP_EINVAL
    with bp.Net((256, 128, 64), 0.1, 0.9, bp.BP_BF16, max_batch=128) as net:
        with pytest.raises(bp.BPError) as e:
            net.set_sigmoid(bp.BP_SIGMOID_TABLE)
        assert e.value.status == bp.BP_EINVAL


def _gap_threshold(G):
    """A guard threshold between two consecutive |G| values near the median,
    far (relative to fp32 rounding) from both, so that both sides zero the same
    changes."""
    a = np.sort(np.abs(G[G != 0]))
    mid = len(a) // 2
    for k in range(mid, len(a) - 1):
        if a[k + 1] > a[k] * (1 + 1e-3):
            return 0.5 * (a[k] + a[k + 1])
    raise AssertionError("no gap")


@pytest.mark.parametrize("B", [512, 2, 16384])
def test_fault_guard_matches_oracle(B):
    """Section 8's guard on the persistent (B = 512), one-CTA (B = 2) and
    balanced (B = 16,384) weight phases: the same changes are zeroed and
    counted, the other weights update as usual."""
    sizes = (203, 120, 26)
    X, T, theta = problem(sizes, B, seed=41)
    probe = O.State(sizes, theta, lr=0.05, momentum=0.9)
    O.backward_accumulate(probe, X, T)
    guard = _gap_threshold(probe.G)
    st = O.State(sizes, theta, lr=0.05, momentum=0.9, guard=guard)
    O.train_batch(st, X, T)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        net.set_guard(guard)
        net.train_batch(dev(X), dev(T), B)
        net.check()
        assert net.get_faults(reset=True) == st.faults > 0
        assert net.get_faults() == 0
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, None, "guarded")


def test_fault_guard_on_backward_then_update_and_off_by_default():
    sizes, B = (64, 33, 17, 9), 300
    X, T, theta = problem(sizes, B, seed=42)
    probe = O.State(sizes, theta, lr=0.1, momentum=0.9)
    O.backward_accumulate(probe, X, T)
    guard = _gap_threshold(probe.G)
    st = O.State(sizes, theta, lr=0.1, momentum=0.9, guard=guard)
    O.backward_accumulate(st, X, T)
    O.apply_update(st)
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        Xd, Td = dev(X), dev(T)
        net.forward(Xd, B)
        net.backward(Td, B)
        net.set_guard(guard)
        net.update()
        net.check()
        assert net.get_faults() == st.faults > 0
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st,
                    kappa(sizes, theta, X, T), "guarded")
        # off again: a step zeroes nothing
        net.set_guard(0.0)
        net.get_faults(reset=True)
        net.train_batch(Xd, Td, B)
        net.check()
        assert net.get_faults() == 0
        with pytest.raises(bp.BPError):
            net.set_guard(-1.0)


@pytest.mark.parametrize("sizes,B", [((203, 120, 26), 64), ((64, 33, 17, 9), 37)])
def test_diagnostic_mode_every_sm_agrees(sizes, B):
    """Section 8's diagnostic mode: every CTA (one per SM) computes the error of
    the same patterns alone; on a healthy GPU they agree bit for bit, with the
    oracle's error sum, and the weights are left alone."""
    X, T, theta = problem(sizes, B, seed=51)
    st = O.State(sizes, theta, lr=0.05, momentum=0.9)
    e_ref = O.sse(O.predict(st, X), T)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        sse, sm, agree = net.diagnose(dev(X), dev(T), B)
        n_sm = torch.cuda.get_device_properties(0).multi_processor_count
        assert len(sse) == n_sm and agree == n_sm
        assert np.all(sse == sse[0]) and abs(float(sse[0]) - e_ref) <= TOL * e_ref
        assert np.all((sm >= 0) & (sm < n_sm))
        np.testing.assert_array_equal(net.get_weights(), theta.astype(np.float32))


@pytest.mark.parametrize("mb", [33, 2])
def test_deepest_net_the_boundary_allows(mb):
    """BP_MAX_SIZES layer sizes (8 weight layers) of odd widths, on the
    persistent kernel (groups of 33) and the one-CTA kernel (groups of 2)."""
    sizes = (7, 9, 5, 11, 6, 8, 4, 10, 3)
    assert len(sizes) == bp.BP_MAX_SIZES
    n = 66
    X, T, theta = problem(sizes, n, seed=61, lo=-1.0, hi=1.0)
    # the first layers' changes are small sums of cancelling terms (kappa up
    # to a few hundred), which the bar takes into account step by step
    stepwise(sizes, X, T, theta, np.zeros_like(theta), mb, 0.3, 0.9)


@pytest.mark.parametrize("B", synth.SWEEP_BATCHES)
def test_batch_sweep_step_matches_oracle(B):
    sizes = (203, 120, 26)
    X, T, theta = problem(sizes, B, seed=11)
    V0 = synth.round_to(np.random.default_rng(2).uniform(-1e-3, 1e-3, theta.size), "f32")
    st = O.State(sizes, theta, lr=0.05, momentum=0.9, V=V0.copy())
    e_ref = O.train_batch(st, X, T)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        net.set_velocity(V0)
        sse = torch.zeros(1, device="cuda")
        net.train_batch(dev(X), dev(T), B, sse)
        net.check()
        assert abs(sse.item() - e_ref) <= TOL * e_ref
        kap = kappa(sizes, theta, X, T)
        W, V = net.get_weights(), net.get_velocity()
        # the step's change lr*G, read back as V - m*V0 in float64
        dv_ref = st.V - 0.9 * V0
        assert_layers(sizes, V.astype(np.float64) - 0.9 * V0, dv_ref, TOL,
                      change_bar(sizes, kap, V, dv_ref), "lr*G")
        assert_layers(sizes, W, st.theta, TOL, None, "W")


def test_mean_scaling():
    sizes, B = (203, 60, 26), 256
    X, T, theta = problem(sizes, B, seed=12)
    st = O.State(sizes, theta, lr=0.1, momentum=0.9, grad_scale=1.0 / B)
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=B, grad_scale=1.0 / B) as net:
        net.set_weights(theta)
        for _ in range(2):
            net.train_batch(dev(X), dev(T), B)
            O.train_batch(st, X, T)
        net.check()
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st,
                    kappa(sizes, theta, X, T), "mean", 2)


def test_zero_learning_rate_keeps_weights_bitwise():
    sizes, B = (203, 60, 26), 64
    X, T, theta = problem(sizes, B, seed=13)
    with bp.Net(sizes, 0.0, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(theta)
        net.train_epoch(dev(X), dev(T), B, 16)
        net.check()
        np.testing.assert_array_equal(net.get_weights(), theta.astype(np.float32))


def test_runs_are_bitwise_reproducible():
    sizes, n, mb = (203, 120, 26), 2048, 512
    X, T, theta = problem(sizes, n, seed=14)
    out = []
    for _ in range(2):
        with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as net:
            net.set_weights(theta)
            net.train_epoch(dev(X), dev(T), n, mb)
            net.check()
            out.append(net.get_weights())
    np.testing.assert_array_equal(out[0], out[1])


def test_pooled_change_is_order_independent_on_gpu():
    # Section 4.1: patterns may be presented in any order
    sizes, B = (203, 120, 26), 512
    X, T, theta = problem(sizes, B, seed=15)
    perm = np.random.default_rng(0).permutation(B)
    Gs = []
    for Xp, Tp in ((X, T), (X[perm], T[perm])):
        with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=B) as net:
            net.set_weights(theta)
            Xd = dev(Xp)
            net.forward(Xd, B)
            net.backward(dev(Tp), B)
            Gs.append(net.get_grads())
    assert_layers(sizes, Gs[1], Gs[0], TOL, kappa(sizes, theta, X, T), "permuted G")


def test_checkpoint_resume_is_exact():
    sizes, n, mb = (203, 60, 26), 1024, 256
    X, T, theta = problem(sizes, n, seed=16)
    Xd, Td = dev(X), dev(T)
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=mb) as a:
        a.set_weights(theta)
        a.train_epoch(Xd, Td, n, mb)
        w, v = a.get_weights(), a.get_velocity()
        a.train_epoch(Xd, Td, n, mb)
        ref = a.get_weights()
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=mb) as b:
        b.set_weights(w)
        b.set_velocity(v)
        b.train_epoch(Xd, Td, n, mb)
        np.testing.assert_array_equal(b.get_weights(), ref)


@pytest.mark.parametrize("n,mb", [(3000, 512), (41, 2), (70000, 512)])
def test_host_buffer_epoch_equals_device_epoch(n, mb):
    """The host-buffer epoch runs in pieces whose copies overlap training: two
    epochs in a row give the same bits as two device-buffer epochs."""
    sizes = (203, 120, 26)
    X, T, theta = problem(sizes, n, seed=17)
    Xh = torch.tensor(X, dtype=torch.float32).pin_memory()
    Th = torch.tensor(T, dtype=torch.float32).pin_memory()
    ns = -(-n // mb)
    sse_h = np.zeros(ns, dtype=np.float32)
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as a:
        a.set_weights(theta)
        a.train_epoch_host(Xh, Th, n, mb, sse_h)
        a.train_epoch_host(Xh, Th, n, mb, sse_h)
        wa = a.get_weights()
    with bp.Net(sizes, 0.05, 0.9, bp.BP_F32, max_batch=mb) as b:
        b.set_weights(theta)
        sse_d = torch.zeros(ns, device="cuda")
        Xd, Td = dev(X), dev(T)
        b.train_epoch(Xd, Td, n, mb, sse_d)
        b.train_epoch(Xd, Td, n, mb, sse_d)
        np.testing.assert_array_equal(b.get_weights(), wa)
        np.testing.assert_array_equal(sse_d.cpu().numpy(), sse_h)


def test_argument_and_state_errors():
    sizes = (203, 60, 26)
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=16) as net:
        X = torch.zeros((32, 203), device="cuda")
        T = torch.zeros((32, 26), device="cuda")
        with pytest.raises(bp.BPError) as e:
            net.forward(X, 32)
        assert e.value.status == bp.BP_EINVAL
        with pytest.raises(bp.BPError) as e:
            net.backward(T, 8)
        assert e.value.status == bp.BP_ESTATE
        net.forward(X, 8)
        with pytest.raises(bp.BPError) as e:
            net.backward(T, 4)
        assert e.value.status == bp.BP_ESTATE
        with pytest.raises(bp.BPError) as e:
            net.train_epoch(X, T, 0, 8)
        assert e.value.status == bp.BP_EINVAL
        with pytest.raises(bp.BPError) as e:
            net.set_hparams(float("nan"), 0.9)
        assert e.value.status == bp.BP_EINVAL
        # float32 rows are read word by word: a buffer off a 4-byte boundary is refused
        with pytest.raises(bp.BPError) as e:
            net.train_batch(X.data_ptr() + 2, T, 8)
        assert e.value.status == bp.BP_EINVAL
        with pytest.raises(bp.BPError) as e:
            net.train_batch(X, T, 8, T.data_ptr() + 1)
        assert e.value.status == bp.BP_EINVAL
        net.check()


def test_nonfinite_error_sum_is_reported():
    sizes, B = (4, 3, 2), 8
    X = np.full((B, 4), np.nan)
    T = np.zeros((B, 2))
    with bp.Net(sizes, 0.1, 0.9, bp.BP_F32, max_batch=B) as net:
        net.set_weights(np.full(bp.connections(sizes), 0.1))
        net.train_batch(dev(X), dev(T), B)
        with pytest.raises(bp.BPError) as e:
            net.check()
        assert e.value.status == bp.BP_ENONFINITE
        net.check()    # the latch is cleared


def test_nettalk60_workload_full():
    """203-60-26, 1,024 patterns, full-batch updates, lr 0.1, momentum 0.9, 10 epochs."""
    sizes, X, T, theta = synth.make_workload("nettalk60")
    w = synth.WORKLOADS["nettalk60"]
    st = O.State(sizes, theta, lr=w["lr"], momentum=w["momentum"])
    n = len(X)
    with bp.Net(sizes, w["lr"], w["momentum"], bp.BP_F32, max_batch=n) as net:
        net.set_weights(theta)
        sse = torch.zeros(w["epochs"], device="cuda")
        Xd, Td = dev(X), dev(T)
        for ep in range(w["epochs"]):
            net.train_epoch(Xd, Td, n, w["minibatch"], sse[ep:ep + 1])
            e_ref = O.train_epoch(st, X, T, w["minibatch"])[0]
            # each epoch's error sum is compared on the trajectory so far
            assert abs(sse[ep].item() - e_ref) <= TOL * e_ref, ep
        net.check()
        check_state(sizes, theta, net.get_weights(), net.get_velocity(), st, None, "10 epochs", 10)


@pytest.mark.slow
def test_nettalk120_workload_full():
    """203-120-26, 65,536 patterns, minibatch 512, lr 0.05, momentum 0.9, 5 epochs,
    launched as the benchmark launches it (one persistent launch per epoch):
    all 640 updates step by step against the oracle from the GPU's own state,
    and the five benchmark launches bit for bit against the launch-per-group
    run.  The end state after 640 updates is printed against the oracle's own
    trajectory (each update's rounding compounds there)."""
    sizes, X, T, theta = synth.make_workload("nettalk120")
    w = synth.WORKLOADS["nettalk120"]
    mb = w["minibatch"]
    W, V = stepwise(sizes, X, T, theta, np.zeros_like(theta), mb, w["lr"], w["momentum"],
                    kap_every=32, epochs=w["epochs"])
    st = O.State(sizes, theta, lr=w["lr"], momentum=w["momentum"])
    for _ in range(w["epochs"]):
        O.train_epoch(st, X, T, mb)
    print("640-update trajectory, W-W0 per part:", layer_errors(sizes, W - theta, st.theta - theta),
          "V per part:", layer_errors(sizes, V, st.V))
