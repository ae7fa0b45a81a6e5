"""The seeded input recipe (CPU): the structure and distributions the
generators promise, the bf16 rounding against torch's own, and determinism.

NETtalk-shaped inputs follow Section 6.3's encoding: 203 inputs as 7 letter
windows of 29 symbols (one symbol on per window) and 26 output features; the
targets carry exactly 3 ones.  The wide nets' inputs are N(0, 1) with
Bernoulli(p) targets, and their weights N(0, 1/fan_in) with zero biases."""
import numpy as np
import pytest

from paper_1801_01554_gb300 import synth


def test_nettalk_patterns_are_one_letter_per_window_and_three_hot_targets():
    X, T = synth.nettalk_patterns(5000, seed=7)
    assert X.shape == (5000, 203) and T.shape == (5000, 26)
    assert set(np.unique(X)) == {0.0, 1.0} and set(np.unique(T)) == {0.0, 1.0}
    blocks = X.reshape(5000, 7, 29)
    assert np.all(blocks.sum(axis=2) == 1)          # one letter in each window
    assert np.all(T.sum(axis=1) == 3)               # three distinct features on
    # letters and features uniform: every symbol of every window and every
    # feature occurs near its expected count (5000/29 and 5000*3/26)
    per_letter = blocks.sum(axis=0)
    assert per_letter.min() > 0.6 * 5000 / 29 and per_letter.max() < 1.4 * 5000 / 29
    per_feature = T.sum(axis=0)
    assert per_feature.min() > 0.8 * 5000 * 3 / 26 and per_feature.max() < 1.2 * 5000 * 3 / 26


def test_nettalk_patterns_reject_other_shapes():
    with pytest.raises(ValueError):
        synth.nettalk_patterns(4, n_in=200)


def test_gaussian_patterns_moments_and_target_rate():
    X, T = synth.gaussian_patterns(4000, 64, 32, 0.1, seed=3)
    assert abs(X.mean()) < 0.01 and abs(X.std() - 1.0) < 0.01
    assert set(np.unique(T)) <= {0.0, 1.0}
    assert abs(T.mean() - 0.1) < 0.005


def test_weight_initialisations():
    sizes = (203, 120, 26)
    offs, total = synth.param_layout(sizes)
    assert total == 204 * 120 + 121 * 26
    assert offs == [(0, 203 * 120), (203 * 120 + 120, 203 * 120 + 120 + 120 * 26)]
    th = synth.init_uniform(sizes, -0.3, 0.3, seed=1)
    assert th.shape == (total,) and th.min() >= -0.3 and th.max() < 0.3
    assert abs(th.mean()) < 0.01                     # biases drawn too: no block of zeros
    for _, b_off in offs:
        assert np.all(th[b_off:b_off + 1] != 0.0)
    wide = (512, 1024, 256)
    thn = synth.init_normal_fanin(wide, seed=2)
    offs, _ = synth.param_layout(wide)
    for l, (w_off, b_off) in enumerate(offs, start=1):
        w = thn[w_off:w_off + wide[l] * wide[l - 1]]
        assert abs(w.std() * np.sqrt(wide[l - 1]) - 1.0) < 0.02
        assert np.all(thn[b_off:b_off + wide[l]] == 0.0)


def test_bf16_round_matches_torch_round_to_nearest_even():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-8, 8, 20000),
                        [0.0, -0.0, 1.0, -2.5, 65504.0, 1e-38, 3.0e38]])
    # exact ties: float32 values whose low 16 bits are 0x8000, with even and odd kept halves
    ties = (np.array([0x3F808000, 0x3F818000, 0xBF808000, 0x40490000 | 0x8000], dtype=np.uint32)
            .view(np.float32).astype(np.float64))
    x = np.concatenate([x, ties])
    ours = synth.bf16_round(x)
    ref = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(ours, ref)


def test_generators_are_deterministic_per_seed():
    a = synth.nettalk_patterns(64, seed=5)
    b = synth.nettalk_patterns(64, seed=5)
    c = synth.nettalk_patterns(64, seed=6)
    assert all(np.array_equal(u, v) for u, v in zip(a, b))
    assert not np.array_equal(a[0], c[0])
    sizes = (16, 8, 4)
    assert np.array_equal(synth.init_uniform(sizes, -1, 1, 3), synth.init_uniform(sizes, -1, 1, 3))
    assert np.array_equal(synth.init_normal_fanin(sizes, 3), synth.init_normal_fanin(sizes, 3))
