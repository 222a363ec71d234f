"""Pins of the oracle's storage helpers and of Eq. 3 (adaptive layer fusion)."""
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- bf16 rounding / decoding

def test_round_bf16_matches_torch_cast():
    rng = np.random.default_rng(1)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        [0.0, -0.0, 1.0, -3.5, 65504.0]]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x.astype(np.float64)), ref)


@pytest.mark.parametrize("x,y", [
    (1.0, 1.0),
    (1.0 + 2.0 ** -8, 1.0),                       # halfway between 1 and 1+2^-7: even wins
    (1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -6),       # halfway between 1+2^-7 (odd) and 1+2^-6
    (1.0 + 2.0 ** -8 + 2.0 ** -20, 1.0 + 2.0 ** -7),
    (-(1.0 + 2.0 ** -8), -1.0),
    (3.0, 3.0),
    (0.1, 0.10009765625),
])
def test_round_bf16_values(x, y):
    assert O.round_bf16(np.array([x]))[0] == y


def test_decode_bf16_bits():
    bits = np.array([0x3F80, 0xC000, 0x3F81, 0x0000, 0x8000, 0x4049], np.uint16)
    np.testing.assert_array_equal(O.decode(bits, "bf16"),
                                  [1.0, -2.0, 1.0 + 2.0 ** -7, 0.0, -0.0, 3.140625])
    np.testing.assert_array_equal(O.decode(np.float32([0.5, -2.25]), "f32"), [0.5, -2.25])


# ----------------------------------------------------------------- Eq. 3, first line

def test_fusion_weight_count_golden():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "fusion_param_count.txt"))
            if l.strip() and not l.startswith("#")]
    for D, T, n in ((int(a), int(b), int(c)) for a, b, c in rows):
        alpha = O.fusion_weights(np.zeros((D, T)))
        assert alpha.size == n


def test_fusion_weights_closed_forms():
    rng = np.random.default_rng(2)
    w = rng.standard_normal((5, 36))
    a = O.fusion_weights(w)
    assert np.all(a > 0)
    np.testing.assert_allclose(a.sum(axis=1), 1.0, rtol=0, atol=1e-15)
    # ratios are exp of logit differences
    np.testing.assert_allclose(a[:, 3] / a[:, 7], np.exp(w[:, 3] - w[:, 7]), rtol=1e-13)
    # shift invariance per row
    np.testing.assert_allclose(O.fusion_weights(w + rng.standard_normal((5, 1)) * 50), a,
                               rtol=1e-12)
    # equal logits: uniform 1/T
    np.testing.assert_allclose(O.fusion_weights(np.full((2, 9), 0.3)), 1 / 9, rtol=1e-15)
    # -Softmax ablation keeps the raw weights
    np.testing.assert_array_equal(O.fusion_weights(w, softmax=False), w)


def test_fusion_weights_match_torch_softmax():
    w = np.random.default_rng(3).standard_normal((8, 24))
    ref = torch.softmax(torch.from_numpy(w), dim=1).numpy()
    np.testing.assert_allclose(O.fusion_weights(w), ref, rtol=1e-13)


# ----------------------------------------------------------------- RMSNorm

def test_rms_norm_values():
    y = O.rms_norm(np.array([3.0, 4.0]), np.ones(2), 0.0)
    np.testing.assert_allclose(y, [0.848528137423857, 1.131370849898476], rtol=1e-14)
    y = O.rms_norm(np.array([[2.0, -2.0, 2.0, -2.0]]), np.array([1.0, 2.0, 3.0, 4.0]), 0.0)
    np.testing.assert_allclose(y, [[1.0, -2.0, 3.0, -4.0]], rtol=1e-15)
    # eps enters under the root: x = [1, 1], eps = 3 -> 1 / sqrt(1 + 3) = 0.5
    np.testing.assert_allclose(O.rms_norm(np.ones(2), np.ones(2), 3.0), [0.5, 0.5], rtol=1e-15)


def test_rms_norm_matches_torch():
    rng = np.random.default_rng(4)
    x, g = rng.standard_normal((7, 96)), rng.standard_normal(96)
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x), (96,), torch.from_numpy(g), eps=1e-6)
    np.testing.assert_allclose(O.rms_norm(x, g, 1e-6), ref.numpy(), rtol=1e-12)


def test_rms_norm_invariants():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((4, 64))
    y = O.rms_norm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=1), 1.0, rtol=1e-13)
    np.testing.assert_allclose(O.rms_norm(7.5 * x, np.ones(64), 0.0), y, rtol=1e-13)


# ----------------------------------------------------------------- Eq. 3, second line

def _hidden(T=6, n=5, d=32, seed=6):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((T, n, d)) * rng.uniform(0.5, 4, (T, 1, 1))


def test_fuse_one_hot_selects_one_layer():
    """alpha one-hot at layer j(i) reproduces RMSNorm(h^(j)) (a logit of -1e4 underflows)."""
    h = _hidden()
    D, T, d = 4, h.shape[0], h.shape[2]
    pick = [5, 0, 3, 1]
    w = np.full((D, T), -1e4)
    for i, j in enumerate(pick):
        w[i, j] = 0.0
    alpha = O.fusion_weights(w)
    assert np.all((alpha == 0) | (alpha == 1))
    g = np.random.default_rng(7).uniform(0.5, 1.5, (D, d))
    F = O.fuse_context(h, alpha, g, 1e-6)
    for i, j in enumerate(pick):
        np.testing.assert_allclose(F[i], O.rms_norm(h[j], g[i], 1e-6), rtol=1e-14)


def test_fuse_uniform_is_layer_mean():
    h = _hidden()
    T, d = h.shape[0], h.shape[2]
    alpha = O.fusion_weights(np.zeros((2, T)))
    F = O.fuse_context(h, alpha, np.ones((2, d)), 0.0)
    mean = h.mean(axis=0)
    np.testing.assert_allclose(F[0], O.rms_norm(mean, np.ones(d), 0.0), rtol=1e-13)
    # with eps = 0 the norm removes the 1/T factor: RMSNorm(mean) = RMSNorm(sum)
    np.testing.assert_allclose(F[1], O.rms_norm(h.sum(axis=0), np.ones(d), 0.0), rtol=1e-13)


def test_fuse_single_target_layer():
    h = _hidden(T=1)
    g = np.full((3, h.shape[2]), 1.25)
    F = O.fuse_context(h, O.fusion_weights(np.random.default_rng(8).standard_normal((3, 1))), g,
                       1e-6)
    for i in range(3):
        np.testing.assert_allclose(F[i], O.rms_norm(h[0], g[i], 1e-6), rtol=1e-14)


def test_fuse_two_layer_mix_by_hand():
    """T = 2, d = 2: s = a h1 + (1-a) h2 computed by hand, then normalised."""
    h = np.array([[[1.0, 0.0]], [[0.0, 1.0]]])         # [T=2][n=1][d=2]
    a1 = 1.0 / (1.0 + np.exp(-np.log(3.0)))              # softmax([log 3, 0]) = [3/4, 1/4]
    alpha = O.fusion_weights(np.array([[np.log(3.0), 0.0]]))
    np.testing.assert_allclose(alpha, [[0.75, 0.25]], rtol=1e-15)
    assert abs(a1 - 0.75) < 1e-15
    F = O.fuse_context(h, alpha, np.ones((1, 2)), 0.0)
    # s = [0.75, 0.25]; mean square = (0.5625 + 0.0625) / 2 = 0.3125
    np.testing.assert_allclose(F[0, 0], np.array([0.75, 0.25]) / np.sqrt(0.3125), rtol=1e-15)


def test_fuse_layer_scale_invariance_with_one_hot():
    h = _hidden(T=3)
    alpha = O.fusion_weights(np.array([[-1e4, 0.0, -1e4]]))
    g = np.ones((1, h.shape[2]))
    h2 = h.copy()
    h2[1] *= 3.7
    np.testing.assert_allclose(O.fuse_context(h2, alpha, g, 0.0), O.fuse_context(h, alpha, g, 0.0),
                               rtol=1e-13)


def test_fuse_bf16_storage_rounds_output_only():
    h = _hidden()
    alpha = O.fusion_weights(np.random.default_rng(9).standard_normal((3, h.shape[0])))
    g = np.ones((3, h.shape[2]))
    F = O.fuse_context(h, alpha, g, 1e-6)
    Fb = O.fuse_context(h, alpha, g, 1e-6, store=O.round_bf16)
    np.testing.assert_array_equal(Fb, O.round_bf16(F))
