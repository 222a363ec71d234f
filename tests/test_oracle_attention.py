"""Pins of the oracle's RoPE, Eq. 4 context projection and bidirectional block attention."""
import numpy as np
import torch

import oracle as O


# ----------------------------------------------------------------- RoPE

def test_rope_position_zero_is_identity():
    x = np.random.default_rng(0).standard_normal((3, 2, 8))
    np.testing.assert_array_equal(O.rope(x, np.zeros(3), 1e6), x)


def test_rope_two_dims_is_plane_rotation():
    """hd = 2: one pair, frequency theta^0 = 1, so position p rotates by p radians."""
    y = O.rope(np.array([[[1.0, 0.0]]]), np.array([1]), 1e6)
    np.testing.assert_allclose(y[0, 0], [0.5403023058681398, 0.8414709848078965], rtol=1e-15)
    y = O.rope(np.array([[[0.0, 2.0]]]), np.array([1]), 1e6)
    np.testing.assert_allclose(y[0, 0], [-2 * 0.8414709848078965, 2 * 0.5403023058681398],
                               rtol=1e-15)


def test_rope_frequency_of_second_pair():
    """hd = 4, theta = 100: pair 1 turns at 100^(-2/4) = 0.1 rad per position."""
    x = np.array([[[0.0, 1.0, 0.0, 0.0]]])       # pair 1 = (x_1, x_3) = (1, 0)
    y = O.rope(x, np.array([10]), 100.0)
    np.testing.assert_allclose(y[0, 0], [0.0, np.cos(1.0), 0.0, np.sin(1.0)], atol=1e-15)


def test_rope_matches_complex_multiplication():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 3, 16))
    pos = rng.integers(0, 40000, 5)
    theta = 1e6
    z = x[..., :8] + 1j * x[..., 8:]
    w = np.exp(1j * pos[:, None, None] * theta ** (-np.arange(8) / 8.0))
    ref = z * w
    y = O.rope(x, pos, theta)
    np.testing.assert_allclose(y[..., :8], ref.real, rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(y[..., 8:], ref.imag, rtol=1e-9, atol=1e-12)


def test_rope_scores_depend_on_offset_only():
    rng = np.random.default_rng(2)
    q, k = rng.standard_normal((1, 1, 64)), rng.standard_normal((1, 1, 64))

    def score(m, n):
        return float(np.sum(O.rope(q, np.array([m]), 1e6) * O.rope(k, np.array([n]), 1e6)))

    np.testing.assert_allclose(score(7, 3), score(1007, 1003), rtol=1e-10)
    np.testing.assert_allclose(score(0, 0), float(np.sum(q * k)), rtol=1e-13)


# ----------------------------------------------------------------- Eq. 4 context part

def test_context_kv_projection_layout():
    rng = np.random.default_rng(3)
    Hkv, hd, d, n = 2, 8, 12, 4
    F = rng.standard_normal((n, d))
    W = rng.standard_normal((2 * Hkv * hd, d))
    k, v = O.context_kv(F, W, np.zeros(n), Hkv, hd, 1e6)     # position 0: no rotation
    np.testing.assert_allclose(k.reshape(n, -1), F @ W[:Hkv * hd].T, rtol=1e-13)
    np.testing.assert_allclose(v.reshape(n, -1), F @ W[Hkv * hd:].T, rtol=1e-13)
    pos = np.arange(10, 10 + n)
    k2, v2 = O.context_kv(F, W, pos, Hkv, hd, 1e6)
    np.testing.assert_allclose(k2, O.rope(k, pos, 1e6), rtol=1e-13)
    np.testing.assert_array_equal(v2, v)                      # values are not rotated


# ----------------------------------------------------------------- attention

def _sdpa(q, k, v):
    """torch's scaled_dot_product_attention in float64 with kv heads repeated in groups."""
    G = q.shape[1] // k.shape[1]
    qt = torch.from_numpy(q).permute(1, 0, 2)                 # [H][B][hd]
    kt = torch.from_numpy(k).repeat_interleave(G, dim=1).permute(1, 0, 2)
    vt = torch.from_numpy(v).repeat_interleave(G, dim=1).permute(1, 0, 2)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)
    return o.permute(1, 0, 2).numpy()


def test_single_query_attention_matches_torch_sdpa():
    """B = 1: the block is one query over [context ; itself] -- textbook attention."""
    rng = np.random.default_rng(4)
    q = rng.standard_normal((1, 8, 64))
    k, v = rng.standard_normal((300, 2, 64)), rng.standard_normal((300, 2, 64))
    np.testing.assert_allclose(O.block_attention(q, k, v), _sdpa(q, k, v), rtol=1e-11, atol=1e-13)


def test_block_attention_is_unmasked():
    """Every query sees every key (no causal mask), for all grouped heads."""
    rng = np.random.default_rng(5)
    q = rng.standard_normal((16, 4, 32))
    k, v = rng.standard_normal((40, 1, 32)), rng.standard_normal((40, 1, 32))
    np.testing.assert_allclose(O.block_attention(q, k, v), _sdpa(q, k, v), rtol=1e-11, atol=1e-13)


def test_attention_closed_forms():
    rng = np.random.default_rng(6)
    q = rng.standard_normal((3, 2, 4))
    # all keys equal -> uniform weights -> mean of the values
    k = np.tile(rng.standard_normal((1, 1, 4)), (5, 1, 1))
    v = rng.standard_normal((5, 1, 4))
    np.testing.assert_allclose(O.block_attention(q, k, v),
                               np.broadcast_to(v.mean(axis=0), (3, 2, 4)), rtol=1e-13)
    # two keys: weights sigmoid(s1 - s2)
    q = np.array([[[1.0, 0.0, 0.0, 0.0]]])
    k = np.array([[[2.0, 0.0, 0.0, 0.0]], [[0.0, 0.0, 0.0, 0.0]]])
    v = np.array([[[1.0, 0.0, 0.0, 0.0]], [[0.0, 1.0, 0.0, 0.0]]])
    w1 = 1.0 / (1.0 + np.exp(-1.0))                  # s1 - s2 = 2 / sqrt(4) = 1
    np.testing.assert_allclose(O.block_attention(q, k, v)[0, 0], [w1, 1 - w1, 0, 0], rtol=1e-15)


def test_attention_key_permutation_invariance():
    rng = np.random.default_rng(7)
    q = rng.standard_normal((4, 4, 16))
    k, v = rng.standard_normal((50, 2, 16)), rng.standard_normal((50, 2, 16))
    p = rng.permutation(50)
    np.testing.assert_allclose(O.block_attention(q, k[p], v[p]), O.block_attention(q, k, v),
                               rtol=1e-12)


def test_attention_grouping_is_contiguous():
    """Query head h uses kv head h // (H_q / H_kv): zeroing kv head 1 only moves heads 2, 3."""
    rng = np.random.default_rng(8)
    q = rng.standard_normal((2, 4, 8))
    k, v = rng.standard_normal((6, 2, 8)), rng.standard_normal((6, 2, 8))
    v2 = v.copy()
    v2[:, 1] = 0
    a, b = O.block_attention(q, k, v), O.block_attention(q, k, v2)
    np.testing.assert_array_equal(a[:, :2], b[:, :2])
    np.testing.assert_array_equal(b[:, 2:], 0)
