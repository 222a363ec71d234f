"""Pins of the oracle's prefix acceptance (Sec. 3.2, verification) and of the synthetic target."""
import itertools

import numpy as np
import pytest

import oracle as O
import synth


def _brute_tau(d, g):
    """Largest a in [0, B-1] such that d_k == g_{k-1} for every k <= a, by trying every a."""
    B = len(g)
    best = 0
    for a in range(B):
        if all(d[k - 1] == g[k - 1] for k in range(1, a + 1)):
            best = a
    return best + 1, g[best]


@pytest.mark.parametrize("B", [1, 2, 3, 4])
def test_verify_brute_force_tiny_alphabet(B):
    for d in itertools.product(range(3), repeat=B - 1):
        for g in itertools.product(range(3), repeat=B):
            assert O.verify_accept(list(d), list(g)) == _brute_tau(d, g)


def test_verify_examples():
    assert O.verify_accept([5, 6, 7], [5, 6, 7, 8]) == (4, 8)      # all accepted + bonus
    assert O.verify_accept([5, 6, 7], [4, 6, 7, 8]) == (1, 4)      # first draft rejected
    assert O.verify_accept([5, 6, 7], [5, 9, 7, 8]) == (2, 9)      # later match does not count


def test_synthetic_target_rule():
    rng = np.random.default_rng(0)
    V, B = 11, 9
    thr = synth.accept_threshold(0.5)
    for _ in range(200):
        d = rng.integers(0, V, B - 1)
        u = rng.integers(0, 2 ** 32, B - 1, dtype=np.uint64)
        r = rng.integers(0, V - 1, B - 1)
        g = O.synthetic_target(d, u, r, 3, thr)
        assert g[-1] == 3
        acc = u < thr
        np.testing.assert_array_equal(g[:-1][acc], d[acc])
        assert np.all(g[:-1][~acc] != d[~acc])
        assert np.all((g >= 0) & (g < V))


@pytest.mark.parametrize("p,B", [(0.85, 16), (0.75, 16), (0.8, 8), (0.6, 16), (0.9, 16)])
def test_expected_accept_length(p, B):
    """Independent matches with probability p: E[tau] = sum_{k<B} p^k = (1 - p^B) / (1 - p)."""
    n = 20000
    w = synth.Workload("t", synth.Shape(d=64, n_draft_layers=1, n_target_layers=1, n_q_heads=1,
                                        n_kv_heads=1, head_dim=64, ffn=64, vocab=1000, block=B),
                       (0,) * n, p)
    u, r, last = synth.target_draws(w, 0)
    d = np.random.default_rng(1).integers(0, 1000, (n, B - 1))
    thr = synth.accept_threshold(p)
    taus = np.array([O.verify_accept(d[b], O.synthetic_target(d[b], u[0, b], r[0, b], last[0, b],
                                                              thr))[0] for b in range(n)])
    mean = (1 - p ** B) / (1 - p)
    sd = taus.std() / np.sqrt(n)
    assert abs(taus.mean() - mean) < 4 * sd, (taus.mean(), mean, sd)
    assert taus.min() >= 1 and taus.max() <= B


def test_verify_from_logits_equals_verify_on_planted_maxima():
    """One planted maximum per row makes the logits route equal verify_accept on those tokens;
    a tie between two planted maxima goes to the lower id."""
    rng = np.random.default_rng(9)
    B, V = 6, 40
    for trial in range(200):
        draft = rng.integers(0, V, B - 1)
        g = rng.integers(0, V, B)
        lg = rng.standard_normal((B, V))
        lg[np.arange(B), g] = 10.0
        assert O.verify_from_logits(draft, lg) == O.verify_accept(draft, g)
    lg = np.zeros((B, V))
    lg[:, 7] = lg[:, 3] = 1.0
    assert O.verify_from_logits([3] * (B - 1), lg) == (B, 3)
    assert O.verify_from_logits([7] * (B - 1), lg) == (1, 3)
