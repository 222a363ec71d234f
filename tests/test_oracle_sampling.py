"""Pins of the oracle's sampled decoding (Table 1, temperature 1): the Philox4x64-10 streams, the
Gumbel-max draw, and the speculative-sampling verification rule.

The generator is checked against numpy's own Philox implementation (a library routine) on
arbitrary counters; the draws against their target distributions with a chi-square bound; the
verification rule against the property that defines it (the first token it emits is distributed
as the target's p, whatever the draft's q), both in closed form and by Monte Carlo."""
import numpy as np
import pytest

import oracle as O

# chi-square critical values at upper tail 1e-4 (df -> value), so a correct sampler fails a given
# test with probability 1e-4
CHI2_1E4 = {3: 21.11, 4: 23.51, 5: 25.74, 6: 27.86, 7: 29.88, 9: 33.72}


def _chi2(counts, probs):
    n = counts.sum()
    e = n * np.asarray(probs)
    keep = e > 0
    assert np.all(counts[~keep] == 0)
    return float(np.sum((counts[keep] - e[keep]) ** 2 / e[keep])), int(keep.sum()) - 1


@pytest.mark.parametrize("seed,purpose,step,row", [(0, 1, 0, 0), (7, 2, 3, 11), (2 ** 63 + 5, 3, 2 ** 40, 2 ** 33)])
def test_uniform_stream_is_philox4x64_10(seed, purpose, step, row):
    """uniforms() (numpy's Philox) and philox4x64() (written from the definition) agree on the
    stream layout: element v comes from word (v div 2) mod 4 of the block at counter
    (1 + v div 8, row, step, purpose), key (seed, 0), bits 63..41 for even v, 31..9 for odd v."""
    n = 23
    u = O.uniforms(seed, purpose, step, row, n)
    for v in range(n):
        x = O.philox4x64([1 + v // 8, row, step, purpose], [seed, 0])[(v // 2) % 4]
        bits = x >> 41 if v % 2 == 0 else (x >> 9) & 0x7FFFFF
        assert u[v] == (bits + 0.5) * 2.0 ** -23


def test_philox_rounds_and_key_schedule_matter():
    a = O.philox4x64([1, 2, 3, 4], [5, 6])
    assert O.philox4x64([1, 2, 3, 4], [5, 6], rounds=9) != a
    assert O.philox4x64([1, 2, 3, 4], [5, 7]) != a
    assert O.philox4x64([1, 2, 3, 5], [5, 6]) != a


def test_uniforms_are_exact_fp32_values_in_open_unit_interval():
    u = O.uniforms(3, 1, 0, 0, 200000)
    assert u.min() > 0 and u.max() < 1
    assert np.all(u.astype(np.float32).astype(np.float64) == u)
    k = u * 2 ** 23 - 0.5
    assert np.all(k == np.floor(k))
    # mean 1/2 and variance 1/12 within 5 standard errors
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / u.size)
    assert abs(u.var() - 1 / 12) < 5 * np.sqrt(1 / 180 / u.size)
    # the two uniforms cut from one 64-bit word (its high and low bits) are uncorrelated
    hi, lo = u[0::2], u[1::2]
    assert abs(np.corrcoef(hi, lo)[0, 1]) < 5 / np.sqrt(hi.size)
    for half in (hi, lo):
        assert abs(half.mean() - 0.5) < 5 * np.sqrt(1 / 12 / half.size)


def test_gumbel_draw_frequencies_follow_the_weights():
    w = np.array([0.05, 0.3, 0.0, 0.15, 0.4, 0.1])
    counts = np.zeros(w.size)
    with np.errstate(divide="ignore"):
        lw = np.log(w)
    for row in range(40000):
        counts[O.gumbel_draw(lw, O.uniforms(11, O.RNG_DRAFT, 0, row, w.size))] += 1
    stat, df = _chi2(counts, w)
    assert counts[2] == 0
    assert stat < CHI2_1E4[df], stat


def test_sample_token_temperature():
    """softmax(l / T): at T = 2 the draws follow softmax(l / 2); -inf logits are never drawn."""
    lg = np.array([1.0, -np.inf, 0.0, 2.0, -1.0])
    p = O.softmax_t(lg, 2.0)
    counts = np.zeros(lg.size)
    for row in range(30000):
        counts[O.sample_token(lg, 2.0, O.uniforms(4, O.RNG_DRAFT, 1, row, lg.size))] += 1
    stat, df = _chi2(counts, p)
    assert stat < CHI2_1E4[df], stat
    np.testing.assert_allclose(O.softmax_t([0.0, np.log(3.0)], 1.0), [0.25, 0.75], rtol=1e-15)


def test_speculative_rule_preserves_the_target_distribution_closed_form():
    """P(emit x) = q(x) min(1, p(x)/q(x)) + (1 - sum_d q(d) min(1, p(d)/q(d))) r(x) = p(x)."""
    rng = np.random.default_rng(3)
    for _ in range(200):
        V = int(rng.integers(2, 9))
        p = rng.dirichlet(np.ones(V) * rng.uniform(0.2, 3))
        q = rng.dirichlet(np.ones(V) * rng.uniform(0.2, 3))
        acc = np.array([q[d] * O.accept_prob(p, q, d) for d in range(V)])
        emit = acc + (1 - acc.sum()) * O.residual_dist(p, q)
        np.testing.assert_allclose(emit, p, rtol=0, atol=1e-12)
    p = np.array([0.2, 0.5, 0.3])
    assert all(O.accept_prob(p, p, d) == 1.0 for d in range(3))


@pytest.mark.parametrize("B", [2, 3])
def test_speculative_verify_first_token_is_target_distributed(B):
    """Monte Carlo over the whole rule: drafts drawn from q, verified against p; the first token
    the step emits (d_1 when kept, else the replacement) follows p_0."""
    V, T = 6, 1.0
    rng = np.random.default_rng(5)
    tl = rng.standard_normal((B, V)) * 1.5
    dl = rng.standard_normal((B - 1, V)) * 1.5
    p0 = O.softmax_t(tl[0], T)
    counts = np.zeros(V)
    n = 30000
    for step in range(n):
        draft = [O.sample_token(dl[k], T, O.uniforms(9, O.RNG_DRAFT, step, k, V)) for k in range(B - 1)]
        tau, nxt = O.speculative_verify(draft, tl, dl, T, O.uniforms(9, O.RNG_ACCEPT, step, 0, B - 1),
                                        O.uniforms(9, O.RNG_RESIDUAL, step, 0, V))
        counts[draft[0] if tau >= 2 else nxt] += 1
    stat, df = _chi2(counts, p0)
    assert stat < CHI2_1E4[df], stat


def test_speculative_verify_edge_cases():
    V = 5
    lg = np.log(np.array([0.1, 0.2, 0.3, 0.25, 0.15]))
    B = 4
    u = O.uniforms(1, O.RNG_RESIDUAL, 0, 0, V)
    r = O.uniforms(1, O.RNG_ACCEPT, 0, 0, B - 1)
    # q = p: every draft is kept; the extra token comes from the last target row
    tl = np.stack([lg] * B)
    tau, nxt = O.speculative_verify([2, 0, 4], tl, tl[:B - 1], 1.0, r, u)
    assert tau == B and nxt == O.gumbel_draw(lg, u)
    # a draft the target gives probability 0 is always rejected and never re-drawn
    tl0 = tl.copy()
    tl0[0, 3] = -np.inf
    for step in range(50):
        tau, nxt = O.speculative_verify([3, 0, 0], tl0, tl[:B - 1], 1.0,
                                        O.uniforms(1, O.RNG_ACCEPT, step, 0, B - 1),
                                        O.uniforms(1, O.RNG_RESIDUAL, step, 0, V))
        assert tau == 1 and nxt != 3
