"""The oracle's pins catch plausible mistakes: each case plants one mistake in the oracle (on the
CPU, through monkeypatching) and checks that at least one pin then fails."""
import numpy as np
import pytest

import oracle
import oracle.dflare_oracle as D
from tests import test_oracle_attention as TA
from tests import test_oracle_block as TB
from tests import test_oracle_fusion as TF
from tests import test_oracle_verify as TV


def _patch(monkeypatch, name, fn):
    monkeypatch.setattr(D, name, fn)
    monkeypatch.setattr(oracle, name, fn)


def _fails(*pins):
    for pin in pins:
        try:
            pin()
        except AssertionError:
            return True
    return False


def test_wrong_rope_sign(monkeypatch):
    orig = D.rope

    def bad(x, positions, theta):
        return orig(x, -np.asarray(positions), theta)
    _patch(monkeypatch, "rope", bad)
    assert _fails(TA.test_rope_two_dims_is_plane_rotation, TA.test_rope_matches_complex_multiplication)


def test_wrong_rope_frequency(monkeypatch):
    orig = D.rope

    def bad(x, positions, theta):
        return orig(x, positions, theta ** 0.5)
    _patch(monkeypatch, "rope", bad)
    assert _fails(TA.test_rope_frequency_of_second_pair, TA.test_rope_matches_complex_multiplication)


def test_transposed_fusion_index(monkeypatch):
    def bad(hidden, alpha, fuse_gain, eps, store=D.exact):
        hidden = np.asarray(hidden, float)
        Dn, T = alpha.shape
        out = np.empty((Dn,) + hidden.shape[1:])
        for i in range(Dn):
            s = sum(alpha[j % Dn, i % T] * hidden[j] for j in range(T))
            out[i] = store(D.rms_norm(s, fuse_gain[i], eps))
        return out
    _patch(monkeypatch, "fuse_context", bad)
    assert _fails(TF.test_fuse_one_hot_selects_one_layer)


def test_dropped_fusion_term(monkeypatch):
    def bad(hidden, alpha, fuse_gain, eps, store=D.exact):
        hidden = np.asarray(hidden, float)
        Dn, T = alpha.shape
        out = np.empty((Dn,) + hidden.shape[1:])
        for i in range(Dn):
            s = sum(alpha[i, j] * hidden[j] for j in range(T - 1))
            out[i] = store(D.rms_norm(s, fuse_gain[i], eps))
        return out
    _patch(monkeypatch, "fuse_context", bad)
    assert _fails(TF.test_fuse_uniform_is_layer_mean)


def test_rmsnorm_without_eps(monkeypatch):
    def bad(x, gain, eps):
        x = np.asarray(x, float)
        return gain * x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True))
    _patch(monkeypatch, "rms_norm", bad)
    assert _fails(TF.test_rms_norm_values)


def test_attention_missing_scale(monkeypatch):
    orig = D.block_attention

    def bad(q, k, v):
        return orig(np.asarray(q) * np.sqrt(np.asarray(q).shape[-1]), k, v)
    _patch(monkeypatch, "block_attention", bad)
    assert _fails(TA.test_single_query_attention_matches_torch_sdpa)


def test_attention_wrong_grouping(monkeypatch):
    def bad(q, k, v):
        q, k, v = (np.asarray(a, float) for a in (q, k, v))
        B, Hq, hd = q.shape
        Hkv = k.shape[1]
        out = np.empty_like(q)
        for h in range(Hq):
            g = h % Hkv                       # interleaved instead of contiguous groups
            s = q[:, h] @ k[:, g].T / np.sqrt(hd)
            p = np.exp(s - s.max(axis=1, keepdims=True))
            out[:, h] = (p / p.sum(axis=1, keepdims=True)) @ v[:, g]
        return out
    _patch(monkeypatch, "block_attention", bad)
    assert _fails(TA.test_attention_grouping_is_contiguous, TA.test_single_query_attention_matches_torch_sdpa)


def test_causal_mask_planted(monkeypatch):
    orig = D.block_attention

    def bad(q, k, v):
        q, k, v = (np.asarray(a, float) for a in (q, k, v))
        B = q.shape[0]
        S = k.shape[0]
        out = np.empty_like(q)
        for r in range(B):                    # row r sees keys up to S - B + r only
            out[r:r + 1] = orig(q[r:r + 1], k[:S - B + r + 1], v[:S - B + r + 1])
        return out
    _patch(monkeypatch, "block_attention", bad)
    assert _fails(TA.test_block_attention_is_unmasked)


def test_missing_mlp_residual(monkeypatch):
    orig = D.draft_layer

    def bad(x, lw, ctx_k, ctx_v, positions, shape, store=D.exact, rope_block=True):
        z = dict(lw, w_down=np.zeros_like(lw["w_down"]))
        return orig(x, z, ctx_k, ctx_v, positions, shape, store, rope_block)
    _patch(monkeypatch, "draft_layer", bad)
    assert _fails(TB.test_draft_layer_matches_torch_assembly)


def test_verify_off_by_one(monkeypatch):
    def bad(draft, target):
        B = len(target)
        a = 0
        while a < B - 1 and draft[a] == target[a + 1 if a + 1 < B else a]:
            a += 1
        return a + 1, int(target[a])
    _patch(monkeypatch, "verify_accept", bad)
    assert _fails(lambda: TV.test_verify_brute_force_tiny_alphabet(3))


def test_verify_missing_bonus(monkeypatch):
    def bad(draft, target):
        B = len(target)
        a = 0
        while a < B - 1 and draft[a] == target[a]:
            a += 1
        return a, int(target[a])
    _patch(monkeypatch, "verify_accept", bad)
    assert _fails(lambda: TV.test_verify_brute_force_tiny_alphabet(2))


def test_argmax_highest_index_ties(monkeypatch):
    def bad(logits):
        lg = np.asarray(logits)
        return (lg.shape[-1] - 1 - np.argmax(lg[..., ::-1], axis=-1)).astype(np.int64)
    _patch(monkeypatch, "argmax_lowest", bad)
    assert _fails(TB.test_argmax_lowest_and_gap)


def test_round_bf16_truncating(monkeypatch):
    def bad(x):
        x = np.asarray(x, float)
        m, e = np.frexp(x)
        return np.ldexp(np.trunc(np.ldexp(m, 8)), e - 8)
    _patch(monkeypatch, "round_bf16", bad)
    assert _fails(TF.test_round_bf16_matches_torch_cast)


def test_dflash_concat_in_reverse_layer_order(monkeypatch):
    from tests import test_oracle_variants as TW

    def bad(hidden, w_fc, b_fc, store=D.exact):
        hidden = np.asarray(hidden, float)
        cat = np.concatenate([hidden[j] for j in reversed(range(hidden.shape[0]))], axis=-1)
        return store(cat @ np.asarray(w_fc, float).T + b_fc)
    _patch(monkeypatch, "dflash_context", bad)
    assert _fails(TW.test_dflash_context_brute_force)


def test_dflash_without_bias(monkeypatch):
    from tests import test_oracle_variants as TW

    def bad(hidden, w_fc, b_fc, store=D.exact):
        hidden = np.asarray(hidden, float)
        cat = np.concatenate(list(hidden), axis=-1)
        return store(cat @ np.asarray(w_fc, float).T)
    _patch(monkeypatch, "dflash_context", bad)
    assert _fails(TW.test_dflash_context_one_hot_block_selects_a_layer)


def test_fusion_fc_transposed_weight(monkeypatch):
    from tests import test_oracle_variants as TW

    def bad(F_i, w_fc_i, b_fc_i, store=D.exact):
        return store(np.asarray(F_i, float) @ np.asarray(w_fc_i, float) + b_fc_i)
    _patch(monkeypatch, "fusion_fc", bad)
    assert _fails(TW.test_fusion_fc_brute_force_and_identity)


def test_acceptance_ratio_inverted(monkeypatch):
    from tests import test_oracle_sampling as TS
    _patch(monkeypatch, "accept_prob", lambda p, q, d: min(1.0, float(q[d]) / float(p[d])))
    assert _fails(TS.test_speculative_rule_preserves_the_target_distribution_closed_form)


def test_residual_without_clipping(monkeypatch):
    from tests import test_oracle_sampling as TS

    def bad(p, q):
        w = np.abs(np.asarray(p, float) - np.asarray(q, float))
        return w / w.sum()
    _patch(monkeypatch, "residual_dist", bad)
    assert _fails(TS.test_speculative_rule_preserves_the_target_distribution_closed_form)


def test_replacement_drawn_from_target_instead_of_residual(monkeypatch):
    """A verification that redraws from p (not max(0, p - q)) after a rejection over-weights the
    tokens the draft already proposes."""
    from tests import test_oracle_sampling as TS
    orig_res = D.residual_dist
    _patch(monkeypatch, "residual_dist", lambda p, q: np.asarray(p, float))
    assert _fails(lambda: TS.test_speculative_verify_first_token_is_target_distributed(2))
    _patch(monkeypatch, "residual_dist", orig_res)


def test_philox_words_swapped(monkeypatch):
    from tests import test_oracle_sampling as TS
    orig = D.philox4x64

    def bad(counter, key, rounds=10):
        c = orig(counter, key, rounds)
        return [c[1], c[0], c[2], c[3]]
    _patch(monkeypatch, "philox4x64", bad)
    assert _fails(lambda: TS.test_uniform_stream_is_philox4x64_10(7, 2, 3, 11))
