"""Pins of the oracle's variants: DFlash's FC fusion (Eq. 1) with its shared KV projection (Eq. 2)
and the "-KVProj" / "+FC" ablations of Sec. 6.3 (Table 2).

Each is checked against brute force on tiny inputs, against special cases with a known result
(a one-hot selection, an identity layer), and against another variant that reaches the same
context keys and values along a different route."""
import dataclasses

import numpy as np

import oracle as O
import synth

SMALL = synth.Shape(d=32, n_draft_layers=2, n_target_layers=3, n_q_heads=4, n_kv_heads=2,
                    head_dim=8, ffn=48, vocab=50, block=6, dtype="f32")


def _workload(shape=SMALL, L=11, seed=3):
    return synth.Workload("variants", shape, (L,), 0.8, seed=seed, scale_layers=False)


def _all_weights(w):
    W = dict(synth.weights(w))
    W.update(synth.variant_weights(w))
    return W


def test_dflash_context_brute_force():
    """c_t[o] = b[o] + sum_j sum_e W[o, j d + e] h^(j)[t, e], written out element by element."""
    rng = np.random.default_rng(0)
    T, n, d = 3, 2, 4
    h = rng.standard_normal((T, n, d))
    W = rng.standard_normal((d, T * d))
    b = rng.standard_normal(d)
    c = O.dflash_context(h, W, b)
    for t in range(n):
        for o in range(d):
            acc = b[o]
            for j in range(T):
                for e in range(d):
                    acc += W[o, j * d + e] * h[j, t, e]
            assert abs(c[t, o] - acc) < 1e-12


def test_dflash_context_one_hot_block_selects_a_layer():
    """W_fc = [0, I, 0]: c_t = h_t^(2) + b_fc."""
    rng = np.random.default_rng(1)
    T, n, d = 3, 5, 8
    h = rng.standard_normal((T, n, d))
    W = np.zeros((d, T * d))
    W[:, d:2 * d] = np.eye(d)
    b = rng.standard_normal(d)
    np.testing.assert_allclose(O.dflash_context(h, W, b), h[1] + b, rtol=0, atol=1e-15)


def test_dflash_fc_spans_the_layer_mix_before_its_norm():
    """W_fc = [a_1 I, ..., a_T I], b_fc = 0 gives c_t = sum_j a_j h_t^(j), the sum that Eq. 3
    normalises: RMSNorm(c) equals the layer-wise fusion with weights a."""
    rng = np.random.default_rng(2)
    T, n, d = 4, 6, 16
    h = rng.standard_normal((T, n, d))
    a = rng.dirichlet(np.ones(T))
    W = np.concatenate([a[j] * np.eye(d) for j in range(T)], axis=1)
    c = O.dflash_context(h, W, np.zeros(d))
    gain = 1 + 0.1 * rng.standard_normal(d)
    F = O.fuse_context(h, a[None, :], gain[None, :], 1e-6)
    np.testing.assert_allclose(O.rms_norm(c, gain, 1e-6), F[0], rtol=1e-12)


def test_fusion_fc_brute_force_and_identity():
    rng = np.random.default_rng(4)
    n, d = 3, 5
    F = rng.standard_normal((n, d))
    W = rng.standard_normal((d, d))
    b = rng.standard_normal(d)
    y = O.fusion_fc(F, W, b)
    for t in range(n):
        for o in range(d):
            assert abs(y[t, o] - (b[o] + sum(W[o, e] * F[t, e] for e in range(d)))) < 1e-12
    np.testing.assert_array_equal(O.fusion_fc(F, np.eye(d), np.zeros(d)), F)


def _run(W, shape, last=7, L=11, w=None, **kw):
    w = w or _workload(shape, L)
    o = O.DraftOracle(W, shape, 1, **kw)
    F = o.fuse_context(0, synth.hidden_states(w, 0, 0, L))
    toks, logits, hid = o.draft_block(0, last)
    return o, F, toks, logits


def test_shared_kv_is_hetero_kv_with_copied_weights():
    """-KVProj projects the context with W^d; giving W^t the values of W^d reproduces it through
    the heterogeneous route of Eq. 4, and with distinct W^t the two differ."""
    w = _workload()
    W = _all_weights(w)
    s = SMALL
    shared, _, t1, l1 = _run(W, s, shared_kv=True)
    W2 = dict(W)
    W2["w_kv_ctx"] = np.ascontiguousarray(W["w_qkv"][:, s.d_q:])
    hetero, _, t2, l2 = _run(W2, s)
    for i in range(s.n_draft_layers):
        np.testing.assert_array_equal(shared.ctx_k[0][i], hetero.ctx_k[0][i])
        np.testing.assert_array_equal(shared.ctx_v[0][i], hetero.ctx_v[0][i])
    np.testing.assert_array_equal(t1, t2)
    np.testing.assert_array_equal(l1, l2)
    plain, _, _, _ = _run(W, s)
    assert not np.allclose(plain.ctx_k[0][0], shared.ctx_k[0][0])


def test_fusion_fc_identity_layer_changes_nothing():
    w = _workload()
    W = _all_weights(w)
    s = SMALL
    W["fusion_fc_w"] = np.stack([np.eye(s.d, dtype=np.float32)] * s.n_draft_layers)
    W["fusion_fc_b"] = np.zeros((s.n_draft_layers, s.d), np.float32)
    a, Fa, ta, la = _run(W, s, fusion_fc=True)
    b, Fb, tb, lb = _run(W, s)
    np.testing.assert_array_equal(Fa, Fb)
    np.testing.assert_array_equal(la, lb)
    # a bias shifts the projected context: F' = F + b, and the keys follow
    W["fusion_fc_b"] = np.full((s.n_draft_layers, s.d), 0.25, np.float32)
    c, Fc, _, _ = _run(W, s, fusion_fc=True)
    np.testing.assert_allclose(Fc, Fb + 0.25, rtol=0, atol=1e-12)


def test_dflash_one_hot_equals_raw_one_hot_fusion_with_shared_kv():
    """Two routes to the same context keys: DFlash with W_fc = [I, 0, ...] (c = h^(1)), and the
    layer-wise fusion with raw weights (1, 0, ...) ("-Softmax"), unit gains, eps 0 and hidden rows
    of unit RMS (so F = RMSNorm(h^(1)) = h^(1)), both projected by W^d ("-KVProj")."""
    s = dataclasses.replace(SMALL, rms_eps=0.0)
    L = 9
    w = _workload(s, L)
    W = _all_weights(w)
    D, T, d = s.n_draft_layers, s.n_target_layers, s.d
    h = synth.hidden_states(w, 0, 0, L).astype(np.float64)
    h /= np.sqrt(np.mean(h * h, axis=-1, keepdims=True))
    hidden = h.astype(np.float32)
    W["fuse_logits"] = np.zeros((D, T), np.float32)
    W["fuse_logits"][:, 0] = 1.0
    W["fuse_norm"] = np.ones((D, d), np.float32)
    W["dflash_fc_w"] = np.zeros((d, T * d), np.float32)
    W["dflash_fc_w"][:, :d] = np.eye(d)
    W["dflash_fc_b"] = np.zeros(d, np.float32)
    a = O.DraftOracle(W, s, 1, dflash_fc=True)
    b = O.DraftOracle(W, s, 1, softmax_fusion=False, shared_kv=True)
    Fa = a.fuse_context(0, hidden)
    Fb = b.fuse_context(0, hidden)
    np.testing.assert_allclose(Fa, Fb, rtol=1e-6, atol=1e-6)
    for i in range(D):
        np.testing.assert_allclose(a.ctx_k[0][i], b.ctx_k[0][i], rtol=1e-6, atol=1e-7)
        np.testing.assert_allclose(a.ctx_v[0][i], b.ctx_v[0][i], rtol=1e-6, atol=1e-7)
    _, la, _ = a.draft_block(0, 3)[:3]
    _, lb, _ = b.draft_block(0, 3)[:3]
    np.testing.assert_allclose(la, lb, rtol=1e-5, atol=1e-6)


def test_dflash_every_layer_projects_the_same_feature():
    w = _workload()
    W = _all_weights(w)
    o = O.DraftOracle(W, SMALL, 1, dflash_fc=True)
    F = o.fuse_context(0, synth.hidden_states(w, 0, 0, 11))
    for i in range(1, SMALL.n_draft_layers):
        np.testing.assert_array_equal(F[i], F[0])
