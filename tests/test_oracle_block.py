"""Pins of the oracle's draft layer, LM head / argmax and the whole block forward (Sec. 3.2)."""
import dataclasses

import numpy as np
import torch

import oracle as O
import synth


SMALL = synth.Shape(d=32, n_draft_layers=2, n_target_layers=3, n_q_heads=4, n_kv_heads=2,
                    head_dim=8, ffn=48, vocab=50, block=6, dtype="f32")


def _layer(shape, seed=0):
    rng = np.random.default_rng(seed)
    d, F = shape.d, shape.ffn
    return {
        "attn_norm": 1 + 0.1 * rng.standard_normal(d),
        "w_qkv": 0.2 * rng.standard_normal((shape.d_q + 2 * shape.d_kv, d)),
        "w_o": 0.2 * rng.standard_normal((d, shape.d_q)),
        "mlp_norm": 1 + 0.1 * rng.standard_normal(d),
        "w_gate": 0.2 * rng.standard_normal((F, d)),
        "w_up": 0.2 * rng.standard_normal((F, d)),
        "w_down": 0.2 * rng.standard_normal((d, F)),
    }


def _ctx(shape, L, seed=1):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((L, shape.n_kv_heads, shape.head_dim)),
            rng.standard_normal((L, shape.n_kv_heads, shape.head_dim)))


def _torch_layer(x, lw, ck, cv, pos, s):
    """The same layer assembled from torch library routines (rms_norm, SDPA, silu)."""
    t = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    X = t(x)
    B = X.shape[0]
    xn = torch.nn.functional.rms_norm(X, (s.d,), t(lw["attn_norm"]), eps=s.rms_eps)
    qkv = xn @ t(lw["w_qkv"]).T
    q = qkv[:, :s.d_q].reshape(B, s.n_q_heads, s.head_dim)
    kd = qkv[:, s.d_q:s.d_q + s.d_kv].reshape(B, s.n_kv_heads, s.head_dim)
    vd = qkv[:, s.d_q + s.d_kv:].reshape(B, s.n_kv_heads, s.head_dim)

    def rot(a):   # complex-number form of the rotary embedding
        h = s.head_dim // 2
        z = torch.complex(a[..., :h], a[..., h:])
        f = torch.tensor(s.rope_theta, dtype=torch.float64) ** (-torch.arange(h, dtype=torch.float64) * 2.0 / s.head_dim)
        w = torch.polar(torch.ones(B, 1, h, dtype=torch.float64),
                        t(pos)[:, None, None] * f[None, None, :])
        z = z * w
        return torch.cat([z.real, z.imag], dim=-1)

    q, kd = rot(q), rot(kd)
    K = torch.cat([t(ck), kd]).repeat_interleave(s.n_q_heads // s.n_kv_heads, dim=1)
    V = torch.cat([t(cv), vd]).repeat_interleave(s.n_q_heads // s.n_kv_heads, dim=1)
    o = torch.nn.functional.scaled_dot_product_attention(q.permute(1, 0, 2), K.permute(1, 0, 2),
                                                         V.permute(1, 0, 2))
    X = X + o.permute(1, 0, 2).reshape(B, s.d_q) @ t(lw["w_o"]).T
    xm = torch.nn.functional.rms_norm(X, (s.d,), t(lw["mlp_norm"]), eps=s.rms_eps)
    a = torch.nn.functional.silu(xm @ t(lw["w_gate"]).T) * (xm @ t(lw["w_up"]).T)
    return (X + a @ t(lw["w_down"]).T).numpy()


def test_silu_closed_forms():
    x = np.linspace(-8, 8, 101)
    np.testing.assert_allclose(O.silu(x) - O.silu(-x), x, rtol=1e-13, atol=1e-15)
    assert O.silu(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(O.silu(x), torch.nn.functional.silu(torch.from_numpy(x)).numpy(),
                               rtol=1e-14)


def test_draft_layer_matches_torch_assembly():
    for B in (1, 6):
        s = dataclasses.replace(SMALL, block=B)
        x = np.random.default_rng(2).standard_normal((B, s.d))
        ck, cv = _ctx(s, 17)
        pos = np.arange(17, 17 + B)
        np.testing.assert_allclose(O.draft_layer(x, _layer(s), ck, cv, pos, s),
                                   _torch_layer(x, _layer(s), ck, cv, pos, s), rtol=1e-10,
                                   atol=1e-12)


def test_draft_layer_mask_permutation_equivariance():
    """RoPE off on the block: permuting the B-1 mask rows permutes the outputs (no mask)."""
    s = SMALL
    rng = np.random.default_rng(3)
    x = rng.standard_normal((s.block, s.d))
    ck, cv = _ctx(s, 9)
    pos = np.arange(9, 9 + s.block)
    y = O.draft_layer(x, _layer(s), ck, cv, pos, s, rope_block=False)
    perm = np.concatenate([[0], 1 + rng.permutation(s.block - 1)])
    yp = O.draft_layer(x[perm], _layer(s), ck, cv, pos, s, rope_block=False)
    np.testing.assert_allclose(yp, y[perm], rtol=1e-12, atol=1e-13)
    # identical mask inputs give identical mask outputs
    x[2:] = x[1]
    y = O.draft_layer(x, _layer(s), ck, cv, pos, s, rope_block=False)
    for k in range(2, s.block):
        np.testing.assert_allclose(y[k], y[1], rtol=1e-13, atol=1e-14)


def test_draft_layer_residual_paths_by_hand():
    """Zero W_O and W_down: the layer is the identity. Zero only W_down: x plus the attention
    sub-layer's contribution, which then equals the layer output minus x."""
    s = SMALL
    lw = _layer(s)
    x = np.random.default_rng(4).standard_normal((s.block, s.d))
    ck, cv = _ctx(s, 5)
    pos = np.arange(5, 5 + s.block)
    z = dict(lw, w_o=np.zeros_like(lw["w_o"]), w_down=np.zeros_like(lw["w_down"]))
    np.testing.assert_array_equal(O.draft_layer(x, z, ck, cv, pos, s), x)
    z = dict(lw, w_down=np.zeros_like(lw["w_down"]))
    y = O.draft_layer(x, z, ck, cv, pos, s)
    xn = O.rms_norm(x, lw["attn_norm"], s.rms_eps)
    qkv = xn @ lw["w_qkv"].T
    B = s.block
    q = O.rope(qkv[:, :s.d_q].reshape(B, s.n_q_heads, s.head_dim), pos, s.rope_theta)
    kd = O.rope(qkv[:, s.d_q:s.d_q + s.d_kv].reshape(B, s.n_kv_heads, s.head_dim), pos,
                s.rope_theta)
    vd = qkv[:, s.d_q + s.d_kv:].reshape(B, s.n_kv_heads, s.head_dim)
    o = O.block_attention(q, np.concatenate([ck, kd]), np.concatenate([cv, vd]))
    np.testing.assert_allclose(y - x, o.reshape(B, -1) @ lw["w_o"].T, rtol=1e-10, atol=1e-12)


def test_hetero_kv_reduces_to_shared_projection():
    """-KVProj (Eq. 2): with W^t = W^d, a context row equal to a block row's normalised input
    at the same position yields the same key and value."""
    s = SMALL
    lw = _layer(s)
    x = np.random.default_rng(5).standard_normal((s.block, s.d))
    xn = O.rms_norm(x, lw["attn_norm"], s.rms_eps)
    w_d = lw["w_qkv"][s.d_q:]                                      # [W_K^d ; W_V^d]
    pos = np.arange(30, 30 + s.block)
    k, v = O.context_kv(xn, w_d, pos, s.n_kv_heads, s.head_dim, s.rope_theta)
    qkv = xn @ lw["w_qkv"].T
    kd = O.rope(qkv[:, s.d_q:s.d_q + s.d_kv].reshape(s.block, s.n_kv_heads, s.head_dim), pos,
                s.rope_theta)
    np.testing.assert_allclose(k, kd, rtol=1e-13)
    np.testing.assert_allclose(v.reshape(s.block, -1), qkv[:, s.d_q + s.d_kv:], rtol=1e-13)


def test_argmax_lowest_and_gap():
    lg = np.array([[0.0, 3.0, 3.0, 1.0], [5.0, -1.0, 5.0, 5.0], [-2.0, -1.0, -3.0, -1.5]])
    np.testing.assert_array_equal(O.argmax_lowest(lg), [1, 0, 1])
    np.testing.assert_allclose(O.top2_gap(lg), [0.0, 0.0, 0.5])
    rng = np.random.default_rng(6)
    lg = rng.standard_normal((5, 1000))
    plant = rng.integers(0, 1000, 5)
    lg[np.arange(5), plant] = 10.0
    np.testing.assert_array_equal(O.argmax_lowest(lg), plant)


def test_lm_head_reads_mask_rows_only():
    rng = np.random.default_rng(7)
    x = rng.standard_normal((6, 16))
    g, W = np.ones(16), rng.standard_normal((40, 16))
    a = O.lm_head_logits(x, g, W, 1e-6)
    x2 = x.copy()
    x2[0] = 100.0
    np.testing.assert_array_equal(O.lm_head_logits(x2, g, W, 1e-6), a)
    assert a.shape == (5, 40)
    np.testing.assert_allclose(a, O.rms_norm(x[1:], g, 1e-6) @ W.T, rtol=1e-13)


def _oracle(shape, seed=0, storage="exact", **kw):
    w = synth.Workload("t", shape, (11,), 0.8, seed=seed, scale_layers=False)
    W = synth.weights(w)
    o = O.DraftOracle(W, shape, 1, storage=storage, **kw)
    o.fuse_context(0, synth.hidden_states(w, 0, 0, 11))
    return o, W


def test_block_input_is_token_then_masks():
    o, W = _oracle(SMALL)
    x0 = o.block_input(7)
    np.testing.assert_array_equal(x0[0], W["embed"][7].astype(np.float64))
    for k in range(1, SMALL.block):
        np.testing.assert_array_equal(x0[k], W["embed"][SMALL.vocab - 1].astype(np.float64))


def test_draft_block_permutation_equivariance_end_to_end():
    """Whole forward with block RoPE off and distinct mask-row inputs: permuting the mask rows
    permutes logits and hidden states."""
    o, W = _oracle(SMALL, rope_block=False)
    x0 = np.random.default_rng(8).standard_normal((SMALL.block, SMALL.d)) * 0.3
    tok, lg, hid = o.draft_block(0, 0, x0=x0)
    perm = np.concatenate([[0], 1 + np.random.default_rng(9).permutation(SMALL.block - 1)])
    tok2, lg2, hid2 = o.draft_block(0, 0, x0=x0[perm])
    np.testing.assert_allclose(hid2, hid[:, perm], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(lg2, lg[perm[1:] - 1], rtol=1e-11, atol=1e-12)


def test_draft_block_single_position_matches_torch():
    """B = 1 through the whole stack: each layer is single-query attention + MLP (torch)."""
    s = dataclasses.replace(SMALL, block=1)
    o, W = _oracle(s)
    x0 = np.random.default_rng(10).standard_normal((1, s.d))
    _, _, hid = o.draft_block(0, 0, x0=x0)
    x = x0
    L = o.ctx_len(0)
    for i in range(s.n_draft_layers):
        x = _torch_layer(x, o.layer(i), o.ctx_k[0][i], o.ctx_v[0][i], np.arange(L, L + 1), s)
        np.testing.assert_allclose(hid[i + 1], x, rtol=1e-10, atol=1e-12)


def test_fuse_then_cache_positions():
    """Context rows are appended in order at absolute positions; two fuse calls equal one."""
    s = SMALL
    w = synth.Workload("t", s, (13,), 0.8, scale_layers=False)
    W = synth.weights(w)
    a = O.DraftOracle(W, s, 1)
    a.fuse_context(0, synth.hidden_states(w, 0, 0, 13))
    b = O.DraftOracle(W, s, 1)
    b.fuse_context(0, synth.hidden_states(w, 0, 0, 8))
    b.fuse_context(0, synth.hidden_states(w, 0, 8, 5))
    for i in range(s.n_draft_layers):
        np.testing.assert_allclose(b.ctx_k[0][i], a.ctx_k[0][i], rtol=1e-13)
        np.testing.assert_allclose(b.ctx_v[0][i], a.ctx_v[0][i], rtol=1e-13)
