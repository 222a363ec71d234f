"""Full-size parity in the benchmark's launch configuration: the Qwen3-4B-shaped drafter (d 2560,
5 draft layers, 36 fused target layers, vocab 151936, context 2048, block 16, batch 1), filled
in 2048-position chunks like bench.py, then one block step, against the float64 oracle with bf16
storage rounding. The other full-size shapes are checked on sampled rows (fused context and
cached keys/values at sampled positions, each computed by the oracle on its own)."""
import numpy as np
import pytest

import oracle as O
import synth
from tests.harness import GpuSide, f64, oracle_for, rel_err, tolerance

pytestmark = pytest.mark.gpu
GAP = 1e-2


def test_qwen3_4b_full_step():
    w = synth.preset("qwen3_4b")
    g = GpuSide(w, max_ctx=4096, max_fuse_rows=2048)
    fused = g.fuse(w.ctx_lens)
    x_t = synth.initial_tokens(w)
    tok, logits, hidden = g.draft(x_t)
    o = oracle_for(w, g.W)
    F = o.fuse_context(0, synth.hidden_states(w, 0, 0, w.ctx_lens[0]))
    assert rel_err(f64(fused)[:, 0], F) <= tolerance(w)
    for i in range(w.shape.n_draft_layers):
        k, v = g.lib.read_kv(i, 0, 0, w.ctx_lens[0])
        assert rel_err(f64(k), o.ctx_k[0][i]) <= tolerance(w), ("K", i)
        assert rel_err(f64(v), o.ctx_v[0][i]) <= tolerance(w), ("V", i)
    ot, ol, oh = o.draft_block(0, int(x_t[0]))
    for i in range(oh.shape[0]):
        assert rel_err(hidden[i, 0], oh[i]) <= tolerance(w), ("hidden", i)
    assert rel_err(logits[0], ol) <= tolerance(w)
    keep = O.top2_gap(ol) >= GAP
    np.testing.assert_array_equal(tok[0][keep], ot[keep])
    np.testing.assert_array_equal(tok[0], O.argmax_lowest(logits[0]))
    assert g.lib.device_error() == 0


@pytest.mark.parametrize("name", ["qwen3_8b_b4", "gptoss_20b_b2"])
def test_sampled_rows_full_size(name):
    """Fill the whole ragged context of the full-size workload and check sampled positions of
    every sequence: the fused context (Eq. 3) and every layer's cached K/V (Eq. 4)."""
    w = synth.preset(name)
    s = w.shape
    chunk = 1024
    g = GpuSide(w, max_ctx=max(w.ctx_lens) + 64, max_fuse_rows=w.batch * chunk)
    import torch
    last_fused = None
    for pos0 in range(0, max(w.ctx_lens), chunk):
        ns = [max(0, min(chunk, L - pos0)) for L in w.ctx_lens]
        last_fused = (pos0, ns, g.fuse(ns, pos0=[pos0] * w.batch))
    assert g.lib.ctx_lens() == list(w.ctx_lens)
    o = oracle_for(w, g.W)
    rng = np.random.default_rng(0)
    pos0, ns, fused = last_fused
    fused = f64(fused)
    for b, L in enumerate(w.ctx_lens):
        # fused rows of the last chunk (the kernel's output buffer of that call)
        if ns[b]:
            r = int(rng.integers(0, ns[b]))
            h = synth.hidden_states(w, b, pos0 + r, 1)
            Fo = O.fuse_context(O.decode(h, s.dtype), o.alpha, o._dec("fuse_norm"), s.rms_eps,
                                o.store)
            assert rel_err(fused[:, b, r], Fo[:, 0]) <= tolerance(w)
        # cached K/V rows at sampled absolute positions, all layers
        for p in list(rng.integers(0, L, 3)) + [L - 1]:
            p = int(p)
            h = synth.hidden_states(w, b, p, 1)
            Fo = O.fuse_context(O.decode(h, s.dtype), o.alpha, o._dec("fuse_norm"), s.rms_eps,
                                o.store)
            for i in range(s.n_draft_layers):
                ko, vo = O.context_kv(Fo[i], o._dec("w_kv_ctx", i), np.array([p]), s.n_kv_heads,
                                      s.head_dim, s.rope_theta, o.store)
                k, v = g.lib.read_kv(i, b, p, 1)
                assert rel_err(f64(k), ko) <= tolerance(w), (b, p, i, "K")
                assert rel_err(f64(v), vo) <= tolerance(w), (b, p, i, "V")
    assert g.lib.device_error() == 0
    del torch
