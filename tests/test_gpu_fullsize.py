"""Full-size parity in the benchmark's launch configuration, on every drafter shape the benchmark
runs: the context filled in 2048-position chunks as bench.py fills it, then two verified block
steps, against the float64 oracle with bf16 storage rounding.

Per workload: every fused row F (Eq. 3) element by element against the oracle on the same target
states; every cached key and value of every layer and sequence (Eq. 4) element by element against
the oracle's projection of the GPU's own F bytes, and row-wise against the oracle's cache built
from its own F; the hidden states after every layer and the logits (row-wise, bf16), draft tokens
(exact outside top-2 gaps below 1e-2), the synthetic target's predictions, tau and the next token
(exact) over two steps whose context grows by tau.

Workloads: Qwen3-4B-shaped (d 2560, D 5, T 36, L 2048, b 1); Qwen3-8B-shaped (d 4096, D 8, T 36)
at L 4096 b 1 and at the ragged batch 4 (contexts 2668, 2687, 3853, 1355); GPT-OSS-20B-shaped
(d 2880, D 8, T 24, 64 query / 8 KV heads of 64, vocab 201088, L 8192, b 2); and the long-context
point of the Qwen3-8B-shaped sweep, L 32768 at b 1, where the attention runs its most key tiles per
CTA. That point keeps 2 of the sweep centre's 8 draft layers so the float64 oracle's fill (about
1.1 TFLOP of context projections per draft layer at L 32768) stays within a minute; the attention
launch configuration depends on the context, batch and heads, not on the depth.
"""
import numpy as np
import pytest

import synth
from tests.harness import (GpuSide, check_elem, check_kv, check_rows, f64, fill_hidden,
                           oracle_for, verified_steps)

pytestmark = pytest.mark.gpu
CHUNK = 2048          # bench.py's context-fill chunk
ORACLE_ROWS = 256     # positions per oracle call (positions are independent in Eq. 3 and Eq. 4)

FULL = {
    "qwen3_4b": synth.preset("qwen3_4b"),
    "qwen3_8b_b1": synth.preset("qwen3_8b_b1"),
    "qwen3_8b_b4": synth.preset("qwen3_8b_b4"),
    "gptoss_20b_b2": synth.preset("gptoss_20b_b2"),
    "sweep_L32768_D2": synth.sweep_point(D=2, L=32768),
}


@pytest.mark.parametrize("name", list(FULL))
def test_full_size_fill_and_steps(name):
    w = FULL[name]
    s = w.shape
    L_max = max(w.ctx_lens)
    g = GpuSide(w, max_ctx=L_max + 4 * s.block + 64, max_fuse_rows=w.batch * max(CHUNK, s.block))
    o = oracle_for(w, g.W)
    for pos0 in range(0, L_max, CHUNK):
        ns = [max(0, min(CHUNK, L - pos0)) for L in w.ctx_lens]
        H = fill_hidden(w, ns, [pos0] * w.batch)
        fused = f64(g.fuse(ns, H=H))
        for b, n in enumerate(ns):
            for r0 in range(0, n, ORACLE_ROWS):
                r1 = min(n, r0 + ORACLE_ROWS)
                F = o.fuse_context(b, H[:, b, r0:r1])
                check_elem(w, fused[:, b, r0:r1], F, f"F seq {b} rows {pos0 + r0}..{pos0 + r1}")
                pos = np.arange(pos0 + r0, pos0 + r1)
                for i in range(s.n_draft_layers):
                    k, v = g.lib.read_kv(i, b, pos0 + r0, r1 - r0)
                    check_kv(w, o, f64(k), f64(v), fused[i, b, r0:r1], pos, i,
                             f"seq {b} layer {i} rows {pos0 + r0}..{pos0 + r1}")
        del H, fused
    assert g.lib.ctx_lens() == list(w.ctx_lens)
    for b, L in enumerate(w.ctx_lens):
        for i in range(s.n_draft_layers):
            k, v = g.lib.read_kv(i, b, 0, L)
            check_rows(w, f64(k), o.ctx_k[b][i], f"seq {b} layer {i} K (end to end)")
            check_rows(w, f64(v), o.ctx_v[b][i], f"seq {b} layer {i} V (end to end)")
    assert verified_steps(w, g, o, n_steps=2) >= w.batch
    assert g.lib.device_error() == 0
