"""The benchmark's roofline numerators (algorithmic bytes per launch) against the weight and cache
sizes computed independently from the drafter's shape: every GEMM streams its weights once, the
attention reads the context keys/values once, the argmax reads the logits once."""
import numpy as np
import pytest

import bench
import synth

GEMMS = {"gemm_qkv": "D", "gemm_o": "D", "gemm_gate_up": "D", "gemm_down": "D",
         "gemm_kv_ctx": 1, "gemm_lm_head": 1}


def _weight_bytes(s):
    e = 2 if s.dtype == "bf16" else 4
    per_layer = (s.d_q + 2 * s.d_kv) * s.d + s.d * s.d_q + 3 * s.d * s.ffn + 2 * s.d_kv * s.d
    return e * (s.n_draft_layers * per_layer + s.vocab * s.d)


@pytest.mark.parametrize("name", ["qwen3_4b", "qwen3_8b_b4", "gptoss_20b_b2"])
def test_gemm_bytes_are_the_weights_plus_small_activations(name):
    w = synth.preset(name)
    s = w.shape
    tau = 6.0
    total = 0.0
    for k, n in GEMMS.items():
        launches = s.n_draft_layers if n == "D" else n
        total += launches * bench.algorithmic_bytes(w, k, tau)
    weights = _weight_bytes(s)
    # activations (inputs, outputs, the fp32 residual) add a few per cent at 16..64 token rows
    assert weights <= total <= 1.05 * weights, (total, weights)


def test_qwen3_4b_step_bytes_and_lower_bound():
    """The Qwen3-4B-shaped step: 1.858 GB of GEMM bytes (weights 1.857 GB), 1.91 GB in all, so
    0.28 ms at the measured 6785 GB/s copy bandwidth."""
    w = synth.preset("qwen3_4b")
    s = w.shape
    tau = 6.4
    gemm = sum((s.n_draft_layers if n == "D" else n) * bench.algorithmic_bytes(w, k, tau)
               for k, n in GEMMS.items())
    assert abs(gemm - 1.858e9) < 0.002e9
    kv = bench.algorithmic_bytes(w, "attention", tau)
    # context keys and values of one layer: (L + B) positions x 2 x d_kv x 2 bytes, plus Q and O
    L = float(np.mean(w.ctx_lens))
    assert kv == pytest.approx((L + s.block) * 2 * s.d_kv * 2 + 2 * s.block * s.d_q * 2)
    step = gemm + s.n_draft_layers * kv + bench.algorithmic_bytes(w, "argmax", tau) + \
        bench.algorithmic_bytes(w, "fuse_layers", tau)
    assert abs(step - 1.91e9) < 0.01e9
    assert abs(step / 6785.2e9 * 1e3 - 0.282) < 0.002


def test_argmax_reads_the_mask_rows_logits_once():
    w = synth.preset("qwen3_4b")
    s = w.shape
    assert bench.algorithmic_bytes(w, "argmax", 6.0) == w.batch * (s.block - 1) * s.vocab * 4
