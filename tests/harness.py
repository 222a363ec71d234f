"""Shared test helpers: run a workload through the GPU library and through the oracle.

The two sides get the same seeded input bytes from ``synth``; neither sees the other's outputs.
"""
from __future__ import annotations

import dataclasses

import numpy as np

import oracle as O
import synth

# workloads small enough for the oracle in seconds, spanning several 128-feature tiles, ragged
# contexts, a vocabulary that is not a multiple of 4 and both head sizes
SMALL_HD128 = synth.Workload(
    "small_bf16_hd128",
    synth.Shape(d=512, n_draft_layers=3, n_target_layers=5, n_q_heads=8, n_kv_heads=2,
                head_dim=128, ffn=1472, vocab=3001, block=16),
    (100, 37, 250), 0.85, seed=11)
SMALL_HD64 = synth.Workload(
    "small_bf16_hd64",
    synth.Shape(d=384, n_draft_layers=2, n_target_layers=4, n_q_heads=8, n_kv_heads=2,
                head_dim=64, ffn=640, vocab=2048, block=8),
    (65, 300), 0.75, seed=12)
# many token rows per projection: batch 16 x block 16 = 256 rows (the widest GEMM token tile and
# a 240-row LM head), and block 32 (31 mask rows, two 64-row query tiles per KV head)
WIDE_B16 = synth.Workload(
    "wide_bf16_b16",
    synth.Shape(d=384, n_draft_layers=2, n_target_layers=3, n_q_heads=8, n_kv_heads=2,
                head_dim=64, ffn=640, vocab=1024, block=16),
    tuple(9 + (37 * b) % 61 for b in range(16)), 0.8, seed=13)
BLOCK32 = synth.Workload(
    "block32_bf16",
    synth.Shape(d=256, n_draft_layers=2, n_target_layers=3, n_q_heads=8, n_kv_heads=2,
                head_dim=128, ffn=512, vocab=1500, block=32),
    (90, 17), 0.8, seed=14)
# more token rows than one GEMM token tile holds: batch 9 x block 32 = 288 block rows (a 256-row
# tile and a ragged 32-row one in every draft projection) and 279 LM-head rows
MULTI_TILE = synth.Workload(
    "multi_tile_bf16_b9_B32",
    synth.Shape(d=256, n_draft_layers=2, n_target_layers=2, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=384, vocab=800, block=32),
    tuple(5 + (23 * b) % 67 for b in range(9)), 0.8, seed=19)
# degenerate and less common shapes: more draft layers than the fusion kernels hold at once
# (D 10), 128 query rows per KV head (G 8: two 64-row query tiles), a single fused target layer
# with block 1 (no mask rows: nothing is drafted), and block 2
D10 = synth.Workload(
    "d10_bf16",
    synth.Shape(d=256, n_draft_layers=10, n_target_layers=2, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=256, vocab=700, block=4),
    (33, 70), 0.8, seed=15)
G8 = synth.Workload(
    "g8_bf16_hd64",
    synth.Shape(d=512, n_draft_layers=2, n_target_layers=3, n_q_heads=16, n_kv_heads=2,
                head_dim=64, ffn=512, vocab=900, block=16),
    (150, 45), 0.75, seed=16)
BLOCK1 = synth.Workload(
    "block1_t1_bf16",
    synth.Shape(d=256, n_draft_layers=2, n_target_layers=1, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=256, vocab=300, block=1),
    (20, 1), 0.8, seed=17)
BLOCK2 = synth.Workload(
    "block2_bf16",
    synth.Shape(d=256, n_draft_layers=2, n_target_layers=2, n_q_heads=4, n_kv_heads=2,
                head_dim=128, ffn=256, vocab=300, block=2),
    (64, 129), 0.8, seed=18)
TINY = synth.preset("tiny_f32")


def rel_err(x, y):
    """Max relative error of the vectors along the last axis: max_r ||x_r - y_r|| / ||y_r||.

    A hidden state, a fused context row, a key or value head vector and a row of logits are each
    compared as one vector. Element-wise ratios are not used: bf16 storage rounding makes any
    upstream perturbation flip single elements by a full bf16 ulp, so near-zero elements of an
    otherwise accurate vector would dominate an element-wise maximum.
    """
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    if not y.size:
        return 0.0
    num = np.sqrt(np.sum((x - y) ** 2, axis=-1))
    den = np.sqrt(np.sum(y * y, axis=-1))
    den = np.where(den == 0, 1.0, den)
    return float(np.max(num / den))


def elem_err(x, y):
    """max_i |x_i - y_i| / max(|y_i|, rms(y)) (reported by the diagnostics, not asserted)."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    rms = float(np.sqrt(np.mean(y * y))) if y.size else 1.0
    return float(np.max(np.abs(x - y) / np.maximum(np.maximum(np.abs(y), rms), 1e-300)))


def tolerance(w: synth.Workload) -> float:
    return 2e-2 if w.shape.dtype == "bf16" else 1e-5


def to_device(a: np.ndarray):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a))
    if a.dtype == np.uint16:
        t = t.view(torch.bfloat16)
    return t.cuda()


def storage_name(w: synth.Workload) -> str:
    return "bf16" if w.shape.dtype == "bf16" else "exact"


def fill_hidden(w: synth.Workload, lens, pos0=None):
    """[T][batch][n_max][d] target states for positions pos0[b] .. pos0[b] + lens[b] - 1."""
    s = w.shape
    n_max = max(max(lens), 1)
    dt = np.uint16 if s.dtype == "bf16" else np.float32
    H = np.zeros((s.n_target_layers, w.batch, n_max, s.d), dt)
    for b, n in enumerate(lens):
        if n:
            H[:, b, :n] = synth.hidden_states(w, b, 0 if pos0 is None else pos0[b], n)
    return H


class GpuSide:
    """The library on one workload: weights uploaded, sequences reset."""

    def __init__(self, w: synth.Workload, flags: int = 0, max_ctx: int | None = None,
                 max_fuse_rows: int | None = None, weights: dict | None = None):
        import torch
        from paper_2606_02091_gb300 import DFlare
        self.w = w
        self.W = synth.weights(w) if weights is None else weights
        s = w.shape
        self.max_ctx = max_ctx or (max(w.ctx_lens) + 8 * s.block + 64)
        mfr = max_fuse_rows or w.batch * max(max(w.ctx_lens), s.block)
        self.lib = DFlare.from_shape(s, max_batch=w.batch, max_ctx=self.max_ctx,
                                     max_fuse_rows=mfr, flags=flags)
        self.dev = {k: to_device(v) for k, v in self.W.items()}
        self.lib.set_weights(self.dev)
        self.lib.reset(w.batch)
        self.torch = torch

    def fuse(self, lens, pos0=None, want_fused=True):
        torch = self.torch
        H = to_device(fill_hidden(self.w, lens, pos0))
        n_new = torch.tensor(list(lens), dtype=torch.int32, device="cuda")
        fused = None
        if want_fused:
            s = self.w.shape
            dt = torch.bfloat16 if s.dtype == "bf16" else torch.float32
            fused = torch.zeros((s.n_draft_layers, self.w.batch, H.shape[2], s.d), dtype=dt,
                                device="cuda")
        self.lib.fuse_context(H, n_new, fused)
        return fused

    def draft(self, last_tokens):
        torch = self.torch
        s = self.w.shape
        bsz = self.w.batch
        last = torch.tensor(np.asarray(last_tokens, np.int32), device="cuda")
        toks = torch.zeros((bsz, s.block - 1), dtype=torch.int32, device="cuda")
        logits = torch.zeros((bsz, s.block - 1, s.vocab), dtype=torch.float32, device="cuda")
        hidden = torch.zeros((s.n_draft_layers + 1, bsz, s.block, s.d), dtype=torch.float32,
                             device="cuda")
        self.lib.draft_block(last, toks, logits, hidden)
        torch.cuda.synchronize()
        return toks.cpu().numpy(), logits.cpu().numpy(), hidden.cpu().numpy()


def f64(t):
    """device tensor -> float64 numpy (bf16 widened exactly)."""
    import torch
    return t.detach().to(torch.float64).cpu().numpy()


def oracle_for(w: synth.Workload, W: dict, **kw):
    return O.DraftOracle(W, w.shape, w.batch, storage=storage_name(w), **kw)
