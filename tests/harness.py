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
# A ragged context fill: one call fills 700, 3 and 40 positions, so 5 of the 9 256-row token
# tiles of the context K/V projection hold no appended row (skipped); the LM head's 500 rows end
# inside the first tile of its second 256-row weight pair.
RAGGED = synth.Workload(
    "ragged_fill_bf16",
    synth.Shape(d=384, n_draft_layers=2, n_target_layers=3, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=512, vocab=500, block=8),
    (700, 3, 40), 0.8, seed=21)
# A context fill over many token tiles (2 layers x 8 weight tiles x 32 token tiles of 256 rows):
# the K/V projection skips the 11 token tiles past the shorter sequence.
LONG_FILL = synth.Workload(
    "long_fill_bf16",
    synth.Shape(d=256, n_draft_layers=2, n_target_layers=2, n_q_heads=8, n_kv_heads=4,
                head_dim=128, ffn=256, vocab=300, block=4),
    (4000, 1200), 0.8, seed=23)
# 240 LM-head rows (batch 16 x 15 mask positions) over a vocabulary of 297 weight tiles: the LM
# head pairs them (149 pairs run in one wave, the single tiles would take two), and the last
# pair's second tile lies past the matrix.
WIDE_VOCAB = synth.Workload(
    "wide_vocab_bf16_b16",
    synth.Shape(d=256, n_draft_layers=1, n_target_layers=1, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=256, vocab=38000, block=16),
    tuple(5 + (13 * b) % 29 for b in range(16)), 0.8, seed=25)
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
# 160 query rows per KV head (G 10, block 16): two 128-row query tiles of the tcgen05 attention,
# the second holding 32 rows, and three 64-row tiles of the mma.sync attention
QT2 = synth.Workload(
    "qt2_bf16_g10",
    synth.Shape(d=512, n_draft_layers=2, n_target_layers=2, n_q_heads=20, n_kv_heads=2,
                head_dim=64, ffn=512, vocab=600, block=16),
    (210, 77), 0.8, seed=20)
TINY = synth.preset("tiny_f32")


def rel_err(x, y):
    """Row-wise relative error: max over rows (vectors along the last axis) of ||x_r - y_r|| / ||y_r||."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    if not y.size:
        return 0.0
    num = np.sqrt(np.sum((x - y) ** 2, axis=-1))
    den = np.sqrt(np.sum(y * y, axis=-1))
    den = np.where(den == 0, 1.0, den)
    return float(np.max(num / den))


def elem_err(x, y, floor_frac: float):
    """Element-wise relative error: max_i |x_i - y_i| / max(|y_i|, floor_frac * rms(y)), rms over
    the whole compared tensor (the floor keeps elements that cancel to near zero from dividing
    by almost nothing)."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    if not y.size:
        return 0.0
    rms = float(np.sqrt(np.mean(y * y)))
    den = np.maximum(np.abs(y), max(floor_frac * rms, 1e-300))
    return float(np.max(np.abs(x - y) / den))


# Element-wise floors. bf16: 1e-3 rms; a tensor computed from the same input bytes on both sides
# differs only where the final bf16 rounding falls the other way (one ulp, <= 2^-7 relative).
# fp32: the tensor's rms; fp32 accumulation leaves an absolute error of a few ulp of the terms
# summed, so an element that cancels to 1e-3 rms carries ~1e-4 relative error on any fp32
# implementation, while |x - y| <= 1e-5 rms holds.
BF16_FLOOR = 1e-3
F32_FLOOR = 1.0


def tolerance(w: synth.Workload) -> float:
    return 2e-2 if w.shape.dtype == "bf16" else 1e-5


def check_elem(w: synth.Workload, x, y, what=""):
    """Element-wise check (floor per the storage type), with the row-wise error in the message."""
    floor = BF16_FLOOR if w.shape.dtype == "bf16" else F32_FLOOR
    e = elem_err(x, y, floor)
    assert e <= tolerance(w), (f"{what}: element-wise {e:.3e} (floor {floor} rms) > "
                               f"{tolerance(w)}; row-wise {rel_err(x, y):.3e}")
    return e


def check_rows(w: synth.Workload, x, y, what=""):
    """Hidden states and logits: element-wise in fp32; in bf16 row-wise, since every bf16 storage
    point of the layers (normalised rows, Q/K/V, attention output, SwiGLU product) can round an
    element to the neighbouring value and the next layer carries that ulp forward."""
    if w.shape.dtype != "bf16":
        return check_elem(w, x, y, what)
    r = rel_err(x, y)
    assert r <= tolerance(w), (f"{what}: row-wise {r:.3e} > {tolerance(w)}; element-wise "
                               f"{elem_err(x, y, BF16_FLOOR):.3e} (floor {BF16_FLOOR} rms)")
    return r


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

    def fuse(self, lens, pos0=None, want_fused=True, H=None):
        """One dflare_fuse_context call on the target states of positions pos0[b] .. + lens[b]
        (generated here, or the [T][batch][n_max][d] array H). Returns the fused rows."""
        torch = self.torch
        H = to_device(fill_hidden(self.w, lens, pos0) if H is None else H)
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


def check_kv(w: synth.Workload, o, k, v, F_gpu_i, pos, i, what=""):
    """Cached keys/values of draft layer i at absolute positions pos against Eq. 4 evaluated by the
    oracle on the GPU's own fused rows F_gpu_i (the same input bytes), element by element. (Against
    the oracle's own F they are compared row-wise: an F element rounded to the other bf16
    neighbour, a rate of ~1e-4 per element, moves every key of its position by ~1e-4 absolute,
    about 0.1 of a 1e-3 rms floor.)"""
    s = w.shape
    w_kv = o._dec("w_qkv", i)[s.d_q:] if o.shared_kv else o._dec("w_kv_ctx", i)
    kx, vx = O.context_kv(F_gpu_i, w_kv, np.asarray(pos), s.n_kv_heads, s.head_dim, s.rope_theta,
                          o.store)
    check_elem(w, k, kx, f"{what} K")
    check_elem(w, v, vx, f"{what} V")


GAP = 1e-2   # near-tie threshold of the token comparison (top-2 logit gap on the oracle's logits)


def check_tokens(w: synth.Workload, o, tok, logits, x_last, ot, ol, what=""):
    """Draft tokens of one sequence (Sec. 3.2, greedy drafting).

    - On the GPU's own fp32 logits the argmax (lowest id among equal maxima) is exact.
    - The LM head and argmax alone: the oracle's final RMSNorm, LM head and argmax applied to the
      GPU's last hidden state x_last give the GPU's tokens except where that oracle's top-2 gap is
      below GAP.
    - End to end, against the oracle's own chain: a token may differ only where the oracle's top-2
      gap is below max(GAP, 3 sqrt(2) rms(logits - oracle logits)) of that row, i.e. where the two
      competing logits' measured discrepancy explains the swap at 3 sigma. With bf16 storage the
      two chains' rounding decisions drift apart layer by layer (the row-wise logit difference of a
      d 4096, 8-layer drafter is ~1.3e-2 of the logits' norm, ~0.015 rms), so gaps a little above
      1e-2 are decided by rounding noise, not by the method.
    Returns the number of end-to-end mismatches (all of them inside the rule)."""
    s = w.shape
    np.testing.assert_array_equal(tok, O.argmax_lowest(logits), err_msg=f"{what}: argmax of own logits")
    hl = O.lm_head_logits(np.asarray(x_last, np.float64), o._dec("final_norm"), o._dec("lm_head"),
                          s.rms_eps, o.store)
    ht = O.argmax_lowest(hl)
    bad = (tok != ht) & (O.top2_gap(hl) >= GAP)
    assert not bad.any(), (f"{what}: LM head + argmax on the GPU's last hidden state differs at "
                           f"{np.nonzero(bad)[0].tolist()} (gaps {O.top2_gap(hl)[bad].tolist()})")
    mism = tok != ot
    if mism.any():
        sigma = np.sqrt(np.mean((np.asarray(logits, np.float64) - ol) ** 2, axis=-1))
        thr = np.maximum(GAP, 3 * np.sqrt(2) * sigma)
        gap = O.top2_gap(ol)
        out = mism & (gap >= thr)
        assert not out.any(), (f"{what}: tokens differ from the oracle at {np.nonzero(out)[0].tolist()} "
                               f"with gaps {gap[out].tolist()} above {thr[out].tolist()}")
    return int(mism.sum())


def verified_steps(w: synth.Workload, g: GpuSide, o, n_steps: int):
    """n_steps block steps on both sides: draft -> synthetic target -> prefix accept -> fuse the
    tau accepted positions. Both sides continue from the GPU's drafts (the synthetic target, tau and
    the next token are integer work on them: exact), so every step of every sequence is compared:
    hidden states after every layer, logits and tokens (check_tokens). Returns the number of
    (step, sequence) pairs compared."""
    import torch
    from paper_2606_02091_gb300 import synthetic_target
    s = w.shape
    x_t = synth.initial_tokens(w).astype(np.int64)
    thr = synth.accept_threshold(w.match_p)
    lens = [o.ctx_len(b) for b in range(w.batch)]
    step_ctr = torch.zeros(1, dtype=torch.int32, device="cuda")
    compared = 0
    for step in range(n_steps):
        tok, logits, hidden = g.draft(x_t)
        u, r, last = synth.target_draws(w, step)
        tgt = torch.zeros((w.batch, s.block), dtype=torch.int32, device="cuda")
        acc = torch.zeros(w.batch, dtype=torch.int32, device="cuda")
        nxt = torch.zeros(w.batch, dtype=torch.int32, device="cuda")
        dt = torch.tensor(tok, device="cuda")
        step_ctr.fill_(0)
        synthetic_target(dt, torch.tensor(u.view(np.int32), device="cuda"),
                         torch.tensor(r, device="cuda"), torch.tensor(last, device="cuda"),
                         step_ctr, thr, w.batch, s.block, tgt)
        g.lib.verify_accept(dt, tgt, acc, nxt)
        tgt_h, acc_h, nxt_h = tgt.cpu().numpy(), acc.cpu().numpy(), nxt.cpu().numpy()
        for b in range(w.batch):
            gt = O.synthetic_target(tok[b], u[0, b], r[0, b], last[0, b], thr)
            np.testing.assert_array_equal(tgt_h[b], gt)
            assert (acc_h[b], nxt_h[b]) == O.verify_accept(tok[b], gt)
            ot, ol, oh = o.draft_block(b, int(x_t[b]))
            for i in range(oh.shape[0]):
                check_rows(w, hidden[i, b], oh[i], f"step {step} seq {b} hidden after layer {i - 1}")
            check_rows(w, logits[b], ol, f"step {step} seq {b} logits")
            check_tokens(w, o, tok[b], logits[b], hidden[-1, b], ot, ol, f"step {step} seq {b}")
            compared += 1
        taus = [int(a) for a in acc_h]
        g.fuse(taus, pos0=lens, want_fused=False)
        for b in range(w.batch):
            o.fuse_context(b, synth.hidden_states(w, b, lens[b], taus[b]))
            lens[b] += taus[b]
        x_t = nxt_h.astype(np.int64)
        assert g.lib.ctx_lens() == lens
    assert g.lib.device_error() == 0
    return compared
