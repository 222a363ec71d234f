"""Input recipes: drafter shapes, workloads and the distributions of every input tensor.

Distributions (the synthetic stand-ins for trained weights and for a real target model):
- every weight matrix and the embedding / LM-head tables: N(0, 0.02^2);
- every RMSNorm gain: 1 + N(0, 0.02^2) (a gain near 1, as in a trained model; gains near 0.02
  would collapse all logits into ties);
- fusion logits W^fuse (D x T, fp32): N(0, 1);
- target hidden states: N(0, 1), times one scale s_j ~ U(0.5, 4) per target layer j when the
  workload asks for layer scaling (all bf16 workloads), shared by all positions and sequences;
- first target decode token of each sequence: uniform over [0, V-1) (never the mask token V-1);
- the synthetic target used for verification: for draft row k (1..B-1) the target's prediction
  g_{k-1} equals the draft token d_k when a uniform uint32 u_k is below floor(p * 2^32),
  otherwise it is r_k + (r_k >= d_k) with r_k uniform over [0, V-1), i.e. a uniform token that
  differs from d_k; g_{B-1} is uniform over [0, V).

Element indexing is fixed per tensor so that any slice can be regenerated on its own: target
hidden states of layer j and sequence b are one stream indexed by position * d + k.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import numpy as np

from . import gen


@dataclass(frozen=True)
class Shape:
    """A drafter's architecture."""

    d: int                  # hidden size
    n_draft_layers: int     # D
    n_target_layers: int    # T
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    block: int              # B
    rms_eps: float = 1e-6
    rope_theta: float = 1e6
    dtype: str = "bf16"     # "bf16" or "f32": storage type of weights and activations

    @property
    def d_q(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def d_kv(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def mask_token_id(self) -> int:
        return self.vocab - 1


@dataclass(frozen=True)
class Workload:
    name: str
    shape: Shape
    ctx_lens: tuple          # context length L_b of each sequence before the first block step
    match_p: float           # probability that the synthetic target agrees with a draft token
    seed: int = 0
    scale_layers: bool = True   # scale target layer j by s_j ~ U(0.5, 4)

    @property
    def batch(self) -> int:
        return len(self.ctx_lens)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


TINY = Shape(d=256, n_draft_layers=4, n_target_layers=8, n_q_heads=4, n_kv_heads=2, head_dim=64,
             ffn=768, vocab=4096, block=8, dtype="f32")
Q3_4B = Shape(d=2560, n_draft_layers=5, n_target_layers=36, n_q_heads=32, n_kv_heads=8,
              head_dim=128, ffn=9728, vocab=151936, block=16)
Q3_8B = Shape(d=4096, n_draft_layers=8, n_target_layers=36, n_q_heads=32, n_kv_heads=8,
              head_dim=128, ffn=12288, vocab=151936, block=16)
GPTOSS = Shape(d=2880, n_draft_layers=8, n_target_layers=24, n_q_heads=64, n_kv_heads=8,
               head_dim=64, ffn=2880 * 4, vocab=201088, block=16)


def _ragged_lens(seed: int, batch: int, lo: int, hi: int) -> tuple:
    return tuple(int(x) for x in gen.randint(seed, "ctx_len", (batch,), lo, hi + 1))


PRESETS = {
    # tiny fp32 drafter: context 128, batch 1, block 8, match probability 0.8
    "tiny_f32": Workload("tiny_f32", TINY, (128,), 0.8, scale_layers=False),
    # Qwen3-4B-shaped drafter: context 2048, batch 1, block 16
    "qwen3_4b": Workload("qwen3_4b", Q3_4B, (2048,), 0.85),
    # Qwen3-8B-shaped drafter: context 4096, batch 1; and batch 4 with lengths U{1024..4096}
    "qwen3_8b_b1": Workload("qwen3_8b_b1", Q3_8B, (4096,), 0.85),
    "qwen3_8b_b4": Workload("qwen3_8b_b4", Q3_8B, _ragged_lens(0, 4, 1024, 4096), 0.85),
    # GPT-OSS-20B-shaped drafter: context 8192, batch 2
    "gptoss_20b_b2": Workload("gptoss_20b_b2", GPTOSS, (8192, 8192), 0.75),
}


def preset(name: str) -> Workload:
    return PRESETS[name]


def sweep_point(*, D: int = 8, T: int = 36, B: int = 16, L: int = 4096, batch: int = 1,
                p: float = 0.85, seed: int = 0) -> Workload:
    """One point of the sweep around the Qwen3-8B shape (defaults are its centre)."""
    shp = dataclasses.replace(Q3_8B, n_draft_layers=D, n_target_layers=T, block=B)
    return Workload(f"sweep_D{D}_T{T}_B{B}_L{L}_b{batch}_p{p}", shp, (L,) * batch, p, seed)


def _mat(w: Workload, name: str, shape, mean=0.0, std=0.02):
    return gen.normal(w.seed, name, shape, mean=mean, std=std, dtype=w.shape.dtype)


def weights(w: Workload) -> dict:
    """All draft weights in the stacked row-major layout the library documents.

    Linear maps are stored as [out_features][in_features]; per-layer tensors are stacked over
    the D draft layers. bf16 tensors are uint16 bit arrays, fp32 tensors float32 arrays.
    """
    s = w.shape
    D, d, F = s.n_draft_layers, s.d, s.ffn
    return {
        "fuse_logits": gen.normal(w.seed, "fuse_logits", (D, s.n_target_layers), dtype="f32"),
        "fuse_norm": _mat(w, "fuse_norm", (D, d), mean=1.0),
        "w_kv_ctx": _mat(w, "w_kv_ctx", (D, 2 * s.d_kv, d)),
        "attn_norm": _mat(w, "attn_norm", (D, d), mean=1.0),
        "w_qkv": _mat(w, "w_qkv", (D, s.d_q + 2 * s.d_kv, d)),
        "w_o": _mat(w, "w_o", (D, d, s.d_q)),
        "mlp_norm": _mat(w, "mlp_norm", (D, d), mean=1.0),
        "w_gate": _mat(w, "w_gate", (D, F, d)),
        "w_up": _mat(w, "w_up", (D, F, d)),
        "w_down": _mat(w, "w_down", (D, d, F)),
        "final_norm": _mat(w, "final_norm", (d,), mean=1.0),
        "embed": _mat(w, "embed", (s.vocab, d)),
        "lm_head": _mat(w, "lm_head", (s.vocab, d)),
    }


def variant_weights(w: Workload) -> dict:
    """Extra weights of the "+FC" ablation and of DFlash's FC fusion, stacked like ``weights``:
    fusion_fc_w [D][d][d] and dflash_fc_w [d][T d] ~ N(0, (1/sqrt(fan_in))^2) (a unit-scale
    output for unit-scale inputs), the biases fusion_fc_b [D][d] and dflash_fc_b [d] ~
    N(0, 0.02^2)."""
    s = w.shape
    D, T, d = s.n_draft_layers, s.n_target_layers, s.d
    return {
        "fusion_fc_w": _mat(w, "fusion_fc_w", (D, d, d), std=d ** -0.5),
        "fusion_fc_b": _mat(w, "fusion_fc_b", (D, d)),
        "dflash_fc_w": _mat(w, "dflash_fc_w", (d, T * d), std=(T * d) ** -0.5),
        "dflash_fc_b": _mat(w, "dflash_fc_b", (d,)),
    }


def layer_scales(w: Workload) -> np.ndarray:
    """Per-target-layer scale s_j ~ U(0.5, 4) (ones when the workload does not scale)."""
    T = w.shape.n_target_layers
    if not w.scale_layers:
        return np.ones(T)
    return 0.5 + 3.5 * gen.uniform(w.seed, "hidden_scale", (T,))


def hidden_states(w: Workload, b: int, pos0: int, n: int, out: np.ndarray | None = None) -> np.ndarray:
    """Target hidden states of sequence b at absolute positions [pos0, pos0 + n): [T][n][d]."""
    s = w.shape
    T, d = s.n_target_layers, s.d
    dt = np.uint16 if s.dtype == "bf16" else np.float32
    if out is None:
        out = np.empty((T, n, d), dt)
    sc = layer_scales(w)
    for j in range(T):
        gen.normal(w.seed, f"hidden/b{b}/j{j}", (n, d), std=float(sc[j]), dtype=s.dtype,
                   offset=pos0 * d, out=out[j])
    return out


def initial_tokens(w: Workload) -> np.ndarray:
    """The first target decode token x_t of each sequence, uniform over [0, V-1)."""
    return gen.randint(w.seed, "x_t", (w.batch,), 0, w.shape.vocab - 1)


def accept_threshold(p: float) -> int:
    """floor(p * 2^32): a uniform uint32 below it has probability p (integer test on both sides)."""
    return min(int(np.floor(p * 4294967296.0)), 0xFFFFFFFF)


def target_draws(w: Workload, step: int, n_steps: int = 1):
    """Random draws of the synthetic target for block steps [step, step + n_steps).

    Returns (u [n][batch][B-1] uint32, r [n][batch][B-1] int32 in [0, V-1),
    last [n][batch] int32 in [0, V)).
    """
    bsz, B, V = w.batch, w.shape.block, w.shape.vocab
    shp = (n_steps, bsz, B - 1)
    off = step * bsz * (B - 1)
    u = gen.uniform_u32(w.seed, "target_u", shp, offset=off)
    r = gen.randint(w.seed, "target_r", shp, 0, V - 1, offset=off)
    last = gen.randint(w.seed, "target_last", (n_steps, bsz), 0, V, offset=step * bsz)
    return u, r, last
