"""Plain CPU oracle of the DFlare per-step draft path -- test infrastructure, not product code.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
this module. The GPU library (``paper_2606_02091_gb300``) never imports it, and the two share no
code: no kernels, helpers, tables or constants. Their only common dependency is the seeded input
generator in ``synth/``, which holds none of the method's arithmetic.

Everything is evaluated in float64 with numpy, one definition at a time, in the paper's order
and notation (arxiv 2606.02091):

* Eq. 3 (Sec. 4.1, adaptive layer fusion): alpha^(i) = softmax(W^fuse_{i,:});
  f_t^(i) = RMSNorm(sum_j alpha_j^(i) h_t^(j)).
* Eq. 4 (Sec. 4.2, heterogeneous KV projections): context keys/values come from F^(i) through
  W_K^t / W_V^t; the block's own keys/values from [x_t; X_hat] through W_K^d / W_V^d;
  queries Q = [x_t; X_hat] W_Q.
* Sec. 3.2 (drafting phase): the block is the target decode token x_t followed by B-1 mask
  positions; attention is bidirectional over [context ; block]; only the B block rows pass from
  layer to layer; logits are taken at the mask positions and greedy drafting takes the argmax.
* Sec. 3.2 (verification phase): accept the longest prefix of drafts that matches the target's
  own predictions, plus one token from the target.
* Variants measured against DFlare: the ablations of Sec. 6.3 / Table 2 ("-Softmax", "-KVProj",
  "+FC") and DFlash's FC fusion (Eq. 1) with one shared KV projection (Eq. 2).
* Sampled decoding (Table 1, temperature 1): drafts drawn from softmax(logits / T) and verified
  by the speculative-sampling rejection rule (the rule is not stated in the paper; see the
  sampling section below).

Where the paper is silent the oracle takes these readings:
pre-norm residual blocks (RMSNorm -> attention -> residual; RMSNorm -> SwiGLU MLP -> residual)
and a final RMSNorm before the LM head; RMSNorm y = g * x / sqrt(mean(x^2) + eps) with one gain
vector per norm; no biases and no QK-norm; rotate-half RoPE on queries and keys, context row r
at position r, block row k at position L + k, context keys cached after rotation; grouped-query
heads in contiguous groups; softmax scale 1/sqrt(head_dim); mask token id V-1; argmax ties go to
the lowest token id.

Storage precision. ``store`` is applied where the GPU path stores a tensor in its storage type:
the fused context F, the cached context keys and values, the normalised activations fed to each
projection, Q / K^d / V^d, the attention output and the SwiGLU product. With ``store=round_bf16``
this is the bf16 path's storage rounding (round to nearest even, from the exact float64 value);
with ``store=exact`` nothing is rounded (the fp32 path's reference). The residual stream and the
logits are never rounded.

Pins (tests/test_oracle_*.py): every function here is checked against something other than
itself -- closed forms, invariants of the definitions, reductions to library routines
(torch's scaled_dot_product_attention, torch's bf16 cast), and brute force on tiny inputs.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64


# --------------------------------------------------------------------------- storage helpers

def exact(x):
    """Storage without rounding (the fp32 path's reference)."""
    return x


def round_bf16(x):
    """Round float64 values to the nearest bfloat16 value (8 significant bits), ties to even.

    x = m * 2^e with 0.5 <= |m| < 1 (frexp); m * 2^8 is rounded to an integer (numpy's round is
    half-to-even) and scaled back. Exact in float64 for every normal bf16 magnitude.
    """
    x = np.asarray(x, F64)
    m, e = np.frexp(x)
    return np.ldexp(np.round(np.ldexp(m, 8)), e - 8)


def decode(a, dtype: str):
    """Input bytes -> float64: bf16 bit patterns (uint16) or float32 values."""
    a = np.asarray(a)
    if dtype == "bf16":
        return (a.astype(np.uint32) << 16).view(np.float32).astype(F64)
    return a.astype(F64)


# --------------------------------------------------------------------------- Eq. 3

def fusion_weights(w_fuse, softmax: bool = True):
    """alpha^(i) = softmax(W^fuse_{i,:}) over the T target layers (Eq. 3, first line).

    softmax=False keeps the raw weights: the "-Softmax" ablation of Sec. 6.3 / Table 2.
    The softmax subtracts the row maximum first (the same value in exact arithmetic).
    """
    w = np.asarray(w_fuse, F64)
    if not softmax:
        return w.copy()
    z = np.exp(w - w.max(axis=1, keepdims=True))
    return z / z.sum(axis=1, keepdims=True)


def rms_norm(x, gain, eps: float):
    """RMSNorm over the last axis: gain * x / sqrt(mean(x^2) + eps)."""
    x = np.asarray(x, F64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return np.asarray(gain, F64) * x / np.sqrt(ms + eps)


def fuse_context(hidden, alpha, fuse_gain, eps: float, store=exact):
    """Eq. 3, second line, for every draft layer i and position t.

    hidden: [T][n][d] target states h_t^(j); alpha: [D][T]; fuse_gain: [D][d].
    Returns F: [D][n][d], F[i][t] = RMSNorm_i(sum_j alpha[i, j] * hidden[j][t]).
    """
    hidden = np.asarray(hidden, F64)
    D, T = alpha.shape
    # s^(i) = sum_j alpha[i, j] h^(j) for every i at once: the [D][T] weights times the T target
    # states taken as a [T][n d] matrix
    rest = hidden.shape[1:]
    s = (np.asarray(alpha, F64) @ hidden.reshape(T, int(np.prod(rest)))).reshape((D,) + rest)
    out = np.empty((D,) + hidden.shape[1:], F64)
    for i in range(D):
        out[i] = store(rms_norm(s[i], fuse_gain[i], eps))
    return out


# --------------------------------------------------------------------------- positions

def rope(x, positions, theta: float):
    """Rotate-half rotary embedding of x: [n][heads][hd] at integer positions [n].

    Pair (x_j, x_{j+hd/2}) is the complex number x_j + i x_{j+hd/2}, multiplied by
    exp(i * pos * theta^(-2j/hd)) for j = 0 .. hd/2 - 1.
    """
    x = np.asarray(x, F64)
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-2.0 * np.arange(half) / hd)
    ang = np.asarray(positions, F64)[:, None] * inv_freq[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


# --------------------------------------------------------------------------- Eq. 4 (context)

def context_kv(F_i, w_kv_ctx_i, positions, n_kv_heads: int, head_dim: int, theta: float,
               store=exact):
    """Context keys/values of draft layer i (Eq. 4): K^t = F^(i) W_K^t, V^t = F^(i) W_V^t.

    w_kv_ctx_i: [2 d_kv][d], rows [0, d_kv) hold W_K^t as out x in, rows [d_kv, 2 d_kv) W_V^t.
    Keys are rotated at their absolute positions before they are cached.
    Returns (K [n][H_kv][hd], V [n][H_kv][hd]).
    """
    F_i = np.asarray(F_i, F64)
    d_kv = n_kv_heads * head_dim
    n = F_i.shape[0]
    k = (F_i @ w_kv_ctx_i[:d_kv].T).reshape(n, n_kv_heads, head_dim)
    v = (F_i @ w_kv_ctx_i[d_kv:].T).reshape(n, n_kv_heads, head_dim)
    return store(rope(k, positions, theta)), store(v)


# --------------------------------------------------------------------------- Sec. 6.3 / Eq. 1 variants

def fusion_fc(F_i, w_fc_i, b_fc_i, store=exact):
    """The "+FC" ablation of Sec. 6.3 (Table 2): one more fully-connected layer applied to the
    fused context of draft layer i before it is projected, F'^(i)_t = W_fc^(i) f_t^(i) + b_fc^(i).

    F_i: [n][d]; w_fc_i: [d][d] (out x in); b_fc_i: [d]. Returns F'^(i): [n][d].
    """
    F_i = np.asarray(F_i, F64)
    return store(F_i @ np.asarray(w_fc_i, F64).T + np.asarray(b_fc_i, F64))


def dflash_context(hidden, w_fc, b_fc, store=exact):
    """DFlash's context feature (Eq. 1): c_t = W_fc [h_t^(1); ...; h_t^(T)] + b_fc.

    hidden: [T][n][d]; w_fc: [d][T d], so column j d + e multiplies element e of h_t^(j+1);
    b_fc: [d]. Returns C: [n][d], one row per position, shared by every draft layer (Eq. 2).
    """
    hidden = np.asarray(hidden, F64)
    T = hidden.shape[0]
    concat = np.concatenate([hidden[j] for j in range(T)], axis=-1)   # [n][T d]
    return store(concat @ np.asarray(w_fc, F64).T + np.asarray(b_fc, F64))


# --------------------------------------------------------------------------- Sec. 3.2 block

def silu(x):
    """SiLU(x) = x / (1 + exp(-x))."""
    x = np.asarray(x, F64)
    return x / (1.0 + np.exp(-x))


def block_attention(q, k, v):
    """Bidirectional softmax attention of every block query over every key (Sec. 3.2).

    q: [B][H_q][hd]; k, v: [S][H_kv][hd] (S = context + block rows). No mask of any kind.
    Query head h reads key/value head h // (H_q / H_kv). Scores are scaled by 1/sqrt(hd).
    """
    q, k, v = (np.asarray(a, F64) for a in (q, k, v))
    B, Hq, hd = q.shape
    Hkv = k.shape[1]
    G = Hq // Hkv
    out = np.empty_like(q)
    for h in range(Hq):
        g = h // G
        s = (q[:, h, :] @ k[:, g, :].T) / np.sqrt(hd)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, g, :]
    return out


def draft_layer(x, lw: dict, ctx_k, ctx_v, positions, shape, store=exact, rope_block: bool = True):
    """One draft layer over the B block rows x: [B][d] (Sec. 3.2 with Eq. 4).

    lw: this layer's float64 weights attn_norm [d], w_qkv [d_q + 2 d_kv][d], w_o [d][d_q],
    mlp_norm [d], w_gate / w_up [F][d], w_down [d][F]. ctx_k / ctx_v: this layer's context
    cache [L][H_kv][hd]. positions: the block rows' positions [B].
    """
    B = x.shape[0]
    Hq, Hkv, hd = shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    d_q, d_kv = Hq * hd, Hkv * hd
    # attention sub-layer: Q = [x_t; X_hat] W_Q and the block's K^d, V^d from W_K^d, W_V^d
    xn = store(rms_norm(x, lw["attn_norm"], shape.rms_eps))
    qkv = xn @ lw["w_qkv"].T
    q = qkv[:, :d_q].reshape(B, Hq, hd)
    kd = qkv[:, d_q:d_q + d_kv].reshape(B, Hkv, hd)
    vd = qkv[:, d_q + d_kv:].reshape(B, Hkv, hd)
    if rope_block:
        q = rope(q, positions, shape.rope_theta)
        kd = rope(kd, positions, shape.rope_theta)
    q, kd, vd = store(q), store(kd), store(vd)
    keys = np.concatenate([ctx_k, kd], axis=0)      # K = [F W_K^t ; x_t W_K^d ; X_hat W_K^d]
    vals = np.concatenate([ctx_v, vd], axis=0)      # V likewise (Eq. 4)
    o = store(block_attention(q, keys, vals).reshape(B, d_q))
    x = x + o @ lw["w_o"].T
    # MLP sub-layer: SwiGLU
    xm = store(rms_norm(x, lw["mlp_norm"], shape.rms_eps))
    a = store(silu(xm @ lw["w_gate"].T) * (xm @ lw["w_up"].T))
    return x + a @ lw["w_down"].T


def lm_head_logits(x, final_norm, lm_head, eps: float, store=exact):
    """Logits at the mask rows (block rows 1..B-1) after the final RMSNorm (Sec. 3.2)."""
    h = store(rms_norm(x[1:], final_norm, eps))
    return h @ np.asarray(lm_head, F64).T


def argmax_lowest(logits):
    """Greedy token choice per row; among equal maxima the lowest token id wins."""
    logits = np.asarray(logits)
    return np.argmax(logits, axis=-1).astype(np.int64)   # numpy returns the first maximum


def top2_gap(logits):
    """Largest minus second-largest logit of each row."""
    s = np.sort(np.asarray(logits, F64), axis=-1)
    return s[..., -1] - s[..., -2]


# --------------------------------------------------------------------------- verification

def verify_accept(draft, target):
    """Prefix acceptance (Sec. 3.2, verification phase) for one sequence.

    draft: the B-1 drafted tokens d_1..d_{B-1}. target: the target's B predictions
    g_0..g_{B-1}, where g_k is its argmax after block row k (so g_{k-1} checks d_k).
    Returns (tau, next_token): tau = a + 1 where a is the length of the longest prefix with
    d_k == g_{k-1} for all k <= a, and next_token = g_a, the target's extra token.
    """
    B = len(target)
    a = 0
    while a < B - 1 and draft[a] == target[a]:
        a += 1
    return a + 1, int(target[a])


def verify_from_logits(draft, target_logits):
    """Verification with the target's greedy predictions taken from its logits (Sec. 3.2):
    g_k = argmax_v target_logits[k][v] (lowest id among equal maxima), then ``verify_accept``."""
    return verify_accept(draft, argmax_lowest(target_logits))


def synthetic_target(draft, u, r, last, threshold: int):
    """Stand-in for the target's verification argmax (not part of the method).

    For k = 1..B-1: g_{k-1} = d_k if u_k < threshold, else r_k + (r_k >= d_k) (a uniform token
    different from d_k); g_{B-1} = last.
    """
    draft = np.asarray(draft, np.int64)
    u = np.asarray(u, np.uint64)
    r = np.asarray(r, np.int64)
    g = np.where(u < threshold, draft, r + (r >= draft))
    return np.concatenate([g, [int(last)]]).astype(np.int64)


# --------------------------------------------------------------------------- sampling (Table 1, temperature 1)
#
# Table 1 also reports sampled decoding (temperature 1) without stating its acceptance rule. The
# oracle takes the rule of the speculative-sampling works the paper builds on: draft token d_k is
# accepted with probability min(1, p(d_k) / q(d_k)), where p is the target's and q the draft's
# distribution at that position; at the first rejection the replacement token is drawn from
# max(0, p - q) renormalised, and when every draft is accepted the extra token is drawn from the
# target's distribution after the last block row. Draws use the Gumbel-max form
# argmax_v (log w_v + G_v), G_v = -log(-log u_v), which samples v with probability w_v / sum w.
#
# Random numbers: the uniforms of stream (purpose, step, row) are cut from Philox4x64-10 words
# (Salmon, Moraes, Dror, Shaw, SC'11): element v comes from word (v div 2) mod 4 of the block at
# counter (1 + v div 8, row, step, purpose) under key (seed, 0), bits 63..41 for even v and
# bits 31..9 for odd v, as (23-bit integer + 1/2) 2^-23, a value in (0, 1) that fp32 represents
# exactly.

RNG_DRAFT, RNG_ACCEPT, RNG_RESIDUAL = 1, 2, 3
_M64 = (1 << 64) - 1
PHILOX_MUL = (0xD2E7470EE14C6C93, 0xCA5A826395121157)
PHILOX_WEYL = (0x9E3779B97F4A7C15, 0xBB67AE8584CAA73B)


def philox4x64(counter, key, rounds: int = 10):
    """One Philox4x64 block from its definition (Python integers): each round multiplies words 0
    and 2 by the two round multipliers (128-bit products split into high and low halves) and
    mixes them with words 1 and 3 and the key; the key is advanced by the two Weyl constants
    between rounds."""
    c = [int(x) & _M64 for x in counter]
    k = [int(x) & _M64 for x in key]
    for r in range(rounds):
        if r:
            k = [(k[0] + PHILOX_WEYL[0]) & _M64, (k[1] + PHILOX_WEYL[1]) & _M64]
        p0 = PHILOX_MUL[0] * c[0]
        p1 = PHILOX_MUL[1] * c[2]
        c = [(p1 >> 64) ^ c[1] ^ k[0], p1 & _M64, (p0 >> 64) ^ c[3] ^ k[1], p0 & _M64]
    return c


def uniforms(seed: int, purpose: int, step: int, row: int, n: int):
    """u_0 .. u_{n-1} of stream (purpose, step, row), float64 values in (0, 1).

    Output word w of the stream is word w mod 4 of the Philox4x64-10 block at counter
    (1 + w div 4, row, step, purpose) under key (seed, 0); it gives two uniforms, u_{2w} from its
    bits 63..41 and u_{2w+1} from its bits 31..9, each as (23-bit integer + 1/2) 2^-23.
    numpy's Philox bit generator computes the same blocks; it advances the counter before its
    first block, so it starts from word 0 = 0 to produce block 1 first.
    """
    u64 = lambda *v: np.array([int(x) & _M64 for x in v], dtype=np.uint64)
    g = np.random.Philox(counter=u64(0, row, step, purpose), key=u64(seed, 0))
    nw = (int(n) + 1) // 2
    x = g.random_raw(nw) if nw else np.zeros(0, np.uint64)
    hi = (x >> np.uint64(41)).astype(F64)
    lo = ((x >> np.uint64(9)) & np.uint64(0x7FFFFF)).astype(F64)
    bits = np.empty(2 * nw, F64)
    bits[0::2], bits[1::2] = hi, lo
    return (bits[:int(n)] + 0.5) * 2.0 ** -23


def softmax_t(logits, temperature: float):
    """softmax(logits / T) over the last axis (max-subtracted)."""
    z = np.asarray(logits, F64) / temperature
    z = np.exp(z - z.max(axis=-1, keepdims=True))
    return z / z.sum(axis=-1, keepdims=True)


def gumbel_draw(log_w, u):
    """argmax_v (log_w[v] - log(-log u[v])): a draw of v with probability proportional to
    exp(log_w[v]); entries with log_w = -inf are never drawn (lowest id among equal scores)."""
    score = np.asarray(log_w, F64) - np.log(-np.log(np.asarray(u, F64)))
    return int(np.argmax(score))


def sample_token(logits, temperature: float, u):
    """A draft token at temperature T: a draw from softmax(logits / T)."""
    return gumbel_draw(np.asarray(logits, F64) / temperature, u)


def accept_prob(p, q, d: int):
    """min(1, p(d) / q(d)): the probability of keeping draft token d."""
    return min(1.0, float(p[d]) / float(q[d]))


def residual_dist(p, q):
    """max(0, p - q) renormalised, the replacement distribution after a rejection (p itself when
    the difference vanishes everywhere)."""
    w = np.maximum(np.asarray(p, F64) - np.asarray(q, F64), 0.0)
    tot = w.sum()
    return w / tot if tot > 0 else np.asarray(p, F64)


def speculative_verify(draft, target_logits, draft_logits, temperature: float, r, u_res):
    """Sampled verification of one block.

    draft: d_1 .. d_{B-1}; target_logits: [B][V], row k-1 predicts the position of d_k (row B-1
    the position after the block); draft_logits: [B-1][V], the draft's logits at the position of
    d_k; r: B-1 acceptance uniforms; u_res: V uniforms for the replacement or extra token.
    d_k is kept when r_k q(d_k) < p(d_k), i.e. r_k < p(d_k)/q(d_k). Returns (tau, next_token).
    """
    target_logits = np.asarray(target_logits, F64)
    B = target_logits.shape[0]
    a = 0
    while a < B - 1:
        p = softmax_t(target_logits[a], temperature)
        q = softmax_t(draft_logits[a], temperature)
        d = int(draft[a])
        if r[a] * q[d] < p[d]:
            a += 1
        else:
            break
    if a < B - 1:
        w = residual_dist(softmax_t(target_logits[a], temperature),
                          softmax_t(draft_logits[a], temperature))
    else:
        w = softmax_t(target_logits[B - 1], temperature)
    with np.errstate(divide="ignore"):
        return a + 1, gumbel_draw(np.log(w), u_res)


# --------------------------------------------------------------------------- the whole path

class DraftOracle:
    """The three calls of the draft path over a batch of sequences, in float64.

    weights: dict of input arrays in the library's stacked layout (bf16 bit patterns or fp32),
    as produced by ``synth.weights``. shape: the drafter's architecture. storage: "bf16" applies
    bf16 storage rounding (the bf16 path's reference), "exact" none (the fp32 path's).

    Variants (Sec. 6.3, Table 2, and the DFlash design of Sec. 2.2-2.3):
    softmax_fusion=False  "-Softmax": alpha = W^fuse as it is;
    shared_kv=True        "-KVProj": context rows are projected by the layer's own W_K^d, W_V^d
                          (the K and V rows of w_qkv) instead of W_K^t, W_V^t;
    fusion_fc=True        "+FC": F'^(i) = W_fc^(i) F^(i) + b_fc^(i) (weights fusion_fc_w,
                          fusion_fc_b) replaces F^(i) before the projection;
    dflash_fc=True        DFlash: every layer projects the same c_t of Eq. 1 (weights
                          dflash_fc_w, dflash_fc_b) with its own W_K, W_V (Eq. 2); the layer-wise
                          fusion and W^t are not used.
    """

    def __init__(self, weights: dict, shape, batch: int, storage: str = "exact",
                 softmax_fusion: bool = True, rope_block: bool = True, shared_kv: bool = False,
                 fusion_fc: bool = False, dflash_fc: bool = False):
        if dflash_fc and (fusion_fc or not softmax_fusion):
            raise ValueError("dflash_fc replaces the layer-wise fusion")
        self.w = weights
        self.s = shape
        self.batch = batch
        self.store = round_bf16 if storage == "bf16" else exact
        self.rope_block = rope_block
        self.shared_kv = shared_kv or dflash_fc
        self.fusion_fc = fusion_fc
        self.dflash_fc = dflash_fc
        self._cache = {}
        self.alpha = None if dflash_fc else fusion_weights(weights["fuse_logits"],
                                                           softmax=softmax_fusion)
        D = shape.n_draft_layers
        empty = np.zeros((0, shape.n_kv_heads, shape.head_dim))
        self.ctx_k = [[empty] * D for _ in range(batch)]
        self.ctx_v = [[empty] * D for _ in range(batch)]

    def _dec(self, name, idx=None):
        """float64 copy of an input weight (decoded once, then kept)."""
        key = (name, idx)
        if key not in self._cache:
            a = self.w[name] if idx is None else self.w[name][idx]
            self._cache[key] = decode(a, self.s.dtype)
        return self._cache[key]

    def layer(self, i: int) -> dict:
        return {k: self._dec(k, i) for k in
                ("attn_norm", "w_qkv", "w_o", "mlp_norm", "w_gate", "w_up", "w_down")}

    def ctx_len(self, b: int) -> int:
        return self.ctx_k[b][0].shape[0]

    def fuse_context(self, b: int, hidden):
        """Fuse n newly committed positions of sequence b (hidden: [T][n][d] input bytes) and
        append their keys/values to every layer's context cache. Returns the representation
        each layer projects, [D][n][d]: F^(i) (Eq. 3), F'^(i) under "+FC", c (Eq. 1) under
        DFlash."""
        s = self.s
        D = s.n_draft_layers
        h = decode(hidden, s.dtype)
        n = h.shape[1]
        if self.dflash_fc:
            C = dflash_context(h, self._dec("dflash_fc_w"), self._dec("dflash_fc_b"), self.store)
            F = np.stack([C] * D)
        else:
            F = fuse_context(h, self.alpha, self._dec("fuse_norm"), s.rms_eps, self.store)
            if self.fusion_fc:
                F = np.stack([fusion_fc(F[i], self._dec("fusion_fc_w", i),
                                        self._dec("fusion_fc_b", i), self.store)
                              for i in range(D)])
        L = self.ctx_len(b)
        pos = np.arange(L, L + n)
        for i in range(D):
            # [W_K ; W_V] of the context rows: W^t (Eq. 4), or the block's own W^d (Eq. 2)
            w_kv = self._dec("w_qkv", i)[s.d_q:] if self.shared_kv else self._dec("w_kv_ctx", i)
            k, v = context_kv(F[i], w_kv, pos, s.n_kv_heads, s.head_dim, s.rope_theta, self.store)
            self.ctx_k[b][i] = np.concatenate([self.ctx_k[b][i], k])
            self.ctx_v[b][i] = np.concatenate([self.ctx_v[b][i], v])
        return F

    def block_input(self, last_token: int):
        """X^0 = [E[x_t]; E[mask] x (B-1)] from the shared token embedding (Sec. 3.2, 3.3)."""
        s = self.s
        ids = [int(last_token)] + [s.mask_token_id] * (s.block - 1)
        return decode(self.w["embed"][ids], s.dtype)

    def draft_block(self, b: int, last_token: int, x0=None):
        """One block forward for sequence b. Returns (tokens [B-1], logits [B-1][V],
        hidden [D+1][B][d]: the block rows after the embedding and after every layer)."""
        s = self.s
        x = self.block_input(last_token) if x0 is None else np.asarray(x0, F64)
        L = self.ctx_len(b)
        pos = np.arange(L, L + s.block)
        hidden = [x]
        for i in range(s.n_draft_layers):
            x = draft_layer(x, self.layer(i), self.ctx_k[b][i], self.ctx_v[b][i], pos, s,
                            self.store, self.rope_block)
            hidden.append(x)
        logits = lm_head_logits(x, self._dec("final_norm"), self._dec("lm_head"), s.rms_eps,
                                self.store)
        return argmax_lowest(logits), logits, np.stack(hidden)

    @staticmethod
    def verify_accept(draft, target):
        return verify_accept(draft, target)
