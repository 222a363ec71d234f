"""GB300 (sm_103a) implementation of DFlare's per-step draft path (arxiv 2606.02091).

The path runs in hand-written CUDA kernels inside ``libdflare.so`` (C ABI in include/dflare.h).
This package holds the CUDA sources (``csrc/``), the in-tree build (``build.py``) and a thin
binding (``_lib.py`` for the raw calls, ``DFlare`` below for torch-tensor arguments). PyTorch is
used only to own device memory and to name the CUDA stream.
"""
from __future__ import annotations

import ctypes

from . import _lib
from ._lib import (  # noqa: F401
    DFlareError, DFLARE_BF16, DFLARE_F32, FLAG_NO_BLOCK_ROPE, FLAG_RAW_FUSION, FLAG_SIMT_GEMM,
    FLAG_SERIAL_LAUNCH, FLAG_SHARED_KV, FLAG_FUSION_FC, FLAG_DFLASH_FC, FLAG_DETERMINISTIC,
    FLAG_MMA_SYNC_ATTENTION,
    DEVERR_TOKEN, DEVERR_CAPACITY, DEVERR_TIMEOUT, EXPORTS, WEIGHT_FIELDS, NOALLOC_MAX_ROWS, load,
)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _need_cuda(name, t, dtype=None, numel=None):
    """A contiguous CUDA tensor of `dtype` holding at least `numel` elements (None: unchecked).
    The C ABI takes bare pointers, so an undersized buffer is caught here, on the host."""
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, needs at least {numel}")


class DFlare:
    """One library context: the draft weights, per-layer context KV caches and work buffers.

    Arguments mirror ``dflare_config`` (include/dflare.h). Device buffers passed to the calls
    are torch CUDA tensors; calls are enqueued on the current torch stream unless one is given.
    """

    def __init__(self, *, d, n_draft_layers, n_target_layers, n_q_heads, n_kv_heads, head_dim,
                 ffn, vocab, block, max_batch, max_ctx, max_fuse_rows, mask_token_id=None,
                 rms_eps=1e-6, rope_theta=1e6, dtype="bf16", flags=0):
        self._L = load()
        self.cfg = _lib.Config(d, n_draft_layers, n_target_layers, n_q_heads, n_kv_heads, head_dim,
                               ffn, vocab, block, max_batch, max_ctx, max_fuse_rows,
                               vocab - 1 if mask_token_id is None else mask_token_id, rms_eps,
                               rope_theta, DFLARE_BF16 if dtype == "bf16" else DFLARE_F32, flags)
        self.dtype = dtype
        self._ctx = ctypes.c_void_p()
        _lib.check(self._L.dflare_create(ctypes.byref(self.cfg), ctypes.byref(self._ctx)))
        self._weights = None
        self.batch = max_batch

    @classmethod
    def from_shape(cls, shape, *, max_batch, max_ctx, max_fuse_rows, flags=0):
        """Build from an object with the fields of ``synth.Shape``."""
        return cls(d=shape.d, n_draft_layers=shape.n_draft_layers,
                   n_target_layers=shape.n_target_layers, n_q_heads=shape.n_q_heads,
                   n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim, ffn=shape.ffn,
                   vocab=shape.vocab, block=shape.block, max_batch=max_batch, max_ctx=max_ctx,
                   max_fuse_rows=max_fuse_rows, mask_token_id=shape.vocab - 1,
                   rms_eps=shape.rms_eps, rope_theta=shape.rope_theta, dtype=shape.dtype,
                   flags=flags)

    def close(self):
        if self._ctx:
            self._L.dflare_destroy(self._ctx)
            self._ctx = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, status):
        return _lib.check(status, self._ctx)

    def _tdtype(self):
        import torch
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def _rows(self):
        """(batch, B, mask rows per sequence B - 1)"""
        return self.batch, self.cfg.block, self.cfg.block - 1

    @property
    def raw(self):
        """The dflare_ctx* handle (for direct C-ABI calls)."""
        return self._ctx

    def set_weights(self, weights: dict, stream=None):
        """weights: name -> CUDA tensor in the layout of ``dflare_weights`` (kept alive here).

        A missing or None entry is passed as NULL; the library rejects a NULL weight that the
        context's flags read."""
        w = _lib.Weights()
        for name in WEIGHT_FIELDS:
            t = weights.get(name)
            if t is None:
                continue
            _need_cuda(name, t)
            setattr(w, name, t.data_ptr())
        self._weights = dict(weights)
        self._check(self._L.dflare_set_weights(self._ctx, ctypes.byref(w), _stream(stream)))

    def reset(self, batch: int, stream=None):
        self._check(self._L.dflare_reset(self._ctx, batch, _stream(stream)))
        self.batch = batch

    def fuse_context(self, hidden, n_new, fused_out=None, stream=None):
        """hidden [T][batch][n_max][d]; n_new int32 [batch] (device)."""
        import torch
        c = self.cfg
        if hidden.dim() != 4 or hidden.shape[0] != c.n_target_layers or hidden.shape[1] != self.batch \
                or hidden.shape[3] != c.d:
            raise ValueError(f"hidden must be [T={c.n_target_layers}][batch={self.batch}][n_max][d={c.d}], "
                             f"got {list(hidden.shape)}")
        n_max = hidden.shape[2]
        _need_cuda("hidden", hidden, self._tdtype())
        _need_cuda("n_new", n_new, torch.int32, self.batch)
        slots = 1 if c.flags & FLAG_DFLASH_FC else c.n_draft_layers   # DFlash: one shared c_t
        _need_cuda("fused_out", fused_out, self._tdtype(), slots * self.batch * n_max * c.d)
        self._check(self._L.dflare_fuse_context(self._ctx, _ptr(hidden), _ptr(n_new), n_max,
                                                _ptr(fused_out), _stream(stream)))

    def draft_block(self, last_token, draft_tokens, logits_out=None, hidden_out=None, stream=None):
        self._check_draft_args(last_token, draft_tokens, logits_out, hidden_out)
        self._check(self._L.dflare_draft_block(self._ctx, _ptr(last_token), _ptr(draft_tokens),
                                               _ptr(logits_out), _ptr(hidden_out), _stream(stream)))

    def _check_draft_args(self, last_token, draft_tokens, logits_out, hidden_out):
        import torch
        b, B, m = self._rows()
        c = self.cfg
        _need_cuda("last_token", last_token, torch.int32, b)
        _need_cuda("draft_tokens", draft_tokens, torch.int32, b * m)
        _need_cuda("logits_out", logits_out, torch.float32, b * m * c.vocab)
        _need_cuda("hidden_out", hidden_out, torch.float32, (c.n_draft_layers + 1) * b * B * c.d)

    def _check_verify_args(self, draft_tokens, accept_len, next_token):
        import torch
        b, _, m = self._rows()
        _need_cuda("draft_tokens", draft_tokens, torch.int32, b * m)
        _need_cuda("accept_len", accept_len, torch.int32, b)
        _need_cuda("next_token", next_token, torch.int32, b)

    def verify_accept(self, draft_tokens, target_argmax, accept_len, next_token, stream=None):
        import torch
        b, B, _ = self._rows()
        self._check_verify_args(draft_tokens, accept_len, next_token)
        _need_cuda("target_argmax", target_argmax, torch.int32, b * B)
        self._check(self._L.dflare_verify_accept(self._ctx, _ptr(draft_tokens), _ptr(target_argmax),
                                                 _ptr(accept_len), _ptr(next_token),
                                                 _stream(stream)))

    def draft_block_sampled(self, last_token, temperature, seed, step, draft_tokens,
                            logits_out=None, hidden_out=None, stream=None):
        """As draft_block, with tokens drawn at `temperature`; step: uint64 device counter
        (a one-element int64 tensor)."""
        import torch
        self._check_draft_args(last_token, draft_tokens, logits_out, hidden_out)
        _need_cuda("step", step, torch.int64, 1)
        self._check(self._L.dflare_draft_block_sampled(
            self._ctx, _ptr(last_token), float(temperature), int(seed) & (2 ** 64 - 1), _ptr(step),
            _ptr(draft_tokens), _ptr(logits_out), _ptr(hidden_out), _stream(stream)))

    def verify_sampled(self, draft_tokens, target_logits, temperature, seed, step, accept_len,
                       next_token, stream=None):
        """Speculative-sampling verification of the last drafted block; advances step by one."""
        import torch
        b, B, _ = self._rows()
        self._check_verify_args(draft_tokens, accept_len, next_token)
        _need_cuda("target_logits", target_logits, torch.float32, b * B * self.cfg.vocab)
        _need_cuda("step", step, torch.int64, 1)
        self._check(self._L.dflare_verify_sampled(
            self._ctx, _ptr(draft_tokens), _ptr(target_logits), float(temperature),
            int(seed) & (2 ** 64 - 1), _ptr(step), _ptr(accept_len), _ptr(next_token),
            _stream(stream)))

    def verify_logits(self, draft_tokens, target_logits, accept_len, next_token, stream=None):
        """target_logits [batch][B][V] fp32: the target's argmax is taken on the device."""
        import torch
        b, B, _ = self._rows()
        self._check_verify_args(draft_tokens, accept_len, next_token)
        _need_cuda("target_logits", target_logits, torch.float32, b * B * self.cfg.vocab)
        self._check(self._L.dflare_verify_logits(self._ctx, _ptr(draft_tokens), _ptr(target_logits),
                                                 _ptr(accept_len), _ptr(next_token),
                                                 _stream(stream)))

    def read_kv(self, layer, seq, pos0, n, stream=None):
        import torch
        dt = torch.bfloat16 if self.dtype == "bf16" else torch.float32
        k = torch.empty((n, self.cfg.n_kv_heads, self.cfg.head_dim), dtype=dt, device="cuda")
        v = torch.empty_like(k)
        self._check(self._L.dflare_read_kv(self._ctx, layer, seq, pos0, n, _ptr(k), _ptr(v),
                                           _stream(stream)))
        return k, v

    def ctx_lens(self, stream=None):
        arr = (ctypes.c_int32 * self.batch)()
        self._check(self._L.dflare_ctx_lens(self._ctx, arr, _stream(stream)))
        return list(arr)

    def set_timing(self, stamps=None, slots: int = 0):
        """Device-side timing of the next `slots` GEMM launches into the int64 device tensor
        `stamps` (3 * slots entries: entry, dependency met, exit; see dflare_set_timing); with no
        arguments timing is turned off."""
        import torch
        if stamps is not None:
            _need_cuda("stamps", stamps, torch.int64, 3 * slots)
        self._check(self._L.dflare_set_timing(self._ctx, _ptr(stamps) if stamps is not None else None,
                                              slots if stamps is not None else 0))

    def device_error(self, stream=None) -> int:
        bits = ctypes.c_uint32(0)
        st = self._L.dflare_device_error(self._ctx, ctypes.byref(bits), _stream(stream))
        if st not in (_lib.DFLARE_OK, _lib.DFLARE_EDEVICE):
            self._check(st)
        return bits.value


def argmax_noalloc(logits, tokens_out, stream=None):
    """Greedy argmax of [rows][vocab] fp32 device logits into int32 tokens_out without any device
    allocation (see dflare_argmax_noalloc: fixed scratch, at most NOALLOC_MAX_ROWS rows)."""
    import torch
    vocab = logits.shape[-1]
    rows = logits.numel() // vocab if vocab else 0
    _need_cuda("logits", logits, torch.float32)
    _need_cuda("tokens_out", tokens_out, torch.int32, rows)
    _lib.check(load().dflare_argmax_noalloc(_ptr(logits), rows, vocab, _ptr(tokens_out),
                                            _stream(stream)))


def synthetic_target(draft_tokens, u, r, last, step, threshold, batch, block, target_out,
                     stream=None):
    """Stand-in for the target's verification argmax (see dflare_synthetic_target)."""
    L = load()
    n_steps = u.shape[0]
    _lib.check(L.dflare_synthetic_target(_ptr(draft_tokens), _ptr(u), _ptr(r), _ptr(last), n_steps,
                                         _ptr(step), ctypes.c_uint32(threshold), batch, block,
                                         _ptr(target_out), _stream(stream)))
