"""ctypes binding of libdflare.so: the C ABI declared in include/dflare.h, argument marshalling only.

Every step of the draft path runs in the library's CUDA kernels; this module converts Python
arguments (torch tensors for device buffers, the current torch CUDA stream) into the plain
pointers and sizes of the C calls. It never computes anything itself and has no fallback: if the
shared library is missing or cannot be loaded, importing a call raises.
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdflare.so")

DFLARE_OK, DFLARE_EINVAL, DFLARE_ECAPACITY, DFLARE_ECUDA, DFLARE_ESTATE, DFLARE_ENOMEM, \
    DFLARE_EDEVICE = range(7)
DFLARE_BF16, DFLARE_F32 = 0, 1
FLAG_NO_BLOCK_ROPE = 0x1
FLAG_RAW_FUSION = 0x2
FLAG_SIMT_GEMM = 0x4
FLAG_SERIAL_LAUNCH = 0x8
FLAG_SHARED_KV = 0x10
FLAG_FUSION_FC = 0x20
FLAG_DFLASH_FC = 0x40
FLAG_DETERMINISTIC = 0x80
FLAG_MMA_SYNC_ATTENTION = 0x100
DEVERR_TOKEN, DEVERR_CAPACITY, DEVERR_TIMEOUT = 0x1, 0x2, 0x4

STATUS_NAMES = {0: "DFLARE_OK", 1: "DFLARE_EINVAL", 2: "DFLARE_ECAPACITY", 3: "DFLARE_ECUDA",
                4: "DFLARE_ESTATE", 5: "DFLARE_ENOMEM", 6: "DFLARE_EDEVICE"}

# every entry point include/dflare.h declares
EXPORTS = ("dflare_create", "dflare_destroy", "dflare_set_weights", "dflare_reset",
           "dflare_fuse_context", "dflare_draft_block", "dflare_verify_accept",
           "dflare_verify_logits", "dflare_draft_block_sampled", "dflare_verify_sampled",
           "dflare_read_kv",
           "dflare_ctx_lens", "dflare_device_error", "dflare_last_error",
           "dflare_synthetic_target", "dflare_set_trace", "dflare_set_timing",
           "dflare_argmax_noalloc")

NOALLOC_MAX_ROWS = 4096

TRACE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_char_p, ctypes.c_int, ctypes.c_void_p)


class Config(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int), ("n_draft_layers", ctypes.c_int),
                ("n_target_layers", ctypes.c_int), ("n_q_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("ffn", ctypes.c_int),
                ("vocab", ctypes.c_int), ("block", ctypes.c_int), ("max_batch", ctypes.c_int),
                ("max_ctx", ctypes.c_int), ("max_fuse_rows", ctypes.c_int),
                ("mask_token_id", ctypes.c_int), ("rms_eps", ctypes.c_float),
                ("rope_theta", ctypes.c_float), ("dtype", ctypes.c_int), ("flags", ctypes.c_uint)]


WEIGHT_FIELDS = ("fuse_logits", "fuse_norm", "w_kv_ctx", "attn_norm", "w_qkv", "w_o", "mlp_norm",
                 "w_gate", "w_up", "w_down", "final_norm", "embed", "lm_head",
                 "fusion_fc_w", "fusion_fc_b", "dflash_fc_w", "dflash_fc_b")


class Weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in WEIGHT_FIELDS]


class DFlareError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None


def load():
    """Load libdflare.so (built in-tree by paper_2606_02091_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2606_02091_gb300.build.build()")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, u32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint32
    P = ctypes.POINTER
    sig = {
        "dflare_create": [P(Config), P(vp)],
        "dflare_destroy": [vp],
        "dflare_set_weights": [vp, P(Weights), vp],
        "dflare_reset": [vp, i32, vp],
        "dflare_fuse_context": [vp, vp, vp, i32, vp, vp],
        "dflare_draft_block": [vp, vp, vp, vp, vp, vp],
        "dflare_verify_accept": [vp, vp, vp, vp, vp, vp],
        "dflare_verify_logits": [vp, vp, vp, vp, vp, vp],
        "dflare_draft_block_sampled": [vp, vp, ctypes.c_float, ctypes.c_uint64, vp, vp, vp, vp, vp],
        "dflare_verify_sampled": [vp, vp, vp, ctypes.c_float, ctypes.c_uint64, vp, vp, vp, vp],
        "dflare_read_kv": [vp, i32, i32, i32, i32, vp, vp, vp],
        "dflare_ctx_lens": [vp, vp, vp],
        "dflare_device_error": [vp, P(u32), vp],
        "dflare_last_error": [vp],
        "dflare_synthetic_target": [vp, vp, vp, vp, i32, vp, u32, i32, i32, vp, vp],
        "dflare_set_trace": [vp, TRACE_FN, vp],
        "dflare_set_timing": [vp, vp, i32],
        "dflare_argmax_noalloc": [vp, i32, i32, vp, vp],
    }
    for name, args in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = ctypes.c_char_p if name == "dflare_last_error" else ctypes.c_int
    _lib = L
    return L


def check(status: int, ctx=None):
    if status != DFLARE_OK:
        msg = load().dflare_last_error(ctx)
        raise DFlareError(status, msg.decode() if msg else "")
    return status
