"""The C-ABI library: it builds, loads without a GPU, exports every entry point include/dflare.h
declares, and rejects bad arguments on the host before touching a device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dflare.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2606_02091_gb300 import build, _lib
    build.build()
    return _lib.load()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dflare_[a-z_]+)\s*\(", src)))


def test_header_declares_the_three_calls():
    names = _declared()
    for n in ("dflare_fuse_context", "dflare_draft_block", "dflare_verify_accept"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2606_02091_gb300 import _lib
    names = _declared()
    assert sorted(_lib.EXPORTS) == names
    for n in names:
        assert hasattr(lib, n), n


def _cfg(**kw):
    from paper_2606_02091_gb300 import _lib
    base = dict(d=256, n_draft_layers=4, n_target_layers=8, n_q_heads=4, n_kv_heads=2,
                head_dim=64, ffn=768, vocab=4096, block=8, max_batch=1, max_ctx=256,
                max_fuse_rows=256, mask_token_id=4095, rms_eps=1e-6, rope_theta=1e6, dtype=1,
                flags=0)
    base.update(kw)
    return _lib.Config(**base)


@pytest.mark.parametrize("field,value", [
    ("d", 100), ("d", 0), ("d", 8192), ("n_draft_layers", 0), ("n_draft_layers", 17),
    ("n_target_layers", 0), ("n_target_layers", 65), ("head_dim", 96), ("n_q_heads", 3),
    ("n_kv_heads", 0), ("ffn", 100), ("vocab", 1), ("mask_token_id", 4096), ("mask_token_id", -1),
    ("block", 0), ("block", 33), ("max_batch", 0), ("max_batch", 65), ("max_ctx", 0),
    ("max_fuse_rows", 0), ("rms_eps", -1.0), ("rope_theta", 0.0), ("dtype", 2), ("flags", 0x200), ("flags", 0x400),
    ("flags", 0x40 | 0x2), ("flags", 0x40 | 0x20),   # DFlash FC with -Softmax / +FC
])
def test_create_rejects_bad_config_on_host(lib, field, value):
    ctx = ctypes.c_void_p()
    st = lib.dflare_create(ctypes.byref(_cfg(**{field: value})), ctypes.byref(ctx))
    assert st == 1                                       # DFLARE_EINVAL, no device touched
    assert not ctx
    assert lib.dflare_last_error(None).startswith(b"invalid config")


def test_binding_structs_follow_the_header():
    """The ctypes mirrors of dflare_weights and dflare_config list the header's fields in the
    header's order, and the flag constants carry the header's values."""
    from paper_2606_02091_gb300 import _lib
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    for struct, mirror in (("dflare_weights", _lib.Weights), ("dflare_config", _lib.Config)):
        body = re.search(r"typedef struct \{([^}]*)\}\s*" + struct + ";", src).group(1)
        fields = re.findall(r"(\w+)\s*;", body)
        assert fields == [f for f, _ in mirror._fields_], struct
    flags = dict(re.findall(r"#define DFLARE_FLAG_(\w+)\s+(0x[0-9a-fA-F]+)u", open(HEADER).read()))
    assert flags and all(getattr(_lib, "FLAG_" + k) == int(v, 16) for k, v in flags.items())


def test_create_null_out(lib):
    assert lib.dflare_create(ctypes.byref(_cfg()), None) == 1


def test_null_context_calls_fail(lib):
    assert lib.dflare_reset(None, 1, None) == 1
    assert lib.dflare_fuse_context(None, None, None, 1, None, None) == 1
    assert lib.dflare_draft_block(None, None, None, None, None, None) == 1
    assert lib.dflare_verify_accept(None, None, None, None, None, None) == 1
    assert lib.dflare_destroy(None) == 0


def test_synthetic_target_argument_checks(lib):
    assert lib.dflare_synthetic_target(None, None, None, None, 1, None, 0, 1, 8, None, None) == 1


def test_valid_config_without_gpu_fails_loudly(lib):
    """With no GPU the valid config is accepted by the checks and then fails in CUDA: the
    library never falls back to the CPU."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    ctx = ctypes.c_void_p()
    st = lib.dflare_create(ctypes.byref(_cfg()), ctypes.byref(ctx))
    assert st == 3                                       # DFLARE_ECUDA
    assert not ctx


class _FakeCuda:
    """Stands in for a CUDA tensor on a machine without one: only what the binding inspects."""

    def __init__(self, numel, dtype, shape=None):
        self._n, self.dtype = numel, dtype
        self.shape = tuple(shape) if shape is not None else (numel,)
        self.is_cuda = True

    def is_contiguous(self):
        return True

    def numel(self):
        return self._n

    def dim(self):
        return len(self.shape)

    def data_ptr(self):
        raise AssertionError("an undersized buffer reached the C call")


class _NoLib:
    def __getattr__(self, name):
        raise AssertionError(f"an undersized buffer reached the C call ({name})")


def _bare_binding(block=4, vocab=11, d=8, D=2, T=3, batch=2, flags=0):
    from paper_2606_02091_gb300 import DFlare, _lib
    o = object.__new__(DFlare)   # no dflare_create: the checks run before any library call
    o.cfg = _lib.Config(d, D, T, 2, 1, 4, 16, vocab, block, batch, 64, 64, vocab - 1, 1e-6, 1e6,
                        _lib.DFLARE_F32, flags)
    o.dtype, o.batch, o._ctx, o._L = "f32", batch, None, _NoLib()
    return o


def test_binding_rejects_undersized_buffers_on_the_host():
    import torch
    o = _bare_binding()
    i32, f32 = torch.int32, torch.float32
    ok_last, ok_toks = _FakeCuda(2, i32), _FakeCuda(2 * 3, i32)
    with pytest.raises(ValueError, match="draft_tokens"):
        o.draft_block(ok_last, _FakeCuda(5, i32))
    with pytest.raises(ValueError, match="last_token"):
        o.draft_block(_FakeCuda(1, i32), ok_toks)
    with pytest.raises(ValueError, match="logits_out"):
        o.draft_block(ok_last, ok_toks, logits_out=_FakeCuda(2 * 3 * 11 - 1, f32))
    with pytest.raises(ValueError, match="hidden_out"):
        o.draft_block(ok_last, ok_toks, hidden_out=_FakeCuda(3 * 2 * 4 * 8 - 1, f32))
    with pytest.raises(ValueError, match="target_argmax"):
        o.verify_accept(ok_toks, _FakeCuda(7, i32), ok_last, ok_last)
    with pytest.raises(ValueError, match="target_logits"):
        o.verify_logits(ok_toks, _FakeCuda(2 * 4 * 11 - 1, f32), ok_last, ok_last)
    with pytest.raises(ValueError, match="must be torch.int32"):
        o.verify_accept(ok_toks, _FakeCuda(8, torch.int64), ok_last, ok_last)
    with pytest.raises(ValueError, match="step"):
        o.draft_block_sampled(ok_last, 1.0, 0, _FakeCuda(0, torch.int64), ok_toks)
    hid = _FakeCuda(3 * 2 * 5 * 8, f32, (3, 2, 5, 8))
    with pytest.raises(ValueError, match="fused_out"):
        o.fuse_context(hid, _FakeCuda(2, i32), _FakeCuda(2 * 2 * 5 * 8 - 1, f32))
    with pytest.raises(ValueError, match="hidden must be"):
        o.fuse_context(_FakeCuda(3 * 2 * 5 * 8, f32, (3, 1, 10, 8)), _FakeCuda(2, i32))
    with pytest.raises(ValueError, match="must be torch.float32"):
        o.fuse_context(_FakeCuda(3 * 2 * 5 * 8, torch.bfloat16, (3, 2, 5, 8)), _FakeCuda(2, i32))
    # DFlash writes one shared context slot, so one slot is enough there
    from paper_2606_02091_gb300 import FLAG_DFLASH_FC
    od = _bare_binding(flags=FLAG_DFLASH_FC)
    with pytest.raises(AssertionError, match="reached the C call"):
        od.fuse_context(hid, _FakeCuda(2, i32), _FakeCuda(2 * 5 * 8, f32))
