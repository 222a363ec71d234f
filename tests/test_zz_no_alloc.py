"""dflare_argmax_noalloc: the greedy argmax that allocates no device memory, for callers that
cannot allocate (serving loops whose memory budget is fixed at start-up, code that must not
trigger the device synchronisation cudaMalloc/cudaFree can cause). Its scratch is a fixed array
compiled into the library. The GPU test checks it against the tokens dflare_draft_block drafts
from the same logits, on two calls in a row (the second call reuses the scratch the first one
left behind)."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
from tests.harness import SMALL_HD128, GpuSide


def test_noalloc_rejects_more_rows_than_its_scratch():
    from paper_2606_02091_gb300 import build, _lib
    build.build()
    lib = _lib.load()
    fake = ctypes.c_void_p(256)            # never dereferenced: the size check comes first
    st = lib.dflare_argmax_noalloc(fake, _lib.NOALLOC_MAX_ROWS + 1, 10, fake, None)
    assert st == _lib.DFLARE_ECAPACITY
    assert b"DFLARE_NOALLOC_MAX_ROWS" in lib.dflare_last_error(None)
    assert lib.dflare_argmax_noalloc(None, 1, 10, fake, None) == _lib.DFLARE_EINVAL


def test_noalloc_source_calls_no_allocator():
    """The entry point's translation unit calls no CUDA allocation or free routine."""
    src = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                            "paper_2606_02091_gb300", "csrc", "argmax_noalloc.cu")).read()
    assert not re.search(r"\bcu(da)?(Mem)?(Malloc|Free|Alloc)\w*\s*\(", src)


@pytest.mark.gpu
def test_noalloc_argmax_matches_draft_block_on_two_calls():
    import torch
    from paper_2606_02091_gb300 import argmax_noalloc
    w = SMALL_HD128
    g = GpuSide(w)
    g.fuse(w.ctx_lens, want_fused=False)
    x_t = synth.initial_tokens(w)
    tok1, logits1, _ = g.draft(x_t)
    tok2, logits2, _ = g.draft((x_t + 7) % (w.shape.vocab - 1))
    assert not np.array_equal(logits1, logits2)
    for tok, lg in ((tok1, logits1), (tok2, logits2)):
        dev = torch.from_numpy(np.ascontiguousarray(lg)).cuda()
        out = torch.full(tok.shape, -1, dtype=torch.int32, device="cuda")
        argmax_noalloc(dev, out)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(out.cpu().numpy(), tok)


@pytest.mark.gpu
def test_noalloc_argmax_rows_without_a_finite_maximum():
    """NaN entries are never chosen; a row with nothing above -inf gets its first -inf entry, a
    row of NaN id 0; ties go to the lowest id."""
    import torch
    from paper_2606_02091_gb300 import argmax_noalloc
    V = 5000
    lg = np.random.default_rng(1).standard_normal((5, V)).astype(np.float32)
    lg[0] = -np.inf
    lg[1] = -np.inf
    lg[1, :3] = np.nan
    lg[2] = np.nan
    lg[3, 17] = lg[3, 4096] = 50.0
    lg[4, V - 1] = 50.0
    lg[4, 5] = np.nan
    dev = torch.from_numpy(lg).cuda()
    out = torch.full((5,), -1, dtype=torch.int32, device="cuda")
    argmax_noalloc(dev, out)
    assert out.cpu().tolist() == [0, 3, 0, 17, V - 1]


@pytest.mark.gpu
def test_noalloc_argmax_across_vocabulary_chunks_allocates_nothing():
    """A 151936-token vocabulary (many CTAs per row, merged through the packed 64-bit atomicMax):
    equal maxima in different chunks (lowest id), a maximum only in the last, partial chunk, rows
    of -inf with NaN in one chunk, random rows; two calls in a row on different logits. After a
    warm-up call, repeated calls change neither torch's allocated bytes nor the device's free
    memory."""
    import torch
    from paper_2606_02091_gb300 import argmax_noalloc
    V = 151936
    rng = np.random.default_rng(7)

    def case(seed):
        lg = np.random.default_rng(seed).standard_normal((8, V)).astype(np.float32)
        want = [int(np.argmax(r)) for r in lg]
        lg[0, 100] = lg[0, 140000] = 60.0
        want[0] = 100
        lg[1, V - 3] = 60.0
        want[1] = V - 3
        lg[2] = -np.inf
        lg[2, 50000:51000] = np.nan
        want[2] = 0
        lg[3] = -np.inf
        lg[3, :10] = np.nan
        lg[3, 90000:90100] = np.nan
        want[3] = 10
        top = int(rng.integers(1, V))
        lg[4, [top, 7, V - 1]] = 70.0
        want[4] = min(top, 7)
        lg[5, 3] = np.nan
        lg[5, 151935] = 80.0
        want[5] = 151935
        return lg, want

    out = torch.full((8,), -1, dtype=torch.int32, device="cuda")
    for seed in (1, 2):
        lg, want = case(seed)
        dev = torch.from_numpy(lg).cuda()
        argmax_noalloc(dev, out)
        assert out.cpu().tolist() == want, seed
    torch.cuda.synchronize()
    alloc0 = torch.cuda.memory_allocated()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(20):
        argmax_noalloc(dev, out)
    torch.cuda.synchronize()
    assert torch.cuda.memory_allocated() == alloc0
    assert torch.cuda.mem_get_info()[0] == free0
    assert out.cpu().tolist() == want
