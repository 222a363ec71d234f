"""dflare_argmax_noalloc: the greedy argmax that allocates no device memory, for callers that
cannot allocate (serving loops whose memory budget is fixed at start-up, code that must not
trigger the device synchronisation cudaMalloc/cudaFree can cause). Its scratch is a fixed array
compiled into the library. The GPU test checks it against the tokens dflare_draft_block drafts
from the same logits, on two calls in a row (the second call reuses the scratch the first one
left behind)."""
import ctypes

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
