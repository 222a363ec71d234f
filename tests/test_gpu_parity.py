"""GPU path vs the CPU oracle on the same seeded inputs (Eq. 3, Eq. 4, Sec. 3.2).

Tolerances: max relative error 2e-2 (bf16 storage) or 1e-5 (fp32 storage).
- Fused context rows: element by element, |x - y| / max(|y|, c rms(y)) with c = 1e-3 (bf16) or 1
  (fp32: fp32 accumulation leaves an absolute error of a few ulp of the summed terms).
- Cached keys/values: element by element against Eq. 4 evaluated by the oracle on the GPU's own
  fused rows (the same input bytes), and row-wise (max over head vectors of ||x - y|| / ||y||)
  against the oracle's cache built from its own fused rows.
- Hidden states and logits: element by element in fp32; row-wise in bf16, where each layer's
  bf16 storage points carry single-element ulp flips forward.
- Acceptance lengths and next tokens bit-exact (integer work on the GPU's drafts); draft tokens as in
  tests.harness.check_tokens."""
import numpy as np
import pytest

import oracle as O
import synth
from tests.harness import (BLOCK1, BLOCK2, BLOCK32, D10, G8, LONG_FILL, MULTI_TILE, QT2, RAGGED, SMALL_HD128,
                           SMALL_HD64, TINY, WIDE_B16, WIDE_VOCAB,
                           GpuSide, check_elem, check_kv, check_rows, check_tokens, f64, oracle_for,
                           rel_err, tolerance, verified_steps)

pytestmark = pytest.mark.gpu
GAP = 1e-2
WORKLOADS = [TINY, SMALL_HD128, SMALL_HD64, D10, G8, BLOCK1, BLOCK2, RAGGED, LONG_FILL]


@pytest.fixture(scope="module", params=WORKLOADS, ids=lambda w: w.name)
def run(request):
    w = request.param
    g = GpuSide(w)
    o = oracle_for(w, g.W)
    fused = g.fuse(w.ctx_lens)
    F = [o.fuse_context(b, synth.hidden_states(w, b, 0, n)) for b, n in enumerate(w.ctx_lens)]
    return w, g, o, fused, F


def test_fusion_matches_oracle(run):
    w, g, o, fused, F = run
    got = f64(fused)
    for b, n in enumerate(w.ctx_lens):
        check_elem(w, got[:, b, :n], F[b], f"F seq {b}")


def test_context_lengths(run):
    w, g, o, fused, F = run
    assert g.lib.ctx_lens() == list(w.ctx_lens)
    assert g.lib.device_error() == 0


def test_context_kv_matches_oracle(run):
    w, g, o, fused, F = run
    got = f64(fused)
    for b, n in enumerate(w.ctx_lens):
        for i in range(w.shape.n_draft_layers):
            k, v = g.lib.read_kv(i, b, 0, n)
            check_kv(w, o, f64(k), f64(v), got[i, b, :n], np.arange(n), i, f"seq {b} layer {i}")
            check_rows(w, f64(k), o.ctx_k[b][i], f"seq {b} layer {i} K (end to end)")
            check_rows(w, f64(v), o.ctx_v[b][i], f"seq {b} layer {i} V (end to end)")


def _check_draft(w, tok, logits, hidden, o_res, o):
    for b, (ot, ol, oh) in enumerate(o_res):
        for i in range(oh.shape[0]):
            check_rows(w, hidden[i, b], oh[i], f"seq {b} hidden after layer {i - 1}")
        check_rows(w, logits[b], ol, f"seq {b} logits")
        check_tokens(w, o, tok[b], logits[b], hidden[-1, b], ot, ol, f"seq {b}")


def test_draft_block_matches_oracle(run):
    w, g, o, fused, F = run
    x_t = synth.initial_tokens(w)
    tok, logits, hidden = g.draft(x_t)
    o_res = [o.draft_block(b, int(x_t[b])) for b in range(w.batch)]
    _check_draft(w, tok, logits, hidden, o_res, o)


def test_steps_with_verification(run):
    """Two more block steps: draft -> synthetic target -> prefix accept -> fuse tau positions."""
    w, g, o, fused, F = run
    assert verified_steps(w, g, o, n_steps=2) >= w.batch


def test_rope_off_block_is_mask_permutation_equivariant():
    """With block RoPE off, all mask rows have the same input, so their hidden states and logits
    coincide (the bidirectional block has no position-dependent mask). Bit-identical rows need
    reductions in a fixed order, hence the deterministic mode."""
    from paper_2606_02091_gb300 import FLAG_DETERMINISTIC, FLAG_NO_BLOCK_ROPE
    w = SMALL_HD64
    g = GpuSide(w, flags=FLAG_NO_BLOCK_ROPE | FLAG_DETERMINISTIC)
    g.fuse(w.ctx_lens, want_fused=False)
    tok, logits, hidden = g.draft(synth.initial_tokens(w))
    o = oracle_for(w, g.W, rope_block=False)
    for b, n in enumerate(w.ctx_lens):
        o.fuse_context(b, synth.hidden_states(w, b, 0, n))
    for b in range(w.batch):
        for k in range(2, w.shape.block):
            np.testing.assert_array_equal(hidden[:, b, k], hidden[:, b, 1])
            np.testing.assert_array_equal(tok[b, k - 1], tok[b, 0])
        ot, ol, oh = o.draft_block(b, int(synth.initial_tokens(w)[b]))
        for i in range(oh.shape[0]):
            check_rows(w, hidden[i, b], oh[i], f"seq {b} hidden after layer {i - 1}")


def test_raw_fusion_ablation():
    """-Softmax (Table 2): alpha = W^fuse as is."""
    from paper_2606_02091_gb300 import FLAG_RAW_FUSION
    w = TINY
    g = GpuSide(w, flags=FLAG_RAW_FUSION)
    fused = f64(g.fuse(w.ctx_lens))
    o = oracle_for(w, g.W, softmax_fusion=False)
    F = o.fuse_context(0, synth.hidden_states(w, 0, 0, w.ctx_lens[0]))
    check_elem(w, fused[:, 0], F, "F (-Softmax)")


def test_empty_and_capacity_edges():
    """n_new = 0 appends nothing; an append past max_ctx is refused by the device and flagged."""
    import torch
    from paper_2606_02091_gb300 import DEVERR_CAPACITY
    w = SMALL_HD64
    g = GpuSide(w, max_ctx=310)
    g.fuse([0, 0], want_fused=False)
    assert g.lib.ctx_lens() == [0, 0]
    # an empty context still drafts (the block attends only to itself)
    tok, logits, hidden = g.draft(synth.initial_tokens(w))
    o = oracle_for(w, g.W)
    for b in range(w.batch):
        ot, ol, oh = o.draft_block(b, int(synth.initial_tokens(w)[b]))
        for i in range(oh.shape[0]):
            check_rows(w, hidden[i, b], oh[i], f"empty context seq {b} hidden after layer {i - 1}")
    g.fuse([65, 300], want_fused=False)
    assert g.lib.device_error() == 0
    g.fuse([5, 11], pos0=[65, 300], want_fused=False)       # 300 + 11 > 310: refused
    assert g.lib.ctx_lens() == [70, 300]
    assert g.lib.device_error() & DEVERR_CAPACITY
    assert g.lib.device_error() == 0                       # the word was cleared


def test_bad_token_is_flagged():
    from paper_2606_02091_gb300 import DEVERR_TOKEN
    w = SMALL_HD64
    g = GpuSide(w)
    g.fuse(w.ctx_lens, want_fused=False)
    g.draft([w.shape.vocab + 5, -1])
    assert g.lib.device_error() & DEVERR_TOKEN


def test_simt_gemm_agrees_with_tcgen05_gemm():
    """The two GEMM implementations give the same path within the bf16 tolerance."""
    from paper_2606_02091_gb300 import FLAG_SIMT_GEMM
    w = SMALL_HD128
    a, b = GpuSide(w), GpuSide(w, flags=FLAG_SIMT_GEMM, weights=None)
    a.fuse(w.ctx_lens, want_fused=False)
    b.fuse(w.ctx_lens, want_fused=False)
    x_t = synth.initial_tokens(w)
    ta, la, ha = a.draft(x_t)
    tb, lb, hb = b.draft(x_t)
    assert rel_err(ha, hb) <= tolerance(w)
    assert rel_err(la, lb) <= tolerance(w)


@pytest.mark.parametrize("w", [SMALL_HD128, G8, QT2, D10, BLOCK1], ids=lambda w: w.name)
@pytest.mark.parametrize("kernel", ["tcgen05", "mma_sync"])
def test_attention_kernels_match_oracle(w, kernel):
    """Both bf16 attention kernels (the tcgen05 one, 128 query rows per CTA, and the mma.sync one,
    64 per CTA) on query-row counts per KV head of 64, 128, 160 (two 128-row tiles, the second
    ragged), 8 (a partial warp) and 2: the drafted block and two verified steps against the
    oracle."""
    from paper_2606_02091_gb300 import FLAG_MMA_SYNC_ATTENTION
    g = GpuSide(w, flags=FLAG_MMA_SYNC_ATTENTION if kernel == "mma_sync" else 0)
    o = oracle_for(w, g.W)
    g.fuse(w.ctx_lens, want_fused=False)
    for b, n in enumerate(w.ctx_lens):
        o.fuse_context(b, synth.hidden_states(w, b, 0, n))
    x_t = synth.initial_tokens(w)
    tok, logits, hidden = g.draft(x_t)
    _check_draft(w, tok, logits, hidden, [o.draft_block(b, int(x_t[b])) for b in range(w.batch)], o)
    assert verified_steps(w, g, o, n_steps=2) >= w.batch
    assert g.lib.device_error() == 0


@pytest.mark.parametrize("w", [WIDE_B16, BLOCK32, MULTI_TILE, WIDE_VOCAB], ids=lambda w: w.name)
def test_wide_token_tiles_match_oracle(w):
    """256 token rows per projection (batch 16, the widest tcgen05 token tile), block 32, 288
    rows (two token tiles, the second ragged), and a 240-row LM head over paired weight tiles:
    fused context, cached K/V and the draft block against the oracle."""
    g = GpuSide(w)
    o = oracle_for(w, g.W)
    fused = f64(g.fuse(w.ctx_lens))
    last = w.shape.n_draft_layers - 1
    for b, n in enumerate(w.ctx_lens):
        F = o.fuse_context(b, synth.hidden_states(w, b, 0, n))
        check_elem(w, fused[:, b, :n], F, f"F seq {b}")
        k, v = g.lib.read_kv(last, b, 0, n)
        check_kv(w, o, f64(k), f64(v), fused[last, b, :n], np.arange(n), last, f"seq {b}")
        check_rows(w, f64(k), o.ctx_k[b][last], f"seq {b} K (end to end)")
    x_t = synth.initial_tokens(w)
    tok, logits, hidden = g.draft(x_t)
    _check_draft(w, tok, logits, hidden, [o.draft_block(b, int(x_t[b])) for b in range(w.batch)], o)
    assert g.lib.device_error() == 0


# (flag name, oracle options): the Sec. 6.3 ablations and DFlash's FC fusion (Eq. 1, Eq. 2)
VARIANTS = [
    ("FLAG_SHARED_KV", dict(shared_kv=True)),
    ("FLAG_FUSION_FC", dict(fusion_fc=True)),
    ("FLAG_DFLASH_FC", dict(dflash_fc=True)),
    ("FLAG_SHARED_KV|FLAG_FUSION_FC", dict(shared_kv=True, fusion_fc=True)),
]


@pytest.mark.parametrize("w", [TINY, SMALL_HD128, WIDE_B16], ids=lambda w: w.name)
@pytest.mark.parametrize("flags,kw", VARIANTS, ids=[v[0] for v in VARIANTS])
def test_variant_matches_oracle(w, flags, kw):
    """Each variant against the oracle: the projected context representation (fused_out), the
    cached context keys/values of every layer and one drafted block. A second context, filled
    without fused_out, checks the library's internal buffers."""
    import paper_2606_02091_gb300 as P
    flag = 0
    for f in flags.split("|"):
        flag |= getattr(P, f)
    W = dict(synth.weights(w))
    W.update(synth.variant_weights(w))
    o = oracle_for(w, W, **kw)
    F = [o.fuse_context(b, synth.hidden_states(w, b, 0, n)) for b, n in enumerate(w.ctx_lens)]
    x_t = synth.initial_tokens(w)
    o_res = [o.draft_block(b, int(x_t[b])) for b in range(w.batch)]
    for want_fused in (True, False):
        g = GpuSide(w, flags=flag, weights=W)
        fused = g.fuse(w.ctx_lens, want_fused=want_fused)
        assert g.lib.ctx_lens() == list(w.ctx_lens)
        got = f64(fused) if fused is not None else None
        slots = 1 if kw.get("dflash_fc") else w.shape.n_draft_layers
        for b, n in enumerate(w.ctx_lens):
            if got is not None:
                # +FC's F' is a product of F, whose single-element bf16 flips it carries: row-wise
                chk = check_rows if kw.get("fusion_fc") else check_elem
                chk(w, got[:slots, b, :n], F[b][:slots], f"projected representation seq {b}")
            for i in range(w.shape.n_draft_layers):
                k, v = g.lib.read_kv(i, b, 0, n)
                if got is not None:
                    check_kv(w, o, f64(k), f64(v), got[0 if kw.get("dflash_fc") else i, b, :n],
                             np.arange(n), i, f"seq {b} layer {i}")
                check_rows(w, f64(k), o.ctx_k[b][i], f"{want_fused} seq {b} layer {i} K (end to end)")
                check_rows(w, f64(v), o.ctx_v[b][i], f"{want_fused} seq {b} layer {i} V (end to end)")
        tok, logits, hidden = g.draft(x_t)
        _check_draft(w, tok, logits, hidden, o_res, o)
        assert g.lib.device_error() == 0


@pytest.mark.parametrize("w", [TINY, SMALL_HD128, WIDE_B16], ids=lambda w: w.name)
def test_verify_from_logits_matches_oracle(w):
    """dflare_verify_logits against the oracle: the target's argmax taken from [batch][B][V]
    logits, then prefix acceptance. Rows planted to agree with a random prefix of the drafts,
    ties between two maxima in different vocabulary chunks, and rows of only -inf (lowest id);
    integer results bit-exact, over several rounds on one context."""
    import torch
    s = w.shape
    g = GpuSide(w)
    rng = np.random.default_rng(21)
    B, V, bsz = s.block, s.vocab, w.batch
    for rnd in range(4):
        draft = rng.integers(0, V, (bsz, B - 1)).astype(np.int32)
        lg = rng.standard_normal((bsz, B, V)).astype(np.float32)
        for b in range(bsz):
            a = int(rng.integers(0, B))              # planted prefix length
            for k in range(a):
                lg[b, k, draft[b, k]] = 20.0
            if rnd == 1 and B > 2:                    # a tie: lowest id wins
                lo, hi = sorted(rng.choice(V, 2, replace=False))
                lg[b, B - 1, lo] = lg[b, B - 1, hi] = 30.0
            if rnd == 2:
                lg[b, int(rng.integers(0, B))] = -np.inf
        acc = torch.zeros(bsz, dtype=torch.int32, device="cuda")
        nxt = torch.zeros(bsz, dtype=torch.int32, device="cuda")
        g.lib.verify_logits(torch.from_numpy(draft).cuda(), torch.from_numpy(lg).cuda(), acc, nxt)
        got = list(zip(acc.cpu().tolist(), nxt.cpu().tolist()))
        want = [O.verify_from_logits(draft[b], lg[b]) for b in range(bsz)]
        assert got == want, (rnd, got, want)
    assert g.lib.device_error() == 0


@pytest.mark.parametrize("w", [SMALL_HD128, WIDE_B16], ids=lambda w: w.name)
def test_deterministic_mode_repeats_bit_for_bit(w):
    """DFLARE_FLAG_DETERMINISTIC: two contexts fed the same inputs draft bit-identical hidden
    states and logits; the default mode (split-K partials added to the residual in L2) agrees
    with it within the tolerance."""
    from paper_2606_02091_gb300 import FLAG_DETERMINISTIC
    x_t = synth.initial_tokens(w)
    runs = []
    for flags in (FLAG_DETERMINISTIC, FLAG_DETERMINISTIC, 0):
        g = GpuSide(w, flags=flags)
        g.fuse(w.ctx_lens, want_fused=False)
        runs.append(g.draft(x_t))
        del g
    (t1, l1, h1), (t2, l2, h2), (t3, l3, h3) = runs
    np.testing.assert_array_equal(h1, h2)
    np.testing.assert_array_equal(l1, l2)
    np.testing.assert_array_equal(t1, t2)
    assert rel_err(h3, h1) <= tolerance(w)
    assert rel_err(l3, l1) <= tolerance(w)


def test_repeated_calls_replay_as_graphs():
    """Calls repeated with the same operands run as CUDA graphs (the second is captured, later ones
    replay it). Two deterministic contexts take the same five steps on a side stream: one reusing
    its buffers every step (replayed graphs), one with fresh buffers every call (direct launches).
    Hidden states, logits, tokens, caches and context lengths agree bit for bit, and a change of
    batch or buffers afterwards runs the new operands, not the old graph."""
    import torch
    from paper_2606_02091_gb300 import FLAG_DETERMINISTIC
    w = SMALL_HD128
    s = w.shape
    bsz, B = w.batch, s.block
    runs = []
    for reuse in (True, False):
        g = GpuSide(w, flags=FLAG_DETERMINISTIC)
        st = torch.cuda.Stream()
        dt = torch.bfloat16
        with torch.cuda.stream(st):
            g.fuse(w.ctx_lens, want_fused=False)
            lens = list(w.ctx_lens)
            mk = lambda: (torch.zeros((s.n_target_layers, bsz, B, s.d), dtype=dt, device="cuda"),
                          torch.zeros(bsz, dtype=torch.int32, device="cuda"),
                          torch.tensor(synth.initial_tokens(w), device="cuda"),
                          torch.zeros((bsz, B - 1), dtype=torch.int32, device="cuda"),
                          torch.zeros((bsz, B - 1, s.vocab), dtype=torch.float32, device="cuda"),
                          torch.zeros((s.n_draft_layers + 1, bsz, B, s.d), dtype=torch.float32, device="cuda"))
            bufs = mk()
            out = []
            for step in range(5):
                if not reuse:
                    fresh = mk()
                    fresh[2].copy_(bufs[2])
                    bufs = fresh
                hid, n_new, last, toks, logits, hidden = bufs
                n = [3 + (step + b) % 4 for b in range(bsz)]
                from tests.harness import fill_hidden
                hid.copy_(torch.from_numpy(fill_hidden(w, [B] * bsz, lens)).view(dt))
                n_new.copy_(torch.tensor(n, dtype=torch.int32))
                g.lib.fuse_context(hid, n_new, stream=st)
                lens = [L + k for L, k in zip(lens, n)]
                g.lib.draft_block(last, toks, logits, hidden, stream=st)
                out.append((toks.clone(), logits.clone(), hidden.clone()))
                last.copy_(toks[:, 0])
        torch.cuda.synchronize()
        kv = [g.lib.read_kv(i, b, 0, lens[b]) for i in range(s.n_draft_layers) for b in range(bsz)]
        runs.append((out, kv, g.lib.ctx_lens(), lens))
        assert g.lib.device_error() == 0
        if reuse:   # a different batch after replays: direct launches for the new operands
            from tests.harness import fill_hidden, to_device
            w1 = w.with_(ctx_lens=w.ctx_lens[:1])
            g.lib.reset(1)
            g.lib.fuse_context(to_device(fill_hidden(w1, [w.ctx_lens[0]])),
                               torch.tensor([w.ctx_lens[0]], dtype=torch.int32, device="cuda"))
            t1, l1, h1 = g.draft(synth.initial_tokens(w)[:1])
            o = oracle_for(w1, g.W)
            o.fuse_context(0, synth.hidden_states(w, 0, 0, w.ctx_lens[0]))
            _, ol, oh = o.draft_block(0, int(synth.initial_tokens(w)[0]))
            assert rel_err(l1[0], ol) <= tolerance(w)
    (oa, kva, la, lens_a), (ob, kvb, lb, lens_b) = runs
    assert la == lb == lens_a == lens_b
    for (ta, lga, ha), (tb, lgb, hb) in zip(oa, ob):
        assert torch.equal(ta, tb) and torch.equal(lga, lgb) and torch.equal(ha, hb)
    for (ka, va), (kb, vb) in zip(kva, kvb):
        assert torch.equal(ka, kb) and torch.equal(va, vb)


def test_gemm_timing_stamps_are_ordered():
    """dflare_set_timing on a drafted block: each of the 5 D + 1 timed launches (Q/K^d/V^d,
    attention, O, gate/up, down per layer, then the LM head) records entry <= dependency met <=
    exit, each launch ends after the one before it, and the slots past the last launch stay
    untouched."""
    import torch
    w = SMALL_HD128
    g = GpuSide(w)
    g.fuse(w.ctx_lens, want_fused=False)
    slots = 64
    st = torch.empty(3 * slots, dtype=torch.int64, device="cuda")
    st[:2 * slots].fill_(-1)
    st[2 * slots:].zero_()
    g.lib.set_timing(st, slots)
    g.draft(synth.initial_tokens(w))
    g.lib.set_timing()
    torch.cuda.synchronize()
    a = st.cpu().numpy().view(np.uint64)
    n = 5 * w.shape.n_draft_layers + 1
    entry, dep, done = a[:slots], a[slots:2 * slots], a[2 * slots:]
    for k in range(n):
        assert 0 < entry[k] <= dep[k] <= done[k], k
        if k:
            assert done[k] > done[k - 1], k
    assert np.all(entry[n:] == np.uint64(2 ** 64 - 1)) and np.all(done[n:] == 0)
    assert g.lib.device_error() == 0
