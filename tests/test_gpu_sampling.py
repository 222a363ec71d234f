"""Sampled decoding on the GPU (Table 1, temperature 1) against the oracle.

Both sides draw from the same Philox4x64-10 streams, so given the same logits they take the same
decisions; a decision is compared exactly unless the oracle's float64 evaluation puts it within
the fp32 rounding margin (a top-2 gap of the Gumbel scores, or r q - p for an acceptance, below
1e-4 relative). The draft logits handed to the oracle's verification are the GPU's own (read back
through logits_out), the same input the GPU's verification reads; the logits themselves are
compared with the oracle's by the parity tests. test_sampled_step_end_to_end instead lets the oracle
take every decision of a step from its own logits (with margins for the logit difference between
the two sides). A Monte Carlo test checks the property that defines the rule: the first token a
step emits follows the target's distribution."""
import numpy as np
import pytest

import oracle as O
import synth
from tests.harness import SMALL_HD128, TINY, WIDE_B16, GpuSide, oracle_for

pytestmark = pytest.mark.gpu
MARGIN = 1e-4
CHI2_1E4 = {1: 15.14, 2: 18.42, 3: 21.11, 4: 23.51, 5: 25.74, 6: 27.86, 7: 29.88, 8: 31.83, 9: 33.72}


def _scores(log_w, u):
    with np.errstate(divide="ignore"):
        return np.asarray(log_w, np.float64) - np.log(-np.log(u))


def _draw_ok(gpu_tok, log_w, u):
    """The GPU's draw equals the oracle's, or both lie within the rounding margin of the top."""
    s = _scores(log_w, u)
    top = float(np.max(s))
    tol = MARGIN * (1.0 + abs(top))
    if int(np.argmax(s)) == gpu_tok:
        return True, False
    return bool(s[gpu_tok] >= top - tol), True


def _sampled_run(w, T, seed, step0):
    import torch
    g = GpuSide(w)
    g.fuse(w.ctx_lens, want_fused=False)
    s = w.shape
    bsz = w.batch
    step = torch.tensor([step0], dtype=torch.int64, device="cuda")
    last = torch.tensor(synth.initial_tokens(w), device="cuda")
    toks = torch.zeros((bsz, s.block - 1), dtype=torch.int32, device="cuda")
    logits = torch.zeros((bsz, s.block - 1, s.vocab), dtype=torch.float32, device="cuda")
    g.lib.draft_block_sampled(last, T, seed, step, toks, logits)
    return g, step, toks, logits


@pytest.mark.parametrize("w", [TINY, SMALL_HD128, WIDE_B16], ids=lambda w: w.name)
@pytest.mark.parametrize("T", [1.0, 0.5, 2.0])
def test_sampled_draft_matches_oracle(w, T):
    seed, step0 = 1234, 77
    g, step, toks, logits = _sampled_run(w, T, seed, step0)
    tok = toks.cpu().numpy()
    lg = logits.cpu().numpy()
    s = w.shape
    near = 0
    for b in range(w.batch):
        for k in range(s.block - 1):
            u = O.uniforms(seed, O.RNG_DRAFT, step0, b * (s.block - 1) + k, s.vocab)
            ok, tie = _draw_ok(int(tok[b, k]), lg[b, k].astype(np.float64) / T, u)
            assert ok, (b, k)
            near += tie
    assert near <= max(1, tok.size // 50)
    assert int(step.item()) == step0            # drafting reads the counter, never advances it
    assert g.lib.device_error() == 0


@pytest.mark.parametrize("w", [TINY, SMALL_HD128, WIDE_B16], ids=lambda w: w.name)
def test_sampled_verification_matches_oracle(w):
    import torch
    T, seed = 1.0, 99
    s = w.shape
    B, V, bsz = s.block, s.vocab, w.batch
    rng = np.random.default_rng(31)
    for rnd, step0 in enumerate((5, 6, 7)):
        g, step, toks, logits = _sampled_run(w, T, seed, step0)
        tok = toks.cpu().numpy()
        dl = logits.cpu().numpy().astype(np.float64)
        # target logits near the draft's (frequent acceptance), with some rows replaced by
        # unrelated logits (frequent rejection) and a planted -inf at a drafted token
        tl = np.empty((bsz, B, V), np.float32)
        for b in range(bsz):
            tl[b, :B - 1] = dl[b] / T * rng.uniform(0.7, 1.3) + 0.3 * rng.standard_normal((B - 1, V))
            tl[b, B - 1] = 2.0 * rng.standard_normal(V)
            for k in range(B - 1):
                if rng.random() < 0.15:
                    tl[b, k] = 2.0 * rng.standard_normal(V)
            if rnd == 2 and B > 2:
                tl[b, 1, tok[b, 1]] = -np.inf
        acc = torch.zeros(bsz, dtype=torch.int32, device="cuda")
        nxt = torch.zeros(bsz, dtype=torch.int32, device="cuda")
        g.lib.verify_sampled(toks, torch.from_numpy(tl).cuda(), T, seed, step, acc, nxt)
        acc_h, nxt_h = acc.cpu().numpy(), nxt.cpu().numpy()
        assert int(step.item()) == step0 + 1
        for b in range(bsz):
            r = O.uniforms(seed, O.RNG_ACCEPT, step0, b, B - 1)
            u = O.uniforms(seed, O.RNG_RESIDUAL, step0, b, V)
            # the oracle's decisions, with their float64 margins
            a, borderline = 0, False
            while a < B - 1:
                p = O.softmax_t(tl[b, a], T)
                q = O.softmax_t(dl[b, a], T)
                d = int(tok[b, a])
                lhs, rhs = r[a] * q[d], p[d]
                if abs(lhs - rhs) <= MARGIN * max(lhs, rhs):
                    borderline = True
                    break
                if lhs < rhs:
                    a += 1
                else:
                    break
            if borderline:
                continue
            tau, nxt_o = O.speculative_verify(tok[b], tl[b], dl[b], T, r, u)
            assert tau == a + 1
            assert acc_h[b] == tau, (rnd, b, acc_h[b], tau)
            if a < B - 1:
                wdist = O.residual_dist(O.softmax_t(tl[b, a], T), O.softmax_t(dl[b, a], T))
            else:
                wdist = O.softmax_t(tl[b, B - 1], T)
            with np.errstate(divide="ignore"):
                ok, _ = _draw_ok(int(nxt_h[b]), np.log(wdist), u)
            # p - q in fp32 loses relative accuracy where p and q nearly cancel: accept a GPU
            # draw whose residual weight is within that cancellation of the oracle's choice
            if not ok and a < B - 1:
                p = O.softmax_t(tl[b, a], T)
                q = O.softmax_t(dl[b, a], T)
                t_g, t_o = int(nxt_h[b]), int(nxt_o)
                slack = 1e-5 * (p + q) / np.maximum(np.maximum(p - q, 0), 1e-30)
                sc = _scores(np.log(np.maximum(p - q, 1e-300)), u)
                ok = sc[t_g] + slack[t_g] >= sc[t_o] - slack[t_o]
            assert ok, (rnd, b, int(nxt_h[b]), int(nxt_o))
        assert g.lib.device_error() == 0


@pytest.mark.parametrize("w", [TINY, SMALL_HD128], ids=lambda w: w.name)
def test_sampled_step_end_to_end(w):
    """One sampled step decided by the oracle alone: it fuses the same target states, computes its
    own draft logits, draws its own tokens and runs its own acceptance on the same Philox streams,
    and the GPU's drafts, accept lengths and next tokens must equal those decisions. The target
    logits are built from the oracle's draft logits. A decision is compared exactly unless the
    oracle's own margin for it lies within what the logit difference between the two sides can
    move: 2 max|l_gpu - l_oracle| / T for a draw, the matching relative change of q(d) for an
    acceptance; such borderline decisions must stay rare."""
    import torch
    T, seed, step0 = 1.0, 4321, 11
    s = w.shape
    B, V, bsz = s.block, s.vocab, w.batch
    g, step, toks, logits = _sampled_run(w, T, seed, step0)
    tok_g = toks.cpu().numpy()
    lg = logits.cpu().numpy().astype(np.float64)
    o = oracle_for(w, g.W)
    for b, n in enumerate(w.ctx_lens):
        o.fuse_context(b, synth.hidden_states(w, b, 0, n))
    x_t = synth.initial_tokens(w)
    rng = np.random.default_rng(5)
    tl = np.empty((bsz, B, V), np.float32)
    tok_o = np.zeros((bsz, B - 1), np.int64)
    dl_o, shift, same = [], [], []
    decided = borderline = 0
    for b in range(bsz):
        _, lo, _ = o.draft_block(b, int(x_t[b]))
        dl_o.append(lo)
        delta = float(np.max(np.abs(lg[b] - lo))) / T   # largest score shift between the sides
        shift.append(delta)
        agree = True
        for k in range(B - 1):
            u = O.uniforms(seed, O.RNG_DRAFT, step0, b * (B - 1) + k, V)
            sc = _scores(lo[k] / T, u)
            t = int(np.argmax(sc))
            tok_o[b, k] = t
            assert t == O.sample_token(lo[k], T, u)
            gap = sc[t] - float(np.max(np.delete(sc, t)))
            if gap > 2.0 * delta + MARGIN * (1.0 + abs(sc[t])):
                assert int(tok_g[b, k]) == t, (b, k, int(tok_g[b, k]), t, gap, delta)
                decided += 1
            else:
                borderline += 1
                agree = agree and int(tok_g[b, k]) == t
        same.append(agree)
        tl[b, :B - 1] = lo / T * rng.uniform(0.7, 1.3) + 0.3 * rng.standard_normal((B - 1, V))
        tl[b, B - 1] = 2.0 * rng.standard_normal(V)
        for k in range(B - 1):
            if rng.random() < 0.15:
                tl[b, k] = 2.0 * rng.standard_normal(V)
    assert decided > 0 and borderline <= max(2, (decided + borderline) // 10), (decided, borderline)
    acc = torch.zeros(bsz, dtype=torch.int32, device="cuda")
    nxt = torch.zeros(bsz, dtype=torch.int32, device="cuda")
    g.lib.verify_sampled(toks, torch.from_numpy(tl).cuda(), T, seed, step, acc, nxt)
    acc_h, nxt_h = acc.cpu().numpy(), nxt.cpu().numpy()
    assert int(step.item()) == step0 + 1
    checked = 0
    for b in range(bsz):
        if not same[b]:
            continue                      # a borderline draw went the other way on the GPU
        r = O.uniforms(seed, O.RNG_ACCEPT, step0, b, B - 1)
        u = O.uniforms(seed, O.RNG_RESIDUAL, step0, b, V)
        rel = np.expm1(2.0 * shift[b])    # bound on the relative change of q(d) between the sides
        a, clear = 0, True
        while a < B - 1:
            p = O.softmax_t(tl[b, a], T)
            q = O.softmax_t(dl_o[b][a], T)
            d = int(tok_o[b, a])
            lhs, rhs = r[a] * q[d], p[d]
            if abs(lhs - rhs) <= (rel + MARGIN) * max(lhs, rhs):
                clear = False
                break
            if lhs < rhs:
                a += 1
            else:
                break
        if not clear:
            continue
        tau, nxt_o = O.speculative_verify(tok_o[b], tl[b], dl_o[b], T, r, u)
        assert tau == a + 1
        assert acc_h[b] == tau, (b, acc_h[b], tau)
        if a < B - 1:
            # the replacement draws from max(0, p - q): q moves by at most rel q between the sides
            p = O.softmax_t(tl[b, a], T)
            q = O.softmax_t(dl_o[b][a], T)
            wgt = np.maximum(p - q, 0)
            slack = (rel + 1e-5) * (p + q) / np.maximum(wgt, 1e-30)
            with np.errstate(divide="ignore"):
                sc = _scores(np.log(np.maximum(wgt, 1e-300)), u)
            t_g, t_o = int(nxt_h[b]), int(nxt_o)
            assert t_g == t_o or sc[t_g] + slack[t_g] >= sc[t_o] - slack[t_o], (b, t_g, t_o)
        else:
            with np.errstate(divide="ignore"):
                ok, _ = _draw_ok(int(nxt_h[b]), np.log(O.softmax_t(tl[b, B - 1], T)), u)
            assert ok, (b, int(nxt_h[b]), int(nxt_o))
        checked += 1
    assert checked >= 1
    assert g.lib.device_error() == 0


def test_first_emitted_token_follows_the_target():
    """3000 sampled steps on one context: whatever the draft proposes, the first token a step
    emits (d_1 when kept, else the replacement) is distributed as softmax(target row 0 / T), and
    the drafted d_1 as softmax(draft row 0 / T). T = 0.05 sharpens the synthetic drafter's nearly
    flat logits so that a few tokens carry most of the mass and both branches of the rule occur."""
    import torch
    w = TINY
    s = w.shape
    T, seed, n = 0.05, 5, 3000
    g, step, toks, logits = _sampled_run(w, T, seed, 0)
    dl = logits.cpu().numpy().astype(np.float64)
    rng = np.random.default_rng(2)
    tl = np.empty((1, s.block, s.vocab), np.float32)
    tl[0] = np.concatenate([dl[0], dl[0, -1:]]) + 0.03 * rng.standard_normal((s.block, s.vocab))
    tl_d = torch.from_numpy(tl).cuda()
    p0 = O.softmax_t(tl[0, 0], T)
    q0 = O.softmax_t(dl[0, 0], T)
    last = torch.tensor(synth.initial_tokens(w), device="cuda")
    acc = torch.zeros(1, dtype=torch.int32, device="cuda")
    nxt = torch.zeros(1, dtype=torch.int32, device="cuda")
    d1 = torch.zeros(n, dtype=torch.int32, device="cuda")
    a = torch.zeros(n, dtype=torch.int32, device="cuda")
    nx = torch.zeros(n, dtype=torch.int32, device="cuda")
    step.zero_()
    for i in range(n):
        g.lib.draft_block_sampled(last, T, seed, step, toks)
        g.lib.verify_sampled(toks, tl_d, T, seed, step, acc, nxt)
        d1[i:i + 1].copy_(toks[0, :1])
        a[i:i + 1].copy_(acc)
        nx[i:i + 1].copy_(nxt)
    d1, a, nx = d1.cpu().numpy(), a.cpu().numpy(), nx.cpu().numpy()
    first = np.where(a >= 2, d1, nx)
    assert int(step.item()) == n
    assert 0.05 < np.mean(a >= 2) < 0.95           # both branches of the rule are exercised

    def chi2(samples, probs):
        order = np.argsort(-probs)
        k = min(max(int(np.sum(probs[order] * n >= 20)), 2), 8)
        bins = list(order[:k])
        e = np.array([probs[t] for t in bins] + [1 - probs[bins].sum()]) * n
        c = np.array([np.sum(samples == t) for t in bins] + [np.sum(~np.isin(samples, bins))])
        keep = e > 0
        return float(np.sum((c[keep] - e[keep]) ** 2 / e[keep])), int(keep.sum()) - 1

    stat, df = chi2(first, p0)
    assert stat < CHI2_1E4[df], (stat, df)
    stat, df = chi2(d1, q0)
    assert stat < CHI2_1E4[df], (stat, df)
    assert g.lib.device_error() == 0


def test_temperature_is_checked_on_the_host():
    import torch
    from paper_2606_02091_gb300 import DFlareError
    w = TINY
    g, step, toks, logits = _sampled_run(w, 1.0, 0, 0)
    last = torch.tensor(synth.initial_tokens(w), device="cuda")
    for bad in (0.0, -1.0, float("inf"), float("nan"), 1e-45):
        with pytest.raises(DFlareError):
            g.lib.draft_block_sampled(last, bad, 0, step, toks)
