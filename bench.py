#!/usr/bin/env python
"""Throughput of the DFlare per-step draft path on one GB300 (or N independent replicas).

One step = one block step of the path on the workload's batch: fuse the previous step's
accepted positions (Eq. 3, Eq. 4) -> draft a block (Sec. 3.2) -> synthetic target argmax ->
prefix acceptance (Sec. 3.2). Inputs are seeded synthetic tensors shaped like the named drafter
(weights N(0, 0.02), target states N(0,1) x U(0.5, 4) per layer). The headline workload is the
largest single-GPU one, the Qwen3-8B-shaped drafter at batch 4: d 4096, 8 draft layers, 36 fused
target layers, block 16, ragged contexts U{1024..4096}; the line's `configs` object holds the same
measurement for the other drafter shapes (tiny fp32, Qwen3-4B, Qwen3-8B batch 1, GPT-OSS-20B
batch 2).

Prints one JSON line (rank 0). `value` = drafted tokens/s (batch x (B-1) per step) over the
timed CUDA-graph replays with inputs resident in HBM; `e2e` = the same metric through the public
calls with the step's inputs copied from pinned host memory and results read back every step;
`roofline` = the dominant kernel's (the projection GEMM's) algorithmic bytes over its
event-timed launch durations vs the measured HBM copy bandwidth; `cpu_baseline` = the CPU oracle
on a bounded sample. `--impl reference` times the CPU oracle alone (the reference arm).
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "drafted tokens/s per GB300 (block 16)"
UNIT = "drafted tokens/s"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=HEADLINE, choices=sorted(synth.PRESETS))
    p.add_argument("--headline-only", action="store_true",
                   help="measure the --workload only (no per-config sub-objects)")
    p.add_argument("--draft-layers", type=int, default=0,
                   help="override D of --workload (a smaller case for profiling); implies --headline-only")
    p.add_argument("--vocab", type=int, default=0,
                   help="override the vocabulary of --workload; implies --headline-only")
    p.add_argument("--batch", type=int, default=0,
                   help="override the batch of --workload (every context as long as the longest); "
                        "implies --headline-only")
    p.add_argument("--ctx", type=int, default=0,
                   help="override every context length of --workload; implies --headline-only")
    p.add_argument("--sub-cpu-seconds", type=float, default=6.0,
                   help="CPU time budget of the oracle steps of each non-headline workload")
    p.add_argument("--e2e-steps", type=int, default=50)
    p.add_argument("--breakdown-steps", type=int, default=30)
    p.add_argument("--cpu-seconds", type=float, default=12.0,
                   help="CPU time budget of the oracle steps timed for cpu_baseline")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--fill-chunk", type=int, default=2048)
    p.add_argument("--serial-launch", action="store_true",
                   help="no programmatic dependent launch between kernels (A/B measurement)")
    p.add_argument("--mma-sync-attention", action="store_true",
                   help="the mma.sync attention kernel instead of the tcgen05 one (A/B measurement)")
    p.add_argument("--sweep", action="store_true",
                   help="throughput sweep around the Qwen3-8B-shaped drafter (one JSON line per point)")
    p.add_argument("--sweep-points", default="",
                   help="comma-separated indexes into the sweep's point list (default: all)")
    p.add_argument("--no-variants", action="store_true",
                   help="skip the context-fusion comparison with the ablations and DFlash's FC")
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return d.get("hbm_gbs", 6800.0), "measured", d
    return 6800.0, "fallback", {}


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


# ----------------------------------------------------------------------------- CPU oracle leg

def oracle_steps(w, W, n_steps, budget_s=None):
    """Time full oracle block steps after an untimed oracle context fill: n_steps of them, or,
    with budget_s, as many as fit in budget_s seconds (at least 2, at most n_steps)."""
    import oracle as O
    s = w.shape
    o = O.DraftOracle(W, s, w.batch, storage="bf16" if s.dtype == "bf16" else "exact")
    for b, L in enumerate(w.ctx_lens):
        o.fuse_context(b, synth.hidden_states(w, b, 0, L))
    # decode the weights once before timing (the oracle keeps float64 copies)
    for i in range(s.n_draft_layers):
        o.layer(i)
    o._dec("lm_head")
    o._dec("final_norm")
    x_t = synth.initial_tokens(w).astype(np.int64)
    taus = [0] * w.batch
    lens = list(w.ctx_lens)
    thr = synth.accept_threshold(w.match_p)
    t0 = time.perf_counter()
    tau_sum = 0
    done = 0
    for step in range(n_steps):
        if budget_s is not None and step >= 2 and time.perf_counter() - t0 >= budget_s:
            break
        done += 1
        u, r, last = synth.target_draws(w, step)
        for b in range(w.batch):
            if taus[b]:
                o.fuse_context(b, synth.hidden_states(w, b, lens[b], taus[b]))
                lens[b] += taus[b]
            tok, _, _ = o.draft_block(b, int(x_t[b]))
            g = O.synthetic_target(tok, u[0, b], r[0, b], last[0, b], thr)
            taus[b], x_t[b] = O.verify_accept(tok, g)
            tau_sum += taus[b]
    dt = time.perf_counter() - t0
    drafted = done * w.batch * (s.block - 1)
    return drafted / dt, dt, tau_sum / (done * w.batch), done


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = synth.preset(args.workload)
    W = synth.weights(w)
    # bounded: at most ~150 s of oracle steps in the whole run
    value, dt, tau, n = oracle_steps(w, W, args.steps, budget_s=150.0)
    sample = (f"{n} of {args.steps} requested block steps of workload {w.name} (oracle fp64, "
              f"bf16 storage rounding) after an untimed oracle fill of {list(w.ctx_lens)} "
              f"positions; warmup: 1 step")
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dt / n, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "impl": "reference",
        "config": config_of(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": host_cores(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "mean_accept_len": tau,
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 200 ms while running."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.out = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.out.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.out:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- cudart events

class Cudart:
    """cudaEvent* from the CUDA runtime torch loaded (events recorded inside captured graphs)."""

    def __init__(self):
        import torch  # noqa: F401  (loads libcudart)
        lib = None
        for name in ("libcudart.so.13", "libcudart.so.12", "libcudart.so"):
            try:
                lib = ctypes.CDLL(name)
                break
            except OSError:
                continue
        if lib is None:
            import glob
            cands = glob.glob("/usr/local/cuda/lib64/libcudart.so*")
            lib = ctypes.CDLL(cands[0])
        self.lib = lib
        lib.cudaEventCreate.argtypes = [ctypes.POINTER(ctypes.c_void_p)]
        lib.cudaEventRecordWithFlags.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint]
        lib.cudaEventElapsedTime.argtypes = [ctypes.POINTER(ctypes.c_float), ctypes.c_void_p,
                                             ctypes.c_void_p]
        lib.cudaEventDestroy.argtypes = [ctypes.c_void_p]

    def event(self):
        e = ctypes.c_void_p()
        assert self.lib.cudaEventCreate(ctypes.byref(e)) == 0
        return e

    def record(self, e, stream, captured=True):
        # cudaEventRecordExternal: inside stream capture this becomes an event-record node; an
        # eager launch takes the default flags
        assert self.lib.cudaEventRecordWithFlags(e, stream, 1 if captured else 0) == 0

    def elapsed(self, a, b):
        ms = ctypes.c_float()
        assert self.lib.cudaEventElapsedTime(ctypes.byref(ms), a, b) == 0
        return ms.value


def kernels_per_trace(shape):
    """Kernel launches behind one traced call site (attention is one launch in bf16, split +
    combine in fp32)."""
    return {"attention": 1 if shape.dtype == "bf16" else 2}


def algorithmic_bytes(w, name, mean_tau, mean_ctx=None):
    """Bytes a launch of `name` must move at minimum (weights, activations, caches, outputs).
    mean_ctx: the sequences' mean context length when the launch ran (default: the workload's
    initial contexts; the benchmark's contexts grow by tau every step)."""
    s = w.shape
    b, B, d, F, V = w.batch, s.block, s.d, s.ffn, s.vocab
    e = 2 if s.dtype == "bf16" else 4
    dq, dkv = s.d_q, s.d_kv
    M = b * B
    Mh = b * (B - 1)
    L = float(np.mean(w.ctx_lens)) if mean_ctx is None else float(mean_ctx)
    if name == "gemm_lm_head":
        return V * d * e + Mh * d * e + Mh * V * 4
    if name == "gemm_gate_up":
        return 2 * F * d * e + M * d * e + M * F * e
    if name == "gemm_down":
        return d * F * e + M * F * e + 2 * M * d * 4
    if name == "gemm_qkv":
        return (dq + 2 * dkv) * d * e + M * d * e + M * (dq + 2 * dkv) * e
    if name == "gemm_o":
        return d * dq * e + M * dq * e + 2 * M * d * 4
    if name == "gemm_kv_ctx":
        n = b * mean_tau
        return s.n_draft_layers * (2 * dkv * d * e + n * d * e + n * 2 * dkv * e)
    if name == "attention":
        return b * (L + B) * 2 * dkv * e + 2 * M * dq * e
    if name == "fuse_layers":
        n = b * mean_tau
        return n * (s.n_target_layers + s.n_draft_layers) * d * e
    if name == "argmax":
        return Mh * V * 4
    return 0


def gemm_traffic(w):
    """DRAM bytes per step of the GEMM kernel from the committed ncu summary, if it was measured
    on this workload and on the current GEMM sources."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"gemm_tc_traffic_{w.name}.json")
    if not os.path.exists(path):
        return None
    d = json.load(open(path))
    csrc = os.path.join(ROOT, "paper_2606_02091_gb300", "csrc")
    src = open(os.path.join(csrc, "gemm_tc.cu"), "rb").read() + \
        open(os.path.join(csrc, "epilogue.cuh"), "rb").read()
    if hashlib.sha256(src).hexdigest()[:16] != d.get("source_sha256_16"):
        return None
    return d.get("dram_bytes_per_step")


FUSION_VARIANTS = (("dflare", ()), ("minus_kvproj", ("FLAG_SHARED_KV",)),
                   ("plus_fc", ("FLAG_FUSION_FC",)), ("dflash_fc", ("FLAG_DFLASH_FC",)))


def fusion_variants(w, dev_w, fill_chunks, hid_step, n_step, reps=100):
    """Time one dflare_fuse_context call (fusion, optional FC, context K/V projection) of DFlare
    and of each variant: at decode (n_step new positions per sequence, a CUDA graph of one call
    replayed `reps` times between events) and at a context fill (the fill chunks, once untimed,
    then timed from an empty context)."""
    import torch
    import paper_2606_02091_gb300 as P
    from paper_2606_02091_gb300 import DFlare
    s = w.shape
    esz = 2 if s.dtype == "bf16" else 4
    extra = {}
    for k, v in synth.variant_weights(w).items():
        t = torch.from_numpy(v)
        extra[k] = (t.view(torch.bfloat16) if v.dtype == np.uint16 else t).cuda()
    n_fill = sum(w.ctx_lens)
    fill_rows = max(Ht.shape[2] for Ht, _ in fill_chunks)
    n_new = torch.full((w.batch,), n_step, dtype=torch.int32, device="cuda")
    out = {}
    for name, flags in FUSION_VARIANTS:
        flag = 0
        for f in flags:
            flag |= getattr(P, f)
        lib = DFlare.from_shape(s, max_batch=w.batch, max_ctx=max(w.ctx_lens) + n_step * (reps + 8),
                                max_fuse_rows=w.batch * max(fill_rows, s.block), flags=flag)
        lib.set_weights({**dev_w, **extra})
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        fill_ms = None
        for timed in (False, True):
            lib.reset(w.batch)
            torch.cuda.synchronize()
            ev[0].record()
            for Ht, nt in fill_chunks:
                lib.fuse_context(Ht, nt)
            ev[1].record()
            torch.cuda.synchronize()
            fill_ms = ev[0].elapsed_time(ev[1])
        lib.reset(w.batch)
        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cs):
            lib.fuse_context(hid_step, n_new)
            torch.cuda.synchronize()
            with torch.cuda.graph(graph, stream=cs):
                lib.fuse_context(hid_step, n_new)
        torch.cuda.synchronize()
        lib.reset(w.batch)
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize()
        ev[2].record()
        for _ in range(reps):
            graph.replay()
        ev[3].record()
        torch.cuda.synchronize()
        if lib.device_error():
            raise RuntimeError(f"device error in the {name} fusion variant")
        step_us = 1e3 * ev[2].elapsed_time(ev[3]) / reps
        wbytes = {"dflare": s.n_draft_layers * 2 * s.d_kv * s.d,
                  "minus_kvproj": s.n_draft_layers * 2 * s.d_kv * s.d,
                  "plus_fc": s.n_draft_layers * (2 * s.d_kv + s.d) * s.d,
                  "dflash_fc": s.n_target_layers * s.d * s.d + s.n_draft_layers * 2 * s.d_kv * s.d}
        out[name] = {"step_us": step_us, "fill_us": 1e3 * fill_ms,
                     "weight_bytes_per_call": wbytes[name] * esz}
        del graph
        lib.close()
    out["note"] = (f"one dflare_fuse_context call per entry: decode = {n_step} new positions per "
                   f"sequence (CUDA graph of one call, {reps} replays); fill = {n_fill} positions "
                   "from empty. dflare: Eq. 3 + Eq. 4; minus_kvproj / plus_fc: the Sec. 6.3 "
                   "ablations; dflash_fc: Eq. 1 (one GEMM over the T stacked target layers) + "
                   "Eq. 2's shared K/V projection")
    return out


def sampled_steps(w, dev_w, fill_chunks, hid_step, x0, reps=100, temperature=1.0, seed=2024):
    """Block steps at temperature 1 (Table 1's sampled rows): fuse the previous step's tau
    positions, draft with dflare_draft_block_sampled, verify with dflare_verify_sampled against
    fixed synthetic target logits ([batch][B][V] N(0, 1), resident in HBM), in a CUDA graph of one
    step replayed `reps` times between events, on a context filled like the main run."""
    import torch
    from paper_2606_02091_gb300 import DFlare
    s = w.shape
    fill_rows = max(Ht.shape[2] for Ht, _ in fill_chunks)
    lib = DFlare.from_shape(s, max_batch=w.batch, max_ctx=max(w.ctx_lens) + s.block * (reps + 8),
                            max_fuse_rows=w.batch * max(fill_rows, s.block))
    lib.set_weights(dev_w)
    lib.reset(w.batch)
    for Ht, nt in fill_chunks:
        lib.fuse_context(Ht, nt)
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    tgt = torch.randn((w.batch, s.block, s.vocab), generator=g, device="cuda")
    step_ctr = torch.zeros(1, dtype=torch.int64, device="cuda")
    acc = torch.zeros(w.batch, dtype=torch.int32, device="cuda")
    nxt = x0.clone()
    draft = torch.zeros((w.batch, s.block - 1), dtype=torch.int32, device="cuda")

    def step():
        lib.fuse_context(hid_step, acc)
        lib.draft_block_sampled(nxt, temperature, seed, step_ctr, draft)
        lib.verify_sampled(draft, tgt, temperature, seed, step_ctr, acc, nxt)

    cs = torch.cuda.Stream()
    cs.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cs):
        step()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph, stream=cs):
            step()
    torch.cuda.synchronize()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    lens0 = lib.ctx_lens()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    lens1 = lib.ctx_lens()
    if lib.device_error():
        raise RuntimeError("device error in the sampled steps")
    out = {"ms_per_step": ms, "drafted_tokens_per_s": w.batch * (s.block - 1) / (ms / 1e3),
           "mean_accept_len": (sum(lens1) - sum(lens0)) / (reps * w.batch),
           "temperature": temperature, "steps": reps, "rng_steps": int(step_ctr.item()),
           "note": "CUDA graph of one step (fuse tau positions, sampled draft, speculative-sampling "
                   "verification); target logits are fixed N(0, 1) draws, so tau reflects an "
                   "unrelated target, not a trained pair"}
    del graph
    lib.close()
    return out


def graph_breakdown(lib, cs, step, nb, only=None):
    """Per-launch durations: a CUDA graph of one step with CUDA events recorded by the library's
    trace hook around every launch (or, with `only`, around the launches whose call-site name it
    accepts; the other launches keep their programmatic dependent launch), replayed nb times.
    Returns (name -> [ms, ...], ms per traced step). An event pair around a launch also holds that
    launch's own launch latency, which inside the untraced graph overlaps the previous kernel."""
    import torch
    import paper_2606_02091_gb300 as P
    cr = Cudart()
    rec = []
    pool = []

    @P._lib.TRACE_FN
    def ev_cb(user, name, phase, stream):
        n = name.decode()
        if only is not None and not only(n):
            return
        if len(pool) <= len(rec):
            pool.append(cr.event())
        e = pool[len(rec)]
        cr.record(e, stream)
        rec.append((n, phase, e))

    L_ = P.load()
    L_.dflare_set_trace(lib.raw, ev_cb, None)
    g2 = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cs):
        with torch.cuda.graph(g2, stream=cs):
            step()
    L_.dflare_set_trace(lib.raw, P._lib.TRACE_FN(), None)
    torch.cuda.synchronize()
    per = {}
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    total = 0.0
    for _ in range(nb):
        t0.record()
        g2.replay()
        t1.record()
        torch.cuda.synchronize()
        total += t0.elapsed_time(t1)
        open_ev = {}
        for name, phase, e in rec:
            if phase == 0:
                open_ev.setdefault(name, []).append(e)
            else:
                st = open_ev[name].pop()
                per.setdefault(name, []).append(cr.elapsed(st, e))
    del g2
    return per, total / max(nb, 1)


def gemm_timeline(lib, cs, step, nb, slots=256):
    """Device-side times of every projection-GEMM and attention launch of one step inside a CUDA
    graph of the step with nothing added between its launches (dflare_set_timing: %globaltimer at
    the first CTA's entry, at the first CTA's met dependency, at the last CTA's exit), replayed nb
    times. Returns (names, [[(entry, ready, exit) ns per launch] per replay])."""
    import torch
    import paper_2606_02091_gb300 as P
    names = []

    @P._lib.TRACE_FN
    def name_cb(user, name, phase, stream):
        n = name.decode()
        if phase == 0 and (n.startswith("gemm_") or n == "attention"):
            names.append(n)

    L_ = P.load()
    stamps = torch.empty(3 * slots, dtype=torch.int64, device="cuda")
    L_.dflare_set_trace(lib.raw, name_cb, None)
    lib.set_timing(stamps, slots)
    g3 = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cs):
        with torch.cuda.graph(g3, stream=cs):
            step()
    lib.set_timing()
    L_.dflare_set_trace(lib.raw, P._lib.TRACE_FN(), None)
    torch.cuda.synchronize()
    n = min(len(names), slots)
    runs = []
    for _ in range(nb):
        stamps[:2 * slots].fill_(-1)
        stamps[2 * slots:].zero_()
        g3.replay()
        torch.cuda.synchronize()
        a = stamps.cpu().numpy().view(np.uint64)
        runs.append([(int(a[k]), int(a[slots + k]), int(a[2 * slots + k])) for k in range(n)])
    del g3
    return names[:n], runs


def union_ns(spans):
    """Total length of the union of [start, end) intervals."""
    tot, cur_s, cur_e = 0, None, None
    for s0, e0 in sorted(spans):
        if cur_e is None or s0 > cur_e:
            if cur_e is not None:
                tot += cur_e - cur_s
            cur_s, cur_e = s0, e0
        else:
            cur_e = max(cur_e, e0)
    if cur_e is not None:
        tot += cur_e - cur_s
    return tot


def replica_aggregate(ms, units_per_step, steps, dist=None, device="cuda"):
    """Weak-scaling aggregate of independent replicas (one per rank, no data-path exchange):
    the job's time is the slowest rank's, its throughput every rank's units over that time.
    Returns (max ms over ranks, units per second of the whole job)."""
    world = 1
    if dist is not None and dist.is_initialized():
        import torch
        t = torch.tensor([float(ms)], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        world = dist.get_world_size()
    return ms, world * units_per_step * steps / (ms / 1e3)


def config_of(w):
    """The `config` object of a bench line (both arms print the same keys)."""
    s = w.shape
    return {"workload": w.name, "dtype": s.dtype, "d": s.d, "draft_layers": s.n_draft_layers,
            "target_layers": s.n_target_layers, "heads": [s.n_q_heads, s.n_kv_heads],
            "head_dim": s.head_dim, "ffn": s.ffn, "vocab": s.vocab, "block": s.block,
            "batch": w.batch, "ctx": list(w.ctx_lens), "match_p": w.match_p}


# the benchmark's workloads: the headline (the largest single-GPU workload: Qwen3-8B-shaped,
# ragged batch 4) and the other drafter shapes, each measured the same way
HEADLINE = "qwen3_8b_b4"
CONFIG_SET = ("tiny_f32", "qwen3_4b", "qwen3_8b_b1", "qwen3_8b_b4", "gptoss_20b_b2")
N_ROT = 4     # per-step target-state buffers rotated through the timed steps


def measure(w, args, steps, warmup, e2e_steps, nb, cpu_seconds, extras, dist=None, world=1,
            rank=0, local=0):
    """One workload: context fill, then `steps` timed block steps (CUDA-graph replays, inputs
    resident in HBM), the per-launch breakdown, the end-to-end loop through the public calls
    and, optionally, the fusion variants, the sampled path and the CPU oracle. Returns the
    measurement as a dict (the fields of a bench line)."""
    import torch
    import paper_2606_02091_gb300 as P
    from paper_2606_02091_gb300 import DFlare, synthetic_target

    s = w.shape
    K, Wm, E = steps, max(warmup, 3), e2e_steps
    W = synth.weights(w)
    dev_w = {}
    for k, v in W.items():
        t = torch.from_numpy(v)
        dev_w[k] = (t.view(torch.bfloat16) if v.dtype == np.uint16 else t).cuda()
    chunk = min(args.fill_chunk, max(w.ctx_lens))
    n_steps_total = Wm + K + E + nb + 16
    max_ctx = max(w.ctx_lens) + s.block * n_steps_total
    lib = DFlare.from_shape(s, max_batch=w.batch, max_ctx=max_ctx,
                            max_fuse_rows=w.batch * max(chunk, s.block),
                            flags=(P.FLAG_SERIAL_LAUNCH if args.serial_launch else 0) |
                            (P.FLAG_MMA_SYNC_ATTENTION if args.mma_sync_attention else 0))
    lib.set_weights(dev_w)
    lib.reset(w.batch)
    # context fill in chunks (the target's prompt states): once untimed, then again from an empty
    # context with CUDA events around the fusion and context-projection launches (the fusion and
    # the context K/V projection are measured at fill, where n = L positions per call)
    dt_np = np.uint16 if s.dtype == "bf16" else np.float32
    fill_chunks = []
    for pos0 in range(0, max(w.ctx_lens), chunk):
        ns = [max(0, min(chunk, L - pos0)) for L in w.ctx_lens]
        H = np.zeros((s.n_target_layers, w.batch, chunk, s.d), dt_np)
        for b, n in enumerate(ns):
            if n:
                H[:, b, :n] = synth.hidden_states(w, b, pos0, n)
        Ht = torch.from_numpy(H)
        fill_chunks.append(((Ht.view(torch.bfloat16) if dt_np == np.uint16 else Ht).cuda(),
                            torch.tensor(ns, dtype=torch.int32, device="cuda")))
        del H, Ht
    fill_ev = []
    crf = Cudart()

    @P._lib.TRACE_FN
    def fill_cb(user, name, phase, stream):
        e = crf.event()
        crf.record(e, stream, captured=False)
        fill_ev.append((name.decode(), phase, e))

    for timed in (False, True):
        lib.reset(w.batch)
        if timed:
            P.load().dflare_set_trace(lib.raw, fill_cb, None)
        for Ht, nt in fill_chunks:
            lib.fuse_context(Ht, nt)
        if timed:
            P.load().dflare_set_trace(lib.raw, P._lib.TRACE_FN(), None)
        torch.cuda.synchronize()
    fill_us = {}
    open_f = {}
    for name, phase, e in fill_ev:
        if phase == 0:
            open_f[name] = e
        else:
            fill_us[name] = fill_us.get(name, 0.0) + 1e3 * crf.elapsed(open_f.pop(name), e)
    n_fill = sum(w.ctx_lens)
    e_sz = 2 if s.dtype == "bf16" else 4
    fuse_bytes = n_fill * (s.n_target_layers + s.n_draft_layers) * s.d * e_sz
    kv_flops = 2.0 * n_fill * s.n_draft_layers * 2 * s.d_kv * s.d
    # per-step buffers: target states of up to B newly committed positions (N_ROT different
    # buffers, used in turn, so no step fuses the rows the step before it fused), draws of the
    # synthetic target for n_tab steps, and the loop state (accept_len doubles as next n_new)
    hid_host = []
    for rot in range(N_ROT):
        Hs = np.zeros((s.n_target_layers, w.batch, s.block, s.d), dt_np)
        for b, L in enumerate(w.ctx_lens):
            Hs[:, b] = synth.hidden_states(w, b, L + rot * s.block, s.block)
        t = torch.from_numpy(Hs)
        hid_host.append(t.view(torch.bfloat16) if dt_np == np.uint16 else t)
    hid_dev = [h.cuda() for h in hid_host]
    n_tab = 1024
    u, r, last = synth.target_draws(w, 0, n_tab)
    u_d = torch.from_numpy(u.view(np.int32)).cuda()
    r_d = torch.from_numpy(r).cuda()
    last_d = torch.from_numpy(last).cuda()
    step_ctr = torch.zeros(1, dtype=torch.int32, device="cuda")
    acc = torch.zeros(w.batch, dtype=torch.int32, device="cuda")
    nxt = torch.from_numpy(synth.initial_tokens(w)).cuda()
    draft = torch.zeros((w.batch, s.block - 1), dtype=torch.int32, device="cuda")
    tgt = torch.zeros((w.batch, s.block), dtype=torch.int32, device="cuda")
    thr = synth.accept_threshold(w.match_p)

    def step_on(hid):
        def step():
            lib.fuse_context(hid, acc)
            lib.draft_block(nxt, draft)
            synthetic_target(draft, u_d, r_d, last_d, step_ctr, thr, w.batch, s.block, tgt)
            lib.verify_accept(draft, tgt, acc, nxt)
        return step

    # launch counting through the trace hook
    counts = {}

    @P._lib.TRACE_FN
    def count_cb(user, name, phase, stream):
        if phase == 0:
            n = name.decode()
            counts[n] = counts.get(n, 0) + 1

    L_ = P.load()
    L_.dflare_set_trace(lib.raw, count_cb, None)
    for i in range(3):
        step_on(hid_dev[i % N_ROT])()
    torch.cuda.synchronize()
    kpt = kernels_per_trace(s)
    launches_per_step = sum(kpt.get(k, 1) * v for k, v in counts.items()) / 3 + 1
    L_.dflare_set_trace(lib.raw, P._lib.TRACE_FN(), None)

    cs = torch.cuda.Stream()
    cs.wait_stream(torch.cuda.current_stream())
    graphs = []
    with torch.cuda.stream(cs):
        for h in hid_dev:
            g = torch.cuda.CUDAGraph()
            step_on(h)()
            torch.cuda.synchronize()
            with torch.cuda.graph(g, stream=cs):
                step_on(h)()
            graphs.append(g)
    torch.cuda.synchronize()
    for i in range(Wm):
        graphs[i % N_ROT].replay()
    torch.cuda.synchronize()
    if lib.device_error():
        raise RuntimeError("device error during warmup")

    # ---------------- timed region: K graph replays (one block step each)
    lens0 = lib.ctx_lens()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    for i in range(K):
        graphs[i % N_ROT].replay()
    ev1.record()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    clk = clocks.stop()
    lens1 = lib.ctx_lens()
    # each step fuses the previous step's tau: the context grows by the accepted positions
    mean_tau = (sum(lens1) - sum(lens0)) / (K * w.batch)
    drafted_per_step = w.batch * (s.block - 1)
    ms, value = replica_aggregate(ms, drafted_per_step, K, dist)
    ms_step = ms / K

    # ---------------- per-kernel durations (CUDA events around every launch, graph replays)
    hbm, peak_src, peaks = measured_peaks()
    step0 = step_on(hid_dev[0])
    ctx_now = float(np.mean(lib.ctx_lens()))   # the contexts the timed steps and breakdowns see
    per, traced_ms = graph_breakdown(lib, cs, step0, nb)
    kernels = {}
    for name, ts in per.items():
        launches = len(ts) / nb
        avg_us = 1e3 * float(np.mean(ts))
        ab = algorithmic_bytes(w, name, mean_tau, ctx_now)
        kernels[name] = {"launches_per_step": launches, "avg_us": avg_us,
                         "us_per_step": avg_us * launches,
                         "algorithmic_bytes": ab,
                         "gbs": (ab / (avg_us * 1e-6) / 1e9) if ab else None}
        if kernels[name]["gbs"]:
            kernels[name]["frac_of_hbm"] = kernels[name]["gbs"] / hbm
        if kernels[name]["us_per_step"] > 1e3 * traced_ms:
            raise RuntimeError(f"{name}: {kernels[name]['us_per_step']:.1f} us per step measured "
                               f"inside a {1e3 * traced_ms:.1f} us traced step")
    # dominant kernel: the tcgen05 projection GEMM (every gemm_* call site launches it), timed on
    # the device inside the step's own graph (no events between launches): each launch's span runs
    # from its first CTA's entry to its last CTA's exit; the step's GEMM time is the union of the
    # spans (a span can start early, next to the previous kernel's tail, under programmatic
    # dependent launch), achieved = the step's algorithmic GEMM bytes over that time
    names, runs = gemm_timeline(lib, cs, step0, nb) if s.dtype == "bf16" else ([], [])
    timed = [run for run in runs if run and all(x[2] > 0 and x[0] < 2 ** 63 for x in run)]
    attn_tl = None
    if timed:
        all_names = names
        gi = [i for i, k in enumerate(all_names) if k.startswith("gemm_")]
        names = [all_names[i] for i in gi]
        g_bytes = sum(algorithmic_bytes(w, k, mean_tau) for k in names)
        g_us = float(np.mean([union_ns([(run[i][0], run[i][2]) for i in gi]) for run in timed])) / 1e3
        g_dep_us = float(np.mean([sum(run[i][2] - min(max(run[i][1], run[i][0]), run[i][2]) for i in gi)
                                  for run in timed])) / 1e3
        span = {}
        dep = {}
        gaps = {}
        for run in timed:
            for li, (lname, st3) in enumerate(zip(all_names, run)):
                span.setdefault(lname, []).append((st3[2] - st3[0]) / 1e3)
                dep.setdefault(lname, []).append((st3[2] - max(st3[1], st3[0])) / 1e3)
                if li + 1 < len(run):   # from this launch's exit to the next timed launch's dependency
                    nx3 = run[li + 1]
                    gaps.setdefault(f"{lname} -> {all_names[li + 1]}", []).append((max(nx3[1], nx3[0]) - st3[2]) / 1e3)
        if "attention" in dep:
            ab = algorithmic_bytes(w, "attention", mean_tau, ctx_now)
            attn_tl = {"avg_after_dependency_us": float(np.mean(dep["attention"])),
                       "avg_span_us": float(np.mean(span["attention"])),
                       "algorithmic_bytes": ab,
                       "frac_of_hbm_after_dependency": ab / (float(np.mean(dep["attention"])) * 1e-6) / 1e9 / hbm,
                       "note": "attention launches timed on the device like the GEMMs (dflare_set_timing)"}
        span = {k: v for k, v in span.items() if k.startswith("gemm_")}
        per_launch = {k: {"launches_per_step": names.count(k),
                          "avg_span_us": float(np.mean(v)),
                          "avg_after_dependency_us": float(np.mean(dep[k])),
                          "frac_of_hbm": algorithmic_bytes(w, k, mean_tau) / (float(np.mean(v)) * 1e-6) / 1e9 / hbm,
                          "frac_of_hbm_after_dependency":
                              algorithmic_bytes(w, k, mean_tau) / (float(np.mean(dep[k])) * 1e-6) / 1e9 / hbm}
                      for k, v in span.items()}
        between = {k: float(np.mean(v)) for k, v in gaps.items()}
        how = ("%globaltimer stamps of every GEMM launch inside the step's CUDA graph "
               "(dflare_set_timing): first-CTA entry to last-CTA exit; us_per_step = union of "
               "the spans over a step")
    else:   # fp32 drafter (CUDA-core GEMM): CUDA events around the GEMM launches
        per_g, _ = graph_breakdown(lib, cs, step0, nb, only=lambda n: n.startswith("gemm_"))
        names = [k for k, ts in per_g.items() for _ in range(len(ts) // nb)]
        g_bytes = sum(algorithmic_bytes(w, k, mean_tau) * len(ts) / nb for k, ts in per_g.items())
        g_us = sum(1e3 * float(np.sum(ts)) / nb for ts in per_g.values())
        g_dep_us = None
        per_launch = {k: {"launches_per_step": len(ts) / nb, "avg_span_us": 1e3 * float(np.mean(ts)),
                          "frac_of_hbm": algorithmic_bytes(w, k, mean_tau) / (1e-3 * float(np.mean(ts))) / 1e9 / hbm}
                      for k, ts in per_g.items()}
        how = "CUDA events around the GEMM launches only, in a replay of the step's graph"
        between = {}
    if g_us > 1e3 * ms_step:
        raise RuntimeError(f"GEMM time {g_us:.1f} us per step exceeds the {1e3 * ms_step:.1f} us step")
    achieved = g_bytes / (g_us * 1e-6) / 1e9
    roofline = {"bound": "hbm", "kernel": "gemm_tc_kernel" if timed else "gemm_simt_kernel",
                "launches_per_step": len(names),
                "algorithmic_bytes_per_step": g_bytes, "us_per_step": g_us,
                "us_per_step_after_dependency": g_dep_us,
                "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "frac_after_dependency": (g_bytes / (g_dep_us * 1e-6) / 1e9 / hbm) if g_dep_us else None,
                "between_gemms_us": between,
                "traffic": gemm_traffic(w), "peak_source": peak_src, "per_launch": per_launch,
                "note": "achieved = algorithmic GEMM bytes of a step / GEMM time of a step, timed "
                        f"by {how}; a span can include a wait for the previous kernel when the "
                        "launch starts early under programmatic dependent launch, so frac is a lower "
                        "bound; frac_after_dependency divides by the time from each launch's first "
                        "met dependency to its exit (weights prefetched before that are not "
                        "counted in the time); between_gemms_us: from a GEMM's exit to the next "
                        "GEMM's dependency (the kernels between them and the launch latencies); "
                        "traffic = ncu DRAM bytes per step from profiles/, null if the GEMM sources "
                        "changed since"}
    # the whole block step against HBM: every kernel's algorithmic bytes over the graph-timed
    # step (no events between launches)
    s_bytes = sum(k["algorithmic_bytes"] * k["launches_per_step"] for k in kernels.values())
    s_gbs = s_bytes / (ms_step * 1e-3) / 1e9
    step_roofline = {"bytes_per_step": s_bytes, "ms_per_step": ms_step, "achieved": s_gbs,
                     "peak": hbm, "unit": "GB/s", "frac": s_gbs / hbm,
                     "lower_bound_ms": s_bytes / (hbm * 1e9) * 1e3,
                     "note": "algorithmic bytes of every kernel of a step (weights, context K/V, "
                             "target states, logits) / the CUDA-graph step time"}

    # ---------------- end to end through the public calls with host buffers
    pin_h = [h.pin_memory() for h in hid_host]
    pin_u = torch.from_numpy(u.view(np.int32)).pin_memory()
    pin_r = torch.from_numpy(r).pin_memory()
    pin_last = torch.from_numpy(last).pin_memory()
    # accept lengths, next tokens and drafts of a step live in one device buffer, read back by
    # one copy per step; two such buffers alternate (step i reads the loop state from the
    # buffer step i - 1 wrote), so a step's read-back on the copy stream overlaps the next step
    nio = w.batch * (s.block + 1)
    io_b = [torch.zeros(nio, dtype=torch.int32, device="cuda") for _ in range(2)]

    def io_parts(io):
        return io[:w.batch], io[w.batch:2 * w.batch], io[2 * w.batch:].view(w.batch, s.block - 1)
    io_parts(io_b[1])[0].copy_(acc)
    io_parts(io_b[1])[1].copy_(nxt)
    out_io = torch.zeros((E, nio), dtype=torch.int32).pin_memory()
    # step inputs double-buffered: while step i computes on the current stream, a copy stream
    # brings step i + 1's target states (from the next of the N_ROT pinned host buffers) and
    # target draws into the other device buffer (events order each buffer's copy after the step
    # that last read it)
    hid_b = [hid_dev[0], hid_dev[1]]
    u_b = [torch.zeros((1,) + u.shape[1:], dtype=torch.int32, device="cuda") for _ in range(2)]
    r_b = [torch.zeros((1,) + r.shape[1:], dtype=torch.int32, device="cuda") for _ in range(2)]
    l_b = [torch.zeros((1,) + last.shape[1:], dtype=torch.int32, device="cuda") for _ in range(2)]
    # each step's draws are a one-row table, so the synthetic target's row counter stays at 0
    zero_ctr = torch.zeros(1, dtype=torch.int32, device="cuda")
    h2d = pin_h[0].numel() * pin_h[0].element_size() + \
        (u_b[0].numel() + r_b[0].numel() + l_b[0].numel()) * 4
    d2h = nio * 4
    cps = torch.cuda.Stream()
    main = torch.cuda.current_stream()
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    used = [torch.cuda.Event(), torch.cuda.Event()]
    done = [torch.cuda.Event(), torch.cuda.Event()]
    read = [torch.cuda.Event(), torch.cuda.Event()]

    def load(i, k):
        with torch.cuda.stream(cps):
            cps.wait_event(used[k])
            j = i % n_tab
            hid_b[k].copy_(pin_h[i % N_ROT], non_blocking=True)
            u_b[k].copy_(pin_u[j:j + 1], non_blocking=True)
            r_b[k].copy_(pin_r[j:j + 1], non_blocking=True)
            l_b[k].copy_(pin_last[j:j + 1], non_blocking=True)
            copied[k].record(cps)

    for k in range(2):
        used[k].record(main)
        read[k].record(main)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wall0 = time.perf_counter()
    e0.record()
    load(0, 0)
    for i in range(E):
        k = i & 1
        if i + 1 < E:
            load(i + 1, k ^ 1)
        main.wait_event(copied[k])
        main.wait_event(read[k])          # io_b[k] was read back (two steps ago)
        acc_p, nxt_p, _ = io_parts(io_b[k ^ 1])
        acc_e, nxt_e, draft_e = io_parts(io_b[k])
        lib.fuse_context(hid_b[k], acc_p)
        lib.draft_block(nxt_p, draft_e)
        synthetic_target(draft_e, u_b[k], r_b[k], l_b[k], zero_ctr, thr, w.batch, s.block, tgt)
        used[k].record(main)
        lib.verify_accept(draft_e, tgt, acc_e, nxt_e)
        done[k].record(main)
        with torch.cuda.stream(cps):      # the step's results to pinned host memory
            cps.wait_event(done[k])
            out_io[i].copy_(io_b[k], non_blocking=True)
            read[k].record(cps)
    main.wait_event(read[(E - 1) & 1])    # the last read-back is inside the timed region
    e1.record()
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    e2e_ms = e0.elapsed_time(e1)
    e2e_value = world * drafted_per_step * E / (max(e2e_ms / 1e3, wall))
    if lib.device_error():
        raise RuntimeError("device error during the benchmark")
    tau_h = out_io[:, :w.batch]
    if not bool(((tau_h >= 1) & (tau_h <= s.block)).all()):
        raise RuntimeError("end-to-end read-back holds accept lengths outside [1, B]")

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": Wm, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": s.dtype, "data": "synthetic",
        "config": {**config_of(w),
                   "l2": "not flushed: each step streams the whole draft weight set "
                         f"({sum(v.nbytes for v in W.values()) / 1e9:.2f} GB) > 129 MB L2",
                   "timing": f"CUDA-graph replays of one block step each ({N_ROT} graphs over "
                             f"{N_ROT} target-state buffers, in turn), K replays between events"},
        "block_steps_per_s": K / (ms / 1e3),
        "mean_accept_len": mean_tau,
        "accepted_tokens_per_s": world * w.batch * mean_tau * K / (ms / 1e3),
        "roofline": roofline,
        "attention_timing": attn_tl,
        "step_roofline": step_roofline,
        "kernels": kernels,
        "kernels_note": "CUDA events around every launch of a step, in a separate replay of the "
                        "step's graph with those events (each duration includes its launch's own "
                        "latency, which the untraced graph overlaps); traced_ms_per_step is that "
                        "replay's step time",
        "traced_ms_per_step": traced_ms,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h), "ms_per_step": 1e3 * max(e2e_ms / 1e3, wall) / E,
                "steps": E, "host_ms_per_step": 1e3 * wall / E, "device_ms_per_step": e2e_ms / E,
                "timing": "eager public calls; every step's inputs copied from pinned host "
                          "memory inside the region on a second stream one step ahead, and its "
                          "outputs copied back to pinned host memory on that stream (both "
                          "double-buffered); the region ends after the last read-back"},
        "fill": {"positions": n_fill, "calls": len(range(0, max(w.ctx_lens), chunk)),
                 "fuse_layers_us": fill_us.get("fuse_layers"),
                 "fuse_layers_gbs": fuse_bytes / (fill_us["fuse_layers"] * 1e-6) / 1e9
                 if fill_us.get("fuse_layers") else None,
                 "fuse_layers_frac_of_hbm": fuse_bytes / (fill_us["fuse_layers"] * 1e-6) / 1e9 / hbm
                 if fill_us.get("fuse_layers") else None,
                 "kv_ctx_us": fill_us.get("gemm_kv_ctx"),
                 "kv_ctx_tflops": kv_flops / (fill_us["gemm_kv_ctx"] * 1e-6) / 1e12
                 if fill_us.get("gemm_kv_ctx") else None,
                 "note": "context fill of every sequence from empty, CUDA events around each launch "
                         "(fusion: (T + D) d bytes per position; K/V projection: 2 n D 2 d_kv d flop)"},
        "gpu_launches": int(round(launches_per_step * K)),
        "launches_per_step": launches_per_step,
        "clocks": clk,
    }
    if s.dtype == "bf16" and fill_us.get("gemm_kv_ctx"):
        bf = peaks.get("bf16_tflops")
        line["fill"]["kv_ctx_frac_of_bf16_peak"] = (line["fill"]["kv_ctx_tflops"] / bf) if bf else None
    if extras:
        line["fusion_variants"] = fusion_variants(w, dev_w, fill_chunks, hid_dev[0],
                                                  max(1, int(round(mean_tau))))
        line["sampled"] = sampled_steps(w, dev_w, fill_chunks, hid_dev[0],
                                        torch.from_numpy(synth.initial_tokens(w)).cuda())
    del fill_chunks, graphs
    lib.close()
    del dev_w, hid_dev
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and cpu_seconds > 0:
        v, dt, tau, n_cpu = oracle_steps(w, W, 10 ** 6, budget_s=cpu_seconds)
        line["cpu_baseline"] = {
            "value": v, "unit": UNIT, "cores": host_cores(), "kind": "oracle",
            "sample": f"{n_cpu} full block steps of {w.name} (fp64, bf16 storage "
                      f"rounding) after an untimed oracle fill of {list(w.ctx_lens)} positions",
            "seconds": dt}
    return line


SUB_KEYS = ("value", "unit", "ms_per_step", "block_steps_per_s", "mean_accept_len",
            "accepted_tokens_per_s", "config", "roofline", "attention_timing", "step_roofline", "e2e", "fill",
            "cpu_baseline", "clocks", "launches_per_step", "kernels")


def run_ours(args):
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    cpu_s = 0.0 if args.no_cpu_baseline else args.cpu_seconds
    w = synth.preset(args.workload)
    if args.draft_layers or args.vocab or args.batch or args.ctx:
        import dataclasses
        shp = dataclasses.replace(w.shape, n_draft_layers=args.draft_layers or w.shape.n_draft_layers,
                                  vocab=args.vocab or w.shape.vocab)
        lens = (max(w.ctx_lens),) * args.batch if args.batch else w.ctx_lens
        if args.ctx:
            lens = (args.ctx,) * len(lens)
        w = w.with_(shape=shp, ctx_lens=lens,
                    name=f"{w.name}_D{shp.n_draft_layers}_V{shp.vocab}_b{len(lens)}_L{max(lens)}")
        args.headline_only = True
    line = measure(w, args, args.steps, args.warmup, args.e2e_steps,
                   args.breakdown_steps, cpu_s, not args.no_variants, dist, world, rank, local)
    # the other drafter shapes, each measured the same way (one GPU only: under torchrun every
    # rank runs the headline workload as an independent replica)
    if world == 1 and not args.headline_only:
        line["configs"] = {}
        for name in CONFIG_SET:
            if name == args.workload:
                continue
            sub = measure(synth.preset(name), args, args.steps, args.warmup, args.e2e_steps,
                          args.breakdown_steps, 0.0 if args.no_cpu_baseline else args.sub_cpu_seconds,
                          False, local=local)
            line["configs"][name] = {k: sub[k] for k in SUB_KEYS if k in sub}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


# one-at-a-time around the centre, then two corners: b16 x B32 x L32768 x D16 (tensor- and
# KV-heavy) and b16 x B16 (the M = 256 GEMM corner)
SWEEP_CENTRE = dict(D=8, T=36, B=16, L=4096, batch=1, p=0.85)
SWEEP_AXES = (("D", (2, 5, 8, 12, 16)), ("T", (4, 12, 36)), ("B", (8, 16, 32)),
              ("L", (512, 2048, 8192, 32768)), ("batch", (1, 4, 16)), ("p", (0.6, 0.9)))
SWEEP_CORNERS = (dict(batch=16, B=32, L=32768, D=16), dict(batch=16, B=16))


def sweep_points():
    pts = [dict(SWEEP_CENTRE)]
    for k, vals in SWEEP_AXES:
        pts += [{**SWEEP_CENTRE, k: v} for v in vals if v != SWEEP_CENTRE[k]]
    return pts + [{**SWEEP_CENTRE, **c} for c in SWEEP_CORNERS]


def run_sweep(args):
    """Block steps per second over the sweep points (throughput only). Weights and target states
    come from torch's device generator (N(0, 0.02^2) matrices, 1 + N(0, 0.02^2) gains, N(0, 1)
    states): the content does not change the work, and the host generator would spend minutes
    on the largest contexts. Each point fills its contexts in 2048-position chunks, then times a
    CUDA graph of one block step (fuse tau positions, draft, synthetic target, verify)."""
    import dataclasses
    import torch
    from paper_2606_02091_gb300 import DFlare, synthetic_target
    torch.cuda.set_device(0)
    K, Wm = args.steps, max(args.warmup, 3)
    dmax = max(v for k, vals in SWEEP_AXES if k == "D" for v in vals)
    top = dataclasses.replace(synth.sweep_point().shape, n_draft_layers=dmax)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(0)

    def rnd(*shape, mean=0.0, std=0.02):
        t = torch.randn(shape, generator=gen, device="cuda", dtype=torch.float32)
        return (t * std + mean).to(torch.bfloat16)
    Dm, d, F, V = top.n_draft_layers, top.d, top.ffn, top.vocab
    W = {"fuse_norm": rnd(Dm, d, mean=1.0), "w_kv_ctx": rnd(Dm, 2 * top.d_kv, d),
         "attn_norm": rnd(Dm, d, mean=1.0), "w_qkv": rnd(Dm, top.d_q + 2 * top.d_kv, d),
         "w_o": rnd(Dm, d, top.d_q), "mlp_norm": rnd(Dm, d, mean=1.0), "w_gate": rnd(Dm, F, d),
         "w_up": rnd(Dm, F, d), "w_down": rnd(Dm, d, F), "final_norm": rnd(d, mean=1.0),
         "embed": rnd(V, d), "lm_head": rnd(V, d)}
    stacked = ("fuse_norm", "w_kv_ctx", "attn_norm", "w_qkv", "w_o", "mlp_norm", "w_gate", "w_up", "w_down")
    pts = sweep_points()
    if args.sweep_points:
        pts = [pts[int(i)] for i in args.sweep_points.split(",")]
    for pt in pts:
        w = synth.sweep_point(D=pt["D"], T=pt["T"], B=pt["B"], L=pt["L"], batch=pt["batch"], p=pt["p"])
        s = w.shape
        bsz, L, B, T = w.batch, pt["L"], s.block, s.n_target_layers
        chunk = min(2048, L)
        lib = DFlare.from_shape(s, max_batch=bsz, max_ctx=L + B * (K + Wm + 16),
                                max_fuse_rows=bsz * max(chunk, B))
        weights = {k: (v[:s.n_draft_layers] if k in stacked else v) for k, v in W.items()}
        weights["fuse_logits"] = torch.randn((s.n_draft_layers, T), generator=gen, device="cuda")
        lib.set_weights(weights)
        lib.reset(bsz)
        t_fill = time.perf_counter()
        for pos0 in range(0, L, chunk):
            H = torch.randn((T, bsz, chunk, d), generator=gen, device="cuda", dtype=torch.bfloat16)
            n = torch.full((bsz,), min(chunk, L - pos0), dtype=torch.int32, device="cuda")
            lib.fuse_context(H, n)
            del H
        torch.cuda.synchronize()
        t_fill = time.perf_counter() - t_fill
        hid = torch.randn((T, bsz, B, d), generator=gen, device="cuda", dtype=torch.bfloat16)
        u, r, last = synth.target_draws(w, 0, 1024)
        u_d, r_d, last_d = (torch.from_numpy(x).cuda() for x in (u.view(np.int32), r, last))
        step_ctr = torch.zeros(1, dtype=torch.int32, device="cuda")
        acc = torch.zeros(bsz, dtype=torch.int32, device="cuda")
        nxt = torch.from_numpy(synth.initial_tokens(w)).cuda()
        draft = torch.zeros((bsz, B - 1), dtype=torch.int32, device="cuda")
        tgt = torch.zeros((bsz, B), dtype=torch.int32, device="cuda")
        thr = synth.accept_threshold(w.match_p)

        def step():
            lib.fuse_context(hid, acc)
            lib.draft_block(nxt, draft)
            synthetic_target(draft, u_d, r_d, last_d, step_ctr, thr, bsz, B, tgt)
            lib.verify_accept(draft, tgt, acc, nxt)

        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cs):
            step()
            torch.cuda.synchronize()
            with torch.cuda.graph(graph, stream=cs):
                step()
        torch.cuda.synchronize()
        for _ in range(Wm):
            graph.replay()
        torch.cuda.synchronize()
        lens0 = lib.ctx_lens()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(K):
            graph.replay()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / K
        tau = (sum(lib.ctx_lens()) - sum(lens0)) / (K * bsz)
        if lib.device_error():
            raise RuntimeError(f"device error at sweep point {pt}")
        kern = {}
        if args.breakdown_steps > 0:
            per, _ = graph_breakdown(lib, cs, step, args.breakdown_steps)
            kern = {n: round(1e3 * float(np.sum(ts)) / args.breakdown_steps, 1) for n, ts in per.items()}
        e = 2
        wbytes = e * (s.n_draft_layers * (d * (s.d_q + 2 * s.d_kv) + s.d_q * d + 3 * d * s.ffn + 2 * s.d_kv * d)
                      + V * d)
        print(json.dumps({"sweep": pt, "ms_per_step": ms, "drafted_tokens_per_s": bsz * (B - 1) / (ms / 1e3),
                          "mean_accept_len": tau, "accepted_tokens_per_s": bsz * tau / (ms / 1e3),
                          "weight_gbs": wbytes / (ms / 1e3) / 1e9, "fill_s": t_fill,
                          "us_per_step_events": kern}), flush=True)
        del graph
        lib.close()
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
