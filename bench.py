"""Benchmark of the draft-then-verify step on the 7B-shape workload.

Workload: 7B-shape Llama target (32 layers, d 4096, 32 MHA heads, FFN 11008,
vocab 32000) with a 160M draft (12 layers, d 768, 12 heads), bf16 weights
N(0, 0.02) from seeds, a prefix of 2048 uniform-random ids, batch 1, K = 4 draft
tokens per step, T = 1.0 with Philox uniforms.  A step is one whole pass of the
hot path: K draft forward passes + samples, one verify pass over K+1 positions,
acceptance / resample / commit.

Metric: accepted (committed) tokens per second over the timed steps.  The verify
pass is also timed on its own (CUDA events around each verify launch inside the
timed region) and reported as achieved HBM bandwidth against the measured copy
peak (roofline).  e2e: the same metric through the public API for a whole
request: prompt copied from pinned host memory, prefill, then decoding with every
step's result copied to pinned host memory and read by the host.

--impl reference times the oracle (plain fp64 CPU implementation) on the same
workload, on a bounded sample: per-layer timings of the target and draft
forward passes at context 2048 plus one acceptance, scaled to full depth.

Multi-GPU (torchrun): replicas only, one independent request per rank; the
value is the sum of all ranks' tokens over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

TARGET, DRAFT = "target_7b", "draft_160m"
PREFIX, K_DRAFT, TEMP = 2048, 4, 1.0
WORKLOAD = "7B-shape target + 160M draft, prefix 2048, K=4, T=1.0, batch 1"
METRIC = "accepted tokens/s (batch 1, 7B-shape, K=4); verify-step HBM GB/s vs peak"


def workload_config(k: int, world: int) -> dict:
    """The workload keys both arms report in `config`."""
    return {"workload": WORKLOAD, "target": TARGET, "draft": DRAFT, "prefix": PREFIX,
            "K": k, "temperature": TEMP, "global_batch": world,
            "parallelism": f"replicas x{world}"}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d.get("hbm_gbs", 6800.0)), "measured"
    return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def verify_bytes(t, ctx: int, K: int) -> int:
    """Algorithmic HBM bytes of one verify pass: every target weight once
    (embedding rows excluded), KV read for positions < ctx, KV written for K+1
    rows, fp32 logits written."""
    d, q, kv, f, v, L = t.d_model, t.q_dim, t.kv_dim, t.d_ffn, t.vocab, t.n_layers
    weights = L * ((q + 2 * kv) * d + d * q + 3 * f * d) * 2 + v * d * 2 + (2 * L + 1) * d * 2
    kv_read = L * 2 * ctx * kv * 2
    kv_write = L * 2 * (K + 1) * kv * 2
    logits = (K + 1) * v * 4
    return weights + kv_read + kv_write + logits


def combine_rank_stats(stats, world: int, device):
    """One rank's [ms, tokens, e2e_s, generated, verify_ms] -> the job's: the
    times (ms, e2e_s, verify_ms) are the maximum over ranks, the counts (tokens,
    generated) the sum.  torch.distributed is initialised when world > 1; the
    collective runs on `device` ("cuda" for NCCL, "cpu" for gloo)."""
    import torch
    import torch.distributed as dist

    if world <= 1:
        return stats.clone()
    mx = stats.clone().to(device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = stats.clone().to(device)
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    out = mx.cpu().clone()
    out[1], out[3] = sm[1].cpu(), sm[3].cpu()
    return out


def run_gpu(args, rank: int, world: int):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2608_10362_gb300 import Engine
    from seeded_inputs import SHAPES, gen_prompt, iter_weights

    dev = int(os.environ.get("LOCAL_RANK", 0))
    torch.cuda.set_device(dev)
    t, dft = SHAPES[TARGET], SHAPES[DRAFT]
    K = args.k
    steps, warm = args.steps, args.warmup
    max_seq = PREFIX + (steps + warm + 8) * (K + 1) + 16
    t0 = time.time()
    eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=K, max_drafts=1,
                 draft_shape_max=dft, draft_budget_bytes=1 << 30, use_graphs=True,
                 launch_mode=args.launch_mode,
                 trace=args.trace_pass if args.trace is not None else None, device=dev,
                 draft_kernel=args.draft_kernel)
    eng.register_draft(0, dft, iter_weights(dft, 1))
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    setup_s = time.time() - t0
    prompt = gen_prompt(100 + rank, PREFIX, t.vocab)
    eng.prefill(0, prompt, seed=1 + rank)
    s = eng.stream
    for _ in range(warm):
        eng.step(K, TEMP)
    eng.sync()
    L0 = int(eng.seq_state()[0, 0])
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    ev_d = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev) as clk:
        torch.cuda.nvtx.range_push("timed")   # for profilers: --nvtx --nvtx-include "timed/"
        start.record(s)
        for i in range(steps):
            ev_d[i].record(s)
            eng.draft_step(K, TEMP)
            ev[i][0].record(s)
            eng.verify_step(K)
            ev[i][1].record(s)
            eng.accept_commit(K, TEMP)
        stop.record(s)
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    bits = eng.sync()
    if args.trace is not None and rank == 0:
        np.save(args.trace, eng.pass_trace())
    ms = start.elapsed_time(stop)
    verify_ms = [a.elapsed_time(b) for a, b in ev]
    draft_ms = sum(d.elapsed_time(v[0]) for d, v in zip(ev_d, ev)) / steps
    launches = eng.launches_per_step()
    draft_fused = bool(eng.info(__import__("paper_2608_10362_gb300")._lib.INFO_DRAFT_FUSED))
    L1 = int(eng.seq_state()[0, 0])
    tokens = L1 - L0
    ctx_mean = L0 + (L1 - L0) / 2
    vb = verify_bytes(t, int(ctx_mean), K)
    v_avg = sum(verify_ms) / len(verify_ms)

    # ---- end to end through the public API: pinned prompt -> prefill -> decode
    # with a device->host read of every step's result
    e2e_steps = steps
    prompt_pinned = torch.from_numpy(gen_prompt(200 + rank, PREFIX, t.vocab)).pin_memory()
    res = eng.results_host
    torch.cuda.synchronize()
    e0 = time.perf_counter()
    eng.prefill(0, prompt_pinned.numpy(), seed=7 + rank)
    generated = 0
    for _ in range(e2e_steps):
        eng.step(K, TEMP, res)
        s.synchronize()
        generated += int(res[0]) + 1
    e2e_s = time.perf_counter() - e0
    eng.sync()
    h2d = PREFIX * 4
    d2h = (K + 2) * 4

    stats = torch.tensor([ms, float(tokens), e2e_s, float(generated), v_avg], dtype=torch.float64)
    if world > 1:
        job = combine_rank_stats(stats, world, "cuda")
        ms, tokens, e2e_s, generated, v_avg = (float(x) for x in job)
    eng.close()
    return dict(ms=ms, tokens=tokens, verify_ms=v_avg, verify_bytes=vb, clocks=clk.summary(),
                e2e_s=e2e_s, generated=generated, h2d=h2d / e2e_steps, d2h=d2h,
                setup_s=setup_s, bits=bits, steps=steps, tokens_per_step=tokens / steps / world,
                launches=launches * steps, launches_per_step=launches, draft_ms=draft_ms,
                draft_fused=draft_fused)


def oracle_step_timer(K: int):
    """The reference arm's step: the oracle's time for one draft-then-verify
    iteration, estimated from five parts - a target layer (alternating between
    two; 5 rows at context 2048), the target LM head, a draft layer (1 row), the
    draft LM head, one acceptance - each weighted by how often an iteration runs
    it.  Every part is timed once at setup; each call re-times one part (in turn),
    so a step is a bounded sample.  The sampled layers are built once."""
    import numpy as np

    from oracle.llama import LlamaOracle
    from oracle.speculative import accept
    from seeded_inputs import SHAPES, gen_kv, gen_logits, gen_tensor

    t, dft = SHAPES[TARGET], SHAPES[DRAFT]

    def build(shape, seed, rows):
        w = {}
        for li in (0, 1):
            for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
                w[(n, li)] = gen_tensor(shape, seed, n, li)
        w[("final_norm", -1)] = gen_tensor(shape, seed, "final_norm")
        w[("lm_head", -1)] = gen_tensor(shape, seed, "lm_head")
        model = LlamaOracle(shape, w)
        cache = model.new_cache(PREFIX + rows)
        kvs = gen_kv(3, (2, PREFIX, shape.n_kv_heads, shape.head_dim), 1.0)
        cache.k[:2, :PREFIX] = kvs
        cache.v[:2, :PREFIX] = kvs[::-1]
        h = np.random.default_rng(0).standard_normal((rows, shape.d_model))
        return model, cache, h, np.arange(PREFIX, PREFIX + rows)

    tgt = build(t, 0, K + 1)
    drf = build(dft, 1, 1)
    zt = gen_logits(5, K + 1, t.vocab).astype(np.float64)
    zd = gen_logits(6, K, t.vocab).astype(np.float64)
    n = [0]

    def t_layer():
        tgt[0].layer(n[0] & 1, tgt[2], tgt[1], tgt[3])

    def d_layer():
        drf[0].layer(n[0] & 1, drf[2], drf[1], drf[3])

    parts = [t_layer, lambda: tgt[0].logits(tgt[2]), d_layer, lambda: drf[0].logits(drf[2]),
             lambda: accept(zt, zd, [1] * K, TEMP, [0.5] * K, 0.5)]
    weight = [t.n_layers, 1, K * dft.n_layers, K, 1]   # times per iteration
    last = [0.0] * len(parts)

    def run_part(i):
        a = time.perf_counter()
        parts[i]()
        last[i] = time.perf_counter() - a

    for i in range(len(parts)):   # every part timed once before the first step
        run_part(i)

    def one() -> float:
        # a step times one part afresh (in turn) and returns the iteration estimate
        run_part(n[0] % len(parts))
        n[0] += 1
        return sum(w * x for w, x in zip(weight, last))

    desc = (f"fp64 numpy oracle: iteration = {t.n_layers} x one target layer (5 rows, context "
            f"{PREFIX}) + LM head + {K} x ({dft.n_layers} x one draft layer (1 row) + LM head) + "
            f"one acceptance (V={t.vocab}); each step re-times one of these five parts in turn")
    return one, desc


def oracle_sample(tokens_per_iter: float, K: int, reps: int = 1):
    """Time the oracle on a bounded sample of the workload and scale to one
    iteration: 2 target layers + LM head at context 2048 (5 rows), 2 draft
    layers + LM head (1 row), one acceptance; full depth = per-layer time x
    layer count."""
    import numpy as np

    from oracle.llama import LlamaOracle
    from oracle.speculative import accept
    from seeded_inputs import SHAPES, gen_kv, gen_logits, gen_tensor

    t, dft = SHAPES[TARGET], SHAPES[DRAFT]

    def model_with_layers(shape, seed, layers):
        w = {}
        for li in layers:
            for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
                w[(n, li)] = gen_tensor(shape, seed, n, li)
        w[("final_norm", -1)] = gen_tensor(shape, seed, "final_norm")
        w[("lm_head", -1)] = gen_tensor(shape, seed, "lm_head")
        return LlamaOracle(shape, w)

    def time_layers(model, shape, rows, ctx):
        cache = model.new_cache(ctx + rows)
        kvs = gen_kv(3, (2, ctx, shape.n_kv_heads, shape.head_dim), 1.0)
        cache.k[:2, :ctx] = kvs
        cache.v[:2, :ctx] = kvs[::-1]
        h = np.random.default_rng(0).standard_normal((rows, shape.d_model))
        pos = np.arange(ctx, ctx + rows)
        best_layer, best_lm = 1e9, 1e9
        for _ in range(reps):
            a = time.perf_counter()
            for li in (0, 1):
                model.layer(li, h, cache, pos)
            best_layer = min(best_layer, (time.perf_counter() - a) / 2)
            a = time.perf_counter()
            model.logits(h)
            best_lm = min(best_lm, time.perf_counter() - a)
        return best_layer, best_lm

    a0 = time.perf_counter()
    tm = model_with_layers(t, 0, (0, 1))
    dm = model_with_layers(dft, 1, (0, 1))
    tl, tlm = time_layers(tm, t, K + 1, PREFIX)
    dl, dlm = time_layers(dm, dft, 1, PREFIX)
    zt = gen_logits(5, K + 1, t.vocab).astype(np.float64)
    zd = gen_logits(6, K, t.vocab).astype(np.float64)
    a = time.perf_counter()
    accept(zt, zd, [1] * K, TEMP, [0.5] * K, 0.5)
    tacc = time.perf_counter() - a
    iter_s = t.n_layers * tl + tlm + K * (dft.n_layers * dl + dlm) + tacc
    wall = time.perf_counter() - a0
    return {
        "value": tokens_per_iter / iter_s,
        "iter_s": iter_s,
        "cores": os.cpu_count(),
        "sample": (f"fp64 numpy oracle: 2 of {t.n_layers} target layers (5 rows, context {PREFIX}) "
                   f"+ LM head, 2 of {dft.n_layers} draft layers (1 row) + LM head, one acceptance "
                   f"(V={t.vocab}); per-layer time x depth = {iter_s:.2f} s per iteration; "
                   f"{tokens_per_iter:.3f} tokens/iteration; sample wall {wall:.1f} s"),
    }


def verify_bytes_batch(t, ctxs, K: int) -> int:
    """verify_bytes for a batch: weights once, each request's KV at its context."""
    L, kv = t.n_layers, t.kv_dim
    weights = verify_bytes(t, 0, 0) - L * 2 * 1 * kv * 2 - t.vocab * 4
    B = len(ctxs)
    return (weights + sum(L * 2 * int(c) * kv * 2 for c in ctxs) + B * L * 2 * (K + 1) * kv * 2
            + B * (K + 1) * t.vocab * 4)


def run_pair_case(args, tname: str, dname: str, prefixes, K: int, T: float, seed: int = 0):
    """Steady-state decoding of len(prefixes) requests with a target/draft pair:
    aggregate committed tokens/s, and the verify pass against the HBM roofline."""
    import numpy as np
    import torch

    from paper_2608_10362_gb300 import Engine, weights_bytes
    from seeded_inputs import SHAPES, gen_prompt, iter_weights
    t, d = SHAPES[tname], SHAPES[dname]
    B = len(prefixes)
    steps, warm = args.steps, args.warmup
    max_seq = int(max(prefixes)) + (steps + warm + 4) * (K + 1) + 16
    eng = Engine(t, iter_weights(t, seed), max_batch=B, max_seq=max_seq, max_k=K, max_drafts=1,
                 draft_shape_max=d, draft_budget_bytes=weights_bytes(d) + (1 << 20), use_graphs=True)
    eng.register_draft(0, d, iter_weights(d, seed + 1))
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    for b, n in enumerate(prefixes):
        eng.prefill(b, gen_prompt(100 + b, int(n), t.vocab), seed=1 + b)
    eng.set_batch(B)
    for _ in range(warm):
        eng.step(K, T)
    eng.sync()
    L0 = eng.seq_state()[:B, 0].astype(np.int64)
    s = eng.stream
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    for i in range(steps):
        eng.draft_step(K, T)
        ev[i][0].record(s)
        eng.verify_step(K)
        ev[i][1].record(s)
        eng.accept_commit(K, T)
    b_.record(s)
    torch.cuda.synchronize()
    bits = eng.sync()
    L1 = eng.seq_state()[:B, 0].astype(np.int64)
    ms = a.elapsed_time(b_)
    v_ms = sum(x.elapsed_time(y) for x, y in ev) / steps
    vb = verify_bytes_batch(t, (L0 + L1) // 2, K)
    eng.close()
    peak, peak_kind = measured_peaks()
    gbs = vb / (v_ms * 1e-3) / 1e9
    return {"target": tname, "draft": dname, "batch": B, "K": K, "T": T,
            "tokens_per_s": float((L1 - L0).sum()) / (ms * 1e-3), "ms_per_step": ms / steps,
            "tokens_per_step": float((L1 - L0).sum()) / steps, "verify_ms": v_ms,
            "verify_GBps": gbs, "verify_frac": gbs / peak, "peak": peak, "peak_kind": peak_kind,
            "algorithmic_bytes": vb, "device_status": bits}


def run_switching_case(args):
    """Draft switching under a 2 GiB draft budget: the 7B target with a pool of
    drafts (68M, 160M, tied 1.1B) in pinned host memory; every 64 committed tokens
    the active draft changes by a seeded schedule, and the next scheduled draft is
    loaded asynchronously (side stream) while the current one decodes."""
    import numpy as np
    import torch

    from paper_2608_10362_gb300 import Engine, weights_bytes
    from seeded_inputs import SHAPES, gen_prompt, iter_weights
    t = SHAPES[TARGET]
    pool = {0: SHAPES["draft_68m"], 1: SHAPES["draft_160m"], 2: SHAPES["draft_1b1_tied"]}
    K, T, prefix, budget = 4, 1.0, 1024, 2 << 30
    rng = np.random.default_rng(3)
    n_switch = max(2, args.steps)
    sched = [int(x) for x in rng.integers(0, 3, n_switch + 1)]
    sched[0] = 0   # start on the smallest draft (the tied 1.1B, 2.07 GB, fits only alone)
    for i in range(1, len(sched)):
        if sched[i] == sched[i - 1]:
            sched[i] = (sched[i] + 1) % 3
    max_seq = prefix + (n_switch + 2) * 64 * 2 + 256
    eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=K, max_drafts=3,
                 draft_shape_max=pool[2], draft_budget_bytes=budget, use_graphs=True)
    for i, sh in pool.items():
        eng.register_draft(i, sh, iter_weights(sh, 10 + i))
    eng.prefill(0, gen_prompt(5, prefix, t.vocab), seed=2)
    resident = []

    def ensure_loaded(i):
        """Make draft i resident (evicting non-active drafts first); False when it
        cannot fit beside the active draft (the active draft is never evicted)."""
        if i in resident:
            return True
        need = weights_bytes(pool[i])
        others = [j for j in resident if j != active[0]]
        if need + sum(weights_bytes(pool[j]) for j in resident if j == active[0]) > budget:
            return False
        while sum(weights_bytes(pool[j]) for j in resident) + need > budget:
            victim = others.pop(0)
            eng.evict_draft(victim)
            resident.remove(victim)
        eng.load_draft_async(i)
        resident.append(i)
        return True

    active = [sched[0]]
    ensure_loaded(sched[0])
    eng.set_active_draft(sched[0])
    eng.sync()
    s = eng.stream
    load_ms, tokens, step_ms, fallbacks = [], 0, [], 0
    L = int(eng.seq_state()[0, 0])
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    for k in range(n_switch):
        if k + 1 < len(sched):
            ensure_loaded(sched[k + 1])          # prefetch the next draft (side stream)
        start = L
        while L - start < 64:
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s)
            eng.step(K, T)
            b.record(s)
            b.synchronize()
            step_ms.append(a.elapsed_time(b))
            L = int(eng.seq_state()[0, 0])
        tokens += L - start
        if k + 1 < len(sched):
            if not ensure_loaded(sched[k + 1]):
                fallbacks += 1                       # stays on the resident draft
                continue
            t0 = time.perf_counter()
            active[0] = sched[k + 1]
            eng.set_active_draft(sched[k + 1])   # waits on the GPU for the copy, catches up
            eng.sync()
            load_ms.append((time.perf_counter() - t0) * 1e3)
    wall = time.perf_counter() - wall0
    bits = eng.sync()
    eng.close()
    return {"case": "switching", "target": TARGET, "pool": ["68M", "160M", "1.1B tied"],
            "budget_GiB": 2, "switch_every_tokens": 64, "switches": n_switch,
            "schedule": sched[:n_switch + 1], "tokens_per_s": tokens / wall,
            "step_ms_median": float(np.median(step_ms)),
            "switch_ms_median": float(np.median(load_ms)) if load_ms else None,
            "fallbacks": fallbacks, "device_status": bits}


def run_case(args):
    """Diagnostic cases (not the headline metric)."""
    import numpy as np
    import torch

    from seeded_inputs import SHAPES, bf16_round, gen_prompt, iter_weights
    if args.case == "gemm":
        from paper_2608_10362_gb300 import op_linear
        rng = np.random.default_rng(0)
        x = torch.from_numpy(bf16_round(rng.standard_normal((args.rows, args.kdim), dtype=np.float32)))
        w = torch.randn(args.n, args.kdim, device="cuda", dtype=torch.bfloat16) * 0.02
        xt = x.to(torch.bfloat16).cuda()
        scratch = torch.zeros(64 << 20, dtype=torch.uint8, device="cuda")
        for _ in range(args.warmup):
            op_linear(xt, w, scratch)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(args.steps):
            op_linear(xt, w, scratch)
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / args.steps
        nbytes = args.n * args.kdim * 2 + args.rows * (args.kdim * 2 + args.n * 4)
        return {"case": "gemm", "n_out": args.n, "k": args.kdim, "rows": args.rows,
                "us_per_launch": ms * 1e3, "GB/s": nbytes / ms / 1e6}
    from paper_2608_10362_gb300 import Engine
    if args.case == "edge":
        return {"case": "edge", **run_pair_case(args, "target_1b1", "draft_68m", [512], 5, args.temp)}
    if args.case == "batched":
        from seeded_inputs import gen_prompt_lengths
        ctx = [int(c) for c in gen_prompt_lengths(11, 16, 512, 4096)]
        return {"case": "batched", **run_pair_case(args, "target_8b", "draft_1b1_v128k", ctx, 8, 1.0)}
    if args.case == "switching":
        return run_switching_case(args)
    if args.case == "prefill":
        # a whole-prompt prefill of the 7B target (chunks of up to 128 rows), timed,
        # inside an NVTX range "prefill"
        t = SHAPES[TARGET]
        eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=PREFIX + 64, max_k=args.k,
                     max_drafts=0, use_graphs=True,
                     trace="prefill" if args.trace is not None else None)
        prompt = gen_prompt(3, PREFIX, t.vocab)
        for _ in range(args.warmup):
            eng.prefill(0, prompt, seed=1)
        eng.sync()
        s = eng.stream
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.nvtx.range_push("prefill")
        a.record(s)
        for _ in range(args.steps):
            eng.prefill(0, prompt, seed=1)
        b.record(s)
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        bits = eng.sync()
        ms = a.elapsed_time(b) / args.steps
        if args.trace is not None:
            np.save(args.trace, eng.pass_trace())
        eng.close()
        return {"case": "prefill", "target": TARGET, "tokens": PREFIX, "ms": ms,
                "tokens_per_s": PREFIX / ms * 1e3, "device_status": bits}
    if args.case == "verify":
        # the 7B verify pass alone, one launch per op and no graph, inside an NVTX
        # range "verify" (for profilers: ncu --nvtx --nvtx-include "verify/")
        t = SHAPES[TARGET]
        K = args.k
        max_seq = PREFIX + (args.steps + args.warmup + 2) * (K + 1) + 16
        eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=K, max_drafts=0,
                     use_graphs=False, launch_mode=args.launch_mode)
        from paper_2608_10362_gb300 import _lib
        eng.prefill(0, gen_prompt(3, PREFIX, t.vocab), seed=1)
        dt = np.zeros((1, eng.max_k), dtype=np.int32)
        dt[0, :K] = gen_prompt(4, K, t.vocab)
        eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
        for _ in range(args.warmup):
            eng.verify_step(K)
        eng.sync()
        s = eng.stream
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.nvtx.range_push("verify")
        a.record(s)
        for _ in range(args.steps):
            eng.verify_step(K)
        b.record(s)
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        bits = eng.sync()
        ms = a.elapsed_time(b) / args.steps
        eng.close()
        return {"case": "verify", "target": TARGET, "K": K, "prefix": PREFIX, "graphs": False,
                "ms_per_verify": ms, "device_status": bits}
    t, d = SHAPES["draft_160m"], SHAPES["draft_68m"]
    K = args.k
    max_seq = 512 + (args.steps + args.warmup + 4) * (K + 1) + 16
    eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=K, max_drafts=1,
                 draft_shape_max=d, draft_budget_bytes=512 << 20, use_graphs=True,
                 launch_mode=args.launch_mode,
                 trace=args.trace_pass if args.trace is not None else None)
    eng.register_draft(0, d, iter_weights(d, 1))
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    eng.prefill(0, gen_prompt(3, 512, t.vocab), seed=1)
    for _ in range(args.warmup):
        eng.step(K, TEMP)
    eng.sync()
    L0 = int(eng.seq_state()[0, 0])
    s = eng.stream
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    for _ in range(args.steps):
        eng.step(K, TEMP)
    b.record(s)
    torch.cuda.synchronize()
    bits = eng.sync()
    L1 = int(eng.seq_state()[0, 0])
    ms = a.elapsed_time(b)
    if args.trace is not None:      # timestamps of the last traced pass
        np.save(args.trace, eng.pass_trace())
    eng.close()
    return {"case": "small", "target": "draft_160m", "draft": "draft_68m", "K": K,
            "ms_per_step": ms / args.steps, "tokens_per_s": (L1 - L0) / ms * 1e3,
            "device_status": bits}


TRAFFIC_PROFILE = os.path.join(ROOT, "profiles", "verify_7b_k4_ctx2048_dram.md")


def kernel_sources_hash() -> str:
    """sha256 over the CUDA sources (name + content, sorted by name)."""
    import glob
    import hashlib
    csrc = os.path.join(ROOT, "paper_2608_10362_gb300", "csrc")
    files = sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cuh")) +
                   glob.glob(os.path.join(csrc, "*.h")))
    h = hashlib.sha256()
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def recorded_traffic():
    """DRAM bytes of one verify pass from the committed ncu summary, if it was
    taken on the kernel sources as they are now (else None)."""
    try:
        with open(TRAFFIC_PROFILE) as fh:
            text = fh.read()
    except OSError:
        return None
    vals = {}
    for ln in text.splitlines():
        if ":" in ln and ln.split(":")[0] in ("traffic_bytes_per_verify", "kernel_sources_sha256"):
            k, v = ln.split(":", 1)
            vals[k.strip()] = v.strip()
    if vals.get("kernel_sources_sha256") != kernel_sources_hash():
        return None
    return int(vals["traffic_bytes_per_verify"]) if "traffic_bytes_per_verify" in vals else None


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--k", type=int, default=K_DRAFT)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--case", default="step", choices=["step", "gemm", "small", "verify", "prefill", "edge", "batched",
                                                          "switching"],
                    help="step: the workload above; gemm / small: diagnostic cases sized for "
                         "profiler captures (one projection GEMM; a 160M target with a 68M draft)")
    ap.add_argument("--temp", type=float, default=0.8, help="(--case edge) temperature")
    ap.add_argument("--launch-mode", default="per_op", choices=["per_op", "pass"],
                    help="one launch per op, or one persistent launch per pass")
    ap.add_argument("--draft-kernel", default="auto", choices=["auto", "per_op", "fused"],
                    help="draft-step kernels (auto: the fused draft kernel when the draft fits it)")
    ap.add_argument("--trace", default=None,
                    help="save per-op timestamps of the last traced pass (.npy); diagnostic, "
                         "not for the headline number")
    ap.add_argument("--trace-pass", default="verify", choices=["verify", "draft"],
                    help="(--case step) the pass to trace; --case prefill traces prefill chunks")
    ap.add_argument("--n", type=int, default=22016)
    ap.add_argument("--kdim", type=int, default=4096)
    ap.add_argument("--rows", type=int, default=5)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.case != "step":
        print(json.dumps(run_case(args)))
        return

    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))

    if args.impl == "reference":
        if rank != 0:
            return
        # The oracle cannot run full-depth 7B iterations fast enough to measure its
        # own acceptance; every iteration commits at least one token, so the
        # reference arm counts 1 token per iteration (a lower bound, stated in the
        # sample description).  W untimed steps, then K timed ones (one part each).
        tok_iter = 1.0
        a0 = time.perf_counter()
        one, desc = oracle_step_timer(args.k)
        for _ in range(args.warmup):
            one()
        iters = [one() for _ in range(args.steps)]
        it = statistics.median(iters)
        v = tok_iter / it
        wall = time.perf_counter() - a0
        cfg = workload_config(args.k, world)
        cfg["timing"] = "oracle on host cores"
        line = {"impl": "reference", "metric": METRIC, "value": v,
                "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": 1000.0 * it, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": cfg,
                "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": os.cpu_count(),
                                 "kind": "oracle",
                                 "sample": desc + f"; median of {args.steps} steps, wall "
                                           f"{wall:.1f} s; tokens/iteration counted as 1 "
                                           "(lower bound: acceptance not measured by the oracle)"},
                "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    r = run_gpu(args, rank, world)
    if rank != 0:
        return
    peak, peak_kind = measured_peaks()
    achieved = r["verify_bytes"] / (r["verify_ms"] * 1e-3) / 1e9
    value = r["tokens"] / (r["ms"] * 1e-3)
    line = {
        "metric": METRIC,
        "value": value, "unit": "tokens/s", "n_gpus": world, "steps": r["steps"],
        "warmup": args.warmup, "ms_per_step": r["ms"] / r["steps"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {**workload_config(args.k, world),
                   "l2": "inputs larger than L2 (13.5 GB of target weights streamed per verify)",
                   "tokens_per_step": r["tokens_per_step"]},
        "roofline": {"kernel": "verify pass (one CUDA graph of the target forward)",
                     "bound": "hbm", "achieved": achieved, "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": recorded_traffic(),
                     "traffic_source": "ncu dram__bytes_read+write of one verify pass "
                                       "(profiles/verify_7b_k4_ctx2048_dram.md); null when the "
                                       "kernels changed since",
                     "verify_ms": r["verify_ms"],
                     "algorithmic_bytes": r["verify_bytes"],
                     "frac_of_8000": achieved / 8000.0},
        "e2e": {"value": r["generated"] / r["e2e_s"], "unit": "tokens/s",
                "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"],
                "scope": "prompt H2D + prefill 2048 + decode, per-step D2H of results"},
        "gpu_launches": r["launches"],
        "draft": {"ms_per_step": r["draft_ms"], "us_per_pass": 1000.0 * r["draft_ms"] / args.k,
                  "kernel": "fused (one launch per draft step)" if r["draft_fused"] else "per-op",
                  "launches_per_step": r["launches_per_step"]},
        "clocks": r["clocks"],
        "device_status": r["bits"],
        "setup_s": r["setup_s"],
    }
    if not args.no_cpu_baseline and world == 1:
        cb = oracle_sample(r["tokens_per_step"], args.k)
        line["cpu_baseline"] = {"value": cb["value"], "unit": "tokens/s", "cores": cb["cores"],
                                "kind": "oracle", "sample": cb["sample"]}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
