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


def cpu_model() -> str:
    """The host CPU's model name (x86 'model name', else Arm 'CPU part' codes)."""
    try:
        with open("/proc/cpuinfo") as fh:
            text = fh.read()
    except OSError:
        return "unknown"
    for key in ("model name", "Model name", "CPU part"):
        for ln in text.splitlines():
            if ln.startswith(key):
                return ln.split(":", 1)[1].strip()
    return "unknown"


class OracleIteration:
    """The CPU baseline: the oracle (plain fp64 NumPy) running whole
    draft-then-verify iterations of the workload at a reduced, stated depth.

    The target keeps n_t of its layers and the draft n_d of its layers, both at
    full width and full vocabulary; the target's KV cache holds PREFIX synthetic
    positions.  One step = K draft passes (1 row each, sampled), one verify pass
    over K+1 rows, acceptance and commit - all of it executed, and its elapsed
    time is the step's time.  The full-depth iteration time is estimated from the
    same step's own per-layer timings (layer time x depth) and is what the
    tokens/s value reports, with the committed tokens per iteration the oracle
    itself measured over its steps."""

    def __init__(self, K: int, n_t: int = 2, n_d: int = 1, seed: int = 0):
        import dataclasses

        import numpy as np

        from oracle.llama import LlamaOracle
        from oracle.speculative import SpecDecoder
        from seeded_inputs import SHAPES, gen_kv, gen_prompt, gen_tensor

        self.np = np
        t, d = SHAPES[TARGET], SHAPES[DRAFT]
        self.full = (t.n_layers, d.n_layers)
        self.K, self.n_t, self.n_d = K, n_t, n_d
        ts, ds = dataclasses.replace(t, n_layers=n_t), dataclasses.replace(d, n_layers=n_d)

        def weights(shape, full_shape, seed_):
            w = {}
            for li in range(shape.n_layers):
                for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
                    w[(n, li)] = gen_tensor(full_shape, seed_, n, li)
            for n in ("tok_emb", "final_norm", "lm_head"):
                w[(n, -1)] = gen_tensor(full_shape, seed_, n)
            return w

        self.to = LlamaOracle(ts, weights(ts, t, seed), keep_f64=True)
        self.do = LlamaOracle(ds, weights(ds, d, seed + 1), keep_f64=True)
        prompt = [int(x) for x in gen_prompt(100, 2, t.vocab)]
        self.sd = SpecDecoder(self.to, self.do, prompt, PREFIX + 4096)
        # a committed sequence of PREFIX tokens: the target cache holds the first
        # PREFIX - 1 positions (position 0 from the prompt's own row, 1..PREFIX-2
        # seeded N(0,1) K/V); the draft cache is as long (its K/V are zeros)
        kv = gen_kv(3, (n_t, 2, PREFIX, t.n_kv_heads, t.head_dim))
        self.sd.tc.k[:, 1:PREFIX - 1] = kv[:, 0, 1:PREFIX - 1]
        self.sd.tc.v[:, 1:PREFIX - 1] = kv[:, 1, 1:PREFIX - 1]
        self.sd.tc.length = PREFIX - 1
        self.sd.tokens = [self.sd.tokens[0]] * (PREFIX - 1) + self.sd.tokens[-1:]
        self.sd.dc.length = PREFIX - 1
        self.step_i = 0
        self.tokens = 0
        # per-part timers wrap the models' layer and logits calls
        self.part = {"t_layer": 0.0, "t_lm": 0.0, "d_layer": 0.0, "d_lm": 0.0}
        for name, model in (("t", self.to), ("d", self.do)):
            self._wrap(model, name)

    def _wrap(self, model, name):
        layer, logits = model.layer, model.logits

        def timed_layer(*a, **k):
            t0 = time.perf_counter()
            r = layer(*a, **k)
            self.part[name + "_layer"] += time.perf_counter() - t0
            return r

        def timed_logits(*a, **k):
            t0 = time.perf_counter()
            r = logits(*a, **k)
            self.part[name + "_lm"] += time.perf_counter() - t0
            return r

        model.layer, model.logits = timed_layer, timed_logits

    def step(self):
        """One executed iteration: (elapsed s, committed tokens, full-depth estimate s)."""
        for k in self.part:
            self.part[k] = 0.0
        t0 = time.perf_counter()
        rec = self.sd.step(self.K, TEMP, 1, 0, self.step_i)
        el = time.perf_counter() - t0
        self.step_i += 1
        n = rec.result.n_accepted + 1
        self.tokens += n
        fixed = el - sum(self.part.values())
        est = (self.part["t_layer"] * self.full[0] / self.n_t + self.part["t_lm"] +
               self.part["d_layer"] * self.full[1] / self.n_d + self.part["d_lm"] + fixed)
        return el, n, est

    def describe(self) -> str:
        return (f"fp64 numpy oracle: whole iterations (K={self.K} draft passes, verify over "
                f"{self.K + 1} rows, acceptance) of the target at {self.n_t} of {self.full[0]} layers and "
                f"the draft at {self.n_d} of {self.full[1]} layers, full width and vocabulary, target "
                f"KV at context {PREFIX}; full-depth time = this step's per-layer times x depth")


def cpu_baseline_run(K: int, warmup: int, steps: int, one_core: bool = True) -> dict:
    """W + K oracle iterations on all host cores (and, optionally, the same in a
    1-core subprocess); tokens/s at full depth from the measured parts."""
    import statistics as st
    a0 = time.perf_counter()
    it = OracleIteration(K)
    setup = time.perf_counter() - a0
    for _ in range(warmup):
        it.step()
    rows = [it.step() for _ in range(steps)]
    el = [r[0] for r in rows]
    est = st.median([r[2] for r in rows])
    tok_iter = sum(r[1] for r in rows) / len(rows)
    out = {"value": tok_iter / est, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
           "cpu_model": cpu_model(), "ms_per_step": 1000.0 * st.mean(el), "steps": steps,
           "full_depth_iteration_s": est, "tokens_per_iteration": tok_iter, "setup_s": setup,
           "sample": it.describe() + f"; {steps} timed steps after {warmup}; "
                     f"{tok_iter:.2f} tokens per iteration (the oracle's own)"}
    if one_core:
        env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
        code = ("import bench, json; r = bench.cpu_baseline_run(%d, 1, 2, one_core=False); "
                "print(json.dumps({'value': r['value'], 'full_depth_iteration_s': r['full_depth_iteration_s']}))" % K)
        try:
            p = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                               text=True, timeout=600)
            one = json.loads(p.stdout.strip().splitlines()[-1])
            out["one_core"] = {"value": one["value"], "full_depth_iteration_s": one["full_depth_iteration_s"]}
        except Exception as e:  # pragma: no cover - reported, not fatal
            out["one_core"] = {"error": str(e)[:200]}
    return out


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
        torch.cuda.nvtx.range_push("verify")   # for profilers: --nvtx --nvtx-include "verify/"
        eng.verify_step(K)
        torch.cuda.nvtx.range_pop()
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


class TimedResidency:
    """The residency mechanism the scheduler acts through: the Engine's draft calls,
    with each side-stream load bracketed by CUDA events (its copy time, and its
    overlap with the steps on the main stream)."""

    def __init__(self, eng, base_event):
        import torch
        self.eng, self.base, self.torch = eng, base_event, torch
        self.loads = []            # (draft, start event, end event)

    def state(self, d):
        return self.eng.query_draft(d)

    def load(self, d):
        from paper_2608_10362_gb300 import MemSpecError, _lib
        if self.eng.query_draft(d) != 0:
            return True
        a = self.torch.cuda.Event(enable_timing=True)
        b = self.torch.cuda.Event(enable_timing=True)
        a.record(self.eng.side)
        try:
            self.eng.load_draft_async(d)
        except MemSpecError as e:
            if e.status == _lib.ERR_BUDGET:
                return False
            raise
        b.record(self.eng.side)
        self.loads.append((d, a, b))
        return True

    def evict(self, d):
        self.eng.evict_draft(d)

    def set_active(self, d):
        self.eng.set_active_draft(d)


def run_switching_case(args):
    """Draft switching under a 2 GiB draft budget: the 7B target with a pool of
    drafts (68M, 160M, tied 1.1B) in pinned host memory.  Every interval (64
    committed tokens) a seeded score stream stands in for the draft predictor;
    the policies of the native scheduler (MemSpec's cache update + best-resident
    selection, MAB-Async's UCB, static) and a blocking baseline (evict, load and
    switch to the top-scored draft at once) run the same stream.  Reported per
    policy: tokens/s over the whole run, desired / fallback / stall time, load
    time per draft, how much of the load time overlapped decoding, and the
    verify pass's GB/s with and without a load in flight."""
    import numpy as np
    import torch

    from paper_2608_10362_gb300 import DraftScheduler, Engine, weights_bytes
    from seeded_inputs import SHAPES, gen_prompt, gen_score_stream, iter_weights
    t = SHAPES[TARGET]
    pool = {0: SHAPES["draft_68m"], 1: SHAPES["draft_160m"], 2: SHAPES["draft_1b1_tied"]}
    K, T, prefix, budget, every = 4, 1.0, 1024, 2 << 30, 64
    n_int = max(3, args.steps)
    scores = gen_score_stream(3, n_int + 1, 3, phase=2)
    max_seq = prefix + (n_int + 2) * (every + 2 * (K + 1)) * 4 + 256
    eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=K, max_drafts=3,
                 draft_shape_max=pool[2], draft_budget_bytes=budget, use_graphs=True)
    for i, sh in pool.items():
        eng.register_draft(i, sh, iter_weights(sh, 10 + i))
    sizes = {i: weights_bytes(sh) for i, sh in pool.items()}
    ctx_now = prefix + 4 * (every + K + 1)
    vb = verify_bytes(t, ctx_now, K)
    s = eng.stream
    results = {}
    for policy in ("memspec", "mab_async", "static", "blocking"):
        # a fresh start: no draft resident, a new request
        eng.set_active_draft(-1)
        for i in pool:
            if eng.query_draft(i) != 0:
                eng.sync()
                while eng.query_draft(i) == 2:
                    time.sleep(0.001)
                eng.evict_draft(i)
        torch.cuda.synchronize()
        base = torch.cuda.Event(enable_timing=True)
        base.record(s)
        mech = TimedResidency(eng, base)
        eng.prefill(0, gen_prompt(5, prefix, t.vocab), seed=2)     # no draft active yet
        sched = None
        if policy != "blocking":
            sched = DraftScheduler(3, 2, policy, ucb_c=2.0, k_draft=K, mechanism=mech)
            sched.start(scores[0])                                  # loads d0, catches it up
        else:
            d0 = int(np.argmax(scores[0]))
            mech.load(d0)
            mech.set_active(d0)
        steps, stall_ms, switches = [], 0.0, 0
        L = int(eng.seq_state()[0, 0])
        torch.cuda.synchronize()
        w0 = time.perf_counter()
        tokens = 0
        for k in range(n_int):
            a0 = time.perf_counter()
            start, it = L, 0
            while L - start < every:
                e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
                e[0].record(s)
                eng.draft_step(K, T)
                e[1].record(s)
                eng.verify_step(K)
                e[2].record(s)
                eng.accept_commit(K, T, eng.results_host)
                s.synchronize()
                L += int(eng.results_host[0]) + 1
                it += 1
                steps.append(e)
            tokens += L - start
            if sched is not None:
                sched.feedback(it, L - start, time.perf_counter() - a0)
                sched.point(scores[k + 1])
            else:                       # blocking: switch to the top draft now
                want = int(np.argmax(scores[k + 1]))
                b0 = time.perf_counter()
                cur = [i for i in pool if eng.query_draft(i) != 0]
                if want not in cur:
                    eng.set_active_draft(-1)
                    for i in cur:
                        free = budget - sum(sizes[j] for j in pool if eng.query_draft(j) != 0)
                        if free >= sizes[want]:
                            break
                        eng.evict_draft(i)
                    mech.load(want)
                    switches += 1
                eng.set_active_draft(want)              # waits for the copy, catches up
                eng.sync()
                stall_ms += (time.perf_counter() - b0) * 1e3
        torch.cuda.synchronize()
        wall = time.perf_counter() - w0
        st = sched.stats() if sched is not None else {}
        # loads: copy time and overlap with the steps (all events against `base`)
        t_of = lambda ev: base.elapsed_time(ev)
        spans = [(t_of(x[0]), t_of(x[2])) for x in steps]
        loads = []
        for d, a, b in mech.loads:
            la, lb = t_of(a), t_of(b)
            ov = sum(max(0.0, min(lb, y) - max(la, x)) for x, y in spans)
            loads.append((d, lb - la, ov))
        ver = [(t_of(x[1]), t_of(x[2])) for x in steps]
        busy = lambda v: any(min(v[1], lb) > max(v[0], la) for _, la, lb in
                             [(d, t_of(a), t_of(b)) for d, a, b in mech.loads])
        v_load = [y - x for x, y in ver if busy((x, y))]
        v_idle = [y - x for x, y in ver if not busy((x, y))]
        load_ms = {}
        for d, ms_, _ in loads:
            load_ms.setdefault(["68M", "160M", "1.1B tied"][d], []).append(round(ms_, 2))
        total_load = sum(x[1] for x in loads)
        res = {"tokens_per_s": tokens / wall, "tokens": tokens, "wall_s": wall,
               "step_ms_median": float(np.median([x[0].elapsed_time(x[2]) for x in steps])),
               "loads": len(loads), "load_ms": load_ms,
               "overlap_fraction": (sum(x[2] for x in loads) / total_load) if total_load > 0 else None,
               "verify_GBps_loading": (vb / (np.median(v_load) * 1e-3) / 1e9) if v_load else None,
               "verify_GBps_idle": (vb / (np.median(v_idle) * 1e-3) / 1e9) if v_idle else None,
               "stall_ms": stall_ms if policy == "blocking" else 0.0, "blocking_switches": switches}
        if st:
            res.update({"desired_s": st["desired_s"], "fallback_s": st["fallback_s"],
                        "policy_s": st["policy_s"], "fallback_intervals": st["fallback_intervals"],
                        "desired_intervals": st["desired_intervals"], "evictions": st["evictions"],
                        "refusals": st["refusals"], "switches": st["switches"]})
            sched.close()
        results[policy] = res
    bits = eng.sync()
    eng.close()
    return {"case": "switching", "target": TARGET, "pool": ["68M", "160M", "1.1B tied"],
            "budget_GiB": 2, "capacity": 2, "interval_tokens": every, "intervals": n_int,
            "prefix": prefix, "K": K, "T": T, "policies": results, "device_status": bits}


def run_int4_case(args):
    """The 7B target's projections as group-wise INT4 weights (the paper's GPTQ
    INT4 targets): 32 layers x (qkv 12288x4096, o 4096x4096, gate_up 22016x4096,
    down 4096x11008) with distinct random codes (3.6 GB packed, far above L2),
    one launch per projection at `rows` activation rows (K + 1 = 5 for one
    verify pass), replayed from a CUDA graph.  Reports each shape's mean launch time over the 32 layers and
    the whole stack's algorithmic bytes / time against the measured HBM peak."""
    import torch

    from paper_2608_10362_gb300 import int4_pack, op_linear_int4
    from seeded_inputs import SHAPES
    t = SHAPES[TARGET]
    shapes = {"qkv": (t.q_dim + 2 * t.kv_dim, t.d_model), "o": (t.d_model, t.q_dim),
              "gate_up": (2 * t.d_ffn, t.d_model), "down": (t.d_model, t.d_ffn)}
    rows = args.rows
    gen = torch.Generator(device="cuda").manual_seed(0)
    n_layers = args.int4_layers or t.n_layers
    layers = []
    for _ in range(n_layers):
        ent = {}
        for name, (n, k) in shapes.items():
            qw = torch.randint(0, 256, (n, k // 2), dtype=torch.uint8, device="cuda", generator=gen)
            sc = (torch.rand(n, k // 128, device="cuda", generator=gen) * 0.006 + 0.002).to(torch.bfloat16)
            zs = torch.randint(0, 16, (n, k // 128), dtype=torch.uint8, device="cuda", generator=gen)
            ent[name] = int4_pack(qw, sc, zs)
            del qw, sc, zs
        layers.append(ent)
    xs = {k: (torch.randn(rows, k, device="cuda", generator=gen)).to(torch.bfloat16)
          for k in {t.d_model, t.q_dim, t.d_ffn}}
    ys = {name: torch.empty(rows, n, device="cuda") for name, (n, k) in shapes.items()}

    def nbytes(name):
        n, k = shapes[name]
        return ((n + 15) // 16) * (k // 128) * 1072 + rows * k * 2 + rows * n * 4

    def run(names):
        for ent in layers:
            for name in names:
                n, k = shapes[name]
                op_linear_int4(xs[k], ent[name], n, y=ys[name])

    out = {"case": "int4", "target": TARGET, "rows": rows, "layers": n_layers, "group": 128, "shapes": {}}
    peak, peak_src = measured_peaks()
    out["peak"] = {"hbm_GBps": peak, "source": peak_src}
    for names in [[nm] for nm in shapes] + [list(shapes)]:
        for _ in range(args.warmup):
            run(names)
        torch.cuda.synchronize()
        # the pass's launches replayed from a CUDA graph: the timing is the
        # kernels', not the Python loop's
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            run(names)
        graph.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(1, args.steps)
        a.record()
        for _ in range(reps):
            graph.replay()
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / reps
        byt = sum(nbytes(nm) for nm in names) * n_layers
        gbs = byt / ms / 1e6
        key = names[0] if len(names) == 1 else "all"
        out["shapes"][key] = {"us_per_launch": ms * 1e3 / (n_layers * len(names)),
                              "ms_per_pass": ms, "bytes_per_pass": byt, "GB/s": gbs,
                              "frac_of_hbm_peak": gbs / peak}
    return out


def run_tree_case(args):
    """Tree verification on the 7B target at prefix 2048 (the engine MemSpec
    builds on verifies draft trees): one step = the tree pass (root + nodes,
    ancestor-masked attention), a draw from every row, the walk, the commit and
    the K/V compaction, replayed from a CUDA graph.  Trees of 4, 8, 15 and 31
    nodes (widths per depth below), random tokens; the chain verify pass at
    K = 4 (5 rows) is timed alongside.  With random weights almost nothing is
    accepted: the line reports cost per step and bytes per second, not
    tokens per step."""
    import numpy as np
    import torch

    from paper_2608_10362_gb300 import Engine, _lib
    from seeded_inputs import SHAPES, gen_prompt, iter_weights
    t = SHAPES[TARGET]
    reps = max(1, args.steps)
    max_seq = PREFIX + (reps + args.warmup + 4) * 33 + 64
    eng = Engine(t, iter_weights(t, 0), max_batch=1, max_seq=max_seq, max_k=args.k, max_drafts=0,
                 use_graphs=True)
    prompt = gen_prompt(3, PREFIX, t.vocab)
    rng = np.random.default_rng(9)
    shapes = {4: (2, 1, 1), 8: (2, 2, 1, 1, 1, 1), 15: (4, 3, 3, 2, 2, 1), 31: (6, 5, 5, 4, 4, 3, 2, 2)}
    out = {"case": "tree", "target": TARGET, "prefix": PREFIX, "graphs": True, "trees": {}}
    s = eng.stream
    for n_nodes, widths in shapes.items():
        # a spine with `w` children per level, continued through the first child
        tokens, parents, cur = [], [], -1
        for w in widths:
            first = len(tokens)
            for _ in range(w):
                tokens.append(int(rng.integers(0, t.vocab)))
                parents.append(cur)
            cur = first
        assert len(tokens) == n_nodes, (n_nodes, len(tokens))
        eng.prefill(0, prompt, seed=1)
        for _ in range(args.warmup):
            eng.tree_step(tokens, parents, TEMP)
        eng.sync()
        L0 = int(eng.seq_state()[0, 0])
        pass_bytes = verify_bytes(t, L0 - 1, n_nodes)   # the pass over n_nodes + 1 rows
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s)
        for _ in range(reps):
            eng.tree_step(tokens, parents, TEMP)
        b.record(s)
        torch.cuda.synchronize()
        bits = eng.sync()
        ms = a.elapsed_time(b) / reps
        L1 = int(eng.seq_state()[0, 0])
        out["trees"][n_nodes] = {"rows": n_nodes + 1, "depth": len(widths), "ms_per_step": ms,
                                 "tokens_per_step": (L1 - L0) / reps, "pass_GBps": pass_bytes / ms / 1e6,
                                 "device_status": bits}
    # the chain verify pass over K + 1 rows, same prefix, for comparison
    eng.prefill(0, prompt, seed=1)
    dt = np.zeros((1, eng.max_k), dtype=np.int32)
    dt[0, :args.k] = gen_prompt(4, args.k, t.vocab)
    eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
    for _ in range(args.warmup):
        eng.verify_step(args.k)
    eng.sync()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    for _ in range(reps):
        eng.verify_step(args.k)
    b.record(s)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / reps
    out["chain_verify"] = {"K": args.k, "rows": args.k + 1, "ms": ms,
                           "pass_GBps": verify_bytes(t, PREFIX - 1, args.k) / ms / 1e6,
                           "device_status": eng.sync()}
    eng.close()
    return out


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
    if args.case == "int4":
        return run_int4_case(args)
    if args.case == "tree":
        return run_tree_case(args)
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
        # range "verify" (for profilers: ncu --nvtx --nvtx-include "verify/");
        # --layers N keeps only N of the 7B target's layers (every per-layer
        # kernel and the LM head keep their full size: a profiler-sized case)
        import dataclasses
        t = SHAPES[TARGET]
        if args.layers:
            t = dataclasses.replace(t, n_layers=args.layers)
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
        return {"case": "verify", "target": TARGET, "layers": t.n_layers, "K": K, "prefix": PREFIX,
                "graphs": False, "ms_per_verify": ms, "device_status": bits}
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


TRAFFIC_PROFILE = os.path.join(ROOT, "profiles", "verify_7b_2layers_k4_ctx2048_dram.md")
# the sources of the kernels a verify pass launches (and of their launch set-up)
VERIFY_SOURCES = ("api.cu", "attention.cu", "attn_body.cuh", "embed.cu", "embed_body.cuh", "gemm.cu",
                  "gemm_epi.cuh", "internal.h", "pack.cu", "ptx.cuh")


def kernel_sources_hash(names=VERIFY_SOURCES) -> str:
    """sha256 over the named CUDA sources (name + content, in name order)."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2608_10362_gb300", "csrc")
    h = hashlib.sha256()
    for name in sorted(names):
        h.update(name.encode())
        with open(os.path.join(csrc, name), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def recorded_traffic():
    """DRAM bytes of one full verify pass, scaled from the committed ncu summary
    of a 2-layer pass (per-layer kernels x 32 + LM head + embedding), if it was
    taken on the verify kernels' sources as they are now (else None)."""
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
                                                          "switching", "int4", "tree"],
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
    ap.add_argument("--layers", type=int, default=0,
                    help="(--case verify) layers of the 7B target to keep (default: all)")
    ap.add_argument("--int4-layers", type=int, default=0,
                    help="(--case int4) layers of INT4 weights (default: all of the 7B target's)")
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
        # K timed oracle iterations after W untimed ones, each executed in full
        # at the stated reduced depth (OracleIteration); ms_per_step is their
        # elapsed time, value the full-depth tokens/s estimated from them
        a0 = time.perf_counter()
        cb = cpu_baseline_run(args.k, args.warmup, args.steps, one_core=False)
        wall = time.perf_counter() - a0
        cfg = workload_config(args.k, world)
        cfg["timing"] = "oracle on host cores"
        v = cb["value"]
        line = {"impl": "reference", "metric": METRIC, "value": v,
                "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": cb["ms_per_step"], "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": cfg,
                "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cb["cores"], "kind": "oracle",
                                 "cpu_model": cb["cpu_model"],
                                 "full_depth_iteration_s": cb["full_depth_iteration_s"],
                                 "tokens_per_iteration": cb["tokens_per_iteration"],
                                 "sample": cb["sample"] + f"; run wall {wall:.1f} s"},
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
                     "traffic_source": "ncu dram__bytes_read+write per kernel of a 2-layer 7B verify "
                                       "pass, scaled to 32 layers (profiles/verify_7b_2layers_k4_"
                                       "ctx2048_dram.md); null when the verify kernels changed since",
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
        cb = cpu_baseline_run(args.k, 1, 3, one_core=True)
        line["cpu_baseline"] = {k: cb[k] for k in ("value", "unit", "cores", "kind", "cpu_model",
                                                   "full_depth_iteration_s", "tokens_per_iteration",
                                                   "sample", "one_core")}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
