"""Parity at the workload sizes (GPU), in the launch configuration bench.py uses
(captured CUDA graphs):

* edge pair (1.1B GQA target, 68M draft, prefix 512, K=5): lock-step against the
  oracle, greedy and T = 0.8;
* 7B-shape target with the 160M draft (the benchmark's pair): a 3-step
  lock-step from a 64-token prefix, and the verify pass at context 2048 with a
  seeded KV cache, K=4 (logits of all K+1 rows and the K/V appended);
* 8B-shape target, batched verify (B=16, K=8, vocab 128256, per-request contexts
  uniform in [512, 4096]): logits of every request, then acceptance /
  resample / commit of all 16 requests on those logits with per-request Philox
  keys;
* draft switching under a byte budget: load / query / evict rules, and lock-step
  parity after switching the active draft mid-generation.
"""
import dataclasses

import numpy as np
import pytest
import torch

from lockstep import LOGIT_TOL, RECORDS, U_TOL, LockstepReport, check_step
from oracle.llama import LlamaOracle
from oracle.philox import step_uniforms
from oracle.speculative import SpecDecoder, accept, argmax_first, sample_inverse_cdf, softmax_t
from seeded_inputs import SHAPES, ModelShape, gen_kv, gen_prompt, gen_prompt_lengths, gen_weights

pytestmark = pytest.mark.gpu


def _kv_view(eng, shape):
    """bf16 view [layer][K|V][request][kv_head][pos][hd] of the engine's KV cache."""
    return eng.kv.view(torch.bfloat16).view(shape.n_layers, 2, eng.max_batch, shape.n_kv_heads,
                                            eng.max_seq, shape.head_dim)


def _fill_kv(eng, shape, req, ctx, seed, oracle_cache=None):
    """Seeded N(0,1) bf16 K/V for positions < ctx of one request (GPU and oracle)."""
    kv = gen_kv(seed, (shape.n_layers, 2, ctx, shape.n_kv_heads, shape.head_dim))
    view = _kv_view(eng, shape)
    t = torch.from_numpy(kv).to(torch.bfloat16)          # exact: values are bf16
    view[:, :, req, :, :ctx, :] = t.permute(0, 1, 3, 2, 4).cuda()
    if oracle_cache is not None:
        oracle_cache.k[:, :ctx] = kv[:, 0].astype(np.float64)
        oracle_cache.v[:, :ctx] = kv[:, 1].astype(np.float64)
        oracle_cache.length = ctx
    return kv


def _set_verify_state(eng, ctxs, K, tokens_last, drafts, seeds=None):
    from paper_2608_10362_gb300 import _lib
    B = len(ctxs)
    state = np.zeros((eng.max_batch, 4), dtype=np.int32)
    toks = np.zeros((eng.max_batch, eng.max_seq), dtype=np.int32)
    dt = np.zeros((eng.max_batch, eng.max_k), dtype=np.int32)
    for b, ctx in enumerate(ctxs):
        state[b] = (ctx + 1, ctx, 0, 0)
        toks[b, ctx] = tokens_last[b]
        dt[b, :K] = drafts[b]
    eng.write_buffer(_lib.BUF_TOKENS, toks)
    eng.write_buffer(_lib.BUF_SEQ_STATE, state)
    eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
    if seeds is not None:
        sd = np.zeros(eng.max_batch, dtype=np.uint64)
        sd[:B] = seeds
        eng.write_buffer(_lib.BUF_SEEDS, sd)
    eng.set_batch(B)


# ---------------------------------------------------------------------- edge pair
@pytest.fixture(scope="module")
def edge():
    from paper_2608_10362_gb300 import Engine
    t, d = SHAPES["target_1b1"], SHAPES["draft_68m"]
    wt, wd = gen_weights(t, 0), gen_weights(d, 1)
    eng = Engine(t, wt, max_batch=1, max_seq=1024, max_k=5, max_drafts=1, draft_shape_max=d,
                 draft_budget_bytes=256 << 20, use_graphs=True)
    eng.register_draft(0, d, wd)
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    yield eng, LlamaOracle(t, wt, keep_f64=True), LlamaOracle(d, wd, keep_f64=True)
    eng.close()


# error-band flags allowed on the edge pair (its logit error is ~10x the tiny pair's)
EDGE_BAND_FLAGS = 2


@pytest.mark.parametrize("T", [0.0, 0.8])
def test_edge_pair_lockstep(edge, T):
    eng, to, do = edge
    prompt = gen_prompt(21, 512, 32000)
    K, steps = 5, 6
    eng.prefill(0, prompt, seed=9)
    sd = SpecDecoder(to, do, prompt, len(prompt) + steps * (K + 1) + 4)
    rep = LockstepReport()
    for step in range(steps):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 9, step, rep)
    line = rep.record(f"edge T={T}")
    assert rep.band_flags <= EDGE_BAND_FLAGS, line


# ---------------------------------------------------------------------- 7B target + 160M draft
@pytest.fixture(scope="module")
def big_pair():
    from paper_2608_10362_gb300 import Engine
    t, d = SHAPES["target_7b"], SHAPES["draft_160m"]
    wt, wd = gen_weights(t, 0), gen_weights(d, 1)
    eng = Engine(t, wt, max_batch=1, max_seq=2048 + 64, max_k=4, max_drafts=1,
                 draft_shape_max=d, draft_budget_bytes=512 << 20, use_graphs=True)
    eng.register_draft(0, d, wd)
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    yield eng, t, wt, LlamaOracle(t, wt), LlamaOracle(d, wd, keep_f64=True)
    eng.close()


def test_7b_160m_lockstep_short_prefix(big_pair):
    """The benchmark's pair, every decision of three whole iterations (T = 1,
    K = 4) compared with the oracle from a 64-token prefix."""
    eng, t, _, to, do = big_pair
    K, T, steps, seed = 4, 1.0, 3, 31
    prompt = gen_prompt(61, 64, t.vocab)
    eng.prefill(0, prompt, seed=seed)
    sd = SpecDecoder(to, do, prompt, len(prompt) + steps * (K + 1) + 4)
    rep = LockstepReport()
    for step in range(steps):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, seed, step, rep)
    line = rep.record("7B + 160M T=1.0 prefix 64")
    assert rep.band_flags == 0, line


def test_7b_verify_pass_full_size(big_pair):
    eng, t, w, oracle, _ = big_pair
    K, ctx = 4, 2048
    cache = oracle.new_cache(ctx + K + 1)
    _fill_kv(eng, t, 0, ctx, 77, cache)
    rng = np.random.default_rng(5)
    last, drafts = int(rng.integers(0, t.vocab)), rng.integers(0, t.vocab, K).astype(np.int32)
    _set_verify_state(eng, [ctx], K, [last], [drafts])
    eng.verify_step(K)
    assert eng.sync() == 0
    zg = eng.target_logits(1, K)[0]
    kv_new = _kv_view(eng, t)[:, :, 0, :, ctx:ctx + K + 1, :].float().cpu().numpy()
    zo = oracle.forward(cache, [last] + list(drafts))
    errs = []
    for i in range(K + 1):
        err = np.abs(zg[i] - zo[i]).max() / np.abs(zo[i]).max()
        errs.append(err)
        assert err <= LOGIT_TOL
        a, b = argmax_first(zo[i]), int(np.argmax(zg[i]))
        assert a == b or zo[i][a] - zo[i][b] <= 2 * np.abs(zg[i] - zo[i]).max()
    RECORDS.append(f"7B verify ctx {ctx} K={K}: max logit err {max(errs):.2e} of max")
    # K/V appended at positions ctx..ctx+K (bf16 storage of the rotated keys / values)
    ko = cache.k[:, ctx:ctx + K + 1].transpose(0, 2, 1, 3)     # [layer][kvh][pos][hd]
    vo = cache.v[:, ctx:ctx + K + 1].transpose(0, 2, 1, 3)
    for got, ref in ((kv_new[:, 0], ko), (kv_new[:, 1], vo)):
        scale = np.abs(ref).max(axis=(1, 2, 3), keepdims=True)
        assert np.all(np.abs(got - ref) <= 0.03 * scale)


# ---------------------------------------------------------------------- batched 8B verify
def test_8b_batched_verify_and_accept_all_requests():
    """Batched verification at its stated size: every request's K+1 logit rows
    against the oracle, then acceptance / resample / commit of all 16 requests
    on the GPU's own logits (identical inputs on both sides, per-request Philox
    keys): n and the final token bit-exact unless the stated tolerance exempts
    the decision, p_i(x_i) and q_i(x_i) within 1e-4 relative."""
    from paper_2608_10362_gb300 import Engine, _lib
    t = SHAPES["target_8b"]
    # a minimal draft with the target's vocabulary: acceptance needs an active draft
    dsh = ModelShape(1, 128, 2, 2, 64, 352, t.vocab)
    B, K, T = 16, 8, 1.0
    ctxs = [int(c) for c in gen_prompt_lengths(11, B, 512, 4096)]
    w = gen_weights(t, 0)
    eng = Engine(t, w, max_batch=B, max_seq=4096 + 64, max_k=K, max_drafts=1,
                 draft_shape_max=dsh, draft_budget_bytes=64 << 20, use_graphs=True)
    eng.register_draft(0, dsh, gen_weights(dsh, 5))
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    oracle = LlamaOracle(t, w)
    rng = np.random.default_rng(6)
    last = rng.integers(0, t.vocab, B)
    drafts = rng.integers(0, t.vocab, (B, K)).astype(np.int32)
    seeds = [1000 + 7 * b for b in range(B)]
    for b in range(B):
        _fill_kv(eng, t, b, ctxs[b], 100 + b)
    _set_verify_state(eng, ctxs, K, last, drafts, seeds)
    eng.verify_step(K)
    assert eng.sync() == 0
    zg = eng.target_logits(B, K)
    # ---- logits: the requests advance in groups of four, layer by layer (each
    # matrix is converted once per group)
    worst = 0.0
    for g0 in range(0, B, 4):
        grp = list(range(g0, g0 + 4))
        caches = {}
        for b in grp:
            caches[b] = oracle.new_cache(ctxs[b] + K + 1)
            kv = gen_kv(100 + b, (t.n_layers, 2, ctxs[b], t.n_kv_heads, t.head_dim))
            caches[b].k[:, :ctxs[b]] = kv[:, 0]
            caches[b].v[:, :ctxs[b]] = kv[:, 1]
            caches[b].length = ctxs[b]
            del kv
        hs = {b: oracle.embed([int(last[b])] + list(drafts[b])) for b in grp}
        pos = {b: np.arange(ctxs[b], ctxs[b] + K + 1) for b in grp}
        for li in range(t.n_layers):
            for b in grp:
                hs[b] = oracle.layer(li, hs[b], caches[b], pos[b])
        for b in grp:
            zo = oracle.logits(hs[b])
            err = max(np.abs(zg[b, i] - zo[i]).max() / np.abs(zo[i]).max() for i in range(K + 1))
            worst = max(worst, err)
            assert err <= LOGIT_TOL, (b, ctxs[b], err)
        del caches, hs
    RECORDS.append(f"8B batched verify B={B} K={K}: max logit err {worst:.2e} of max "
                   f"(all {B} requests)")
    # ---- acceptance on the GPU's logits: drafts drawn from q = softmax(zd / T),
    # zd = the target's logits plus noise (so that acceptance is neither certain nor rare)
    zt64 = zg.astype(np.float64)
    zd = np.empty((B, K, t.vocab), dtype=np.float32)
    xs = np.zeros((B, K), dtype=np.int32)
    for b in range(B):
        u_d, _, _ = step_uniforms(seeds[b], b, 0, K)
        sd_row = zt64[b, :K].std(axis=1, keepdims=True)
        noise = np.random.default_rng([7, b]).standard_normal((K, t.vocab))
        zd[b] = (zt64[b, :K] + 0.7 * sd_row * noise).astype(np.float32)
        for i in range(K):
            xs[b, i] = sample_inverse_cdf(softmax_t(zd[b, i].astype(np.float64), T), u_d[i])
    eng.write_buffer(_lib.BUF_DRAFT_LOGITS, zd)
    dt = np.zeros((B, eng.max_k), dtype=np.int32)
    dt[:, :K] = xs
    eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
    eng.accept_commit(K, T, eng.results_host)
    assert eng.sync() == 0
    res = eng.results_host.numpy()[:B * (K + 2)].reshape(B, K + 2)
    dbg = eng.accept_debug(B, K)
    state = eng.seq_state()
    rep = LockstepReport()
    for b in range(B):
        _, u_a, u_f = step_uniforms(seeds[b], b, 0, K)
        ro = accept(zt64[b], zd[b].astype(np.float64), xs[b], T, u_a, u_f)
        n_g = int(res[b, 0])
        y_g = int(res[b, n_g + 1])
        rep.decisions += 2
        # p_i(x_i), q_i(x_i) of every draft position, from the same logits
        np.testing.assert_allclose(dbg[b, :K], ro.p_of_x, rtol=1e-4)
        np.testing.assert_allclose(dbg[b, K:2 * K], ro.q_of_x, rtol=1e-4)
        if n_g != ro.n_accepted:
            i = min(n_g, ro.n_accepted)
            dist = abs(u_a[i] - ro.p_of_x[i] / ro.q_of_x[i])
            assert dist < U_TOL, (b, n_g, ro.n_accepted, dist)
            rep.tol_flags += 1
            rep.flag_notes.append(("n", b, i, f"|u-p/q| {dist:.2e}"))
        elif y_g != ro.token:
            n = n_g
            p = softmax_t(zt64[b, n], T)
            w_ = np.maximum(p - softmax_t(zd[b, n].astype(np.float64), T), 0.0) if n < K else p
            c = np.cumsum(w_)
            dist = abs(u_f - c[min(y_g, ro.token)] / c[-1])
            assert dist < U_TOL, (b, y_g, ro.token, dist)
            rep.tol_flags += 1
            rep.flag_notes.append(("y", b, n, f"|u-F| {dist:.2e}"))
        # commit: L grows by n + 1, the accepted drafts and y are appended
        assert int(state[b, 0]) == ctxs[b] + 1 + n_g + 1
        assert list(res[b, 1:n_g + 1]) == list(xs[b, :n_g])
        toks = eng.committed_tokens(b)
        assert list(toks[ctxs[b] + 1:]) == list(xs[b, :n_g]) + [y_g]
        rep.tokens_committed += n_g + 1
    rep.steps = 1
    line = rep.record(f"8B batched acceptance B={B} K={K} V={t.vocab}")
    eng.close()
    assert rep.band_flags == 0, line


# ---------------------------------------------------------------------- draft switching
def test_draft_switching_under_budget():
    from paper_2608_10362_gb300 import Engine, MemSpecError, _lib, weights_bytes
    t = SHAPES["tiny_target"]
    d0 = SHAPES["tiny_draft"]
    d1 = dataclasses.replace(d0, n_layers=3)
    d2 = dataclasses.replace(d0, n_layers=1)
    ws = {0: gen_weights(d0, 1), 1: gen_weights(d1, 2), 2: gen_weights(d2, 3)}
    shapes = {0: d0, 1: d1, 2: d2}
    sizes = {i: weights_bytes(s) for i, s in shapes.items()}
    budget = sizes[0] + sizes[1] + 1024            # fits drafts 0 and 1, not all three
    wt = gen_weights(t, 0)
    eng = Engine(t, wt, max_batch=1, max_seq=512, max_k=4, max_drafts=3, draft_shape_max=d1,
                 draft_budget_bytes=budget, use_graphs=True)
    for i in range(3):
        eng.register_draft(i, shapes[i], ws[i])
        assert eng.query_draft(i) == 0
    eng.load_draft_async(0)
    eng.load_draft_async(1)
    with pytest.raises(MemSpecError) as ex:
        eng.load_draft_async(2)                     # over budget: refused, nothing changes
    assert ex.value.status == _lib.ERR_BUDGET
    eng.set_active_draft(0)
    assert eng.query_draft(0) == 1
    with pytest.raises(MemSpecError) as ex:
        eng.evict_draft(0)                          # the active draft is never evicted
    assert ex.value.status == _lib.ERR_BUSY
    prompt = gen_prompt(31, 100, 2048)
    eng.prefill(0, prompt, seed=4)
    to = LlamaOracle(t, wt, keep_f64=True)
    K, T = 4, 1.0
    sd = SpecDecoder(to, LlamaOracle(d0, ws[0], keep_f64=True), prompt, 400)
    rep = LockstepReport()
    step = 0
    for _ in range(3):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    # switch: evict draft 1 to make room for draft 2, load it, make it active
    eng.evict_draft(1)
    assert eng.query_draft(1) == 0
    eng.load_draft_async(2)
    eng.set_active_draft(2)                         # waits for the copy on the GPU, catches up
    assert eng.query_draft(2) == 1
    do2 = LlamaOracle(d2, ws[2], keep_f64=True)
    sd.draft = do2
    sd.dc = do2.new_cache(400)
    do2.forward(sd.dc, sd.tokens[:-1], want_logits=False)   # the new draft's catch-up
    for _ in range(3):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    # draft 0 is still resident and becomes active again: it catches up from its old length
    eng.set_active_draft(0)
    sd.draft = LlamaOracle(d0, ws[0], keep_f64=True)
    sd.dc = sd.draft.new_cache(400)
    sd.draft.forward(sd.dc, sd.tokens[:-1], want_logits=False)
    for _ in range(2):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    line = rep.record("tiny draft switching T=1.0")
    eng.close()
    assert rep.band_flags == 0, line
