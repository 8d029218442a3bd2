"""Oracle for the draft-then-verify step of speculative decoding (MemSpec).

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, float64 CPU
restatement of what the GPU path computes.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline`` /
``--impl reference`` legs may import it.  The CUDA library never calls it and
shares no code with it; both sides receive the same seeded inputs from
``seeded_inputs`` and nothing else.

What it restates, and where it comes from:

* ``philox``  - Philox4x32-10 counter-based uniforms (Salmon, Moraes, Dror,
  Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11, Section 5).
* ``llama``   - the Llama-style decoder used as target and draft (MemSpec
  Section 4.1 evaluates LLaMA-2-7B / Qwen2.5-7B targets with small drafts):
  RMSNorm, rotary position embedding, causal grouped-query attention over a
  KV cache that holds bf16 values (the workload's KV precision), SwiGLU
  feed-forward, LM head.
* ``int4`` - the group-wise INT4 weight-only linear layer of the paper's GPTQ
  INT4 targets (Section 4.1): w = (q - z) s per group of inputs, y = x W^T.
* ``scheduler`` - MemSpec's draft cache update and runtime loop (Sections
  3.3-3.4, Algorithms 2-3) and the MAB-Async baseline (Sections 2.3, 4.1).
* ``tree`` - verification of a draft tree in one target pass and the walk that
  accepts a path of it, as in the engine MemSpec is built on (Section 3.5,
  "System Implementation"); pinned against a tree-masked attention pass
  (torch SDPA), chi-square draws from the target and E[accepted] in closed
  form (tests/test_oracle_tree.py).
* ``speculative`` - the draft-and-verify iteration that MemSpec runs unchanged
  (Section 3.5: "the standard draft-and-verify process"; Section 2.1, Eq. 1:
  throughput ~ E[A] / L_iter), with the acceptance rule of the speculative
  sampling papers it cites (Leviathan, Kalman, Matias, ICML 2023, Algorithm 1;
  Chen et al. 2023, Algorithm 2): accept draft token x with probability
  min(1, p(x)/q(x)), otherwise resample from norm(max(0, p - q)); when every
  draft token is accepted, draw one more token from the target.

Pins (tests/test_oracle_*.py, run with ``-m "not gpu"``): Philox known-answer
vectors; bf16 rounding of the KV cache against hand-worked ties and PyTorch's
conversion; attention / RMSNorm / SiLU against PyTorch library routines; RoPE
closed forms; KV-cached decoding equals full recomputation; causality;
greedy speculative output equals greedy target-only output; a draft equal to
the target accepts every token; emitted tokens follow the target
distribution (chi-square, 1e5 trials at vocab 64); acceptance rate equals
sum_x min(p, q) and E[tokens/iteration] = (1 - a^(K+1)) / (1 - a).
"""
