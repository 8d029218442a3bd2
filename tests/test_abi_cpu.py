"""The C-ABI library on a machine without a GPU: it builds, loads, exports every
symbol the headers declare, validates arguments on the host, and its host-side
logic (blob layout, stream-K schedule, Philox) is consistent."""
import ctypes as C
import os
import re
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in ("memspec.h", "memspec_ops.h", "memspec_sched.h")]

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and
                                not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="CUDA toolkit not installed")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_10362_gb300 import build, _lib
    build.build()
    return _lib.load()


def _declared():
    names = set()
    for h in HEADERS:
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(memspec_\w+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    from paper_2608_10362_gb300 import _lib
    declared = _declared()
    assert len(declared) >= 24
    for name in declared:
        assert hasattr(lib, name), name
    assert declared == set(_lib.EXPORTS), declared ^ set(_lib.EXPORTS)


def _cfg(**kw):
    from paper_2608_10362_gb300.engine import model_cfg
    from seeded_inputs import SHAPES
    import dataclasses
    return model_cfg(dataclasses.replace(SHAPES["tiny_target"], **kw))


def test_weight_blob_layout(lib):
    from paper_2608_10362_gb300 import _lib
    from seeded_inputs import SHAPES
    for name in ("tiny_target", "draft_68m", "target_7b", "draft_1b1_tied"):
        s = SHAPES[name]
        from paper_2608_10362_gb300.engine import model_cfg
        cfg = model_cfg(s)
        total = C.c_size_t()
        assert lib.memspec_weights_bytes(C.byref(cfg), C.byref(total)) == 0
        # documented sizes: row-major bf16, or packed 16 KB tiles of 128 (pairs:
        # 64 + 64) rows x 64 columns, zero-padded
        def packed(n, k, pair=False):
            rows = 64 if pair else 128
            return -(-n // rows) * -(-k // 64) * 16384
        d, q, kv, f, v = s.d_model, s.n_heads * s.head_dim, s.n_kv_heads * s.head_dim, s.d_ffn, s.vocab
        expect = {_lib.T_TOK_EMB: v * d * 2, _lib.T_ATTN_NORM: d * 2, _lib.T_WQKV: packed(q + 2 * kv, d),
                  _lib.T_WO: packed(d, q), _lib.T_FFN_NORM: d * 2, _lib.T_WGATE: packed(f, d, True),
                  _lib.T_WUP: 0, _lib.T_WDOWN: packed(d, f), _lib.T_FINAL_NORM: d * 2,
                  _lib.T_LM_HEAD: v * d * 2 if s.tied else packed(v, d)}
        spans = []
        for t in range(10):
            layers = range(s.n_layers) if 1 <= t <= 7 else [0]
            for l in layers:
                off, nb = C.c_size_t(), C.c_size_t()
                assert lib.memspec_weights_offset(C.byref(cfg), t, l, C.byref(off), C.byref(nb)) == 0
                assert off.value % 256 == 0
                assert nb.value == expect[t], (name, t, nb.value, expect[t])
                if t == _lib.T_WUP:   # inside the gate/up pair tiles
                    g = C.c_size_t()
                    lib.memspec_weights_offset(C.byref(cfg), _lib.T_WGATE, l, C.byref(g), C.byref(nb))
                    assert g.value == off.value
                elif not (t == _lib.T_LM_HEAD and s.tied):
                    spans.append((off.value, expect[t]))
        spans.sort()
        for (o1, n1), (o2, _) in zip(spans, spans[1:]):
            assert o1 + n1 <= o2
        assert spans[-1][0] + spans[-1][1] <= total.value
        assert total.value - sum(n for _, n in spans) < 256 * len(spans)
        if s.tied:
            a, b, n = C.c_size_t(), C.c_size_t(), C.c_size_t()
            lib.memspec_weights_offset(C.byref(cfg), _lib.T_LM_HEAD, 0, C.byref(a), C.byref(n))
            lib.memspec_weights_offset(C.byref(cfg), _lib.T_TOK_EMB, 0, C.byref(b), C.byref(n))
            assert a.value == b.value


def test_host_validation_rejects_bad_arguments(lib):
    from paper_2608_10362_gb300 import _lib
    n = C.c_size_t()
    assert lib.memspec_weights_bytes(None, C.byref(n)) == _lib.ERR_INVALID_ARG
    bad = _cfg(n_kv_heads=3)
    assert lib.memspec_weights_bytes(C.byref(bad), C.byref(n)) == _lib.ERR_INVALID_ARG
    cfg = _cfg()
    off = C.c_size_t()
    assert lib.memspec_weights_offset(C.byref(cfg), 2, 99, C.byref(off), C.byref(n)) == _lib.ERR_INVALID_ARG
    assert lib.memspec_weights_offset(C.byref(cfg), 42, 0, C.byref(off), C.byref(n)) == _lib.ERR_INVALID_ARG
    assert lib.memspec_kv_bytes(C.byref(cfg), 0, 10, C.byref(n)) == _lib.ERR_INVALID_ARG
    assert lib.memspec_kv_bytes(C.byref(cfg), 2, 100, C.byref(n)) == 0
    assert n.value == 4 * 2 * 2 * 4 * 100 * 64 * 2

    p = _lib.InitParams()
    p.target = _cfg()
    p.max_batch, p.max_seq, p.max_k, p.max_drafts = 1, 256, 4, 0
    assert lib.memspec_workspace_bytes(C.byref(p), C.byref(n)) == 0 and n.value > 0
    for field, val, code in [("max_batch", 0, _lib.ERR_INVALID_ARG), ("max_k", 16, _lib.ERR_INVALID_ARG),
                             ("max_seq", 1, _lib.ERR_INVALID_ARG), ("max_drafts", 17, _lib.ERR_INVALID_ARG)]:
        q = _lib.InitParams.from_buffer_copy(p)
        setattr(q, field, val)
        assert lib.memspec_workspace_bytes(C.byref(q), C.byref(n)) == code, field
    q = _lib.InitParams.from_buffer_copy(p)
    q.max_batch, q.max_k = 32, 8                      # 32 * 9 rows > 256
    assert lib.memspec_workspace_bytes(C.byref(q), C.byref(n)) == _lib.ERR_UNSUPPORTED
    q = _lib.InitParams.from_buffer_copy(p)
    q.target = _cfg(head_dim=96, n_heads=8, n_kv_heads=8, d_model=768)
    assert lib.memspec_workspace_bytes(C.byref(q), C.byref(n)) == _lib.ERR_UNSUPPORTED
    out = C.c_void_p()
    assert lib.memspec_init(C.byref(p), None, C.byref(out)) == _lib.ERR_INVALID_ARG
    assert lib.memspec_op_linear(None, None, None, 1, 1, 8, None, 0, None, None) == _lib.ERR_INVALID_ARG
    assert lib.memspec_op_sample(None, 1, 10, C.c_float(1.0), None, None, None) == _lib.ERR_INVALID_ARG
    assert b"invalid" in lib.memspec_op_last_error()
    # a null context is rejected by every context call
    assert lib.memspec_draft_step(None, 4, C.c_float(1.0)) == _lib.ERR_INVALID_ARG
    assert lib.memspec_verify_step(None, 4) == _lib.ERR_INVALID_ARG
    assert lib.memspec_accept_commit(None, 4, C.c_float(1.0), None) == _lib.ERR_INVALID_ARG
    assert lib.memspec_load_draft_async(None, 0, None) == _lib.ERR_INVALID_ARG


HOST_PROBE = r"""
#include <cstdio>
#include "internal.h"
using namespace memspec;
int main() {
  // stream-K: ranges partition [0, T) and sk_cta_of inverts sk_begin
  for (int T = 1; T <= 700; T += (T < 64 ? 1 : 37))
    for (int G = 1; G <= T && G <= 300; G += (G < 20 ? 1 : 13)) {
      if (sk_begin(0, T, G) != 0 || sk_begin(G, T, G) != T) { printf("BAD range %d %d\n", T, G); return 1; }
      for (int c = 0; c < G; ++c) {
        if (sk_begin(c + 1, T, G) <= sk_begin(c, T, G)) { printf("BAD empty %d %d %d\n", T, G, c); return 1; }
        for (int t = sk_begin(c, T, G); t < sk_begin(c + 1, T, G); ++t)
          if (sk_cta_of(t, T, G) != c) { printf("BAD owner %d %d %d\n", T, G, t); return 1; }
      }
    }
  // device Philox, compiled for the host: (seed, req, step, slot) -> uniform
  const unsigned long long seeds[3] = {0ull, 3ull, 0x123456789abcdefull};
  for (int s = 0; s < 3; ++s)
    for (int r = 0; r < 3; ++r)
      for (int st = 0; st < 3; ++st)
        for (int k = 0; k < 9; ++k)
          printf("%llu %d %d %d %.17g\n", seeds[s], r, st * 1000, k, (double)philox_uniform(seeds[s], r, st * 1000, k));
  return 0;
}
"""


def test_host_logic_schedule_and_philox(tmp_path):
    """Stream-K partition of the GEMM tiles, and the CUDA-side Philox compiled for
    the host agreeing with the oracle's independent implementation."""
    from oracle.philox import uniform
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("no g++")
    src = tmp_path / "probe.cpp"
    src.write_text(HOST_PROBE)
    exe = tmp_path / "probe"
    csrc = os.path.join(ROOT, "paper_2608_10362_gb300", "csrc")
    res = subprocess.run([gxx, "-std=c++17", "-O1", "-I", csrc, "-I", "/usr/local/cuda/include",
                          str(src), "-o", str(exe)], capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout
    lines = out.stdout.strip().splitlines()
    assert len(lines) == 3 * 3 * 3 * 9
    for line in lines:
        s, r, st, k, u = line.split()
        assert float(u) == pytest.approx(uniform(int(s), int(r), int(st), int(k)), rel=0, abs=0)
