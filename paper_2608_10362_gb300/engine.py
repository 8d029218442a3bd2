"""Thin Python binding over the C ABI: device memory comes from PyTorch, every
step of the draft-then-verify path runs in libmemspec.so.

The binding only marshals arguments: it allocates the weight blobs, KV caches,
workspace and draft arena with torch, copies bf16 weights into the blob layout
the library reports (memspec_weights_offset), and forwards calls.
"""
from __future__ import annotations

import ctypes as C
from typing import Iterable, Mapping

import numpy as np
import torch

from . import _lib
from ._lib import MemSpecError, ModelCfg, InitParams


def model_cfg(shape) -> ModelCfg:
    """memspec_model_cfg from any object with the Llama shape attributes."""
    return ModelCfg(int(shape.n_layers), int(shape.d_model), int(shape.n_heads),
                    int(shape.n_kv_heads), int(shape.head_dim), int(shape.d_ffn),
                    int(shape.vocab), int(bool(getattr(shape, "tied", False))),
                    float(getattr(shape, "rope_base", 10000.0)),
                    float(getattr(shape, "norm_eps", 1e-5)))


def _check(lib, status: int, ctx=None):
    if status != _lib.OK:
        msg = lib.memspec_last_error(ctx).decode() if ctx is not None else \
            lib.memspec_op_last_error().decode()
        raise MemSpecError(status, msg)


def weights_bytes(shape) -> int:
    lib = _lib.load()
    cfg = model_cfg(shape)
    n = C.c_size_t()
    _check(lib, lib.memspec_weights_bytes(C.byref(cfg), C.byref(n)))
    return n.value


def tensor_offset(shape, tensor: int, layer: int = 0):
    lib = _lib.load()
    cfg = model_cfg(shape)
    off, nb = C.c_size_t(), C.c_size_t()
    _check(lib, lib.memspec_weights_offset(C.byref(cfg), tensor, layer, C.byref(off), C.byref(nb)))
    return off.value, nb.value


def kv_bytes(shape, max_batch: int, max_seq: int) -> int:
    lib = _lib.load()
    cfg = model_cfg(shape)
    n = C.c_size_t()
    _check(lib, lib.memspec_kv_bytes(C.byref(cfg), max_batch, max_seq, C.byref(n)))
    return n.value


_ROW_MAJOR = {"tok_emb": _lib.T_TOK_EMB, "attn_norm": _lib.T_ATTN_NORM,
              "ffn_norm": _lib.T_FFN_NORM, "final_norm": _lib.T_FINAL_NORM}
_PACKED = {"wo": _lib.T_WO, "w_down": _lib.T_WDOWN, "lm_head": _lib.T_LM_HEAD}


def _bf16(arr, device) -> torch.Tensor:
    t = arr if isinstance(arr, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(arr))
    return t.to(device=device, dtype=torch.bfloat16).contiguous()


def pack_matrix(src: torch.Tensor, dst: torch.Tensor, src2: torch.Tensor = None,
                stream=None) -> None:
    """Pack row-major bf16 device matrices (src [n][k], and src2 for a gate/up
    pair) into the blob's packed-tile format at dst (a uint8 device view)."""
    lib = _lib.load()
    n, k = src.shape
    s = stream.cuda_stream if stream is not None else torch.cuda.current_stream(src.device).cuda_stream
    _check(lib, lib.memspec_pack_matrix(C.c_void_p(src.data_ptr()),
                                        C.c_void_p(src2.data_ptr() if src2 is not None else 0),
                                        int(n), int(k), C.c_void_p(dst.data_ptr()), dst.numel(),
                                        C.c_void_p(s)))


def fill_blob(shape, blob: torch.Tensor, tensors: Iterable, device=None) -> None:
    """Copy (name, layer, array) weights (float32 arrays holding bf16 values, or
    bf16 torch tensors) into a uint8 blob at the library's offsets: norms and the
    embedding row-major, projection matrices packed on the GPU (memspec_pack_matrix).
    A host blob (pinned) is packed on `device` and copied back."""
    dev = blob.device if blob.device.type == "cuda" else torch.device(device or "cuda")
    pending = {}   # (layer, group) -> {name: device tensor}

    def place(tensor_id, layer, fill):
        off, nb = tensor_offset(shape, tensor_id, max(layer, 0))
        if blob.device.type == "cuda":
            fill(blob[off:off + nb])
        else:   # pack into a device buffer, then copy to the host blob
            tmp = torch.empty(nb, dtype=torch.uint8, device=dev)
            fill(tmp)
            blob[off:off + nb].copy_(tmp.cpu())

    for name, layer, arr in tensors:
        if name in _ROW_MAJOR:
            off, nb = tensor_offset(shape, _ROW_MAJOR[name], max(layer, 0))
            t = _bf16(arr, blob.device).view(-1)
            assert nb == t.numel() * 2, (name, nb, t.numel())
            blob[off:off + nb].view(torch.bfloat16).copy_(t)
        elif name in _PACKED:
            t = _bf16(arr, dev)
            place(_PACKED[name], layer, lambda view, t=t: pack_matrix(t, view))
        elif name in ("wq", "wk", "wv"):
            g = pending.setdefault((layer, "qkv"), {})
            g[name] = _bf16(arr, dev)
            if len(g) == 3:
                w = torch.cat([g["wq"], g["wk"], g["wv"]], dim=0)
                place(_lib.T_WQKV, layer, lambda view, w=w: pack_matrix(w, view))
                del pending[(layer, "qkv")]
        elif name in ("w_gate", "w_up"):
            g = pending.setdefault((layer, "ffn"), {})
            g[name] = _bf16(arr, dev)
            if len(g) == 2:
                gt, up = g["w_gate"], g["w_up"]
                place(_lib.T_WGATE, layer, lambda view, gt=gt, up=up: pack_matrix(gt, view, up))
                del pending[(layer, "ffn")]
        else:
            raise KeyError(f"unknown tensor {name}")
    if pending:
        raise ValueError(f"incomplete matrix groups: {sorted(pending)}")
    torch.cuda.synchronize(dev)


class Engine:
    """One target, a set of registered drafts, and the device memory they use."""

    def __init__(self, target_shape, target_weights, *, max_batch: int = 1, max_seq: int = 1024,
                 max_k: int = 8, max_drafts: int = 4, draft_shape_max=None,
                 draft_budget_bytes: int = 0, use_graphs: bool = True,
                 launch_mode: str = "per_op", trace=None, device: int = 0,
                 draft_kernel: str = "auto"):
        """launch_mode "per_op": one kernel launch per op of a pass; "pass": each
        draft step and verify pass as one persistent launch.  ``trace``
        ("verify", "draft" or "prefill") records per-op timestamps of that pass, see
        ``pass_trace``.  draft_kernel ("auto", "per_op", "fused") picks the kernels
        of the per-op draft step, see memspec_init_params.draft_kernel."""
        if launch_mode not in ("per_op", "pass"):
            raise ValueError(f"launch_mode must be 'per_op' or 'pass', not {launch_mode!r}")
        self.lib = _lib.load()
        self.device = torch.device("cuda", device)
        torch.cuda.set_device(self.device)
        self.shape = target_shape
        self.max_batch, self.max_seq, self.max_k = max_batch, max_seq, max_k
        self.vocab = target_shape.vocab
        self.stream = torch.cuda.Stream(self.device)
        self.side = torch.cuda.Stream(self.device, priority=0)
        self.blob = torch.empty(weights_bytes(target_shape), dtype=torch.uint8, device=self.device)
        fill_blob(target_shape, self.blob, _as_triples(target_weights))
        self.kv = torch.empty(kv_bytes(target_shape, max_batch, max_seq), dtype=torch.uint8,
                              device=self.device)
        self.arena = torch.empty(max(draft_budget_bytes, 256), dtype=torch.uint8,
                                 device=self.device)
        dmax = draft_shape_max if draft_shape_max is not None else target_shape
        p = InitParams()
        p.target = model_cfg(target_shape)
        p.target_weights_dev = self.blob.data_ptr()
        p.target_kv_dev = self.kv.data_ptr()
        p.max_batch, p.max_seq, p.max_k, p.max_drafts = max_batch, max_seq, max_k, max_drafts
        p.draft_shape_max = model_cfg(dmax)
        p.draft_arena_dev = self.arena.data_ptr()
        p.draft_budget_bytes = draft_budget_bytes
        p.stream_main = self.stream.cuda_stream
        p.stream_side = self.side.cuda_stream
        p.use_graphs = int(use_graphs)
        p.launch_mode = _lib.LAUNCH_PASS if launch_mode == "pass" else _lib.LAUNCH_PER_OP
        if trace not in (None, "verify", "draft", "prefill"):
            raise ValueError(f"trace must be None, 'verify', 'draft' or 'prefill', not {trace!r}")
        p.trace = {None: 0, "verify": 1, "draft": 2, "prefill": 3}[trace]
        kinds = {"auto": _lib.DRAFT_KERNEL_AUTO, "per_op": _lib.DRAFT_KERNEL_PER_OP,
                 "fused": _lib.DRAFT_KERNEL_FUSED}
        if draft_kernel not in kinds:
            raise ValueError(f"draft_kernel must be one of {sorted(kinds)}, not {draft_kernel!r}")
        p.draft_kernel = kinds[draft_kernel]
        self.params = p
        n = C.c_size_t()
        _check(self.lib, self.lib.memspec_workspace_bytes(C.byref(p), C.byref(n)))
        self.workspace = torch.empty(n.value + 256, dtype=torch.uint8, device=self.device)
        ws_ptr = (self.workspace.data_ptr() + 255) // 256 * 256
        torch.cuda.synchronize(self.device)
        ctx = C.c_void_p()
        _check(self.lib, self.lib.memspec_init(C.byref(p), C.c_void_p(ws_ptr), C.byref(ctx)))
        self.ctx = ctx
        self.drafts = {}
        self.results_host = torch.zeros(max_batch * (max_k + 2), dtype=torch.int32,
                                        pin_memory=True)

    # -------------------------------------------------------------- helpers
    def _call(self, fn, *args):
        st = fn(self.ctx, *args)
        if st != _lib.OK:
            raise MemSpecError(st, self.lib.memspec_last_error(self.ctx).decode())

    def close(self):
        if getattr(self, "ctx", None):
            torch.cuda.synchronize(self.device)
            self.lib.memspec_destroy(self.ctx)
            self.ctx = None

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass

    # -------------------------------------------------------------- drafts
    def register_draft(self, draft_id: int, shape, weights):
        blob = torch.empty(weights_bytes(shape), dtype=torch.uint8, pin_memory=True)
        fill_blob(shape, blob, _as_triples(weights), device=self.device)
        kv = torch.empty(kv_bytes(shape, self.max_batch, self.max_seq), dtype=torch.uint8,
                         device=self.device)
        cfg = model_cfg(shape)
        self._call(self.lib.memspec_register_draft, draft_id, C.byref(cfg), blob.data_ptr(),
                   kv.data_ptr())
        self.drafts[draft_id] = (shape, blob, kv)

    def load_draft_async(self, draft_id: int) -> int:
        off = C.c_size_t()
        self._call(self.lib.memspec_load_draft_async, draft_id, C.byref(off))
        return off.value

    def query_draft(self, draft_id: int) -> int:
        s = C.c_int32()
        self._call(self.lib.memspec_query_draft, draft_id, C.byref(s))
        return s.value

    def evict_draft(self, draft_id: int):
        self._call(self.lib.memspec_evict_draft, draft_id)

    def set_active_draft(self, draft_id: int):
        self._call(self.lib.memspec_set_active_draft, draft_id)

    # -------------------------------------------------------------- requests / steps
    def prefill(self, req: int, tokens, seed: int = 0):
        arr = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32))
        self._call(self.lib.memspec_prefill, req, arr.ctypes.data_as(C.POINTER(C.c_int32)),
                   len(arr), C.c_uint64(seed))

    def set_batch(self, batch: int):
        self._call(self.lib.memspec_set_batch, batch)

    def draft_step(self, K: int, temperature: float):
        self._call(self.lib.memspec_draft_step, K, C.c_float(temperature))

    def verify_step(self, K: int):
        self._call(self.lib.memspec_verify_step, K)

    def accept_commit(self, K: int, temperature: float, results: torch.Tensor | None = None):
        ptr = None if results is None else results.data_ptr()
        self._call(self.lib.memspec_accept_commit, K, C.c_float(temperature), ptr)

    def tree_step(self, tokens, parents, temperature: float, results: torch.Tensor | None = None):
        """One tree verification step (request 0, batch 1): node i carries
        tokens[i] and parents[i] (-1: child of the root).  With `results` (int32
        [66], pinned) the outcome {n_emit, L_before, emitted[32], rows[32]} is
        copied there; read it after sync()."""
        t = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32))
        p = np.ascontiguousarray(np.asarray(parents, dtype=np.int32))
        if t.shape != p.shape or t.ndim != 1:
            raise ValueError("tokens and parents must be 1-D of equal length")
        ptr = None if results is None else results.data_ptr()
        self._call(self.lib.memspec_tree_step, len(t), t.ctypes.data, p.ctypes.data, C.c_float(temperature), ptr)

    def sync(self, timeout_ms: int = -1) -> int:
        bits = C.c_uint32()
        st = self.lib.memspec_sync(self.ctx, timeout_ms, C.byref(bits))
        if st != _lib.OK:
            raise MemSpecError(st, self.lib.memspec_last_error(self.ctx).decode()
                               + f" (device bits 0x{bits.value:x})")
        return bits.value

    def step(self, K: int, temperature: float, results: torch.Tensor | None = None):
        self.draft_step(K, temperature)
        self.verify_step(K)
        self.accept_commit(K, temperature, results)

    # -------------------------------------------------------------- inspection
    def info(self, what: int) -> int:
        v = C.c_int64()
        self._call(self.lib.memspec_query_info, what, C.byref(v))
        return v.value

    def launches_per_step(self) -> int:
        """Kernel launches of the last draft step + verify pass + acceptance."""
        return sum(self.info(w) for w in (_lib.INFO_DRAFT_LAUNCHES, _lib.INFO_VERIFY_LAUNCHES,
                                          _lib.INFO_ACCEPT_LAUNCHES))

    def read_buffer(self, buf: int, dtype, count: int) -> np.ndarray:
        out = np.empty(count, dtype=dtype)
        self._call(self.lib.memspec_read_buffer, buf, out.ctypes.data, out.nbytes)
        return out

    def write_buffer(self, buf: int, arr: np.ndarray):
        arr = np.ascontiguousarray(arr)
        self._call(self.lib.memspec_write_buffer, buf, arr.ctypes.data, arr.nbytes)

    def seq_state(self) -> np.ndarray:
        return self.read_buffer(_lib.BUF_SEQ_STATE, np.int32, self.max_batch * 4).reshape(-1, 4)

    def committed_tokens(self, req: int = 0) -> np.ndarray:
        L = int(self.seq_state()[req, 0])
        toks = self.read_buffer(_lib.BUF_TOKENS, np.int32, self.max_batch * self.max_seq)
        return toks.reshape(self.max_batch, self.max_seq)[req, :L]

    def pass_trace(self) -> np.ndarray:
        """Timestamps (ns) of the last traced pass, [n_ops][SMs][16] =
        worker start, worker end, activation loads issued, first MMA issued,
        partials stored, arrival counted, reduction inputs loaded, reduction
        done, then epilogue-internal points (entries an op did not reach keep
        older values)."""
        head = self.read_buffer(_lib.BUF_PASS_TRACE, np.uint64, 2)
        n_ops, grid = int(head[0]), int(head[1])
        n = min(n_ops, _lib.PASS_TRACE_OPS)
        t = self.read_buffer(_lib.BUF_PASS_TRACE, np.uint64, 2 + n * grid * 16)
        return t[2:].reshape(n, grid, 16)

    def target_logits(self, batch: int, K: int) -> np.ndarray:
        n = batch * (K + 1) * self.vocab
        return self.read_buffer(_lib.BUF_TARGET_LOGITS, np.float32, n).reshape(batch, K + 1, -1)

    def draft_logits(self, batch: int, K: int) -> np.ndarray:
        n = batch * K * self.vocab
        return self.read_buffer(_lib.BUF_DRAFT_LOGITS, np.float32, n).reshape(batch, K, -1)

    def draft_tokens(self, batch: int) -> np.ndarray:
        n = batch * self.max_k
        return self.read_buffer(_lib.BUF_DRAFT_TOKENS, np.int32, n).reshape(batch, self.max_k)

    def accept_debug(self, batch: int, K: int) -> np.ndarray:
        n = batch * (2 * K + 2)
        return self.read_buffer(_lib.BUF_ACCEPT_DEBUG, np.float32, n).reshape(batch, 2 * K + 2)


def _as_triples(weights):
    """Accept {(name, layer): array} or an iterable of (name, layer, array)."""
    if isinstance(weights, Mapping):
        return [(n, l, a) for (n, l), a in weights.items()]
    return weights


# ------------------------------------------------------------------ op-level calls
def op_linear(x: torch.Tensor, w: torch.Tensor, scratch: torch.Tensor | None = None,
              stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """y = x . w^T on the weight-streaming GEMM kernel (x, w bf16 on cuda)."""
    lib = _lib.load()
    rows, k = x.shape
    n_out = w.shape[0]
    nb = C.c_size_t()
    _check(lib, lib.memspec_op_linear_scratch_bytes(rows, n_out, k, C.byref(nb)))
    if scratch is None:
        scratch = torch.zeros(nb.value + 256, dtype=torch.uint8, device=x.device)
    base = (scratch.data_ptr() + 255) // 256 * 256
    y = torch.empty(rows, n_out, dtype=torch.float32, device=x.device)
    s = stream or torch.cuda.current_stream(x.device)
    _check(lib, lib.memspec_op_linear(x.data_ptr(), w.data_ptr(), y.data_ptr(), rows, n_out, k,
                                      base, nb.value, None, s.cuda_stream))
    return y


def op_linear_noalloc(x: torch.Tensor, w: torch.Tensor, y: torch.Tensor | None = None,
                      status: torch.Tensor | None = None,
                      stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """y = x . w^T through memspec_op_linear_noalloc (no scratch argument; the
    library's fixed device array is used).  rows <= 16.  ``y`` (fp32 [rows][n_out])
    may be given so that the call itself allocates nothing; ``status`` (one
    int32/uint32 on the device) receives the kernel's error bits."""
    lib = _lib.load()
    rows, k = x.shape
    n_out = w.shape[0]
    if y is None:
        y = torch.empty(rows, n_out, dtype=torch.float32, device=x.device)
    s = stream or torch.cuda.current_stream(x.device)
    _check(lib, lib.memspec_op_linear_noalloc(x.data_ptr(), w.data_ptr(), y.data_ptr(), rows,
                                              n_out, k,
                                              None if status is None else status.data_ptr(),
                                              s.cuda_stream))
    return y


def int4_pack(qweight: torch.Tensor, scales: torch.Tensor, zeros: torch.Tensor,
              stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """Repack GPTQ-style INT4 weights (qweight uint8 [n][k/2], scales bf16
    [n][k/128], zeros uint8 [n][k/128], all on cuda) into the layout
    op_linear_int4 reads; returns the packed uint8 buffer."""
    lib = _lib.load()
    n_out, half_k = qweight.shape
    k = 2 * half_k
    nbytes = lib.memspec_int4_packed_bytes(n_out, k)
    if nbytes < 0:
        raise MemSpecError(_lib.ERR_INVALID_ARG, f"bad INT4 shape n={n_out} k={k}")
    packed = torch.empty(nbytes, dtype=torch.uint8, device=qweight.device)
    s = stream or torch.cuda.current_stream(qweight.device)
    _check(lib, lib.memspec_int4_pack(qweight.data_ptr(), scales.data_ptr(), zeros.data_ptr(), n_out, k,
                                      packed.data_ptr(), s.cuda_stream))
    return packed


def op_linear_int4(x: torch.Tensor, packed: torch.Tensor, n_out: int, y: torch.Tensor | None = None,
                   status: torch.Tensor | None = None,
                   stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """y = x . W^T (fp32 [rows][n_out]) for x bf16 [rows][k] and W packed by
    int4_pack; `status` (int32 [1] on cuda, optional) receives the kernel's
    error bits."""
    lib = _lib.load()
    rows, k = x.shape
    if y is None:
        y = torch.empty(rows, n_out, dtype=torch.float32, device=x.device)
    s = stream or torch.cuda.current_stream(x.device)
    _check(lib, lib.memspec_op_linear_int4(x.data_ptr(), packed.data_ptr(), y.data_ptr(), rows, n_out, k,
                                           None if status is None else status.data_ptr(), s.cuda_stream))
    return y


def op_sample(logits: torch.Tensor, temperature: float, u: torch.Tensor | None = None):
    lib = _lib.load()
    rows, vocab = logits.shape
    out = torch.empty(rows, dtype=torch.int32, device=logits.device)
    s = torch.cuda.current_stream(logits.device)
    _check(lib, lib.memspec_op_sample(logits.data_ptr(), rows, vocab, C.c_float(temperature),
                                      None if u is None else u.data_ptr(), out.data_ptr(),
                                      s.cuda_stream))
    return out
