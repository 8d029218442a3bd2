/*
 * memspec_ops.h - op-level entry points of the same library (libmemspec.so).
 *
 * These expose single kernels of the draft-then-verify step so that each can
 * be checked and timed on its own.  Same conventions as memspec.h: device
 * pointers are caller-owned, work is enqueued on the given stream, arguments
 * are validated before anything is enqueued.
 */
#ifndef MEMSPEC_OPS_H_
#define MEMSPEC_OPS_H_

#include "memspec.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Scratch bytes that memspec_op_linear needs for (rows, n_out, k): split-K
 * partial sums and per-row-tile arrival counters. */
memspec_status memspec_op_linear_scratch_bytes(int32_t rows, int32_t n_out, int32_t k,
                                               size_t* bytes);

/* y[rows][n_out] (fp32) = x[rows][k] (bf16, row-major) . w[n_out][k]^T (bf16).
 * This is the weight-streaming GEMM every projection of the verify and draft
 * passes runs (Q/K/V, O, gate/up, down, LM head): TMA-staged weight tiles,
 * tcgen05 MMA into TMEM, stream-K over all SMs, deterministic split-K
 * reduction (above 16 rows, split row tiles are finished by a second launch
 * on the same stream, one CTA per row tile and 16-row chunk).
 * rows in 1..256, k a multiple of 8, n_out >= 1, and
 * ceil(n_out/128) * ceil(k/64) * (SMs + 1) below 2^32.
 * scratch_dev: memspec_op_linear_scratch_bytes bytes, 256-byte aligned; its
 * counters must be zero on entry and are left zero on exit (zero it once).
 * status_dev: uint32 device word, bits set on in-kernel errors (may be NULL).
 * x, w: 16-byte aligned.  Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
memspec_status memspec_op_linear(const void* x_dev, const void* w_dev, float* y_dev,
                                 int32_t rows, int32_t n_out, int32_t k,
                                 void* scratch_dev, size_t scratch_bytes,
                                 uint32_t* status_dev, void* stream);

/* The same GEMM as memspec_op_linear (y = x . w^T, fp32 out), for callers
 * that cannot allocate device memory: plug-ins whose host application owns all
 * device memory, fixed-budget deployments that allocate only at start-up, and
 * latency-critical loops that cannot afford cudaMalloc / cudaFree (which may
 * synchronise the device).  The paper has no counterpart; this is a property
 * of the library's interface.
 * Instead of a scratch argument it uses one file-scope device array of about
 * 2.6 MB that every GPU loading the library keeps until the process exits.
 * Limits: rows in 1..16, n_out in 1..131072, k a positive multiple of 8 up to
 * 2^20; x and w 16-byte aligned.  Larger sizes return MEMSPEC_ERR_INVALID_ARG
 * (message in memspec_op_last_error) and enqueue nothing.  The call allocates
 * nothing; it enqueues a clear of the array's counters and the kernel on
 * `stream`.  Its split-K grid differs from memspec_op_linear's, so results
 * agree with it within rounding, not bit for bit.
 * All calls share the array: calls that overlap on the GPU (other streams,
 * other host threads) race - serialise them.  The first call on a device looks
 * up the array's address on that device; make it before any stream capture.
 * status_dev: optional uint32 device word for in-kernel error bits (NULL: an
 * internal word that the caller cannot read is used). */
memspec_status memspec_op_linear_noalloc(const void* x_dev, const void* w_dev, float* y_dev,
                                         int32_t rows, int32_t n_out, int32_t k,
                                         uint32_t* status_dev, void* stream);

/* Group-wise INT4 weight-only linear layer (the paper's targets are GPTQ INT4
 * models, Section 4.1).  The weights W[n_out][k] are given GPTQ-style,
 *   W[r][c] = (q[r][c] - zeros[r][c/128]) * scales[r][c/128],
 *   qweight: uint8 [n_out][k/2], byte j of row r = q[r][2j] | q[r][2j+1] << 4
 *   scales:  bf16  [n_out][k/128];   zeros: uint8 [n_out][k/128], values 0..15
 * and are repacked once, by memspec_int4_pack, into the kernel's layout (one
 * 1072-byte record per 16-row tile and 128-column group, codes regrouped
 * within each 32-bit word; rows past n_out are zero-filled).  The layout is private to this library: only
 * memspec_op_linear_int4 reads it.
 *
 * memspec_int4_packed_bytes: bytes of the packed copy, or -1 for bad sizes
 * (n_out >= 1, k a positive multiple of 128). */
int64_t memspec_int4_packed_bytes(int32_t n_out, int32_t k);

/* Repack on `stream` (device pointers; qweight 4-byte, scales 2-byte, packed
 * 16-byte aligned; packed holds memspec_int4_packed_bytes).  The caller owns
 * every buffer; nothing is allocated.  Errors: INVALID_ARG (n_out outside
 * 1..1048576, k not a positive multiple of 128, NULL, misalignment), CUDA. */
memspec_status memspec_int4_pack(const void* qweight_dev, const void* scales_dev, const void* zeros_dev,
                                 int32_t n_out, int32_t k, void* packed_dev, void* stream);

/* y[rows][n_out] (fp32) = x[rows][k] (bf16, row-major) . W^T, enqueued on
 * `stream`.  rows in 1..16; x and packed 16-byte aligned, y 4-byte aligned;
 * the activations (rows (2k + 64) bytes) plus a ring of at least two
 * 1072-byte records per warp (16 warps) must fit in 220 KB of shared memory
 * (else UNSUPPORTED: e.g. rows 9..16 at k = 11008).  Results are
 * deterministic.  status_dev: optional uint32 device word; bit 0 is set if a
 * wait for a bulk copy ran out (about a second; y is then incomplete).
 * Allocates nothing and keeps no state between calls.
 * Errors: INVALID_ARG (sizes, NULL, misalignment), UNSUPPORTED, CUDA. */
memspec_status memspec_op_linear_int4(const void* x_dev, const void* packed_dev, float* y_dev, int32_t rows,
                                      int32_t n_out, int32_t k, uint32_t* status_dev, void* stream);

/* Categorical sampling of each row of logits[rows][vocab] (fp32): with T > 0,
 * out[r] = smallest j with sum_{i<=j} exp(z_i/T - m) > u[r] * sum_i exp(z_i/T - m);
 * with T == 0, out[r] = argmax (lowest id on ties).  u_dev: fp32 [rows] in
 * (0,1) (ignored for T == 0).  This is the draft-token sampler of
 * memspec_draft_step. */
memspec_status memspec_op_sample(const float* logits_dev, int32_t rows, int32_t vocab,
                                 float temperature, const float* u_dev, int32_t* out_dev,
                                 void* stream);

/* Message describing the last failed op-level call (or memspec_init) on this
 * host thread; never NULL. */
const char* memspec_op_last_error(void);

/* Overwrite an internal buffer of ctx (same ids as memspec_read_buffer) from
 * host memory; synchronous.  Lets tests feed the acceptance step synthetic
 * logits and set sequence state.  Writable: TARGET_LOGITS, DRAFT_LOGITS,
 * DRAFT_TOKENS, TOKENS, SEQ_STATE, SEEDS. */
memspec_status memspec_write_buffer(memspec_ctx* ctx, int32_t buffer, const void* src_host,
                                    size_t bytes);

#ifdef __cplusplus
}
#endif
#endif /* MEMSPEC_OPS_H_ */
