/*
 * memspec.h - C ABI of the GB300 (sm_103a) draft-then-verify step.
 *
 * The library implements the data-parallel hot path of speculative decoding
 * as MemSpec runs it (arxiv 2608.10362, Section 3.5: "the standard
 * draft-and-verify process"; throughput ~ E[A] / L_iter, Section 2.1 Eq. 1):
 *
 *   memspec_draft_step    the draft model's K autoregressive M=1 proposals
 *   memspec_verify_step   one target pass over the K+1 positions
 *                         [last committed token, x_1..x_K] against its KV cache
 *   memspec_tree_step     (alternative to the three calls above) one target
 *                         pass over a caller-built draft tree, the
 *                         root-down acceptance walk and the commit
 *   memspec_accept_commit speculative-sampling acceptance (accept x_i with
 *                         probability min(1, p_i(x_i)/q_i(x_i)), else resample
 *                         from norm(max(0, p - q)); bonus token when all K are
 *                         accepted; Leviathan et al. ICML'23 Alg. 1, cited by
 *                         the paper in Section 1) and KV commit / rollback
 *   memspec_load_draft_async  side-stream load of a non-resident draft's
 *                         weights into the device draft arena (Section 3.3,
 *                         Algorithm 2: "asynchronously prefetch d"; Section 3.5:
 *                         prefetching overlapped with decoding)
 *
 * The scheduling policy of MemSpec (Algorithms 1-3: prediction, cache update,
 * best-resident selection) is host-side control logic that sits ABOVE this
 * ABI and calls it.
 *
 * Conventions for every call:
 *  - Device memory is owned by the caller (weights, KV caches, workspace, draft
 *    arena).  The library borrows pointers and never frees them.
 *  - Pointers named *_dev are device pointers; *_host are host pointers
 *    (pinned where stated).  Streams are cudaStream_t passed as void*.
 *  - Step calls only enqueue work on the main stream and return; results are
 *    ready after memspec_sync() or a caller-side stream synchronisation.
 *  - Every call returns a memspec_status; nothing throws across the ABI.
 *    On error, memspec_last_error() describes the first failure of the call.
 *    Arguments are validated before any work is enqueued: a call that returns
 *    MEMSPEC_ERR_INVALID_ARG has enqueued nothing.
 *  - Device-side errors (a bounded wait that ran out, an out-of-range token)
 *    set a status word that memspec_sync() returns as
 *    MEMSPEC_ERR_DEVICE_STATUS.  Kernels never trap.
 *  - One context per host thread.
 */
#ifndef MEMSPEC_H_
#define MEMSPEC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum memspec_status {
  MEMSPEC_OK = 0,
  MEMSPEC_ERR_INVALID_ARG = 1,
  MEMSPEC_ERR_CUDA = 2,
  MEMSPEC_ERR_BUDGET = 3,        /* draft does not fit the arena without evicting the active draft */
  MEMSPEC_ERR_NOT_RESIDENT = 4,  /* draft named by a step is not loaded */
  MEMSPEC_ERR_BUSY = 5,          /* draft is loading / in use */
  MEMSPEC_ERR_TIMEOUT = 6,       /* host-side wait ran out */
  MEMSPEC_ERR_DEVICE_STATUS = 7, /* a kernel reported an error in the device status word */
  MEMSPEC_ERR_UNSUPPORTED = 8    /* shape outside what the kernels implement */
} memspec_status;

/* Device status word bits (memspec_sync / memspec_device_status). */
#define MEMSPEC_DEV_TIMEOUT    0x1u  /* a bounded in-kernel wait gave up */
#define MEMSPEC_DEV_BAD_TOKEN  0x2u  /* a token id outside [0, vocab) was fed */
#define MEMSPEC_DEV_BAD_LENGTH 0x4u  /* sequence would exceed max_seq / draft not caught up */

/* Llama-style decoder hyper-parameters (RMSNorm, RoPE on pairs (i, i+hd/2),
 * grouped-query attention, SwiGLU).  Constraints checked by memspec_init /
 * memspec_register_draft: head_dim in {64, 128}; n_heads % n_kv_heads == 0;
 * n_heads*head_dim and n_kv_heads*head_dim multiples of 128; d_model a
 * multiple of 128; d_ffn a multiple of 8; vocab >= 2. */
typedef struct memspec_model_cfg {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t d_ffn;
  int32_t vocab;
  int32_t tied_embeddings;  /* 1: LM head reuses the token embedding */
  float rope_base;          /* theta_i = rope_base^(-2i/head_dim) */
  float norm_eps;           /* RMSNorm epsilon */
} memspec_model_cfg;

/* ---- weight blob layout ------------------------------------------------
 * A model's weights live in ONE contiguous blob (device memory for the
 * target, pinned host memory for drafts that get loaded into the arena), every
 * tensor 256-byte aligned inside it:
 *   TOK_EMB [vocab][d] bf16 row-major; ATTN_NORM, FFN_NORM, FINAL_NORM [d] bf16;
 *   projection matrices in PACKED TILES (below): per layer WQKV (n = (H + 2 Hkv)
 *   hd rows: q, then k, then v; k = d), WO (n = d, k = H hd), WGATE (the gate/up
 *   pair, n = F, k = d; WUP reports 0 bytes at WGATE's offset), WDOWN (n = d,
 *   k = F); LM_HEAD (n = vocab, k = d; absent if tied: the LM head then reads
 *   TOK_EMB).  Linear weights are [out][in], i.e. y = x W^T.
 * Packed tiles: the [n][k] matrix is cut into tiles of 128 rows x 64 columns;
 * tile (rt, kt) is 16384 contiguous bytes at (rt * ceil(k/64) + kt) * 16384;
 * row r of a tile starts at byte 128 r and its 16-byte column chunk c (columns
 * 64 kt + 8c .. + 7) is stored at chunk position c ^ (r % 8); entries beyond n
 * or k are zero.  For the gate/up pair a tile's rows 0..63 are gate rows
 * 64 rt .. 64 rt + 63 and rows 64..127 the same rows of up (ceil(F/64) row
 * tiles).  This is the shared-memory image the tensor cores read, in the order
 * the GEMM streams it, so weights move by 1-D bulk copies of whole tiles.
 * memspec_pack_matrix writes a packed tensor from row-major device arrays. */
typedef enum memspec_tensor {
  MEMSPEC_T_TOK_EMB = 0,
  MEMSPEC_T_ATTN_NORM = 1,
  MEMSPEC_T_WQKV = 2,
  MEMSPEC_T_WO = 3,
  MEMSPEC_T_FFN_NORM = 4,
  MEMSPEC_T_WGATE = 5,
  MEMSPEC_T_WUP = 6,
  MEMSPEC_T_WDOWN = 7,
  MEMSPEC_T_FINAL_NORM = 8,
  MEMSPEC_T_LM_HEAD = 9
} memspec_tensor;

/* Total blob bytes for cfg.  The blob layout is this library's (the paper
 * prescribes none).  Errors: INVALID_ARG (null / bad cfg). */
memspec_status memspec_weights_bytes(const memspec_model_cfg* cfg, size_t* bytes);

/* Byte offset and size of one tensor inside the blob.  layer is ignored for
 * the non-layer tensors.  LM_HEAD of a tied model reports TOK_EMB's offset.
 * Errors: INVALID_ARG (bad tensor id / layer). */
memspec_status memspec_weights_offset(const memspec_model_cfg* cfg, int32_t tensor,
                                      int32_t layer, size_t* offset, size_t* bytes);

/* Pack row-major bf16 src [n][k] (device) into packed tiles at dst (device,
 * dst_bytes >= ceil(n/128) * ceil(k/64) * 16384); with src2 non-NULL, src and
 * src2 are the gate and up matrices of a pair (dst_bytes >= ceil(n/64) *
 * ceil(k/64) * 16384).  k a positive multiple of 8; all pointers 16-byte
 * aligned.  Enqueued on `stream` (cudaStream_t).  Errors (message in
 * memspec_op_last_error): INVALID_ARG, CUDA. */
memspec_status memspec_pack_matrix(const void* src_dev, const void* src2_dev, int32_t n,
                                   int32_t k, void* dst_dev, size_t dst_bytes, void* stream);

/* Bytes of one model's KV cache: n_layers * 2 * max_batch * n_kv_heads *
 * max_seq * head_dim bf16, layout [layer][K|V][request][kv_head][pos][hd]. */
memspec_status memspec_kv_bytes(const memspec_model_cfg* cfg, int32_t max_batch,
                                int32_t max_seq, size_t* bytes);

/* ---- context --------------------------------------------------------------*/
typedef struct memspec_ctx memspec_ctx;

typedef struct memspec_init_params {
  memspec_model_cfg target;
  const void* target_weights_dev;   /* blob, memspec_weights_bytes(target) bytes */
  void* target_kv_dev;              /* memspec_kv_bytes(target, max_batch, max_seq) */
  int32_t max_batch;                /* requests verified together (1..64) */
  int32_t max_seq;                  /* prefix + generated tokens per request */
  int32_t max_k;                    /* largest draft length K (1..15) */
  int32_t max_drafts;               /* draft ids 0..max_drafts-1 (<= 16) */
  memspec_model_cfg draft_shape_max;/* largest draft shape that will be registered
                                       (sizes the activation workspace) */
  void* draft_arena_dev;            /* device arena for resident draft weights */
  size_t draft_budget_bytes;        /* arena size = the enforced draft budget */
  void* stream_main;                /* cudaStream_t for all step calls */
  void* stream_side;                /* cudaStream_t for draft loads (may equal main) */
  int32_t use_graphs;               /* 1: capture each step once and replay it */
  int32_t launch_mode;              /* MEMSPEC_LAUNCH_PER_OP (0): one kernel launch per
                                       op of a pass; MEMSPEC_LAUNCH_PASS (1): each draft
                                       step and verify pass as one persistent launch */
  int32_t trace;                    /* per-op timestamps (MEMSPEC_BUF_PASS_TRACE) of
                                       1: verify passes, 2: draft steps, 3: prefill
                                       chunks (the last one); 0: off */
  int32_t draft_kernel;             /* draft step with launch_mode PER_OP:
                                       MEMSPEC_DRAFT_KERNEL_AUTO (0): the fused draft
                                       kernel when the draft and batch fit it (below),
                                       else per-op kernels; PER_OP (1): always per-op
                                       kernels; FUSED (2): the fused kernel, init or the
                                       draft step fails with UNSUPPORTED if it cannot */
} memspec_init_params;

enum { MEMSPEC_LAUNCH_PER_OP = 0, MEMSPEC_LAUNCH_PASS = 1 };
enum { MEMSPEC_DRAFT_KERNEL_AUTO = 0, MEMSPEC_DRAFT_KERNEL_PER_OP = 1, MEMSPEC_DRAFT_KERNEL_FUSED = 2 };

/* Device workspace bytes memspec_init needs for these params (all device memory
 * is the caller's; the paper has no counterpart).  Errors: INVALID_ARG,
 * UNSUPPORTED. */
memspec_status memspec_workspace_bytes(const memspec_init_params* p, size_t* bytes);

/* Create a context: the target model is loaded once and stays resident
 * (Section 3.4, Algorithm 3: "load target model" before the runtime loop).
 * workspace_dev: device memory of memspec_workspace_bytes
 * bytes, 256-byte aligned, caller-owned, untouched by the caller afterwards.
 * Builds TMA descriptors for the target weights.  Errors: INVALID_ARG,
 * UNSUPPORTED (shape), CUDA. */
memspec_status memspec_init(const memspec_init_params* p, void* workspace_dev,
                            memspec_ctx** out);

/* Release host-side resources (graphs, events).  Does not free caller memory.
 * (Library lifetime; no counterpart in the paper.) */
void memspec_destroy(memspec_ctx* ctx);

/* Message describing the last error of this context (never NULL; no counterpart
 * in the paper). */
const char* memspec_last_error(const memspec_ctx* ctx);

/* ---- drafts (Section 3.3: candidate set D, resident set G under a budget) --*/

/* Register draft draft_id of the candidate set D (Section 3.1) with its weights
 * in pinned host memory - the backing storage tier of Section 3.3 - and its own
 * device KV cache (memspec_kv_bytes(cfg, max_batch, max_seq)).  The host blob must stay valid while the draft is registered.
 * Errors: INVALID_ARG, UNSUPPORTED, BUSY (id already registered). */
memspec_status memspec_register_draft(memspec_ctx* ctx, int32_t draft_id,
                                      const memspec_model_cfg* cfg,
                                      const void* weights_host_pinned,
                                      void* kv_dev);

/* Start copying draft_id's weights into the arena on the side stream
 * (non-blocking): Algorithm 2's "asynchronously prefetch d" (Section 3.3), the
 * load overlapped with decoding (Section 3.5).  Places the draft first-fit in the arena.  If it does not
 * fit, returns MEMSPEC_ERR_BUDGET and changes nothing: the caller chooses what
 * to evict (the active draft is never evicted implicitly).  Already resident
 * or loading: returns OK.  *slot_offset (optional) receives the arena offset. */
memspec_status memspec_load_draft_async(memspec_ctx* ctx, int32_t draft_id,
                                        size_t* slot_offset);

/* *state: 0 = not resident, 1 = resident, 2 = loading (copy in flight): the
 * residency state and prefetch status each draft keeps (Section 3.5).
 * Errors: INVALID_ARG (unregistered id), CUDA. */
memspec_status memspec_query_draft(memspec_ctx* ctx, int32_t draft_id, int32_t* state);

/* Drop draft_id from the arena: Algorithm 2's "evict d_evict" (Section 3.3),
 * which never evicts the active draft d_i.  Refuses (BUSY) while its copy is in
 * flight or while it is the active draft (the draft of the last draft step that has
 * not been followed by memspec_set_active_draft to another draft). */
memspec_status memspec_evict_draft(memspec_ctx* ctx, int32_t draft_id);

/* Make draft_id the active draft d_i of the next interval (Section 3.4,
 * Algorithm 3: the best resident draft is selected at each scheduling point).
 * draft_id = -1 leaves no draft active (then any draft may be evicted and draft
 * steps return NOT_RESIDENT until a draft is made active again).
 * It must be resident or loading (a loading
 * draft makes the next draft step wait on the GPU, never on the host).  The
 * new draft's KV cache is brought up to date with the committed tokens by a
 * chunked prefill on the main stream (host-synchronising: it reads the
 * committed lengths). */
memspec_status memspec_set_active_draft(memspec_ctx* ctx, int32_t draft_id);

/* ---- requests ----------------------------------------------------------- */

/* Start request req with prompt tokens_host[0..n) (n >= 1) and Philox seed (the
 * prompt that precedes the runtime loop of Algorithm 3; its prefill is excluded
 * from steady-state throughput, Section 4.1):
 * copies the prompt, runs the target and the active draft over all prompt
 * tokens but the last (chunks of up to 128 rows), and resets the request's
 * iteration counter.  Host-synchronising.  Errors: INVALID_ARG, CUDA. */
memspec_status memspec_prefill(memspec_ctx* ctx, int32_t req, const int32_t* tokens_host,
                               int32_t n, uint64_t seed);

/* Number of requests stepped together by the step calls (1..max_batch). All
 * of them must have been prefilled.  (Batching is this library's; the paper
 * evaluates batch 1.)  Errors: INVALID_ARG. */
memspec_status memspec_set_batch(memspec_ctx* ctx, int32_t batch);

/* ---- the draft-then-verify step ----------------------------------------- */

/* Algorithm 3 "run draft d_i" (Section 3.4) - the draft half of the standard
 * draft-and-verify iteration (Section 2.1, Eq. 1; Section 3.5).
 * The active draft proposes x_1..x_K for every request: K forward passes of
 * one position each (two for the first pass after a fully accepted step),
 * each followed by sampling x_j ~ softmax(z/T) with Philox uniform slot j-1
 * (T == 0: argmax).  Draft logits are kept for acceptance.  Enqueue only. */
memspec_status memspec_draft_step(memspec_ctx* ctx, int32_t K, float temperature);

/* Algorithm 3 "verify with target model" (Section 3.4; Section 2.1).
 * One target pass over [t_{L-1}, x_1..x_K] at positions L-1..L-1+K per request,
 * appending their K,V to the target cache and writing fp32 logits for
 * positions L..L+K.  Enqueue only. */
memspec_status memspec_verify_step(memspec_ctx* ctx, int32_t K);

/* The accept step of the draft-and-verify iteration (Section 3.5; the
 * speculative sampling rule the paper cites in Section 1), which yields the
 * accepted count A of Eq. 1.
 * Acceptance, resampling and commit for every request (see the file header):
 * n accepted tokens, the correction/bonus token y, L += n + 1, KV rollback by
 * length (target KV valid below L-1; draft KV below L-1, or L-2 when n = K).
 * If results_host_pinned is not NULL, an async copy of int32
 * [batch][K+2] = {n, x_1..x_n, y, unused...} to it is enqueued.  Enqueue only. */
memspec_status memspec_accept_commit(memspec_ctx* ctx, int32_t K, float temperature,
                                     int32_t* results_host_pinned);

/* Tree verification step, as in the speculative-decoding engine MemSpec is
 * built on (Section 3.5, "System Implementation"; that engine verifies draft
 * trees, the paper's own runs use a chain).  Request 0, batch 1.
 * The caller's tree: node i has token tokens_host[i] and parent
 * parents_host[i] (-1: a child of the root, the last committed token t_{L-1};
 * else a smaller node index); 1 <= n_nodes <= 31.  One target pass scores the
 * root and every node: the root at position L-1, node i at L + depth(i) (depth
 * 0 below the root), each row attending to the committed prefix, its
 * ancestors and itself; the nodes' K,V go to the scratch slots L..L-1+n_nodes.
 * Then a token is drawn from each row's softmax(z/T) (Philox slot 64 + e for
 * the step's e-th emitted token; T == 0: argmax), and the walk descends from
 * the root while the drawn token is a child's token (lowest index among equal
 * siblings); the first drawn token that is no child is the step's final
 * token.  Commit: the accepted tokens and the final token (L += accepted + 1),
 * the accepted nodes' K,V moved to consecutive positions after the root.
 * The drafts' caches are not advanced (a following memspec_draft_step catches
 * up at most two tokens; more is reported as device status 0x4).
 * If results_host is not NULL, an async copy of int32 [66] =
 * {n_emit, L_before, emitted[32], accepted_rows[32]} (rows: node index + 1;
 * n_emit = accepted + 1, or 0 if the sequence would pass max_seq) is enqueued.
 * Needs batch 1.  Errors: INVALID_ARG (tree, tokens, T), UNSUPPORTED (batch),
 * CUDA.  Enqueue only. */
memspec_status memspec_tree_step(memspec_ctx* ctx, int32_t n_nodes, const int32_t* tokens_host,
                                 const int32_t* parents_host, float temperature, int32_t* results_host);

/* Host synchronisation (no counterpart in the paper).
 * Wait for the main stream (timeout_ms < 0: no limit) and return the device
 * status word as MEMSPEC_ERR_DEVICE_STATUS if any bit is set (the word is then
 * cleared; *bits, if given, receives it).  Errors: TIMEOUT, CUDA. */
memspec_status memspec_sync(memspec_ctx* ctx, int32_t timeout_ms, uint32_t* bits);

/* ---- inspection (tests, tooling) ----------------------------------------- */
typedef enum memspec_buffer {
  MEMSPEC_BUF_TARGET_LOGITS = 0, /* fp32 [batch][K+1][vocab] of the last verify */
  MEMSPEC_BUF_DRAFT_LOGITS = 1,  /* fp32 [batch][K][vocab] of the last draft step */
  MEMSPEC_BUF_DRAFT_TOKENS = 2,  /* int32 [batch][max_k] */
  MEMSPEC_BUF_TOKENS = 3,        /* int32 [max_batch][max_seq] committed tokens */
  MEMSPEC_BUF_SEQ_STATE = 4,     /* int32 [max_batch][4] = {L, Lt, step, active Ld} */
  MEMSPEC_BUF_ACCEPT_DEBUG = 5,  /* fp32 [batch][2K+2] = {p_i(x_i), q_i(x_i), residual mass, u'} */
  MEMSPEC_BUF_RESIDUAL = 6,      /* fp32 residual stream [rows][d] of the last forward */
  MEMSPEC_BUF_PASS_TRACE = 7,    /* u64 trace of the last traced pass (init param trace):
                                    {n_ops, grid, then [n_ops][grid][16] globaltimer ns =
                                    worker start, worker end, activation loads issued,
                                    first MMA issued, partials stored, arrival counted,
                                    reduction inputs loaded, reduction done, then
                                    epilogue-internal points}; 2048 ops at most */
  MEMSPEC_BUF_SEEDS = 8,         /* u64 [max_batch] Philox keys of the requests (set by prefill) */
  MEMSPEC_BUF_TREE_LOGITS = 9    /* fp32 [32][vocab] rows of the last tree step (row 0 = the root) */
} memspec_buffer;

/* Facts about the last step calls (host-side, no wait).  what:
 *   MEMSPEC_INFO_DRAFT_LAUNCHES  kernel launches of the last draft step
 *   MEMSPEC_INFO_VERIFY_LAUNCHES kernel launches of the last verify pass
 *   MEMSPEC_INFO_ACCEPT_LAUNCHES kernel launches of the last acceptance
 *   MEMSPEC_INFO_DRAFT_FUSED     1 if the last draft step ran the fused draft kernel
 * Errors: INVALID_ARG (unknown id). */
enum { MEMSPEC_INFO_DRAFT_LAUNCHES = 0, MEMSPEC_INFO_VERIFY_LAUNCHES = 1,
       MEMSPEC_INFO_ACCEPT_LAUNCHES = 2, MEMSPEC_INFO_DRAFT_FUSED = 3 };
memspec_status memspec_query_info(memspec_ctx* ctx, int32_t what, int64_t* value);

/* Synchronously copy `bytes` of an internal buffer to host memory (waits for
 * the main stream first).  Errors: INVALID_ARG (bytes too large), CUDA. */
memspec_status memspec_read_buffer(memspec_ctx* ctx, int32_t buffer, void* dst_host,
                                   size_t bytes);

#ifdef __cplusplus
}
#endif
#endif /* MEMSPEC_H_ */
