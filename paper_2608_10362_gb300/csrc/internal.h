// internal.h - launch-parameter structs shared by the host runtime (api.cu) and
// the kernels.  Not part of the public ABI.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace memspec {

typedef __nv_bfloat16 bf16;

constexpr int kMaxGroups = 64;      // requests stepped together
constexpr int kMaxRows = 256;       // rows of one forward pass (MMA N <= 256)
constexpr int kPrefillChunk = 128;  // rows per prefill forward
constexpr int kMaxK = 15;           // largest draft length
constexpr int kMaxDrafts = 16;
constexpr int kStateInts = 4;       // per request: L, Lt, step, unused

// Which rows a forward pass processes.  Row r belongs to group g = r / R
// (a request), index i = r % R; it is valid iff i < valid[g]; its position is
// pos0[g] + i.  Written by the embedding kernel, read by every later kernel of
// the same forward pass.
constexpr int kTreeRows = 32;       // a tree pass: the root and up to 31 draft-tree nodes

struct RowPlan {
  int n_groups;
  int rows_per_group;  // R
  int rows_total;      // n_groups * R
  int max_pos;         // largest valid position of the pass
  int req[kMaxGroups];
  int valid[kMaxGroups];
  int pos0[kMaxGroups];
  // tree passes (one group): row r holds KV slot pos0 + r but sits at RoPE
  // position pos0 + rope_off[r] and sees, beyond pos0, only the rows of anc[r]
  int tree;
  int rope_off[kTreeRows];
  uint32_t anc[kTreeRows];   // bit j: row r sees row j (its ancestors and itself)
};

// A draft tree, written by the host before a tree step (row 0 = the root, the
// last committed token; row i + 1 = node i).
struct TreeDesc {
  int n_rows;
  int tokens[kTreeRows];       // rows >= 1: the node's token
  int parent_row[kTreeRows];   // row of the parent (0 = the root); -1 for row 0
  int rope_off[kTreeRows];     // 0 for the root, 1 + depth for a node
  uint32_t anc[kTreeRows];
};

// The walk's outcome (device), also copied back to the host.
struct TreeResult {
  int n_emit;                  // accepted nodes + the final token (0: nothing committed)
  int L_before;                // committed length before the step
  int emitted[kTreeRows];      // accepted tokens, then the final token
  int rows[kTreeRows];         // rows of the accepted nodes, in path order
};

constexpr int kTreeSlot0 = 64;   // Philox slot of the step's emitted token e: kTreeSlot0 + e

struct TreeWalkArgs {            // tree.cu: the root-down walk and the commit (request 0)
  const TreeDesc* tree;
  const int* samples;            // [n_rows]: the token drawn from each row
  int* seq_state;                // request 0: L, Lt, step
  int* tokens;                   // request 0's committed tokens [max_seq]
  int max_seq;
  TreeResult* result;
  uint32_t* status;
};

struct TreeCompactArgs {         // tree.cu: the accepted nodes' K / V moved to consecutive slots
  bf16* kv;                      // layer l: K at kv + l * 2 * layer_kv, V layer_kv further
  size_t layer_kv;               // elements of one layer's K (request-major [B][Hkv][max_seq][hd])
  int Hkv, hd, max_seq;
  const TreeResult* result;
};
cudaError_t launch_tree_walk(const TreeWalkArgs& a, cudaStream_t s);
cudaError_t launch_tree_compact(const TreeCompactArgs& a, int n_layers, cudaStream_t s);

__host__ __device__ inline bool plan_row_valid(const RowPlan* p, int r) {
  if (r >= p->rows_total) return false;
  const int g = r / p->rows_per_group;
  return (r - g * p->rows_per_group) < p->valid[g];
}

enum PlanMode : int { PLAN_VERIFY = 0, PLAN_DRAFT_FIRST = 1, PLAN_DRAFT_NEXT = 2, PLAN_PREFILL = 3, PLAN_TREE = 4 };

struct EmbedArgs {
  int mode;
  int n_groups;
  int R;
  int j;               // draft pass index (1-based) for PLAN_DRAFT_NEXT
  int prefill_req, prefill_start, prefill_count;
  const int* seq_state;     // [max_batch][kStateInts]
  const int* draft_len;     // [max_batch] processed count of the model being run (drafts)
  const int* tokens;        // [max_batch][max_seq]
  int max_seq;
  const int* draft_tokens;  // [max_batch][max_k]
  int max_k;
  const bf16* emb;          // [vocab][d]
  int d, vocab;
  float* h;                 // [rows][d] residual stream
  bf16* xg;                 // [rows][d] bf16(h * gain) for the first projection
  bf16* xg_lo;              // its low-order plane
  const bf16* gain;         // first RMSNorm gain
  float* ss;                // [ss_tiles][ss_stride]: row sums of squares (partial)
  int ss_stride;
  RowPlan* plan;
  const TreeDesc* tree;     // PLAN_TREE: the tree of this pass
  uint32_t* status;
};

enum GemmEpi : int { EPI_F32 = 0, EPI_RESIDUAL = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };
enum L2Hint : int { L2_EVICT_FIRST = 0, L2_EVICT_NORMAL = 1, L2_EVICT_LAST = 2 };

struct GemmArgs {
  CUtensorMap map_a;        // weights [n_out][k] bf16, box {64, 128} (or {64, 64} for pairs)
  CUtensorMap map_a2;       // second matrix of a SwiGLU pair (up), box {64, 64}
  const uint8_t* a_packed;  // non-null: weights as packed 16 KB tiles in stream-K order
                            // (tile t at a_packed + t * 16384; map_a, map_a2 unused)
  CUtensorMap map_b;        // activations [rows_total][k] bf16, box {64, n_pad}
  CUtensorMap map_b2;       // low-order plane of the activations (split), same shape
  int split;                // 1: activations = hi + lo bf16 planes, two MMAs per k-step
  int n_out;                // output features (F for pairs)
  int k_in;
  int pair;                 // 1: tile = 64 rows of map_a + 64 rows of map_a2
  int rows_total;           // rows of B (activations)
  int n_pad;                // MMA N: rows_total rounded up to 16
  int row_tiles, k_tiles, stages;
  int l2_hint;
  // RMSNorm folded into the epilogue: B = bf16(h * gain) was written by the
  // previous epilogue; y[r] *= rsqrt(sum_i ss[i][r] / k_in + eps)
  int rms;
  const float* ss;          // [ss_count][ss_stride]
  int ss_count, ss_stride;
  float eps;
  // split-K scratch
  float* partials;          // [2 * grid][n_pad * 128]
  int* counters;            // [row_tiles], zero on entry, left zero
  int split_epi;            // 1: contributors to a split row tile only store their partials;
                            // gemm_split_epi_kernel (the next launch) sums them and runs the
                            // epilogue, one CTA per (row tile, 16-row chunk)
  int csk;                  // > 1: launched in clusters of csk CTAs (n_pad == 16 only); a
                            // row tile whose contributors share a cluster is summed by
                            // its first contributor from partials the others push into
                            // its shared memory (no global partials, no counter)
  // epilogue
  int epi;
  float* out;               // EPI_F32
  int out_ld;
  int last_only;            // EPI_F32: only the last valid row of each group
  long long out_group_stride;
  float* h;                 // EPI_RESIDUAL: residual [rows][h_ld], updated in place
  int h_ld;
  float* ss_out;            // EPI_RESIDUAL: [row_tiles][ss_stride]
  const bf16* gain_next;    // EPI_RESIDUAL: gain of the next RMSNorm (nullptr: no xg)
  bf16* xg_out;             // EPI_RESIDUAL: bf16(h_new * gain_next) [rows][h_ld]
  bf16* xg_lo_out;          // EPI_RESIDUAL: low-order plane (nullptr: none)
  bf16* act;                // EPI_SWIGLU: [rows][act_ld]
  bf16* act_lo;             // EPI_SWIGLU: low-order plane (nullptr: none)
  int act_ld;
  float* q_out;             // EPI_QKV: fp32 [rows][q_dim]
  int q_dim, kv_dim, head_dim, n_kv_heads, max_seq;
  bf16* kcache;             // [req][kv_head][max_seq][hd] for this layer
  bf16* vcache;
  const float* rope_cos;    // [max_seq][hd/2]
  const float* rope_sin;
  const RowPlan* plan;      // nullptr: rows < rows_total are valid, no positions
  uint32_t* status;
  unsigned long long* trace;  // nullptr, or this op's trace row (16 slots per CTA)
  int trace_ctas;           // split epilogue kernel: CTAs (linear index) that record
  int warm;                 // 1: dry run of the tail before griddepcontrol.wait
  int ctx_early;            // 1: every kernel before the previous one has completed when
                            // this one starts (an earlier launch of the pass had a full
                            // dependency after the row-plan writer), so the row plan
                            // may be read before griddepcontrol.wait
};

struct AttnArgs {
  CUtensorMap kmap;         // tma: this layer's K cache as [max_batch * Hkv * max_seq][hd] bf16,
  CUtensorMap vmap;         //   box {64, 64}, 128-byte swizzle; V likewise
  int tma;                  // 1: K/V tiles by cp.async.bulk.tensor into mbarrier stages
  const float* q;           // [rows][H][hd] fp32, rotated
  const bf16* kcache;       // [req][Hkv][max_seq][hd]
  const bf16* vcache;
  int H, Hkv, hd, max_seq;
  int rows_per_block;       // query rows (positions) per CTA
  int row_blocks;           // blocks per group
  int chunk;                // keys per split at max_seq (the kernel spreads the actual
                            // context over n_splits, in whole 64-key tiles)
  int n_splits;             // gridDim.x
  float scale_log2;         // log2(e) / sqrt(hd)
  float* part_o;            // [groups][Hkv][row_blocks][n_splits][qmax][hd]
  float* part_ml;           // [groups][Hkv][row_blocks][n_splits][qmax][2]
  int qmax;                 // group_size * rows_per_block
  int* counters;            // [groups][Hkv][row_blocks]
  bf16* out;                // [rows][H][hd]
  bf16* out_lo;             // low-order plane of out
  const RowPlan* plan;
  uint32_t* status;
  unsigned long long* trace;  // nullptr, or this op's trace row (16 slots per CTA)
  int trace_ctas;             // CTAs (linear index) that record
  int ctx_early;              // 1: as GemmArgs::ctx_early; the row plan and the cached
                              // keys / values of positions before this pass's first
                              // new position may be read before griddepcontrol.wait
};

struct SampleArgs {         // draft sampling of pass j
  const float* logits;      // [groups][row_stride] (row for this pass)
  long long row_stride;
  int vocab;
  int n_groups;
  float inv_temp;           // 0: greedy
  int greedy;
  int slot;                 // Philox slot (j-1)
  const int* seq_state;     // for Philox step; nullptr for explicit uniforms
  const unsigned long long* seeds;
  const float* u_explicit;  // [groups] (op-level entry)
  const int* row_slots;     // tree steps: group g is row g of request 0, Philox slot row_slots[g]
  int* out_tok;             // [groups] at stride out_stride
  int out_stride;
  float* part;              // [groups][chunks][4] scratch
  int* counters;            // [groups]
  int chunks;               // CTAs per group (gridDim.x)
  uint32_t* status;
};

struct AcceptArgs {
  const float* zt;          // [groups][K+1][vocab]
  const float* zd;          // [groups][K][vocab]
  const int* draft_tokens;  // [groups][max_k]
  int max_k;
  int K, vocab, n_groups;
  float inv_temp;
  int greedy;
  int chunks;               // CTAs per row
  float* part;              // [groups][2K+1][chunks][4]
  int* counters;            // [groups]
  int* seq_state;           // [max_batch][kStateInts]
  const unsigned long long* seeds;
  int* draft_len;           // [max_batch] Ld of the active draft
  int* tokens;              // [max_batch][max_seq]
  int max_seq;
  int* results;             // [groups][K+2]
  float* debug;             // [groups][2K+2]
  uint32_t* status;
};

// Fused draft step (draft_fused.cu): all K forward passes of a small draft and
// their samples in one cooperative launch, one CTA per SM, grid-wide barriers
// between the ops of a pass.  Rows: at most 2 per request (catch-up) and at most
// kDfMaxGroups requests.
constexpr int kDfMaxGroups = 4;
constexpr int kDfMaxSplits = 12;   // key splits per head of the fused draft attention
constexpr int kDfMaxRows = 2 * kDfMaxGroups;
constexpr int kDfSlotBytes = 16384;     // weight ring slot
constexpr int kDfMaxSlots = 16;
constexpr int kDfComputeWarps = 8;
constexpr int kDfThreads = (kDfComputeWarps + 1) * 32;   // + one copy-issuing warp
constexpr int kDfMaxLayers = 32;
constexpr int kDfMapsPerDraft = kDfMaxLayers * 4 + 1;

struct DraftFusedArgs {
  const CUtensorMap* maps;   // device: per layer {QKV, O, gate/up, down} boxes over the packed
                             // tiles, then the LM head (kDfMaxLayers * 4 + 1 at most)
  const uint8_t* w;          // draft weight blob
  // tensor offsets in the blob; per-layer tensors at off + layer * lstride
  long long off_emb, off_attn_norm, off_wqkv, off_wo, off_ffn_norm, off_wgate, off_wdown,
      off_final_norm, off_lm, lstride;
  int tied;                  // LM head = row-major embedding
  int n_layers, d, H, Hkv, hd, F, V;
  float eps;
  bf16* kv;                  // draft KV cache [layer][K|V][req][kv_head][pos][hd]
  long long layer_kv;        // elements of one layer's K (or V) block
  int max_seq, max_k;
  const float* rope_cos;     // [max_seq][hd/2]
  const float* rope_sin;
  int K, B;                  // passes, requests
  float inv_temp;            // 1/T (0: greedy)
  int greedy;
  const int* seq_state;      // [max_batch][kStateInts]
  const int* draft_len;      // [max_batch] processed count of this draft
  const int* tokens;         // [max_batch][max_seq]
  int* draft_tokens;         // [max_batch][max_k]
  const unsigned long long* seeds;
  float* zd;                 // draft logits [B][K][V]
  // scratch
  float* h;                  // residual stream [kDfMaxRows][d]
  float* qb;                 // rotated queries [kDfMaxRows][H * hd]
  float* att;                // attention partials [kDfMaxRows][H][n_splits][hd + 4]
  float* act;                // SwiGLU output [kDfMaxRows][F]
  float* lm_part;            // per-CTA LM-head statistics [B][grid][4]
  unsigned int* bar;         // [0] barrier arrivals, [1] exits, [2] abort flag
  uint32_t* status;
  int n_splits;              // attention key splits per (request, head)
  int ring_slots;            // weight ring slots of kDfSlotBytes
  int act_floats;            // activation buffer (floats) per row in shared memory (rows: 2B)
  unsigned long long* trace; // optional: {phases, grid, [phase][grid][16] globaltimer ns}: slot 0
                             // phase start, 1 barrier arrival, 13 barrier passed
  int trace_phases;          // phases the trace holds
};
size_t draft_fused_smem_bytes(int ring_slots, int act_rows, int act_floats);
size_t draft_fused_static_smem();
constexpr int kDfScratchFloatsHost = 2 * 256 + 2 * 128 + 8 * 2 * 128;   // == kDfScratchFloats
cudaError_t draft_fused_set_max_smem();
cudaError_t launch_draft_fused(const DraftFusedArgs& a, int grid, cudaStream_t s, bool cooperative);

// Group-wise INT4 weight-only linear layer (int4.cu): y = x (q - z) s^T over a
// repacked weight copy of one 1072-byte record per (16-row tile, 128-column group).
constexpr int kInt4MaxRows = 16;
constexpr int kInt4RecordBytes = 1072;
constexpr int kInt4MaxSmem = 220 * 1024;
struct Int4Args {
  const bf16* x;            // [rows][k] bf16
  const uint8_t* packed;    // records, tile-major
  float* y;                 // [rows][n]
  int rows, n, k;
  int tiles_per_cta;        // whole 16-row tiles per CTA
  uint32_t* status;         // optional device word: bit 0 = a copy wait ran out
};
size_t int4_packed_bytes(long long n, int k);
int int4_pick_depth(int rows, int k);   // cp.async ring slots per warp; 0: does not fit
cudaError_t int4_set_max_smem();
struct Int4Plan {
  int depth;           // record slots per warp (0: does not fit)
  int tiles_per_cta;
  int grid;
};
Int4Plan int4_plan(int rows, int n, int k, int sms);
cudaError_t launch_int4_linear(const Int4Args& a, const Int4Plan& p, cudaStream_t s);
cudaError_t launch_int4_pack(const uint8_t* qweight, const bf16* scales, const uint8_t* zeros, uint8_t* out,
                             int n, int k, cudaStream_t s);

// launchers (each returns the launch's cudaError_t)
cudaError_t launch_embed(const EmbedArgs& a, int rows, cudaStream_t s, bool pdl);
cudaError_t launch_gemm(const GemmArgs& a, int grid, size_t smem, cudaStream_t s, bool pdl);
size_t gemm_smem_bytes(int n_pad, int stages, int planes = 1, int csk = 0);
int gemm_pick_stages(int n_pad, int planes = 1, int csk = 0);
// Thread-block clusters of `csk` CTAs of the GEMM kernel with epilogue `epi` and
// `smem` bytes of dynamic shared memory that can be resident at once (0: none).
int gemm_max_active_clusters(int epi, int csk, size_t smem);
cudaError_t gemm_set_max_smem();
cudaError_t launch_gemm_split_epi(const GemmArgs& a, int gemm_grid, cudaStream_t s, bool pdl);
cudaError_t launch_attention(const AttnArgs& a, int n_groups, cudaStream_t s, bool pdl);
size_t attention_smem_bytes(const AttnArgs& a);
cudaError_t attention_set_max_smem();
cudaError_t launch_sample(const SampleArgs& a, cudaStream_t s, bool pdl);
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s, bool pdl);
cudaError_t launch_rope_table(float* cos_t, float* sin_t, int max_seq, int half, float base,
                              cudaStream_t s);

// x ~= hi + lo with hi = bf16(x), lo = bf16(x - hi): two bf16 planes carry about
// 16 significant bits, so bf16 tensor-core products see (almost) fp32 inputs.
// x = hi + lo in two bf16 planes.  The references must be registers or shared
// memory: with global references the compiler re-read hi from memory (a round
// trip per call, measured); use store_split_bf16 for global outputs.
__device__ __forceinline__ void split_bf16(float x, bf16& hi, bf16& lo) {
  const bf16 h = __float2bfloat16_rn(x);
  hi = h;
  lo = __float2bfloat16_rn(x - __bfloat162float(h));
}
// Store x as bf16 at hi_p and (lo_p != nullptr) its low-order part at lo_p.
__device__ __forceinline__ void store_split_bf16(bf16* hi_p, bf16* lo_p, float x) {
  const bf16 h = __float2bfloat16_rn(x);
  *hi_p = h;
  if (lo_p != nullptr) *lo_p = __float2bfloat16_rn(x - __bfloat162float(h));
}

// Message returned by memspec_op_last_error() on this host thread.
void set_op_error(const char* msg);
inline void set_op_error(const std::string& msg) { set_op_error(msg.c_str()); }

// Philox4x32-10 (Salmon et al., SC'11), device side.
__host__ __device__ inline uint32_t philox_u01_bits(uint32_t c0, uint32_t c1, uint32_t c2,
                                                    uint32_t c3, uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u, W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += W0;
      k1 += W1;
    }
    const uint64_t p0 = static_cast<uint64_t>(M0) * c0;
    const uint64_t p1 = static_cast<uint64_t>(M1) * c2;
    const uint32_t hi0 = static_cast<uint32_t>(p0 >> 32), lo0 = static_cast<uint32_t>(p0);
    const uint32_t hi1 = static_cast<uint32_t>(p1 >> 32), lo1 = static_cast<uint32_t>(p1);
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return c0;
}

// Uniform for (seed, request, step, slot): odd multiple of 2^-24 in (0, 1).
__host__ __device__ inline float philox_uniform(unsigned long long seed, int req, int step,
                                                int slot) {
  const uint32_t w = philox_u01_bits(static_cast<uint32_t>(req), static_cast<uint32_t>(step), 0u,
                                     static_cast<uint32_t>(slot),
                                     static_cast<uint32_t>(seed & 0xFFFFFFFFull),
                                     static_cast<uint32_t>(seed >> 32));
  return static_cast<float>(2u * (w >> 9) + 1u) * (1.0f / 16777216.0f);
}

// Stream-K schedule: CTA c of G processes global tiles [begin(c), begin(c+1)).
// Packed weight tiles: a [n][k] matrix as tiles of 128 rows x 64 columns, tile
// (rt, kt) = 16384 contiguous bytes at (rt * ceil(k/64) + kt) * 16384; row r of a
// tile at byte 128 r, its 16-byte column chunk c at chunk position c ^ (r % 8)
// (the 128-byte-swizzled K-major image the tensor cores read); zero beyond n, k.
// Pairs (gate/up): tile rows 0..63 from the first matrix, 64..127 from the second.
constexpr int kPackTileBytes = 16384;
inline size_t packed_bytes(long long n, long long k, bool pair) {
  const long long rt = pair ? (n + 63) / 64 : (n + 127) / 128;
  return static_cast<size_t>(rt * ((k + 63) / 64)) * kPackTileBytes;
}
cudaError_t launch_pack(const bf16* src, const bf16* src2, int n, int k, uint8_t* dst,
                        cudaStream_t s);

// 32-bit arithmetic: the host guarantees (T + 1) * (G + 1) < 2^32 for every GEMM
// (sk_fits).
inline bool sk_fits(long long T, int G) { return (T + 1) * (G + 1) < (1LL << 32); }
__host__ __device__ inline int sk_begin(int c, int T, int G) {
  return static_cast<int>((static_cast<unsigned>(c) * static_cast<unsigned>(T)) /
                          static_cast<unsigned>(G));
}
// The CTA whose range contains tile t.
__host__ __device__ inline int sk_cta_of(int t, int T, int G) {
  return static_cast<int>(((static_cast<unsigned>(t) + 1u) * static_cast<unsigned>(G) +
                           static_cast<unsigned>(T) - 1u) /
                          static_cast<unsigned>(T)) -
         1;
}

}  // namespace memspec
