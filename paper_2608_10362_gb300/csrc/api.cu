// api.cu - host runtime behind the C ABI of include/memspec.h and memspec_ops.h.
//
// Responsibilities: validate arguments, carve the caller's workspace, encode TMA
// descriptors for every weight matrix, enqueue the forward passes of the
// draft-then-verify step (optionally captured once as CUDA graphs and
// replayed), manage the draft arena (first-fit placement under the byte budget,
// side-stream copies fenced by events), and report errors as status codes.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <ctime>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/memspec.h"
#include "../../include/memspec_ops.h"
#include "internal.h"
#include "pass.h"

using namespace memspec;

namespace {

thread_local std::string g_op_error;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2D bf16 tensor map over a row-major [rows][cols] matrix, box {64 cols, box_rows},
// 128-byte swizzle, zero fill out of bounds.
bool encode_map(CUtensorMap* map, const void* base, int rows, int cols, int box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (fn == nullptr) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) != 0 || (cols * 2) % 16 != 0) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D bf16 tensor map, no swizzle (the bytes are copied as stored), zero fill
// out of bounds: dims {d0, d1, d2} elements, strides of dims 1 and 2 in bytes,
// box {b0, b1, b2}.
bool encode_box3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                  uint64_t s1, uint64_t s2, uint32_t b0, uint32_t b1, uint32_t b2) {
  EncodeTiledFn fn = get_encode_fn();
  if (fn == nullptr || (reinterpret_cast<uintptr_t>(base) & 15) != 0 || s1 % 16 || s2 % 16) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
int round_up(int x, int m) { return (x + m - 1) / m * m; }
int ceil_div(int a, int b) { return (a + b - 1) / b; }

int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

std::string g_attr_error;

bool ensure_func_attrs() {
  static bool done = false;
  if (done) return true;
  cudaError_t e = gemm_set_max_smem();
  if (e != cudaSuccess) {
    g_attr_error = std::string("gemm smem attribute: ") + cudaGetErrorString(e);
    return false;
  }
  e = attention_set_max_smem();
  if (e != cudaSuccess) {
    g_attr_error = std::string("attention smem attribute: ") + cudaGetErrorString(e);
    return false;
  }
  e = pass_set_max_smem();
  if (e != cudaSuccess) {
    g_attr_error = std::string("pass kernel smem attribute: ") + cudaGetErrorString(e);
    return false;
  }
  e = draft_fused_set_max_smem();
  if (e != cudaSuccess) {
    g_attr_error = std::string("fused draft kernel smem attribute: ") + cudaGetErrorString(e);
    return false;
  }
  e = int4_set_max_smem();
  if (e != cudaSuccess) {
    g_attr_error = std::string("int4 kernel smem attribute: ") + cudaGetErrorString(e);
    return false;
  }
  done = true;
  return true;
}

// ---------------------------------------------------------------- blob layout
struct Layout {
  size_t emb, final_norm, lm_head, total;
  std::vector<size_t> attn_norm, wqkv, wo, ffn_norm, wgate, wup, wdown;
};

bool cfg_valid(const memspec_model_cfg* c, std::string* why) {
  if (c == nullptr) {
    *why = "null model cfg";
    return false;
  }
  if (c->n_layers < 1 || c->d_model < 128 || c->n_heads < 1 || c->n_kv_heads < 1 ||
      c->head_dim < 1 || c->d_ffn < 8 || c->vocab < 2) {
    *why = "model cfg: a dimension is out of range";
    return false;
  }
  if (c->n_heads % c->n_kv_heads != 0) {
    *why = "model cfg: n_heads must be a multiple of n_kv_heads";
    return false;
  }
  if (!(c->rope_base > 0.f) || !(c->norm_eps >= 0.f)) {
    *why = "model cfg: rope_base must be > 0 and norm_eps >= 0";
    return false;
  }
  return true;
}

memspec_status cfg_supported(const memspec_model_cfg* c, std::string* why) {
  if (c->head_dim != 64 && c->head_dim != 128) {
    *why = "head_dim must be 64 or 128";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  if (c->d_model % 128 || (c->n_heads * c->head_dim) % 128 || (c->n_kv_heads * c->head_dim) % 128) {
    *why = "d_model, n_heads*head_dim and n_kv_heads*head_dim must be multiples of 128";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  if (c->d_ffn % 8) {
    *why = "d_ffn must be a multiple of 8";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  if (c->vocab > 131072) {
    *why = "vocab must be <= 131072";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  return MEMSPEC_OK;
}

Layout make_layout(const memspec_model_cfg& c) {
  Layout L;
  const size_t d = c.d_model, q = static_cast<size_t>(c.n_heads) * c.head_dim,
               kv = static_cast<size_t>(c.n_kv_heads) * c.head_dim, f = c.d_ffn, v = c.vocab;
  size_t off = 0;
  auto take = [&](size_t elems) {   // row-major bf16
    const size_t o = off;
    off = align256(off + elems * 2);
    return o;
  };
  auto take_packed = [&](size_t n, size_t k, bool pair) {
    const size_t o = off;
    off = align256(off + packed_bytes(static_cast<long long>(n), static_cast<long long>(k), pair));
    return o;
  };
  L.emb = take(v * d);
  for (int l = 0; l < c.n_layers; ++l) {
    L.attn_norm.push_back(take(d));
    L.wqkv.push_back(take_packed(q + 2 * kv, d, false));
    L.wo.push_back(take_packed(d, q, false));
    L.ffn_norm.push_back(take(d));
    L.wgate.push_back(take_packed(f, d, true));   // gate/up pair tiles
    L.wup.push_back(L.wgate.back());
    L.wdown.push_back(take_packed(d, f, false));
  }
  L.final_norm = take(d);
  L.lm_head = c.tied_embeddings ? L.emb : take_packed(v, d, false);
  L.total = off;
  return L;
}

size_t kv_bytes(const memspec_model_cfg& c, int max_batch, int max_seq) {
  return static_cast<size_t>(c.n_layers) * 2 * max_batch * c.n_kv_heads * max_seq * c.head_dim * 2;
}

// ---------------------------------------------------------------- attention launch geometry
struct AttnGeo {
  int rows_per_block, row_blocks, n_splits, chunk, qmax;
};

AttnGeo attn_geometry(const memspec_model_cfg& c, int groups, int R, int max_seq) {
  AttnGeo g;
  const int gs = c.n_heads / c.n_kv_heads;
  // query vectors per CTA: at most 64 (4 m-tiles of 16); decode-sized GQA passes
  // (2..8 query heads per KV head, at most 64 vectors in all) take row blocks of
  // at most 8 vectors for the transposed form - every warp busy, three CTAs per
  // SM; the blocks of a head re-read its keys, mostly from L2 (batched 8B verify,
  // 36 vectors per head: 11.0 -> 9.8 ms)
  const int qlimit = (gs >= 2 && gs <= 8 && gs * R <= 64) ? 8 : 64;
  int rpb = std::max(1, qlimit / gs);
  rpb = std::min(rpb, R);
  g.rows_per_block = rpb;
  g.row_blocks = ceil_div(R, rpb);
  g.qmax = gs * rpb;
  const int units = groups * c.n_kv_heads * g.row_blocks;
  const int max_splits = ceil_div(max_seq, 64);
  // one wave of CTAs: the transposed form (at most 8 query vectors per CTA, 2
  // stages) fits three per SM, the 16-row form (3 stages) two (an extra partial
  // wave would double the time); at most 16 splits (the combine fetches 16
  // splits' outputs per round trip)
  const bool tq = g.qmax <= 8;
  const int per_sm = tq ? 3 : 2;
  int want = std::max(1, std::min(16, (per_sm * sm_count()) / units));
  want = std::min(want, max_splits);
  g.chunk = round_up(ceil_div(max_seq, want), 64);
  g.n_splits = ceil_div(max_seq, g.chunk);
  // the combine keeps (2 n_splits + 1) x qmax floats of split statistics in the
  // CTA's shared memory (stages x 64 keys x hd x 2 x 2 bytes, last 16 bytes reserved)
  const size_t smem = static_cast<size_t>(tq ? 2 : 3) * 2 * 64 * c.head_dim * 2 - 16;
  while (static_cast<size_t>(2 * g.n_splits + 1) * g.qmax * 4 > smem) {
    g.chunk *= 2;
    g.n_splits = ceil_div(max_seq, g.chunk);
  }
  return g;
}

size_t attn_part_floats(const memspec_model_cfg& c, const AttnGeo& g, int groups) {
  const size_t units = static_cast<size_t>(groups) * c.n_kv_heads * g.row_blocks;
  return units * g.n_splits * g.qmax * c.head_dim;
}
size_t attn_units(const memspec_model_cfg& c, const AttnGeo& g, int groups) {
  return static_cast<size_t>(groups) * c.n_kv_heads * g.row_blocks;
}

// ---------------------------------------------------------------- models
struct ModelRT {
  memspec_model_cfg cfg{};
  Layout lay;
  const uint8_t* w = nullptr;  // device blob
  bf16* kv = nullptr;
  CUtensorMap m_lm{};   // tied LM head: the row-major embedding
  int l2_hint = L2_EVICT_FIRST;
  bool ready = false;
};

bool build_maps(ModelRT& m, std::string* why) {
  const memspec_model_cfg& c = m.cfg;
  const int d = c.d_model, q = c.n_heads * c.head_dim, kv = c.n_kv_heads * c.head_dim,
            f = c.d_ffn;
  (void)q;
  (void)kv;
  (void)f;
  // projection weights are packed tiles (bulk copies, no tensor map); only a
  // tied LM head reads the row-major embedding through a tensor map
  bool ok = true;
  if (c.tied_embeddings) ok = encode_map(&m.m_lm, m.w + m.lay.lm_head, c.vocab, d, 128);
  if (!ok) *why = "cuTensorMapEncodeTiled failed (driver entry point or alignment)";
  m.ready = ok;
  return ok;
}

struct DraftRec {
  bool registered = false;
  memspec_model_cfg cfg{};
  const void* host_blob = nullptr;
  size_t bytes = 0;
  int state = 0;  // 0 not resident, 1 resident, 2 loading
  size_t arena_off = 0;
  cudaEvent_t ev = nullptr;
  ModelRT rt;
  int* d_len = nullptr;  // device [max_batch]
  // TMA boxes of the fused draft kernel (host copy, and the weights they were built for)
  std::vector<CUtensorMap> df_maps;
  const uint8_t* df_maps_for = nullptr;
};

struct GraphKey {
  int kind, draft, K;
  uint32_t tbits;
  int batch;
  bool operator<(const GraphKey& o) const {
    return std::tie(kind, draft, K, tbits, batch) < std::tie(o.kind, o.draft, o.K, o.tbits, o.batch);
  }
};

}  // namespace

struct memspec_ctx {
  memspec_init_params p{};
  bool pdl = true;   // programmatic dependent launch between the kernels of a pass
  cudaStream_t main = nullptr, side = nullptr;
  std::string err;
  // workspace
  float* h = nullptr;
  bf16* xg = nullptr;
  bf16* xg_lo = nullptr;   // low-order planes of the bf16 activations
  bf16* o_lo = nullptr;
  bf16* act_lo = nullptr;
  float* ss = nullptr;
  int ss_stride = kMaxRows;
  float* q = nullptr;
  bf16* o = nullptr;
  bf16* act = nullptr;
  float* gemm_part = nullptr;
  int* gemm_cnt = nullptr;
  size_t gemm_cnt_bytes = 0;
  float* att_po = nullptr;
  float* att_pml = nullptr;
  int* att_cnt = nullptr;
  size_t att_po_cap = 0, att_cnt_cap = 0;
  float* zt = nullptr;
  float* zd = nullptr;
  int* tokens = nullptr;
  int* state = nullptr;
  int* draft_tokens = nullptr;
  int* d_len_all = nullptr;
  unsigned long long* seeds = nullptr;
  RowPlan* plan = nullptr;
  uint32_t* status = nullptr;
  int* results = nullptr;
  float* acc_part = nullptr;
  float* acc_dbg = nullptr;
  int* acc_cnt = nullptr;
  int* smp_cnt = nullptr;
  TreeDesc* tree_desc = nullptr;            // tree steps: the tree, its rows' draws,
  int* tree_samples = nullptr;              // the walk's outcome and the rows' logits
  TreeResult* tree_result = nullptr;
  float* tree_z = nullptr;
  float* rope_cos[2] = {nullptr, nullptr};  // hd 64, hd 128
  float* rope_sin[2] = {nullptr, nullptr};
  size_t ws_bytes = 0;
  int max_rows = 0;
  int vocab = 0;
  // models
  ModelRT target;
  DraftRec drafts[kMaxDrafts];
  int active = -1;
  int batch = 1;
  int last_K = 0;
  std::map<GraphKey, cudaGraphExec_t> graphs;
  std::map<GraphKey, int> graph_launches;   // kernel launches inside each captured graph
  int last_launches[3] = {0, 0, 0};         // of the last draft step, verify pass, acceptance
  bool last_draft_fused = false;            // the last draft step ran the fused kernel
  // op tables of the pass kernel (workspace areas, bump-allocated per graph)
  uint8_t* op_area = nullptr;
  size_t op_area_bytes = 0, op_area_used = 0;
  int* done_area = nullptr;
  size_t done_area_ints = 0, done_area_used = 0;
  bool pass_kernel = false;  // draft / verify passes as one persistent launch
  bool cooperative = false;
  unsigned long long* trace = nullptr;   // per-op trace (init param trace = 1: verify, 2: draft)
  // fused draft step scratch
  float* df_att = nullptr;
  size_t df_att_floats = 0;
  float* df_lm = nullptr;
  unsigned int* df_bar = nullptr;
  CUtensorMap* df_maps = nullptr;   // [kMaxDrafts][kDfMapsPerDraft], 64-byte aligned
  bool df_coop = true;       // cooperative launch attribute (cleared if capture refuses it)
  std::map<std::tuple<const void*, int, int, int>, CUtensorMap> bmaps;
};

namespace {

memspec_status fail(memspec_ctx* c, memspec_status s, const std::string& why) {
  if (c) c->err = why;
  return s;
}
memspec_status cuda_fail(memspec_ctx* c, cudaError_t e, const char* where) {
  std::string m = std::string(where) + ": " + cudaGetErrorString(e);
  if (c) c->err = m;
  return MEMSPEC_ERR_CUDA;
}

struct WsPlan {
  size_t off = 0;
  size_t take(size_t bytes) {
    const size_t o = off;
    off = align256(off + bytes);
    return o;
  }
};

int model_q(const memspec_model_cfg& c) { return c.n_heads * c.head_dim; }
int model_kv(const memspec_model_cfg& c) { return c.n_kv_heads * c.head_dim; }

// Computes (and optionally binds) the workspace layout.
size_t layout_workspace(const memspec_init_params* p, memspec_ctx* c, uint8_t* base) {
  const memspec_model_cfg& t = p->target;
  const memspec_model_cfg& dm = p->draft_shape_max;
  const bool has_draft = p->max_drafts > 0;
  auto mx = [&](int a, int b) { return has_draft ? std::max(a, b) : a; };
  const int dmax = mx(t.d_model, dm.d_model);
  const int qmax_dim = mx(model_q(t), model_q(dm));
  const int fmax = mx(t.d_ffn, dm.d_ffn);
  const int B = p->max_batch, K = p->max_k;
  const int rows = std::max({B * (K + 1), kPrefillChunk, 2 * B});
  const int V = t.vocab;
  const int nsm = sm_count();
  // attention partial sizing: max over the passes this context runs
  size_t po = 0, cnt = 0;
  auto acc_att = [&](const memspec_model_cfg& m, int groups, int R) {
    AttnGeo g = attn_geometry(m, groups, R, p->max_seq);
    po = std::max(po, attn_part_floats(m, g, groups));
    cnt = std::max(cnt, attn_units(m, g, groups));
  };
  acc_att(t, B, K + 1);
  acc_att(t, 1, kPrefillChunk);
  if (has_draft) {
    acc_att(dm, B, 2);
    acc_att(dm, B, 1);
    acc_att(dm, 1, kPrefillChunk);
  }
  const int max_rt = std::max({ceil_div(V, 128), ceil_div(fmax, 64),
                               ceil_div(model_q(t) + 2 * model_kv(t), 128),
                               has_draft ? ceil_div(model_q(dm) + 2 * model_kv(dm), 128) : 1,
                               ceil_div(dmax, 128)});
  WsPlan w;
  const size_t o_h = w.take(static_cast<size_t>(kMaxRows) * dmax * 4);
  const size_t o_xg = w.take(static_cast<size_t>(kMaxRows) * dmax * 2);
  const size_t o_xgl = w.take(static_cast<size_t>(kMaxRows) * dmax * 2);
  const size_t o_ss = w.take(static_cast<size_t>(ceil_div(dmax, 128)) * kMaxRows * 4);
  const size_t o_q = w.take(static_cast<size_t>(kMaxRows) * qmax_dim * 4);
  const size_t o_o = w.take(static_cast<size_t>(kMaxRows) * qmax_dim * 2);
  const size_t o_ol = w.take(static_cast<size_t>(kMaxRows) * qmax_dim * 2);
  const size_t o_act = w.take(static_cast<size_t>(kMaxRows) * fmax * 2);
  const size_t o_actl = w.take(static_cast<size_t>(kMaxRows) * fmax * 2);
  const size_t o_gp = w.take(static_cast<size_t>(2) * nsm * kMaxRows * 128 * 4);
  const size_t o_gc = w.take(static_cast<size_t>(max_rt) * 4);   // split-K arrival counters
  const size_t o_apo = w.take(po * 4);
  const size_t o_apml = w.take(po / 64 * 2 * 4 + 1024);
  const size_t o_acnt = w.take(cnt * 4);
  const size_t o_zt = w.take(static_cast<size_t>(B) * (K + 1) * V * 4);
  const size_t o_zd = w.take(static_cast<size_t>(B) * K * V * 4);
  const size_t o_tok = w.take(static_cast<size_t>(B) * p->max_seq * 4);
  const size_t o_st = w.take(static_cast<size_t>(B) * kStateInts * 4);
  const size_t o_dt = w.take(static_cast<size_t>(B) * K * 4);
  const size_t o_dl = w.take(static_cast<size_t>(std::max(1, p->max_drafts)) * B * 4);
  const size_t o_seed = w.take(static_cast<size_t>(B) * 8);
  const size_t o_plan = w.take(sizeof(RowPlan));
  const size_t o_status = w.take(4);
  const size_t o_res = w.take(static_cast<size_t>(B) * (K + 2) * 4);
  const size_t o_ap = w.take(static_cast<size_t>(B) * (2 * K + 1) * 4 * 4);
  const size_t o_ad = w.take(static_cast<size_t>(B) * (2 * K + 2) * 4);
  const size_t o_ac = w.take(static_cast<size_t>(B) * 4);
  const size_t o_sc = w.take(static_cast<size_t>(B) * 4);
  const size_t o_td = w.take(sizeof(TreeDesc));
  const size_t o_ts = w.take(static_cast<size_t>(kTreeRows) * 4);
  const size_t o_tr = w.take(sizeof(TreeResult));
  const size_t o_tz = w.take(static_cast<size_t>(kTreeRows) * V * 4);
  const size_t o_rc64 = w.take(static_cast<size_t>(p->max_seq) * 32 * 4);
  const size_t o_rs64 = w.take(static_cast<size_t>(p->max_seq) * 32 * 4);
  const size_t o_rc128 = w.take(static_cast<size_t>(p->max_seq) * 64 * 4);
  const size_t o_rs128 = w.take(static_cast<size_t>(p->max_seq) * 64 * 4);
  const size_t op_bytes = static_cast<size_t>(24) << 20;     // pass-kernel op tables
  const size_t done_ints = static_cast<size_t>(64) << 10;
  // fused draft step: attention partials [rows][H][splits][hd + 4], LM-head
  // statistics [groups][SMs][4], barrier words
  const int dhd = has_draft ? dm.head_dim : 64;
  const size_t df_att_floats = static_cast<size_t>(kDfMaxRows) *
                               std::max<size_t>(nsm, static_cast<size_t>(kDfMaxGroups) *
                                                         (has_draft ? dm.n_heads : 1)) *
                               (dhd + 4);
  const size_t o_dfa = w.take(df_att_floats * 4);
  const size_t o_dfl = w.take(static_cast<size_t>(kDfMaxGroups) * nsm * 4 * 4);
  const size_t o_dfb = w.take(64);
  const size_t o_dfm = w.take(has_draft ? static_cast<size_t>(kMaxDrafts) * kDfMapsPerDraft * sizeof(CUtensorMap) : 0);
  const size_t o_ops = w.take(op_bytes);
  const size_t o_done = w.take(done_ints * 4);
  const size_t trace_bytes =
      (p->trace >= 1 && p->trace <= 3)
          ? (2 + static_cast<size_t>(kPassTraceOps) * nsm * kPassTraceSlots) * 8
          : 0;
  const size_t o_trace = w.take(trace_bytes);
  if (c != nullptr) {
    c->trace = trace_bytes ? reinterpret_cast<unsigned long long*>(base + o_trace) : nullptr;
    c->h = reinterpret_cast<float*>(base + o_h);
    c->xg = reinterpret_cast<bf16*>(base + o_xg);
    c->xg_lo = reinterpret_cast<bf16*>(base + o_xgl);
    c->o_lo = reinterpret_cast<bf16*>(base + o_ol);
    c->act_lo = reinterpret_cast<bf16*>(base + o_actl);
    c->ss = reinterpret_cast<float*>(base + o_ss);
    c->q = reinterpret_cast<float*>(base + o_q);
    c->o = reinterpret_cast<bf16*>(base + o_o);
    c->act = reinterpret_cast<bf16*>(base + o_act);
    c->gemm_part = reinterpret_cast<float*>(base + o_gp);
    c->gemm_cnt = reinterpret_cast<int*>(base + o_gc);
    c->gemm_cnt_bytes = static_cast<size_t>(max_rt) * 4;
    c->att_po = reinterpret_cast<float*>(base + o_apo);
    c->att_pml = reinterpret_cast<float*>(base + o_apml);
    c->att_cnt = reinterpret_cast<int*>(base + o_acnt);
    c->att_po_cap = po;
    c->att_cnt_cap = cnt;
    c->zt = reinterpret_cast<float*>(base + o_zt);
    c->zd = reinterpret_cast<float*>(base + o_zd);
    c->tokens = reinterpret_cast<int*>(base + o_tok);
    c->state = reinterpret_cast<int*>(base + o_st);
    c->draft_tokens = reinterpret_cast<int*>(base + o_dt);
    c->d_len_all = reinterpret_cast<int*>(base + o_dl);
    c->seeds = reinterpret_cast<unsigned long long*>(base + o_seed);
    c->plan = reinterpret_cast<RowPlan*>(base + o_plan);
    c->status = reinterpret_cast<uint32_t*>(base + o_status);
    c->results = reinterpret_cast<int*>(base + o_res);
    c->acc_part = reinterpret_cast<float*>(base + o_ap);
    c->acc_dbg = reinterpret_cast<float*>(base + o_ad);
    c->acc_cnt = reinterpret_cast<int*>(base + o_ac);
    c->smp_cnt = reinterpret_cast<int*>(base + o_sc);
    c->tree_desc = reinterpret_cast<TreeDesc*>(base + o_td);
    c->tree_samples = reinterpret_cast<int*>(base + o_ts);
    c->tree_result = reinterpret_cast<TreeResult*>(base + o_tr);
    c->tree_z = reinterpret_cast<float*>(base + o_tz);
    c->rope_cos[0] = reinterpret_cast<float*>(base + o_rc64);
    c->rope_sin[0] = reinterpret_cast<float*>(base + o_rs64);
    c->rope_cos[1] = reinterpret_cast<float*>(base + o_rc128);
    c->rope_sin[1] = reinterpret_cast<float*>(base + o_rs128);
    c->df_att = reinterpret_cast<float*>(base + o_dfa);
    c->df_att_floats = df_att_floats;
    c->df_lm = reinterpret_cast<float*>(base + o_dfl);
    c->df_bar = reinterpret_cast<unsigned int*>(base + o_dfb);
    c->df_maps = has_draft ? reinterpret_cast<CUtensorMap*>(base + o_dfm) : nullptr;
    c->op_area = base + o_ops;
    c->op_area_bytes = op_bytes;
    c->done_area = reinterpret_cast<int*>(base + o_done);
    c->done_area_ints = done_ints;
    c->max_rows = rows;
    c->vocab = V;
  }
  return w.off;
}

memspec_status validate_params(const memspec_init_params* p, std::string* why) {
  if (p == nullptr) {
    *why = "null params";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (!cfg_valid(&p->target, why)) return MEMSPEC_ERR_INVALID_ARG;
  memspec_status s = cfg_supported(&p->target, why);
  if (s != MEMSPEC_OK) return s;
  if (p->max_batch < 1 || p->max_batch > kMaxGroups) {
    *why = "max_batch must be in 1..64";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (p->max_k < 1 || p->max_k > kMaxK) {
    *why = "max_k must be in 1..15";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (p->max_batch * (p->max_k + 1) > kMaxRows) {
    *why = "max_batch * (max_k + 1) must be <= 256";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  if (p->max_seq < 2 || p->max_seq > (1 << 20)) {
    *why = "max_seq must be in 2..2^20";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (p->max_drafts < 0 || p->max_drafts > kMaxDrafts) {
    *why = "max_drafts must be in 0..16";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (p->draft_kernel < MEMSPEC_DRAFT_KERNEL_AUTO || p->draft_kernel > MEMSPEC_DRAFT_KERNEL_FUSED) {
    *why = "draft_kernel must be AUTO, PER_OP or FUSED";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (p->max_drafts > 0) {
    if (!cfg_valid(&p->draft_shape_max, why)) return MEMSPEC_ERR_INVALID_ARG;
    s = cfg_supported(&p->draft_shape_max, why);
    if (s != MEMSPEC_OK) return s;
  }
  return MEMSPEC_OK;
}

// Tensor map over a bf16 activation buffer [rows][cols] with box {64, n_pad}:
// rows >= `rows` read as zero.  Cached per (buffer, rows, cols, n_pad).
bool act_map(memspec_ctx* c, const void* ptr, int rows, int cols, int n_pad, CUtensorMap* out) {
  auto key = std::make_tuple(ptr, rows, cols, n_pad);
  auto it = c->bmaps.find(key);
  if (it == c->bmaps.end()) {
    CUtensorMap m;
    if (!encode_map(&m, ptr, rows, cols, n_pad)) return false;
    it = c->bmaps.emplace(key, m).first;
  }
  *out = it->second;
  return true;
}

// ---------------------------------------------------------------- forward pass
struct FwdSpec {
  int mode, n_groups, R, j;
  int pre_req, pre_start, pre_count;
  const int* d_len;  // draft pass 1: processed counts of the draft
  float* logits;     // nullptr: no LM head
  int last_only;
  long long out_group_stride;
};

// Stream-K grid: at most one CTA per SM, and at least ceil(k_tiles / 4) tiles per
// CTA so that a row tile is shared by at most ~4 CTAs (the last of them sums the
// partials; more contributors lengthen that serial tail more than they add
// bandwidth on small matrices).  kGemmSpareSms SMs stay free: with every SM
// streaming, some SMs stream 1-2 us slower than the rest and the CTAs that start
// on SMs still held by the previous launch start late, and a static partition
// waits for the slowest; with 16 SMs free the verify pass measured 3.34 ms
// instead of 3.42 (QKV launch 21 us instead of 25).
constexpr int kGemmSpareSms = 16;

int env_int(const char* name, int dflt) {
  const char* e = std::getenv(name);
  return e != nullptr ? std::atoi(e) : dflt;
}
// MEMSPEC_SK_MAXC overrides the contributor limit (measurement).
int gemm_grid(int row_tiles, int k_tiles) {
  static const int max_contrib = std::max(1, env_int("MEMSPEC_SK_MAXC", 4));
  static const int max_grid = env_int("MEMSPEC_GEMM_MAXG", 0);   // > 0: overrides (measurement)
  const int T = row_tiles * k_tiles;
  const int min_tiles = std::max(1, (k_tiles + max_contrib - 1) / max_contrib);
  const int sms = max_grid > 0 ? std::min(max_grid, sm_count())
                               : (sm_count() > 4 * kGemmSpareSms ? sm_count() - kGemmSpareSms
                                                                 : sm_count());
  return std::max(1, std::min({T, sms, T / min_tiles}));
}

// Whether a GEMM launch dry-runs its tail before griddepcontrol.wait: worth it
// when the launch starts early (while its predecessor's CTAs drain); the down
// projection follows gate/up, whose CTAs nearly all reduce and leave late.
// MEMSPEC_WARM_DOWN / MEMSPEC_WARM_OTHER = 0 or 1 override (measurement).
int warm_default(const char* env, int dflt) {
  const char* e = std::getenv(env);
  return e != nullptr ? (e[0] == '1') : dflt;
}
int warm_down() {
  static int v = -1;
  if (v < 0) v = warm_default("MEMSPEC_WARM_DOWN", 1);
  return v;
}
int warm_other() {
  static int v = -1;
  if (v < 0) v = warm_default("MEMSPEC_WARM_OTHER", 1);
  return v;
}

// Cluster exchange for decode GEMMs (16 padded rows): a grid of Q clusters of C
// CTAs whose stream-K ranges put every split row tile inside one cluster, so that
// the split-K partials move through distributed shared memory instead of global
// memory (no store, counter or reload on the critical tail).  Taken when its
// largest range is at most kCskTailTiles - 1 tiles longer than plain stream-K's:
// a global-memory exchange costs about as much as streaming that many tiles
// (~1.5 us, measured).  Clusters of at most four CTAs: larger ones (fewer ring
// stages for the receive slots, longer sums) made the draft step slower, measured.
// MEMSPEC_CSK=0 disables it; MEMSPEC_CSK_MAX sets the largest C (measurement).
constexpr int kCskTailTiles = 4;
bool sk_split_free(int T, int KT, int G) {   // no row tile is shared by two CTAs
  for (int c = 1; c < G; ++c)
    if (sk_begin(c, T, G) % KT != 0) return false;
  return true;
}
bool csk_aligned(int R, int KT, int G, int C) {
  const int T = R * KT;
  for (int rt = 0; rt < R; ++rt)
    if (sk_cta_of(rt * KT, T, G) / C != sk_cta_of(rt * KT + KT - 1, T, G) / C) return false;
  return true;
}
struct CskPick {
  int grid, csk;
};
CskPick pick_csk(const GemmArgs& a, int planes, int g0) {
  static const int enabled = env_int("MEMSPEC_CSK", 1);
  static const int c_max = std::min(8, env_int("MEMSPEC_CSK_MAX", 4));
  const int R = a.row_tiles, KT = a.k_tiles, T = R * KT;
  CskPick best{g0, 0};
  if (!enabled || a.n_pad != 16 || sk_split_free(T, KT, g0)) return best;
  int best_cost = ceil_div(T, g0) + kCskTailTiles;
  int dev = 0;
  cudaGetDevice(&dev);
  static std::map<std::tuple<int, int, int, size_t>, int> fit;   // (device, epi, C, smem) -> clusters
  static std::mutex fit_mu;
  std::lock_guard<std::mutex> lock(fit_mu);
  for (int C = 2; C <= c_max; ++C) {
    const size_t smem = gemm_smem_bytes(a.n_pad, gemm_pick_stages(a.n_pad, planes, C), planes, C);
    const auto key = std::make_tuple(dev, a.epi, C, smem);
    auto it = fit.find(key);
    if (it == fit.end()) it = fit.emplace(key, gemm_max_active_clusters(a.epi, C, smem)).first;
    // never more CTAs than plain stream-K: clusters must all be resident while the
    // previous launch still holds SMs (a larger clustered grid measured far slower)
    const int q_max = std::min({it->second, g0 / C, T / C});
    for (int Q = q_max; Q >= 1; --Q) {
      const int G = Q * C;
      if (!sk_fits(T, G)) continue;
      const int cost = ceil_div(T, G);
      if (cost >= best_cost) break;   // smaller grids only cost more
      if (!csk_aligned(R, KT, G, C)) continue;
      best = {G, C};
      best_cost = cost;
      break;
    }
  }
  return best;
}

void emit_gemm(memspec_ctx* c, GemmArgs& a, std::vector<PassOp>& ops) {
  const int planes = a.split ? 2 : 1;
  if (a.warm < 0) a.warm = warm_down();   // the down projection marks itself with -1
  else a.warm = warm_other();
  int grid = gemm_grid(a.row_tiles, a.k_tiles);
  a.csk = 0;
  if (!c->pass_kernel) {   // the persistent kernel runs every op on its own grid
    const CskPick pk = pick_csk(a, planes, grid);
    grid = pk.grid;
    a.csk = pk.csk;
  }
  a.stages = gemm_pick_stages(a.n_pad, planes, a.csk);
  a.partials = c->gemm_part;
  a.counters = c->gemm_cnt;
  a.status = c->status;
  // Two or more 16-row chunks (trees, batched verify, prefill): split row tiles
  // get their own epilogue launch, one CTA per (row tile, 16-row chunk), instead
  // of one contributor folding every chunk in turn (a 31-node tree step 5.02 ->
  // 4.81 ms, batched 8B verify 17.6 -> 12.0 ms).  MEMSPEC_SPLIT_EPI_ROWS sets the
  // threshold (0: never; measurement).
  static const int split_rows = env_int("MEMSPEC_SPLIT_EPI_ROWS", 32);
  a.split_epi = (!c->pass_kernel && a.csk == 0 && split_rows > 0 && a.n_pad >= split_rows &&
                 !sk_split_free(a.row_tiles * a.k_tiles, a.k_tiles, grid))
                    ? 1
                    : 0;
  PassOp op{};
  op.type = OP_GEMM;
  op.grid = grid;
  op.smem = static_cast<int>(gemm_smem_bytes(a.n_pad, a.stages, planes, a.csk));
  op.u.g = a;
  ops.push_back(op);
  if (a.split_epi) {
    PassOp ep{};
    ep.type = OP_GEMM_EPI;
    ep.grid = grid;
    ep.u.g = a;
    ops.push_back(ep);
  }
}

// Launches as separate kernels: the op after the embedding kernel (which writes
// the row plan) waits for every earlier kernel (no programmatic dependent
// launch), so every later op starts after the plan - and the KV cache of earlier
// positions - is final and may read them before griddepcontrol.wait (ctx_early).
// MEMSPEC_CTX_EARLY=0 turns this off (measurement).
void mark_ctx_early(std::vector<PassOp>& ops, size_t first) {
  static const int enabled = env_int("MEMSPEC_CTX_EARLY", 1);
  if (!enabled || ops.size() < first + 2 || ops[first].type != OP_EMBED) return;
  ops[first + 1].full_dep = 1;
  for (size_t i = first + 2; i < ops.size(); ++i) {
    if (ops[i].type == OP_GEMM) ops[i].u.g.ctx_early = 1;
    if (ops[i].type == OP_ATTN) ops[i].u.at.ctx_early = 1;
  }
}

memspec_status emit_forward(memspec_ctx* c, ModelRT& m, const FwdSpec& f,
                            std::vector<PassOp>& ops) {
  const size_t first_op = ops.size();
  const memspec_model_cfg& cf = m.cfg;
  const int d = cf.d_model, qd = model_q(cf), kvd = model_kv(cf), F = cf.d_ffn;
  const int rows = f.n_groups * f.R;
  const int n_pad = round_up(rows, 16);
  const int hsel = cf.head_dim == 128 ? 1 : 0;
  EmbedArgs ea{};
  ea.mode = f.mode;
  ea.n_groups = f.n_groups;
  ea.R = f.R;
  ea.j = f.j;
  ea.prefill_req = f.pre_req;
  ea.prefill_start = f.pre_start;
  ea.prefill_count = f.pre_count;
  ea.seq_state = c->state;
  ea.draft_len = f.d_len;
  ea.tokens = c->tokens;
  ea.max_seq = c->p.max_seq;
  ea.draft_tokens = c->draft_tokens;
  ea.max_k = c->p.max_k;
  ea.emb = reinterpret_cast<const bf16*>(m.w + m.lay.emb);
  ea.d = d;
  ea.vocab = cf.vocab;
  ea.h = c->h;
  ea.xg = c->xg;
  ea.xg_lo = c->xg_lo;
  ea.gain = reinterpret_cast<const bf16*>(m.w + m.lay.attn_norm[0]);
  ea.ss = c->ss;
  ea.ss_stride = c->ss_stride;
  ea.plan = c->plan;
  ea.status = c->status;
  {
    PassOp op{};
    op.type = OP_EMBED;
    op.n_units = rows;
    op.u.e = ea;
    ops.push_back(op);
  }

  const size_t layer_kv = static_cast<size_t>(c->p.max_batch) * cf.n_kv_heads * c->p.max_seq * cf.head_dim;
  AttnGeo geo = attn_geometry(cf, f.n_groups, f.R, c->p.max_seq);
  if (attn_part_floats(cf, geo, f.n_groups) > c->att_po_cap ||
      attn_units(cf, geo, f.n_groups) > c->att_cnt_cap)
    return fail(c, MEMSPEC_ERR_UNSUPPORTED, "attention partial buffer too small for this pass");
  int ss_count = 1;
  for (int l = 0; l < cf.n_layers; ++l) {
    bf16* kl = m.kv + static_cast<size_t>(l) * 2 * layer_kv;
    bf16* vl = kl + layer_kv;
    {  // QKV + RoPE + KV append, RMSNorm fused into the activation producer
      GemmArgs a{};
      a.a_packed = m.w + m.lay.wqkv[l];
      a.n_out = qd + 2 * kvd;
      a.k_in = d;
      a.pair = 0;
      a.rows_total = rows;
      a.n_pad = n_pad;
      a.row_tiles = ceil_div(a.n_out, 128);
      a.k_tiles = ceil_div(d, 64);
      a.l2_hint = m.l2_hint;
      if (!act_map(c, c->xg, rows, d, n_pad, &a.map_b) ||
          !act_map(c, c->xg_lo, rows, d, n_pad, &a.map_b2))
        return fail(c, MEMSPEC_ERR_CUDA, "activation tensor map");
      a.split = 1;
      a.rms = 1;
      a.ss = c->ss;
      a.ss_count = ss_count;
      a.ss_stride = c->ss_stride;
      a.eps = cf.norm_eps;
      a.epi = EPI_QKV;
      a.q_out = c->q;
      a.q_dim = qd;
      a.kv_dim = kvd;
      a.head_dim = cf.head_dim;
      a.n_kv_heads = cf.n_kv_heads;
      a.max_seq = c->p.max_seq;
      a.kcache = kl;
      a.vcache = vl;
      a.rope_cos = c->rope_cos[hsel];
      a.rope_sin = c->rope_sin[hsel];
      a.plan = c->plan;
      emit_gemm(c, a, ops);
    }
    {  // attention
      AttnArgs at{};
      at.q = c->q;
      at.kcache = kl;
      at.vcache = vl;
      at.H = cf.n_heads;
      at.Hkv = cf.n_kv_heads;
      at.hd = cf.head_dim;
      at.max_seq = c->p.max_seq;
      at.rows_per_block = geo.rows_per_block;
      at.row_blocks = geo.row_blocks;
      at.chunk = geo.chunk;
      at.n_splits = geo.n_splits;
      at.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(cf.head_dim));
      at.part_o = c->att_po;
      at.part_ml = c->att_pml;
      at.qmax = geo.qmax;
      at.counters = c->att_cnt;
      at.out = c->o;
      at.out_lo = c->o_lo;
      at.plan = c->plan;
      at.status = c->status;
      // per-op launches stream K/V tiles by TMA (the persistent pass kernel keeps cp.async)
      if (!c->pass_kernel) {
        const int kv_rows = c->p.max_batch * cf.n_kv_heads * c->p.max_seq;
        if (!encode_map(&at.kmap, kl, kv_rows, cf.head_dim, 64) ||
            !encode_map(&at.vmap, vl, kv_rows, cf.head_dim, 64))
          return fail(c, MEMSPEC_ERR_CUDA, "KV tensor map");
        at.tma = 1;
      }
      PassOp op{};
      op.type = OP_ATTN;
      op.n_units = at.n_splits * at.Hkv * at.row_blocks * f.n_groups;
      op.grid = f.n_groups;
      op.u.at = at;
      ops.push_back(op);
    }
    {  // O projection + residual
      GemmArgs a{};
      a.a_packed = m.w + m.lay.wo[l];
      a.n_out = d;
      a.k_in = qd;
      a.rows_total = rows;
      a.n_pad = n_pad;
      a.row_tiles = ceil_div(d, 128);
      a.k_tiles = ceil_div(qd, 64);
      a.l2_hint = m.l2_hint;
      if (!act_map(c, c->o, rows, qd, n_pad, &a.map_b) ||
          !act_map(c, c->o_lo, rows, qd, n_pad, &a.map_b2))
        return fail(c, MEMSPEC_ERR_CUDA, "activation tensor map");
      a.split = 1;
      a.epi = EPI_RESIDUAL;
      a.h = c->h;
      a.h_ld = d;
      a.ss_out = c->ss;
      a.gain_next = reinterpret_cast<const bf16*>(m.w + m.lay.ffn_norm[l]);
      a.xg_out = c->xg;
      a.xg_lo_out = c->xg_lo;
      a.ss_stride = c->ss_stride;
      a.plan = c->plan;
      emit_gemm(c, a, ops);
      ss_count = ceil_div(d, 128);
    }
    {  // gate/up + SwiGLU
      GemmArgs a{};
      a.a_packed = m.w + m.lay.wgate[l];
      a.pair = 1;
      a.n_out = F;
      a.k_in = d;
      a.rows_total = rows;
      a.n_pad = n_pad;
      a.row_tiles = ceil_div(F, 64);
      a.k_tiles = ceil_div(d, 64);
      a.l2_hint = m.l2_hint;
      if (!act_map(c, c->xg, rows, d, n_pad, &a.map_b) ||
          !act_map(c, c->xg_lo, rows, d, n_pad, &a.map_b2))
        return fail(c, MEMSPEC_ERR_CUDA, "activation tensor map");
      a.split = 1;
      a.rms = 1;
      a.ss = c->ss;
      a.ss_count = ss_count;
      a.ss_stride = c->ss_stride;
      a.eps = cf.norm_eps;
      a.epi = EPI_SWIGLU;
      a.act = c->act;
      a.act_lo = c->act_lo;
      a.act_ld = F;
      a.plan = c->plan;
      emit_gemm(c, a, ops);
    }
    {  // down projection + residual
      GemmArgs a{};
      a.warm = -1;
      a.a_packed = m.w + m.lay.wdown[l];
      a.n_out = d;
      a.k_in = F;
      a.rows_total = rows;
      a.n_pad = n_pad;
      a.row_tiles = ceil_div(d, 128);
      a.k_tiles = ceil_div(F, 64);
      a.l2_hint = m.l2_hint;
      if (!act_map(c, c->act, rows, F, n_pad, &a.map_b) ||
          !act_map(c, c->act_lo, rows, F, n_pad, &a.map_b2))
        return fail(c, MEMSPEC_ERR_CUDA, "activation tensor map");
      a.split = 1;
      a.epi = EPI_RESIDUAL;
      a.h = c->h;
      a.h_ld = d;
      a.ss_out = c->ss;
      a.gain_next = reinterpret_cast<const bf16*>(
          m.w + (l + 1 < cf.n_layers ? m.lay.attn_norm[l + 1] : m.lay.final_norm));
      a.xg_out = c->xg;
      a.xg_lo_out = c->xg_lo;
      a.ss_stride = c->ss_stride;
      a.plan = c->plan;
      emit_gemm(c, a, ops);
    }
  }
  if (f.logits != nullptr) {  // final RMSNorm + LM head -> fp32 logits
    GemmArgs a{};
    if (cf.tied_embeddings)
      a.map_a = m.m_lm;
    else
      a.a_packed = m.w + m.lay.lm_head;
    a.n_out = cf.vocab;
    a.k_in = d;
    a.rows_total = rows;
    a.n_pad = n_pad;
    a.row_tiles = ceil_div(cf.vocab, 128);
    a.k_tiles = ceil_div(d, 64);
    a.l2_hint = m.l2_hint;
    if (!act_map(c, c->xg, rows, d, n_pad, &a.map_b) ||
        !act_map(c, c->xg_lo, rows, d, n_pad, &a.map_b2))
      return fail(c, MEMSPEC_ERR_CUDA, "activation tensor map");
    a.split = 1;
    a.rms = 1;
    a.ss = c->ss;
    a.ss_count = ss_count;
    a.ss_stride = c->ss_stride;
    a.eps = cf.norm_eps;
    a.epi = EPI_F32;
    a.out = f.logits;
    a.out_ld = cf.vocab;
    a.last_only = f.last_only;
    a.out_group_stride = f.out_group_stride;
    a.plan = c->plan;
    emit_gemm(c, a, ops);
  }
  if (!c->pass_kernel) mark_ctx_early(ops, first_op);
  return MEMSPEC_OK;
}

// ---------------------------------------------------------------- running op lists
// Each op as its own kernel launch (programmatic dependent launch between them).
memspec_status run_ops_separately(memspec_ctx* c, const std::vector<PassOp>& ops) {
  for (const PassOp& op : ops) {
    cudaError_t e = cudaSuccess;
    switch (op.type) {
      case OP_EMBED: e = launch_embed(op.u.e, op.n_units, c->main, c->pdl); break;
      case OP_GEMM: e = launch_gemm(op.u.g, op.grid, op.smem, c->main, c->pdl && !op.full_dep); break;
      case OP_GEMM_EPI: e = launch_gemm_split_epi(op.u.g, op.grid, c->main, c->pdl); break;
      case OP_ATTN: e = launch_attention(op.u.at, op.grid, c->main, c->pdl && !op.full_dep); break;
      case OP_SAMPLE: e = launch_sample(op.u.s, c->main, c->pdl); break;
      case OP_ACCEPT: e = launch_accept(op.u.acc, c->main, false); break;
      case OP_TREE_WALK: e = launch_tree_walk(op.u.tw, c->main); break;
      case OP_TREE_COMPACT: e = launch_tree_compact(op.u.tc, op.n_units, c->main); break;
      default: return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown op");
    }
    if (e != cudaSuccess) return cuda_fail(c, e, "op launch");
  }
  return MEMSPEC_OK;
}

// An op table in the workspace (device copy of the ops + completion counters).
struct OpTable {
  PassOp* ops = nullptr;
  int* done = nullptr;   // [n_ops + 1]: counters, then the exit counter
  int n_ops = 0;
  PassArgs args{};
};

// Place `ops` in the workspace: synchronous copy (the table must be in place
// before a graph that uses it is captured).
memspec_status place_table(memspec_ctx* c, const std::vector<PassOp>& ops, OpTable* t,
                           unsigned long long* trace) {
  const size_t bytes = ops.size() * sizeof(PassOp);
  const size_t ints = ops.size() + 1;
  if (bytes > c->op_area_bytes || ints > c->done_area_ints)
    return fail(c, MEMSPEC_ERR_UNSUPPORTED, "pass has more ops than the op-table area holds");
  if (c->op_area_used + bytes > c->op_area_bytes || c->done_area_used + ints > c->done_area_ints) {
    // area full: drop every captured graph (their tables go with them)
    cudaError_t e = cudaStreamSynchronize(c->main);
    if (e != cudaSuccess) return cuda_fail(c, e, "sync");
    for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
    c->graphs.clear();
    c->op_area_used = 0;
    c->done_area_used = 0;
  }
  t->ops = reinterpret_cast<PassOp*>(c->op_area + c->op_area_used);
  t->done = c->done_area + c->done_area_used;
  t->n_ops = static_cast<int>(ops.size());
  c->op_area_used += (bytes + 255) & ~static_cast<size_t>(255);
  c->done_area_used += (ints + 63) & ~static_cast<size_t>(63);
  cudaError_t e = cudaMemcpy(t->ops, ops.data(), bytes, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "op table copy");
  // shared-memory layout of the pass: deepest activation stage, attention region
  int b_bytes = 0, hd = 0;
  uint32_t cols = 32;
  for (const PassOp& op : ops) {
    if (op.type == OP_GEMM) {
      const GemmArgs& a = op.u.g;
      const int planes = a.split ? 2 : 1;
      b_bytes = std::max(b_bytes, a.n_pad * 128 * planes);
      const int acols = (a.split && 2 * a.n_pad <= 256) ? 2 * a.n_pad : a.n_pad;
      while (cols < static_cast<uint32_t>(2 * acols)) cols <<= 1;
    } else if (op.type == OP_ATTN) {
      hd = std::max(hd, op.u.at.hd);
    }
  }
  PassArgs& p = t->args;
  p.ops = t->ops;
  p.n_ops = t->n_ops;
  p.done = t->done;
  p.exit_cnt = t->done + t->n_ops;
  p.b_stage_bytes = b_bytes;
  p.attn_bytes = hd ? static_cast<int>(pass_attn_bytes(hd)) : 0;
  p.stages = pass_pick_stages(b_bytes, p.attn_bytes);
  p.tmem_cols = cols;
  p.status = c->status;
  p.trace = trace;
  if (p.stages < 2) return fail(c, MEMSPEC_ERR_UNSUPPORTED, "pass kernel: shared memory too small");
  return MEMSPEC_OK;
}

// Per-op launches record into the trace too: op n's row starts at
// 2 + n * SMs * 16; the header {n_ops, SMs} is written now (before any capture).
memspec_status attach_trace(memspec_ctx* c, std::vector<PassOp>& ops) {
  const int nsm = sm_count();
  for (size_t n = 0; n < ops.size() && n < static_cast<size_t>(kPassTraceOps); ++n) {
    unsigned long long* row = c->trace + 2 + n * nsm * kPassTraceSlots;
    if (ops[n].type == OP_GEMM) ops[n].u.g.trace = row;
    if (ops[n].type == OP_GEMM_EPI) {
      ops[n].u.g.trace = row;
      ops[n].u.g.trace_ctas = nsm;
    }
    if (ops[n].type == OP_ATTN) {
      ops[n].u.at.trace = row;
      ops[n].u.at.trace_ctas = nsm;
    }
  }
  const unsigned long long head[2] = {static_cast<unsigned long long>(ops.size()),
                                      static_cast<unsigned long long>(nsm)};
  cudaError_t e = cudaMemcpy(c->trace, head, sizeof(head), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "trace header");
  return MEMSPEC_OK;
}

memspec_status launch_table(memspec_ctx* c, const OpTable& t) {
  cudaError_t e = launch_pass(t.args, sm_count(), c->main, c->cooperative);
  if (e != cudaSuccess) return cuda_fail(c, e, "pass kernel launch");
  return MEMSPEC_OK;
}

// Build the op list, then run it: one persistent launch (pass kernel) or one
// launch per op; captured once as a CUDA graph per key and replayed when graphs
// are on.  `use_pass` = false always runs separate launches.
template <class Emit>
memspec_status run_pass(memspec_ctx* c, const GraphKey& key, bool use_pass, Emit&& emit) {
  const bool pass = use_pass && c->pass_kernel;
  const int slot = (key.kind == 1 || key.kind == 4) ? 1 : (key.kind == 2 ? 2 : 0);
  if (c->p.use_graphs) {
    auto it = c->graphs.find(key);
    if (it != c->graphs.end()) {
      cudaError_t e = cudaGraphLaunch(it->second, c->main);
      if (e != cudaSuccess) return cuda_fail(c, e, "graph launch");
      c->last_launches[slot] = c->graph_launches[key];
      return MEMSPEC_OK;
    }
  }
  std::vector<PassOp> ops;
  memspec_status s = emit(ops);
  if (s != MEMSPEC_OK) return s;
  const int n_launch = pass ? 1 : static_cast<int>(ops.size());
  c->last_launches[slot] = n_launch;
  // tracing: init param trace = 1 records verify passes, 2 draft steps
  const bool traced = c->trace != nullptr && ((c->p.trace == 1 && key.kind == 1) ||
                                              (c->p.trace == 2 && key.kind == 0));
  OpTable t;
  if (pass) {
    s = place_table(c, ops, &t, traced ? c->trace : nullptr);
    if (s != MEMSPEC_OK) return s;
  } else if (traced) {
    s = attach_trace(c, ops);
    if (s != MEMSPEC_OK) return s;
  }
  if (!c->p.use_graphs) return pass ? launch_table(c, t) : run_ops_separately(c, ops);
  cudaError_t e = cudaStreamBeginCapture(c->main, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return cuda_fail(c, e, "begin capture");
  s = pass ? launch_table(c, t) : run_ops_separately(c, ops);
  cudaGraph_t g = nullptr;
  e = cudaStreamEndCapture(c->main, &g);
  if (s != MEMSPEC_OK) {
    if (g) cudaGraphDestroy(g);
    return s;
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "end capture");
  cudaGraphExec_t ex = nullptr;
  e = cudaGraphInstantiate(&ex, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return cuda_fail(c, e, "graph instantiate");
  c->graphs.emplace(key, ex);
  c->graph_launches[key] = n_launch;
  e = cudaGraphLaunch(ex, c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "graph launch");
  return MEMSPEC_OK;
}

// A forward pass run with separate launches and no graph (prefill, catch-up).
memspec_status enqueue_forward(memspec_ctx* c, ModelRT& m, const FwdSpec& f) {
  std::vector<PassOp> ops;
  memspec_status s = emit_forward(c, m, f, ops);
  if (s != MEMSPEC_OK) return s;
  if (c->trace != nullptr && c->p.trace == 3 && f.mode == PLAN_PREFILL) {   // each chunk overwrites
    s = attach_trace(c, ops);
    if (s != MEMSPEC_OK) return s;
  }
  return run_ops_separately(c, ops);
}

void drop_graphs_of_draft(memspec_ctx* c, int draft) {
  for (auto it = c->graphs.begin(); it != c->graphs.end();) {
    if (it->first.draft == draft) {
      cudaGraphExecDestroy(it->second);
      it = c->graphs.erase(it);
    } else {
      ++it;
    }
  }
}

uint32_t fbits(float x) {
  uint32_t u;
  std::memcpy(&u, &x, 4);
  return u;
}

memspec_status draft_wait_ready(memspec_ctx* c, DraftRec& dr) {
  if (dr.state == 2) {
    cudaError_t e = cudaStreamWaitEvent(c->main, dr.ev, 0);
    if (e != cudaSuccess) return cuda_fail(c, e, "wait for draft load");
  }
  return MEMSPEC_OK;
}

// Bring draft `id`'s KV cache up to the committed tokens of requests [0, batch).
memspec_status draft_catch_up(memspec_ctx* c, int id) {
  DraftRec& dr = c->drafts[id];
  const int B = c->p.max_batch;
  std::vector<int> st(static_cast<size_t>(B) * kStateInts), dl(B);
  cudaError_t e = cudaStreamSynchronize(c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "sync");
  e = cudaMemcpy(st.data(), c->state, st.size() * 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(dl.data(), dr.d_len, dl.size() * 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "read lengths");
  for (int b = 0; b < c->batch; ++b) {
    const int L = st[b * kStateInts];
    for (int start = dl[b]; start < L - 1; start += kPrefillChunk) {
      FwdSpec f{};
      f.mode = PLAN_PREFILL;
      f.n_groups = 1;
      f.R = kPrefillChunk;
      f.pre_req = b;
      f.pre_start = start;
      f.pre_count = std::min(kPrefillChunk, L - 1 - start);
      memspec_status s = enqueue_forward(c, dr.rt, f);
      if (s != MEMSPEC_OK) return s;
    }
    if (L - 1 > dl[b]) {
      const int v = L - 1;
      e = cudaMemcpyAsync(dr.d_len + b, &v, 4, cudaMemcpyHostToDevice, c->main);
      if (e == cudaSuccess) e = cudaStreamSynchronize(c->main);
      if (e != cudaSuccess) return cuda_fail(c, e, "set draft length");
    }
  }
  return MEMSPEC_OK;
}


// ---------------------------------------------------------------- fused draft step
// Launch parameters of the fused draft kernel for the active draft, or false
// (with the reason) when the draft or batch does not fit it: at most
// kDfMaxGroups requests, and a shared-memory ring of at least 8 weight slots
// beside the activation rows.
bool fused_draft_plan(memspec_ctx* c, DraftRec& dr, int K, float T, DraftFusedArgs* out,
                      std::string* why) {
  const memspec_model_cfg& m = dr.cfg;
  const Layout& lay = dr.rt.lay;
  const int B = c->batch, G = sm_count();
  if (B > kDfMaxGroups) {
    *why = "more than 4 requests";
    return false;
  }
  const int hq = m.n_heads * m.head_dim;
  const int f_pad = round_up(m.d_ffn, 64);
  const int act_floats = std::max({m.d_model, hq, f_pad});
  const size_t fixed = draft_fused_smem_bytes(0, 2 * B, act_floats) + draft_fused_static_smem() + 1024;
  const long long room = 227LL * 1024 - static_cast<long long>(fixed);
  const int slots = static_cast<int>(std::min<long long>(kDfMaxSlots, room / kDfSlotBytes));
  if (slots < 4) {
    *why = "activation rows leave no room for the weight ring";
    return false;
  }
  int S = std::max(1, G / (B * m.n_heads));
  S = std::min({S, kDfMaxSplits, std::max(1, ceil_div(c->p.max_seq, 64))});
  if (static_cast<size_t>(2 * B) * m.n_heads * S * (m.head_dim + 4) > c->df_att_floats) {
    *why = "too many attention units for the scratch";
    return false;
  }
  // the sampler scans one CTA's vocabulary slice with 32 ids per lane at most
  if (ceil_div(ceil_div(m.vocab, 8), G) * 8 > 1024 || G > 256) {
    *why = "vocabulary slice per SM above 1024 ids";
    return false;
  }
  if (m.n_layers > 1) {   // per-layer tensors at a fixed stride
    const size_t st = lay.attn_norm[1] - lay.attn_norm[0];
    for (int l = 1; l < m.n_layers; ++l)
      if (lay.attn_norm[l] - lay.attn_norm[l - 1] != st || lay.wqkv[l] - lay.wqkv[l - 1] != st ||
          lay.wo[l] - lay.wo[l - 1] != st || lay.ffn_norm[l] - lay.ffn_norm[l - 1] != st ||
          lay.wgate[l] - lay.wgate[l - 1] != st || lay.wdown[l] - lay.wdown[l - 1] != st) {
        *why = "irregular layer layout";
        return false;
      }
  }
  if (m.n_layers > kDfMaxLayers || c->df_maps == nullptr) {
    *why = "more than 32 layers";
    return false;
  }
  // TMA boxes over this draft's weights where they are now (rebuilt after a move)
  const int id = static_cast<int>(&dr - c->drafts);
  CUtensorMap* dev_maps = c->df_maps + static_cast<size_t>(id) * kDfMapsPerDraft;
  if (dr.df_maps_for != dr.rt.w) {
    dr.df_maps.assign(kDfMapsPerDraft, CUtensorMap{});
    const int d = m.d_model, q = m.n_heads * m.head_dim, kv = m.n_kv_heads * m.head_dim, F = m.d_ffn;
    auto packed = [&](CUtensorMap* mp, size_t off, long long n, long long k, bool pair, uint32_t rows,
                      uint32_t tiles) {
      const uint64_t nt = packed_bytes(n, k, pair) / kPackTileBytes;
      return encode_box3d(mp, dr.rt.w + off, 64, 128, nt, 128, kPackTileBytes, 64, rows, tiles);
    };
    bool ok = true;
    for (int l = 0; l < m.n_layers && ok; ++l) {
      CUtensorMap* mp = dr.df_maps.data() + l * 4;
      ok = packed(mp + 0, lay.wqkv[l], q + 2 * kv, d, false, 8, 8) &&
           packed(mp + 1, lay.wo[l], d, q, false, 8, 16) && packed(mp + 2, lay.wgate[l], F, d, true, 8, 8) &&
           packed(mp + 3, lay.wdown[l], d, F, false, 8, 16);
    }
    CUtensorMap* lm = dr.df_maps.data() + m.n_layers * 4;
    if (ok)
      ok = m.tied_embeddings
               ? encode_box3d(lm, dr.rt.w + lay.lm_head, static_cast<uint64_t>(d), static_cast<uint64_t>(m.vocab), 1,
                              static_cast<uint64_t>(d) * 2, static_cast<uint64_t>(d) * 2 * m.vocab, 256, 8, 1)
               : packed(lm, lay.lm_head, m.vocab, d, false, 8, 16);
    if (!ok) {
      *why = "tensor map encoding";
      return false;
    }
    if (cudaMemcpyAsync(dev_maps, dr.df_maps.data(), kDfMapsPerDraft * sizeof(CUtensorMap),
                        cudaMemcpyHostToDevice, c->main) != cudaSuccess) {
      *why = "tensor map copy";
      return false;
    }
    dr.df_maps_for = dr.rt.w;
  }
  DraftFusedArgs& a = *out;
  a.maps = dev_maps;
  a.w = dr.rt.w;
  a.off_emb = static_cast<long long>(lay.emb);
  a.off_attn_norm = static_cast<long long>(lay.attn_norm[0]);
  a.off_wqkv = static_cast<long long>(lay.wqkv[0]);
  a.off_wo = static_cast<long long>(lay.wo[0]);
  a.off_ffn_norm = static_cast<long long>(lay.ffn_norm[0]);
  a.off_wgate = static_cast<long long>(lay.wgate[0]);
  a.off_wdown = static_cast<long long>(lay.wdown[0]);
  a.off_final_norm = static_cast<long long>(lay.final_norm);
  a.off_lm = static_cast<long long>(lay.lm_head);
  a.lstride = m.n_layers > 1 ? static_cast<long long>(lay.attn_norm[1] - lay.attn_norm[0]) : 0;
  a.tied = m.tied_embeddings;
  a.n_layers = m.n_layers;
  a.d = m.d_model;
  a.H = m.n_heads;
  a.Hkv = m.n_kv_heads;
  a.hd = m.head_dim;
  a.F = m.d_ffn;
  a.V = m.vocab;
  a.eps = m.norm_eps;
  a.kv = dr.rt.kv;
  a.layer_kv = static_cast<long long>(c->p.max_batch) * m.n_kv_heads * c->p.max_seq * m.head_dim;
  a.max_seq = c->p.max_seq;
  a.max_k = c->p.max_k;
  a.rope_cos = c->rope_cos[m.head_dim == 128 ? 1 : 0];
  a.rope_sin = c->rope_sin[m.head_dim == 128 ? 1 : 0];
  a.K = K;
  a.B = B;
  a.greedy = T == 0.f;
  a.inv_temp = T == 0.f ? 0.f : 1.f / T;
  a.seq_state = c->state;
  a.draft_len = dr.d_len;
  a.tokens = c->tokens;
  a.draft_tokens = c->draft_tokens;
  a.seeds = c->seeds;
  a.zd = c->zd;
  a.h = c->h;
  a.qb = c->q;
  a.att = c->df_att;
  a.act = reinterpret_cast<float*>(c->act);
  a.lm_part = c->df_lm;
  a.bar = c->df_bar;
  a.status = c->status;
  a.n_splits = S;
  a.ring_slots = slots;
  a.act_floats = act_floats;
  // per-phase timestamps of the draft step (init param trace = 2)
  a.trace = (c->trace != nullptr && c->p.trace == 2) ? c->trace : nullptr;
  a.trace_phases = std::min(kPassTraceOps, K * (5 * m.n_layers + 1));
  if (a.trace != nullptr) {
    const unsigned long long head[2] = {static_cast<unsigned long long>(a.trace_phases),
                                        static_cast<unsigned long long>(G)};
    if (cudaMemcpy(c->trace, head, sizeof(head), cudaMemcpyHostToDevice) != cudaSuccess) {
      *why = "trace header";
      return false;
    }
  }
  return true;
}

// One launch (captured once per key as a CUDA graph when graphs are on).  The
// launch is cooperative, so that every CTA of the grid is resident for the
// grid-wide barriers; if stream capture refuses the attribute, a plain launch of
// one CTA per SM is used (the kernel's barrier waits are bounded either way).
memspec_status run_fused_draft(memspec_ctx* c, const GraphKey& key, const DraftFusedArgs& a) {
  const int G = sm_count();
  c->last_launches[0] = 1;
  if (!c->p.use_graphs) {
    cudaError_t e = launch_draft_fused(a, G, c->main, c->df_coop);
    if (e != cudaSuccess) return cuda_fail(c, e, "fused draft launch");
    return MEMSPEC_OK;
  }
  auto it = c->graphs.find(key);
  if (it != c->graphs.end()) {
    cudaError_t e = cudaGraphLaunch(it->second, c->main);
    if (e != cudaSuccess) return cuda_fail(c, e, "graph launch");
    return MEMSPEC_OK;
  }
  for (int attempt = 0; attempt < 2; ++attempt) {
    cudaError_t e = cudaStreamBeginCapture(c->main, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return cuda_fail(c, e, "begin capture");
    const cudaError_t le = launch_draft_fused(a, G, c->main, c->df_coop);
    cudaGraph_t g = nullptr;
    e = cudaStreamEndCapture(c->main, &g);
    cudaGraphExec_t ex = nullptr;
    if (le == cudaSuccess && e == cudaSuccess) e = cudaGraphInstantiate(&ex, g, 0);
    if (g) cudaGraphDestroy(g);
    if (le == cudaSuccess && e == cudaSuccess) {
      c->graphs.emplace(key, ex);
      e = cudaGraphLaunch(ex, c->main);
      if (e != cudaSuccess) return cuda_fail(c, e, "graph launch");
      return MEMSPEC_OK;
    }
    (void)cudaGetLastError();
    if (!c->df_coop) return cuda_fail(c, le != cudaSuccess ? le : e, "fused draft capture");
    c->df_coop = false;   // retry without the cooperative attribute
  }
  return fail(c, MEMSPEC_ERR_CUDA, "fused draft capture");
}

}  // namespace

// =================================================================== C ABI
extern "C" {

memspec_status memspec_weights_bytes(const memspec_model_cfg* cfg, size_t* bytes) {
  std::string why;
  if (!cfg_valid(cfg, &why) || bytes == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  *bytes = make_layout(*cfg).total;
  return MEMSPEC_OK;
}

memspec_status memspec_weights_offset(const memspec_model_cfg* cfg, int32_t tensor, int32_t layer,
                                      size_t* offset, size_t* bytes) {
  std::string why;
  if (!cfg_valid(cfg, &why) || offset == nullptr || bytes == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  const Layout L = make_layout(*cfg);
  const size_t d = cfg->d_model, q = static_cast<size_t>(model_q(*cfg)),
               kv = static_cast<size_t>(model_kv(*cfg)), f = cfg->d_ffn, v = cfg->vocab;
  const bool per_layer = tensor >= MEMSPEC_T_ATTN_NORM && tensor <= MEMSPEC_T_WDOWN;
  if (per_layer && (layer < 0 || layer >= cfg->n_layers)) return MEMSPEC_ERR_INVALID_ARG;
  switch (tensor) {
    case MEMSPEC_T_TOK_EMB: *offset = L.emb; *bytes = v * d * 2; break;
    case MEMSPEC_T_ATTN_NORM: *offset = L.attn_norm[layer]; *bytes = d * 2; break;
    case MEMSPEC_T_WQKV: *offset = L.wqkv[layer]; *bytes = packed_bytes(q + 2 * kv, d, false); break;
    case MEMSPEC_T_WO: *offset = L.wo[layer]; *bytes = packed_bytes(d, q, false); break;
    case MEMSPEC_T_FFN_NORM: *offset = L.ffn_norm[layer]; *bytes = d * 2; break;
    case MEMSPEC_T_WGATE: *offset = L.wgate[layer]; *bytes = packed_bytes(f, d, true); break;
    case MEMSPEC_T_WUP: *offset = L.wup[layer]; *bytes = 0; break;   // inside WGATE's pair tiles
    case MEMSPEC_T_WDOWN: *offset = L.wdown[layer]; *bytes = packed_bytes(d, f, false); break;
    case MEMSPEC_T_FINAL_NORM: *offset = L.final_norm; *bytes = d * 2; break;
    case MEMSPEC_T_LM_HEAD:
      *offset = L.lm_head;
      *bytes = cfg->tied_embeddings ? v * d * 2 : packed_bytes(v, d, false);
      break;
    default: return MEMSPEC_ERR_INVALID_ARG;
  }
  return MEMSPEC_OK;
}

memspec_status memspec_kv_bytes(const memspec_model_cfg* cfg, int32_t max_batch, int32_t max_seq,
                                size_t* bytes) {
  std::string why;
  if (!cfg_valid(cfg, &why) || bytes == nullptr || max_batch < 1 || max_seq < 1)
    return MEMSPEC_ERR_INVALID_ARG;
  *bytes = kv_bytes(*cfg, max_batch, max_seq);
  return MEMSPEC_OK;
}

memspec_status memspec_workspace_bytes(const memspec_init_params* p, size_t* bytes) {
  std::string why;
  memspec_status s = validate_params(p, &why);
  if (s != MEMSPEC_OK) return s;
  if (bytes == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  *bytes = layout_workspace(p, nullptr, nullptr);
  return MEMSPEC_OK;
}

memspec_status memspec_init(const memspec_init_params* p, void* workspace_dev, memspec_ctx** out) {
  std::string why;
  if (out == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  *out = nullptr;
  memspec_status s = validate_params(p, &why);
  if (s != MEMSPEC_OK) {
    g_op_error = why;
    return s;
  }
  if (workspace_dev == nullptr || (reinterpret_cast<uintptr_t>(workspace_dev) & 255) != 0 ||
      p->target_weights_dev == nullptr || p->target_kv_dev == nullptr ||
      (p->max_drafts > 0 && p->draft_arena_dev == nullptr && p->draft_budget_bytes > 0)) {
    g_op_error = "null or misaligned device pointer";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  memspec_ctx* c = new memspec_ctx();
  c->p = *p;
  c->main = static_cast<cudaStream_t>(p->stream_main);
  // MEMSPEC_NO_PDL=1 launches every kernel without programmatic dependent launch
  // (for measuring what the overlap buys)
  const char* no_pdl = std::getenv("MEMSPEC_NO_PDL");
  c->pdl = !(no_pdl != nullptr && no_pdl[0] == '1');
  // MEMSPEC_COOPERATIVE=1 launches the pass kernel cooperatively (its grid is
  // one CTA per SM either way)
  c->pass_kernel = p->launch_mode == MEMSPEC_LAUNCH_PASS;
  const char* coop = std::getenv("MEMSPEC_COOPERATIVE");
  c->cooperative = coop != nullptr && coop[0] == '1';
  c->side = p->stream_side ? static_cast<cudaStream_t>(p->stream_side) : c->main;
  c->ws_bytes = layout_workspace(p, c, static_cast<uint8_t*>(workspace_dev));
  if (!ensure_func_attrs()) {
    g_op_error = g_attr_error;
    delete c;
    return MEMSPEC_ERR_CUDA;
  }
  c->target.cfg = p->target;
  c->target.lay = make_layout(p->target);
  c->target.w = static_cast<const uint8_t*>(p->target_weights_dev);
  c->target.kv = static_cast<bf16*>(p->target_kv_dev);
  c->target.l2_hint = L2_EVICT_FIRST;
  if (!build_maps(c->target, &why)) {
    g_op_error = why;
    delete c;
    return MEMSPEC_ERR_CUDA;
  }
  cudaError_t e = cudaMemsetAsync(workspace_dev, 0, c->ws_bytes, c->main);
  if (e == cudaSuccess)
    e = launch_rope_table(c->rope_cos[0], c->rope_sin[0], p->max_seq, 32, p->target.rope_base, c->main);
  if (e == cudaSuccess)
    e = launch_rope_table(c->rope_cos[1], c->rope_sin[1], p->max_seq, 64, p->target.rope_base, c->main);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->main);
  if (e != cudaSuccess) {
    g_op_error = std::string("init: ") + cudaGetErrorString(e);
    delete c;
    return MEMSPEC_ERR_CUDA;
  }
  for (int i = 0; i < kMaxDrafts; ++i) c->drafts[i].d_len = c->d_len_all + i * p->max_batch;
  *out = c;
  return MEMSPEC_OK;
}

void memspec_destroy(memspec_ctx* c) {
  if (c == nullptr) return;
  for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
  for (auto& d : c->drafts)
    if (d.ev) cudaEventDestroy(d.ev);
  delete c;
}

const char* memspec_last_error(const memspec_ctx* c) {
  if (c == nullptr) return g_op_error.c_str();
  return c->err.c_str();
}

memspec_status memspec_register_draft(memspec_ctx* c, int32_t id, const memspec_model_cfg* cfg,
                                      const void* host_blob, void* kv_dev) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  std::string why;
  if (id < 0 || id >= c->p.max_drafts) return fail(c, MEMSPEC_ERR_INVALID_ARG, "draft id out of range");
  if (!cfg_valid(cfg, &why)) return fail(c, MEMSPEC_ERR_INVALID_ARG, why);
  memspec_status s = cfg_supported(cfg, &why);
  if (s != MEMSPEC_OK) return fail(c, s, why);
  if (cfg->vocab != c->p.target.vocab)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "draft and target must share the vocabulary");
  if (cfg->rope_base != c->p.target.rope_base)
    return fail(c, MEMSPEC_ERR_UNSUPPORTED, "draft rope_base must equal the target's");
  const memspec_model_cfg& dm = c->p.draft_shape_max;
  if (cfg->d_model > dm.d_model || model_q(*cfg) > model_q(dm) || cfg->d_ffn > dm.d_ffn)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "draft larger than draft_shape_max");
  if (host_blob == nullptr || kv_dev == nullptr)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "null draft weights or KV pointer");
  DraftRec& d = c->drafts[id];
  if (d.registered) return fail(c, MEMSPEC_ERR_BUSY, "draft id already registered");
  // the draft's attention passes must fit the partial buffers
  for (int R : {1, 2}) {
    AttnGeo g = attn_geometry(*cfg, c->p.max_batch, R, c->p.max_seq);
    if (attn_part_floats(*cfg, g, c->p.max_batch) > c->att_po_cap ||
        attn_units(*cfg, g, c->p.max_batch) > c->att_cnt_cap)
      return fail(c, MEMSPEC_ERR_UNSUPPORTED, "draft attention does not fit the workspace");
  }
  d.registered = true;
  d.cfg = *cfg;
  d.host_blob = host_blob;
  d.bytes = make_layout(*cfg).total;
  d.state = 0;
  d.rt = ModelRT();
  d.rt.cfg = *cfg;
  d.rt.lay = make_layout(*cfg);
  d.rt.kv = static_cast<bf16*>(kv_dev);
  d.rt.l2_hint = L2_EVICT_NORMAL;
  if (d.ev == nullptr) {
    cudaError_t e = cudaEventCreateWithFlags(&d.ev, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(c, e, "event create");
  }
  cudaError_t e = cudaMemsetAsync(d.d_len, 0, c->p.max_batch * 4, c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "reset draft lengths");
  return MEMSPEC_OK;
}

memspec_status memspec_load_draft_async(memspec_ctx* c, int32_t id, size_t* slot_offset) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (id < 0 || id >= c->p.max_drafts || !c->drafts[id].registered)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown draft id");
  DraftRec& d = c->drafts[id];
  if (d.state != 0) {
    if (slot_offset) *slot_offset = d.arena_off;
    return MEMSPEC_OK;
  }
  // first fit over the resident / loading drafts, sorted by offset
  std::vector<std::pair<size_t, size_t>> used;
  for (int i = 0; i < kMaxDrafts; ++i)
    if (c->drafts[i].registered && c->drafts[i].state != 0)
      used.push_back({c->drafts[i].arena_off, align256(c->drafts[i].bytes)});
  std::sort(used.begin(), used.end());
  size_t pos = 0;
  const size_t need = align256(d.bytes);
  bool found = false;
  for (auto& u : used) {
    if (u.first >= pos + need) {
      found = true;
      break;
    }
    pos = std::max(pos, u.first + u.second);
  }
  if (!found && pos + need <= c->p.draft_budget_bytes) found = true;
  if (!found || pos + need > c->p.draft_budget_bytes)
    return fail(c, MEMSPEC_ERR_BUDGET, "draft does not fit the draft budget; evict first");
  uint8_t* dst = static_cast<uint8_t*>(c->p.draft_arena_dev) + pos;
  cudaError_t e = cudaMemcpyAsync(dst, d.host_blob, d.bytes, cudaMemcpyHostToDevice, c->side);
  if (e == cudaSuccess) e = cudaEventRecord(d.ev, c->side);
  if (e != cudaSuccess) return cuda_fail(c, e, "draft copy");
  d.arena_off = pos;
  d.state = 2;
  d.rt.w = dst;
  std::string why;
  if (!build_maps(d.rt, &why)) return fail(c, MEMSPEC_ERR_CUDA, why);
  drop_graphs_of_draft(c, id);
  if (slot_offset) *slot_offset = pos;
  return MEMSPEC_OK;
}

memspec_status memspec_query_draft(memspec_ctx* c, int32_t id, int32_t* state) {
  if (c == nullptr || state == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (id < 0 || id >= c->p.max_drafts || !c->drafts[id].registered)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown draft id");
  DraftRec& d = c->drafts[id];
  if (d.state == 2) {
    cudaError_t e = cudaEventQuery(d.ev);
    if (e == cudaSuccess) d.state = 1;
    else if (e != cudaErrorNotReady) return cuda_fail(c, e, "event query");
  }
  *state = d.state;
  return MEMSPEC_OK;
}

memspec_status memspec_evict_draft(memspec_ctx* c, int32_t id) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (id < 0 || id >= c->p.max_drafts || !c->drafts[id].registered)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown draft id");
  DraftRec& d = c->drafts[id];
  if (id == c->active) return fail(c, MEMSPEC_ERR_BUSY, "the active draft is never evicted");
  if (d.state == 2) {
    cudaError_t e = cudaEventQuery(d.ev);
    if (e == cudaErrorNotReady) return fail(c, MEMSPEC_ERR_BUSY, "draft copy in flight");
    if (e != cudaSuccess) return cuda_fail(c, e, "event query");
  }
  // work already enqueued on the main stream may still read the weights
  cudaError_t e = cudaStreamSynchronize(c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "sync");
  d.state = 0;
  d.rt.w = nullptr;
  d.rt.ready = false;
  drop_graphs_of_draft(c, id);
  return MEMSPEC_OK;
}

memspec_status memspec_set_active_draft(memspec_ctx* c, int32_t id) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (id == -1) {   // no active draft: every draft may be evicted; draft steps are refused
    c->active = -1;
    return MEMSPEC_OK;
  }
  if (id < 0 || id >= c->p.max_drafts || !c->drafts[id].registered)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown draft id");
  DraftRec& d = c->drafts[id];
  if (d.state == 0) return fail(c, MEMSPEC_ERR_NOT_RESIDENT, "draft is not resident");
  memspec_status s = draft_wait_ready(c, d);
  if (s != MEMSPEC_OK) return s;
  c->active = id;
  return draft_catch_up(c, id);
}

memspec_status memspec_prefill(memspec_ctx* c, int32_t req, const int32_t* tokens, int32_t n,
                               uint64_t seed) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (req < 0 || req >= c->p.max_batch) return fail(c, MEMSPEC_ERR_INVALID_ARG, "request out of range");
  if (tokens == nullptr || n < 1 || n >= c->p.max_seq)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "prompt length must be in 1..max_seq-1");
  for (int i = 0; i < n; ++i)
    if (tokens[i] < 0 || tokens[i] >= c->vocab)
      return fail(c, MEMSPEC_ERR_INVALID_ARG, "prompt token outside the vocabulary");
  cudaError_t e = cudaStreamSynchronize(c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "sync");
  int st[kStateInts] = {n, n - 1, 0, 0};
  const unsigned long long sd = seed;
  e = cudaMemcpy(c->tokens + static_cast<size_t>(req) * c->p.max_seq, tokens,
                 static_cast<size_t>(n) * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(c->state + req * kStateInts, st, sizeof(st), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(c->seeds + req, &sd, 8, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "prefill copies");
  for (int start = 0; start < n - 1; start += kPrefillChunk) {
    FwdSpec f{};
    f.mode = PLAN_PREFILL;
    f.n_groups = 1;
    f.R = kPrefillChunk;
    f.pre_req = req;
    f.pre_start = start;
    f.pre_count = std::min(kPrefillChunk, n - 1 - start);
    memspec_status s = enqueue_forward(c, c->target, f);
    if (s != MEMSPEC_OK) return s;
  }
  // every registered draft restarts from zero for this request; the active one
  // is brought up to date now, the others when they become active
  for (int i = 0; i < c->p.max_drafts; ++i) {
    if (!c->drafts[i].registered) continue;
    const int zero = 0;
    e = cudaMemcpy(c->drafts[i].d_len + req, &zero, 4, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(c, e, "reset draft length");
  }
  if (c->active >= 0) {
    DraftRec& d = c->drafts[c->active];
    memspec_status s = draft_wait_ready(c, d);
    if (s != MEMSPEC_OK) return s;
    for (int start = 0; start < n - 1; start += kPrefillChunk) {
      FwdSpec f{};
      f.mode = PLAN_PREFILL;
      f.n_groups = 1;
      f.R = kPrefillChunk;
      f.pre_req = req;
      f.pre_start = start;
      f.pre_count = std::min(kPrefillChunk, n - 1 - start);
      s = enqueue_forward(c, d.rt, f);
      if (s != MEMSPEC_OK) return s;
    }
    const int v = n - 1;
    e = cudaMemcpyAsync(d.d_len + req, &v, 4, cudaMemcpyHostToDevice, c->main);
    if (e != cudaSuccess) return cuda_fail(c, e, "set draft length");
  }
  e = cudaStreamSynchronize(c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "prefill sync");
  return MEMSPEC_OK;
}

memspec_status memspec_set_batch(memspec_ctx* c, int32_t batch) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (batch < 1 || batch > c->p.max_batch) return fail(c, MEMSPEC_ERR_INVALID_ARG, "batch out of range");
  c->batch = batch;
  return MEMSPEC_OK;
}

memspec_status memspec_draft_step(memspec_ctx* c, int32_t K, float T) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (K < 1 || K > c->p.max_k) return fail(c, MEMSPEC_ERR_INVALID_ARG, "K out of range");
  if (!(T >= 0.f)) return fail(c, MEMSPEC_ERR_INVALID_ARG, "temperature must be >= 0");
  if (c->active < 0) return fail(c, MEMSPEC_ERR_NOT_RESIDENT, "no active draft");
  DraftRec& d = c->drafts[c->active];
  if (d.state == 0) return fail(c, MEMSPEC_ERR_NOT_RESIDENT, "active draft not resident");
  memspec_status s = draft_wait_ready(c, d);
  if (s != MEMSPEC_OK) return s;
  const int B = c->batch;
  const int id = c->active;
  if (!c->pass_kernel && c->p.draft_kernel != MEMSPEC_DRAFT_KERNEL_PER_OP) {
    DraftFusedArgs fa{};
    std::string why;
    const bool fits = fused_draft_plan(c, d, K, T, &fa, &why);
    if (fits) {
      c->last_draft_fused = true;
      return run_fused_draft(c, GraphKey{3, id, K, fbits(T), B}, fa);
    }
    if (c->p.draft_kernel == MEMSPEC_DRAFT_KERNEL_FUSED)
      return fail(c, MEMSPEC_ERR_UNSUPPORTED, "fused draft kernel: " + why);
  }
  c->last_draft_fused = false;
  GraphKey key{0, id, K, fbits(T), B};
  return run_pass(c, key, true, [&](std::vector<PassOp>& ops) -> memspec_status {
    for (int j = 1; j <= K; ++j) {
      FwdSpec f{};
      f.mode = j == 1 ? PLAN_DRAFT_FIRST : PLAN_DRAFT_NEXT;
      f.n_groups = B;
      f.R = j == 1 ? 2 : 1;
      f.j = j;
      f.d_len = d.d_len;
      f.logits = c->zd + static_cast<size_t>(j - 1) * c->vocab;
      f.last_only = 1;
      f.out_group_stride = static_cast<long long>(K) * c->vocab;
      memspec_status st = emit_forward(c, d.rt, f, ops);
      if (st != MEMSPEC_OK) return st;
      SampleArgs sa{};
      sa.logits = f.logits;
      sa.row_stride = f.out_group_stride;
      sa.vocab = c->vocab;
      sa.n_groups = B;
      sa.greedy = T == 0.f;
      sa.inv_temp = T == 0.f ? 0.f : 1.f / T;
      sa.slot = j - 1;
      sa.seq_state = c->state;
      sa.seeds = c->seeds;
      sa.out_tok = c->draft_tokens + (j - 1);
      sa.out_stride = c->p.max_k;
      sa.counters = c->smp_cnt;
      sa.status = c->status;
      PassOp op{};
      op.type = OP_SAMPLE;
      op.n_units = B;
      op.u.s = sa;
      ops.push_back(op);
    }
    return MEMSPEC_OK;
  });
}

memspec_status memspec_verify_step(memspec_ctx* c, int32_t K) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (K < 1 || K > c->p.max_k) return fail(c, MEMSPEC_ERR_INVALID_ARG, "K out of range");
  const int B = c->batch;
  GraphKey key{1, -1, K, 0, B};
  return run_pass(c, key, true, [&](std::vector<PassOp>& ops) -> memspec_status {
    FwdSpec f{};
    f.mode = PLAN_VERIFY;
    f.n_groups = B;
    f.R = K + 1;
    f.logits = c->zt;
    f.last_only = 0;
    return emit_forward(c, c->target, f, ops);
  });
}

memspec_status memspec_accept_commit(memspec_ctx* c, int32_t K, float T, int32_t* results_host) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (K < 1 || K > c->p.max_k) return fail(c, MEMSPEC_ERR_INVALID_ARG, "K out of range");
  if (!(T >= 0.f)) return fail(c, MEMSPEC_ERR_INVALID_ARG, "temperature must be >= 0");
  const int B = c->batch;
  const int id = c->active;
  if (id < 0) return fail(c, MEMSPEC_ERR_NOT_RESIDENT, "no active draft");
  GraphKey key{2, id, K, fbits(T), B};
  memspec_status s = run_pass(c, key, false, [&](std::vector<PassOp>& ops) -> memspec_status {
    AcceptArgs a{};
    a.zt = c->zt;
    a.zd = c->zd;
    a.draft_tokens = c->draft_tokens;
    a.max_k = c->p.max_k;
    a.K = K;
    a.vocab = c->vocab;
    a.n_groups = B;
    a.greedy = T == 0.f;
    a.inv_temp = T == 0.f ? 0.f : 1.f / T;
    a.part = c->acc_part;
    a.counters = c->acc_cnt;
    a.seq_state = c->state;
    a.seeds = c->seeds;
    a.draft_len = c->drafts[id].d_len;
    a.tokens = c->tokens;
    a.max_seq = c->p.max_seq;
    a.results = c->results;
    a.debug = c->acc_dbg;
    a.status = c->status;
    PassOp op{};
    op.type = OP_ACCEPT;
    op.n_units = (2 * K + 1) * B;
    op.u.acc = a;
    ops.push_back(op);
    return MEMSPEC_OK;
  });
  if (s != MEMSPEC_OK) return s;
  c->last_K = K;
  if (results_host != nullptr) {
    cudaError_t e = cudaMemcpyAsync(results_host, c->results, static_cast<size_t>(B) * (K + 2) * 4,
                                    cudaMemcpyDeviceToHost, c->main);
    if (e != cudaSuccess) return cuda_fail(c, e, "results copy");
  }
  return MEMSPEC_OK;
}

memspec_status memspec_tree_step(memspec_ctx* c, int32_t n_nodes, const int32_t* tokens_host,
                                 const int32_t* parents_host, float T, int32_t* results_host) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (tokens_host == nullptr || parents_host == nullptr)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "tree tokens and parents required");
  if (n_nodes < 1 || n_nodes > kTreeRows - 1) return fail(c, MEMSPEC_ERR_INVALID_ARG, "tree of 1..31 nodes");
  if (!(T >= 0.f)) return fail(c, MEMSPEC_ERR_INVALID_ARG, "temperature must be >= 0");
  if (c->batch != 1) return fail(c, MEMSPEC_ERR_UNSUPPORTED, "tree steps run one request (batch 1)");
  // the tree as rows: row 0 = the root, row i + 1 = node i
  TreeDesc t{};
  t.n_rows = n_nodes + 1;
  t.parent_row[0] = -1;
  t.rope_off[0] = 0;
  t.anc[0] = 1u;
  for (int i = 0; i < n_nodes; ++i) {
    const int p = parents_host[i];
    if (p < -1 || p >= i) return fail(c, MEMSPEC_ERR_INVALID_ARG, "tree parent must be -1 or a smaller node");
    if (tokens_host[i] < 0 || tokens_host[i] >= c->vocab)
      return fail(c, MEMSPEC_ERR_INVALID_ARG, "tree token out of the vocabulary");
    const int r = i + 1, pr = p + 1;
    t.tokens[r] = tokens_host[i];
    t.parent_row[r] = pr;
    t.rope_off[r] = t.rope_off[pr] + 1;
    t.anc[r] = t.anc[pr] | (1u << r);
  }
  // outside any captured graph: the graph reads only the device copy
  cudaError_t e = cudaMemcpyAsync(c->tree_desc, &t, sizeof(TreeDesc), cudaMemcpyHostToDevice, c->main);
  if (e != cudaSuccess) return cuda_fail(c, e, "tree copy");
  const int R = t.n_rows;
  const ModelRT& tm = c->target;
  GraphKey key{4, -1, R, fbits(T), 1};
  memspec_status s = run_pass(c, key, false, [&](std::vector<PassOp>& ops) -> memspec_status {
    FwdSpec f{};
    f.mode = PLAN_TREE;
    f.n_groups = 1;
    f.R = R;
    f.logits = c->tree_z;
    f.last_only = 0;
    memspec_status st = emit_forward(c, c->target, f, ops);
    if (st != MEMSPEC_OK) return st;
    if (!ops.empty() && ops.front().type == OP_EMBED) ops.front().u.e.tree = c->tree_desc;
    SampleArgs sa{};
    sa.logits = c->tree_z;
    sa.row_stride = c->vocab;
    sa.vocab = c->vocab;
    sa.n_groups = R;
    sa.greedy = T == 0.f;
    sa.inv_temp = T == 0.f ? 0.f : 1.f / T;
    sa.slot = kTreeSlot0;
    sa.row_slots = c->tree_desc->rope_off;
    sa.seq_state = c->state;
    sa.seeds = c->seeds;
    sa.out_tok = c->tree_samples;
    sa.out_stride = 1;
    sa.counters = c->smp_cnt;
    sa.status = c->status;
    PassOp op{};
    op.type = OP_SAMPLE;
    op.n_units = R;
    op.u.s = sa;
    ops.push_back(op);
    PassOp w{};
    w.type = OP_TREE_WALK;
    w.n_units = 1;
    w.u.tw = TreeWalkArgs{c->tree_desc, c->tree_samples, c->state, c->tokens, c->p.max_seq, c->tree_result,
                          c->status};
    ops.push_back(w);
    PassOp k{};
    k.type = OP_TREE_COMPACT;
    k.n_units = tm.cfg.n_layers;
    k.u.tc = TreeCompactArgs{tm.kv,
                             static_cast<size_t>(c->p.max_batch) * tm.cfg.n_kv_heads * c->p.max_seq * tm.cfg.head_dim,
                             tm.cfg.n_kv_heads, tm.cfg.head_dim, c->p.max_seq, c->tree_result};
    ops.push_back(k);
    return MEMSPEC_OK;
  });
  if (s != MEMSPEC_OK) return s;
  if (results_host != nullptr) {
    e = cudaMemcpyAsync(results_host, c->tree_result, sizeof(TreeResult), cudaMemcpyDeviceToHost, c->main);
    if (e != cudaSuccess) return cuda_fail(c, e, "tree results copy");
  }
  return MEMSPEC_OK;
}

memspec_status memspec_sync(memspec_ctx* c, int32_t timeout_ms, uint32_t* bits) {
  if (c == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  cudaError_t e;
  if (timeout_ms < 0) {
    e = cudaStreamSynchronize(c->main);
  } else {
    cudaEvent_t ev;
    e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(c, e, "event create");
    e = cudaEventRecord(ev, c->main);
    int waited = 0;
    while (e == cudaSuccess || e == cudaErrorNotReady) {
      e = cudaEventQuery(ev);
      if (e != cudaErrorNotReady) break;
      if (waited >= timeout_ms) {
        cudaEventDestroy(ev);
        return fail(c, MEMSPEC_ERR_TIMEOUT, "sync timed out");
      }
      struct timespec ts = {0, 1000000};
      nanosleep(&ts, nullptr);
      ++waited;
    }
    cudaEventDestroy(ev);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "sync");
  uint32_t st = 0;
  e = cudaMemcpy(&st, c->status, 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "status read");
  if (bits) *bits = st;
  if (st != 0) {
    // a kernel gave up part-way: clear the status and the arrival counters so the
    // context can be used again
    cudaMemset(c->status, 0, 4);
    cudaMemset(c->gemm_cnt, 0, c->gemm_cnt_bytes);
    cudaMemset(c->att_cnt, 0, c->att_cnt_cap * 4);
    cudaMemset(c->acc_cnt, 0, static_cast<size_t>(c->p.max_batch) * 4);
    cudaMemset(c->smp_cnt, 0, static_cast<size_t>(c->p.max_batch) * 4);
    return fail(c, MEMSPEC_ERR_DEVICE_STATUS, "device status word set");
  }
  return MEMSPEC_OK;
}

memspec_status memspec_query_info(memspec_ctx* c, int32_t what, int64_t* value) {
  if (c == nullptr || value == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  switch (what) {
    case MEMSPEC_INFO_DRAFT_LAUNCHES: *value = c->last_launches[0]; break;
    case MEMSPEC_INFO_VERIFY_LAUNCHES: *value = c->last_launches[1]; break;
    case MEMSPEC_INFO_ACCEPT_LAUNCHES: *value = c->last_launches[2]; break;
    case MEMSPEC_INFO_DRAFT_FUSED: *value = c->last_draft_fused ? 1 : 0; break;
    default: return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown info id");
  }
  return MEMSPEC_OK;
}

static memspec_status buffer_span(memspec_ctx* c, int32_t buf, void** ptr, size_t* cap) {
  const int B = c->p.max_batch, K = c->p.max_k, V = c->vocab;
  switch (buf) {
    case MEMSPEC_BUF_TARGET_LOGITS: *ptr = c->zt; *cap = static_cast<size_t>(B) * (K + 1) * V * 4; break;
    case MEMSPEC_BUF_DRAFT_LOGITS: *ptr = c->zd; *cap = static_cast<size_t>(B) * K * V * 4; break;
    case MEMSPEC_BUF_DRAFT_TOKENS: *ptr = c->draft_tokens; *cap = static_cast<size_t>(B) * K * 4; break;
    case MEMSPEC_BUF_TOKENS: *ptr = c->tokens; *cap = static_cast<size_t>(B) * c->p.max_seq * 4; break;
    case MEMSPEC_BUF_SEQ_STATE: *ptr = c->state; *cap = static_cast<size_t>(B) * kStateInts * 4; break;
    case MEMSPEC_BUF_ACCEPT_DEBUG: *ptr = c->acc_dbg; *cap = static_cast<size_t>(B) * (2 * K + 2) * 4; break;
    case MEMSPEC_BUF_RESIDUAL: *ptr = c->h; *cap = static_cast<size_t>(kMaxRows) * c->p.target.d_model * 4; break;
    case MEMSPEC_BUF_SEEDS: *ptr = c->seeds; *cap = static_cast<size_t>(B) * 8; break;
    case MEMSPEC_BUF_TREE_LOGITS: *ptr = c->tree_z; *cap = static_cast<size_t>(kTreeRows) * V * 4; break;
    case MEMSPEC_BUF_PASS_TRACE:
      if (c->trace == nullptr) return fail(c, MEMSPEC_ERR_INVALID_ARG, "tracing is off (init param trace)");
      *ptr = c->trace;
      *cap = (2 + static_cast<size_t>(kPassTraceOps) * sm_count() * kPassTraceSlots) * 8;
      break;
    default: return fail(c, MEMSPEC_ERR_INVALID_ARG, "unknown buffer id");
  }
  return MEMSPEC_OK;
}

memspec_status memspec_read_buffer(memspec_ctx* c, int32_t buf, void* dst, size_t bytes) {
  if (c == nullptr || dst == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  void* p;
  size_t cap;
  memspec_status s = buffer_span(c, buf, &p, &cap);
  if (s != MEMSPEC_OK) return s;
  if (bytes > cap) return fail(c, MEMSPEC_ERR_INVALID_ARG, "read larger than the buffer");
  cudaError_t e = cudaStreamSynchronize(c->main);
  if (e == cudaSuccess) e = cudaMemcpy(dst, p, bytes, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "read buffer");
  if (buf == MEMSPEC_BUF_SEQ_STATE && c->active >= 0) {
    // slot 3 of each request reports the active draft's processed count
    std::vector<int> dl(c->p.max_batch);
    e = cudaMemcpy(dl.data(), c->drafts[c->active].d_len, dl.size() * 4, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "read draft lengths");
    int* out = static_cast<int*>(dst);
    for (size_t b = 0; b < dl.size() && (b * kStateInts + 3) * 4 < bytes; ++b) out[b * kStateInts + 3] = dl[b];
  }
  return MEMSPEC_OK;
}

memspec_status memspec_write_buffer(memspec_ctx* c, int32_t buf, const void* src, size_t bytes) {
  if (c == nullptr || src == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (buf != MEMSPEC_BUF_TARGET_LOGITS && buf != MEMSPEC_BUF_DRAFT_LOGITS &&
      buf != MEMSPEC_BUF_DRAFT_TOKENS && buf != MEMSPEC_BUF_TOKENS && buf != MEMSPEC_BUF_SEQ_STATE &&
      buf != MEMSPEC_BUF_SEEDS)
    return fail(c, MEMSPEC_ERR_INVALID_ARG, "buffer is not writable");
  void* p;
  size_t cap;
  memspec_status s = buffer_span(c, buf, &p, &cap);
  if (s != MEMSPEC_OK) return s;
  if (bytes > cap) return fail(c, MEMSPEC_ERR_INVALID_ARG, "write larger than the buffer");
  cudaError_t e = cudaStreamSynchronize(c->main);
  if (e == cudaSuccess) e = cudaMemcpy(p, src, bytes, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "write buffer");
  if (buf == MEMSPEC_BUF_SEQ_STATE && c->active >= 0) {
    // slot 3 sets the active draft's processed count
    const int* in = static_cast<const int*>(src);
    for (size_t b = 0; (b * kStateInts + 3) * 4 < bytes && b < static_cast<size_t>(c->p.max_batch); ++b) {
      e = cudaMemcpy(c->drafts[c->active].d_len + b, in + b * kStateInts + 3, 4, cudaMemcpyHostToDevice);
      if (e != cudaSuccess) return cuda_fail(c, e, "write draft length");
    }
  }
  return MEMSPEC_OK;
}

// ---------------------------------------------------------------- op-level entry points
const char* memspec_op_last_error(void) { return g_op_error.c_str(); }
}  // extern "C"

void memspec::set_op_error(const char* msg) { g_op_error = msg; }

extern "C" {

static size_t op_linear_scratch(int rows, int n_out, int k) {
  const int n_pad = round_up(rows, 16);
  const int rt = ceil_div(n_out, 128);
  (void)k;
  // partials, then one arrival counter per row tile
  return align256(static_cast<size_t>(2) * sm_count() * n_pad * 128 * 4) +
         align256(static_cast<size_t>(rt) * 4) + 256;
}

memspec_status memspec_op_linear_scratch_bytes(int32_t rows, int32_t n_out, int32_t k, size_t* bytes) {
  if (bytes == nullptr || rows < 1 || rows > kMaxRows || n_out < 1 || k < 8) return MEMSPEC_ERR_INVALID_ARG;
  *bytes = op_linear_scratch(rows, n_out, k);
  return MEMSPEC_OK;
}

memspec_status memspec_pack_matrix(const void* src, const void* src2, int32_t n, int32_t k,
                                   void* dst, size_t dst_bytes, void* stream) {
  if (src == nullptr || dst == nullptr) {
    g_op_error = "null pointer";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (n < 1 || k < 8 || k % 8 != 0) {
    g_op_error = "n >= 1 and k a positive multiple of 8";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(src) & 15) || (reinterpret_cast<uintptr_t>(src2) & 15) ||
      (reinterpret_cast<uintptr_t>(dst) & 15)) {
    g_op_error = "src, src2 and dst must be 16-byte aligned";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (dst_bytes < packed_bytes(n, k, src2 != nullptr)) {
    g_op_error = "dst smaller than the packed size";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  cudaError_t e = launch_pack(static_cast<const bf16*>(src), static_cast<const bf16*>(src2), n, k,
                              static_cast<uint8_t*>(dst), static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    g_op_error = std::string("pack launch: ") + cudaGetErrorString(e);
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

memspec_status memspec_op_linear(const void* x, const void* w, float* y, int32_t rows, int32_t n_out,
                                 int32_t k, void* scratch, size_t scratch_bytes, uint32_t* status,
                                 void* stream) {
  if (x == nullptr || w == nullptr || y == nullptr || scratch == nullptr) {
    g_op_error = "null pointer";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (rows < 1 || rows > kMaxRows || n_out < 1 || k < 8 || k % 8 != 0 ||
      !sk_fits(static_cast<long long>(ceil_div(n_out, 128)) * ceil_div(k, 64), sm_count())) {
    g_op_error = "rows must be in 1..256, n_out >= 1, k a positive multiple of 8, "
                 "and ceil(n_out/128) * ceil(k/64) below 2^32 / (SMs + 1)";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(w) & 15) ||
      (reinterpret_cast<uintptr_t>(scratch) & 255)) {
    g_op_error = "x and w must be 16-byte aligned, scratch 256-byte aligned";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (scratch_bytes < op_linear_scratch(rows, n_out, k)) {
    g_op_error = "scratch too small";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (!ensure_func_attrs()) {
    g_op_error = g_attr_error;
    return MEMSPEC_ERR_CUDA;
  }
  GemmArgs a{};
  if (!encode_map(&a.map_a, w, n_out, k, 128)) {
    g_op_error = "cuTensorMapEncodeTiled failed";
    return MEMSPEC_ERR_CUDA;
  }
  const int n_pad = round_up(rows, 16);
  a.n_out = n_out;
  a.k_in = k;
  a.rows_total = rows;
  a.n_pad = n_pad;
  a.row_tiles = ceil_div(n_out, 128);
  a.k_tiles = ceil_div(k, 64);
  a.stages = gemm_pick_stages(n_pad);
  a.l2_hint = L2_EVICT_FIRST;
  if (!encode_map(&a.map_b, x, rows, k, n_pad)) {
    g_op_error = "cuTensorMapEncodeTiled failed for x";
    return MEMSPEC_ERR_CUDA;
  }
  a.epi = EPI_F32;
  a.out = y;
  a.out_ld = n_out;
  uint8_t* sb = static_cast<uint8_t*>(scratch);
  a.partials = reinterpret_cast<float*>(sb);
  const size_t part_bytes = align256(static_cast<size_t>(2) * sm_count() * n_pad * 128 * 4);
  a.counters = reinterpret_cast<int*>(sb + part_bytes);
  a.status = status != nullptr ? status
                               : reinterpret_cast<uint32_t*>(sb + part_bytes +
                                                             align256(static_cast<size_t>(a.row_tiles) * 4));
  a.plan = nullptr;
  const int grid = gemm_grid(a.row_tiles, a.k_tiles);
  // more than 16 rows: split row tiles finished by the split epilogue kernel (as
  // in the passes)
  a.split_epi = (n_pad >= 32 && !sk_split_free(a.row_tiles * a.k_tiles, a.k_tiles, grid)) ? 1 : 0;
  cudaError_t e = launch_gemm(a, grid, gemm_smem_bytes(n_pad, a.stages),
                              static_cast<cudaStream_t>(stream), false);
  if (e == cudaSuccess && a.split_epi)
    e = launch_gemm_split_epi(a, grid, static_cast<cudaStream_t>(stream), false);
  if (e != cudaSuccess) {
    g_op_error = std::string("gemm launch: ") + cudaGetErrorString(e);
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

int64_t memspec_int4_packed_bytes(int32_t n_out, int32_t k) {
  if (n_out < 1 || k < 128 || k % 128 != 0) return -1;
  return static_cast<int64_t>(int4_packed_bytes(n_out, k));
}

memspec_status memspec_int4_pack(const void* qweight, const void* scales, const void* zeros, int32_t n_out,
                                 int32_t k, void* packed, void* stream) {
  if (qweight == nullptr || scales == nullptr || zeros == nullptr || packed == nullptr) {
    g_op_error = "null pointer";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (n_out < 1 || k < 128 || k % 128 != 0 || n_out > (1 << 20)) {
    g_op_error = "n_out in 1..1048576 and k a positive multiple of 128 required";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(qweight) & 3) || (reinterpret_cast<uintptr_t>(scales) & 1) ||
      (reinterpret_cast<uintptr_t>(packed) & 15)) {
    g_op_error = "qweight must be 4-byte, scales 2-byte and packed 16-byte aligned";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  cudaError_t e = launch_int4_pack(static_cast<const uint8_t*>(qweight), static_cast<const bf16*>(scales),
                                   static_cast<const uint8_t*>(zeros), static_cast<uint8_t*>(packed), n_out, k,
                                   static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    g_op_error = std::string("int4 pack launch: ") + cudaGetErrorString(e);
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

memspec_status memspec_op_linear_int4(const void* x, const void* packed, float* y, int32_t rows,
                                      int32_t n_out, int32_t k, uint32_t* status, void* stream) {
  if (x == nullptr || packed == nullptr || y == nullptr) {
    g_op_error = "null pointer";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (rows < 1 || rows > kInt4MaxRows || n_out < 1 || k < 128 || k % 128 != 0 || n_out > (1 << 20)) {
    g_op_error = "rows in 1..16, n_out in 1..1048576 and k a positive multiple of 128 required";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(packed) & 15) ||
      (reinterpret_cast<uintptr_t>(y) & 3)) {
    g_op_error = "x and packed must be 16-byte aligned, y 4-byte aligned";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (int4_pick_depth(rows, k) == 0) {
    g_op_error = "rows x k too large for the activations and a 2-record ring per warp in shared memory";
    return MEMSPEC_ERR_UNSUPPORTED;
  }
  if (!ensure_func_attrs()) {
    g_op_error = g_attr_error;
    return MEMSPEC_ERR_CUDA;
  }
  // whole 16-row tiles, the same number per CTA, at most one CTA per SM
  const Int4Plan plan = int4_plan(rows, n_out, k, sm_count());
  Int4Args a{};
  a.x = static_cast<const bf16*>(x);
  a.packed = static_cast<const uint8_t*>(packed);
  a.y = y;
  a.rows = rows;
  a.n = n_out;
  a.k = k;
  a.tiles_per_cta = plan.tiles_per_cta;
  a.status = status;
  cudaError_t e = launch_int4_linear(a, plan, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    g_op_error = std::string("int4 launch: ") + cudaGetErrorString(e);
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

memspec_status memspec_op_sample(const float* logits, int32_t rows, int32_t vocab, float T,
                                 const float* u, int32_t* out, void* stream) {
  if (logits == nullptr || out == nullptr || rows < 1 || rows > 65535 || vocab < 1 ||
      vocab > 131072 || !(T >= 0.f) || (T > 0.f && u == nullptr)) {
    g_op_error = "invalid sampling arguments";
    return MEMSPEC_ERR_INVALID_ARG;
  }
  SampleArgs sa{};
  sa.logits = logits;
  sa.row_stride = vocab;
  sa.vocab = vocab;
  sa.n_groups = rows;
  sa.greedy = T == 0.f;
  sa.inv_temp = T == 0.f ? 0.f : 1.f / T;
  sa.u_explicit = u;
  sa.out_tok = out;
  sa.out_stride = 1;
  cudaError_t e = launch_sample(sa, static_cast<cudaStream_t>(stream), false);
  if (e != cudaSuccess) {
    g_op_error = std::string("sample launch: ") + cudaGetErrorString(e);
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

}  // extern "C"
