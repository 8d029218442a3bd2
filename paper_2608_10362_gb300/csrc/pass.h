// pass.h - op list of a forward pass, shared by the host runtime (which builds it)
// and the persistent pass kernel (which executes it).  Every op can also be run
// as its own kernel launch (prefill, and the separate-launch mode).
#pragma once
#include "internal.h"

namespace memspec {

// OP_TREE_WALK / OP_TREE_COMPACT run only as their own launches (tree steps)
enum OpType : int { OP_EMBED = 0, OP_GEMM = 1, OP_ATTN = 2, OP_SAMPLE = 3, OP_ACCEPT = 4, OP_TREE_WALK = 5,
                    OP_TREE_COMPACT = 6, OP_GEMM_EPI = 7 };   // OP_GEMM_EPI: u.g, grid = the GEMM's

struct alignas(64) PassOp {
  int type;
  int grid;       // OP_GEMM: stream-K grid (CTAs with tiles)
  int n_units;    // OP_EMBED rows, OP_ATTN units, OP_SAMPLE groups, OP_ACCEPT rows x groups
  int smem;       // OP_GEMM as its own launch: dynamic shared memory bytes
  int full_dep;   // as its own launch: without programmatic dependent launch, so it
                  // starts after every earlier kernel has completed
  int pad[11];
  union U {
    GemmArgs g;
    AttnArgs at;
    EmbedArgs e;
    SampleArgs s;
    AcceptArgs acc;
    TreeWalkArgs tw;
    TreeCompactArgs tc;
  } u;
};

struct PassArgs {
  const PassOp* ops;   // device memory, n_ops entries
  int n_ops;
  int* done;           // [n_ops] completion counters, zero at launch (reset on exit)
  int* exit_cnt;       // zero at launch (reset on exit)
  int stages;          // weight/activation stage ring depth
  int b_stage_bytes;   // activation bytes per stage (max over the GEMM ops)
  int attn_bytes;      // attention shared memory (0: no attention op)
  uint32_t tmem_cols;  // TMEM columns allocated (power of two)
  uint32_t* status;
  // nullptr, or per-op timestamps (globaltimer ns) of this launch:
  // trace[0] = n_ops, trace[1] = grid, then [n_ops][grid][kPassTraceSlots] =
  // {worker start, worker end, activation loads issued, first MMA issued,
  //  partials / split outputs stored, arrival counted, reduction inputs loaded,
  //  reduction epilogue done, then epilogue-internal points 8..15} (slots an op
  //  does not reach keep older values)
  unsigned long long* trace;
};

constexpr int kPassTraceOps = 2048;   // ops a trace buffer holds
constexpr int kPassTraceSlots = 16;

size_t pass_smem_bytes(const PassArgs& p);
int pass_pick_stages(int b_stage_bytes, int attn_bytes);
size_t pass_attn_bytes(int hd);
cudaError_t pass_set_max_smem();
cudaError_t launch_pass(const PassArgs& p, int grid, cudaStream_t s, bool cooperative);

}  // namespace memspec
