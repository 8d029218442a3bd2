// tree.cu - the end of a tree verification step (the engine MemSpec is built on
// verifies draft trees, Section 3.5): after the tree pass has scored the root
// and every node, and one token has been drawn from each row's target
// distribution (the sampler, Philox slot kTreeSlot0 + emitted index), the walk
// descends from the root: while the drawn token is the token of a child of the
// current row, that child is accepted; the first drawn token that is no child
// ends the step.  Every emitted token is a draw from the target's own
// conditional distribution.  The accepted nodes' K / V then move to the
// consecutive slots after the root, so the cache is what a chain of the
// committed tokens would have written.
#include "internal.h"
#include "pass.h"

namespace memspec {

namespace {

// One thread: at most kTreeRows steps over a tree of at most kTreeRows rows.
__global__ void tree_walk_kernel(const TreeWalkArgs a) {
  if (threadIdx.x != 0) return;
  const TreeDesc& t = *a.tree;
  const int n_rows = t.n_rows;
  const int L = a.seq_state[0];
  TreeResult* r = a.result;
  int v = 0, n = 0;
  for (int e = 0; e < n_rows; ++e) {
    const int x = a.samples[v];
    r->emitted[n++] = x;
    int next = -1;
    for (int c = v + 1; c < n_rows; ++c)   // children follow their parent; the lowest index wins
      if (t.parent_row[c] == v && t.tokens[c] == x) {
        next = c;
        break;
      }
    if (next < 0) break;
    r->rows[n - 1] = next;
    v = next;
  }
  r->L_before = L;
  if (L < 1 || L + n > a.max_seq) {   // nothing committed
    r->n_emit = 0;
    atomicOr(a.status, 0x4u);
  } else {
    for (int e = 0; e < n; ++e) a.tokens[L + e] = r->emitted[e];
    r->n_emit = n;
    a.seq_state[0] = L + n;       // committed length
    a.seq_state[1] = L + n - 1;   // target KV valid below: the root and the accepted nodes
  }
  a.seq_state[2] += 1;            // step counter (Philox)
}

// Grid (Hkv, layers, K|V); 32 threads copy one hd-element row at a time.  The
// accepted rows ascend (children follow parents) and row rows[e] sits at slot
// L - 1 + rows[e] >= L + e, so copying in ascending e never overwrites a row
// that a later copy still has to read.
__global__ void tree_compact_kernel(const TreeCompactArgs a) {
  const TreeResult& r = *a.result;
  const int n_acc = r.n_emit - 1;
  if (n_acc <= 0) return;
  const int head = blockIdx.x, layer = blockIdx.y, kv = blockIdx.z;
  bf16* base = a.kv + static_cast<size_t>(layer) * 2 * a.layer_kv + (kv ? a.layer_kv : 0) +
               static_cast<size_t>(head) * a.max_seq * a.hd;   // request 0
  const int L = r.L_before;
  for (int e = 0; e < n_acc; ++e) {
    const int src = L - 1 + r.rows[e], dst = L + e;
    if (src != dst) {
      for (int i = threadIdx.x * 8; i < a.hd; i += 32 * 8)
        *reinterpret_cast<uint4*>(base + static_cast<size_t>(dst) * a.hd + i) =
            *reinterpret_cast<const uint4*>(base + static_cast<size_t>(src) * a.hd + i);
    }
    __syncwarp();
  }
}

}  // namespace

cudaError_t launch_tree_walk(const TreeWalkArgs& a, cudaStream_t s) {
  tree_walk_kernel<<<1, 32, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_tree_compact(const TreeCompactArgs& a, int n_layers, cudaStream_t s) {
  tree_compact_kernel<<<dim3(a.Hkv, n_layers, 2), 32, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace memspec
