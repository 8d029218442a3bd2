// attention.cu - split-KV flash-decode attention for the verify / draft / prefill
// passes: causal grouped-query attention of a few query positions per request
// against that request's KV cache.
//
// Grid: (key split, kv_head x row_block, request group).  A CTA takes the query
// vectors of one KV head's group of query heads for a block of rows (at most 64
// vectors, 16 per m-tile), streams its share of the keys/values (the context
// spread evenly over the splits, whole 64-key tiles) once through a ring of TMA
// boxes (128-byte swizzle, mbarrier per stage, 3 stages; 2 in the transposed
// form; the tiles below the pass's first new position are requested before the
// launch waits for its predecessor) and computes on tensor cores (mma.sync
// m16n8k16, bf16 in, fp32 accumulate):
//   S = Q K^T (Q pre-scaled by log2(e)/sqrt(hd), loaded straight into the
//   A-operand registers), online softmax in registers (running max m, sum l),
//   O += P V with P re-packed from the S fragments.
// Q and P are carried as two bf16 planes (hi + lo, two MMAs each), so only the
// bf16 K/V cache limits the precision; the output is written as hi + lo planes.
// With few query vectors the four warps split each 64-key tile between them
// and are merged at the end.  Each split writes (m, l, o) to a partial buffer;
// the last-arriving split CTA of each (group, kv head, row block) lands every
// split's partial in shared memory and combines them in split order
// (deterministic, no float atomics):
//   o = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s.
// Query row i of a group sits at position pos0 + i and sees keys 0..pos0+i.
#include "attn_body.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace memspec {

namespace {

using namespace attn;

template <int HD, bool TQ>
__global__ void __launch_bounds__(kAttThreads, TQ ? 3 : 2) attn_kernel(const __grid_constant__ AttnArgs a) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  __shared__ uint64_t bars[kStages];   // TMA stages
  if (a.tma && threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
    tma_prefetch_desc(&a.kmap);
    tma_prefetch_desc(&a.vmap);
  }
  __syncthreads();
  pdl_launch_dependents();
  const int lin = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
  unsigned long long* trace =
      (a.trace != nullptr && threadIdx.x == 0 && lin < a.trace_ctas) ? a.trace + lin * 16 : nullptr;
  trace_at(trace, 0);
  auto sync = [] { __syncthreads(); };
  // dry run while the previous kernel finishes: warms this code, writes no
  // global memory (see attention_cta)
  attention_cta<HD, TQ>(a, 0, 0, 0, 0, smem_raw, threadIdx.x, sync, [] {}, false, nullptr, true);
  __syncthreads();
  // the dry run wrote the stages through the generic proxy; the copies into them
  // come through the async proxy
  if (a.tma && threadIdx.x == 0) fence_proxy_async_smem();
  auto wait = [&] {
    pdl_wait();
    trace_at(trace, 13);
  };
  const int kvh = blockIdx.y / a.row_blocks, rb = blockIdx.y - kvh * a.row_blocks;
  attention_cta<HD, TQ>(a, blockIdx.z, kvh, rb, blockIdx.x, smem_raw, threadIdx.x, sync, wait,
                    a.ctx_early != 0, trace, false, a.tma ? bars : nullptr);
  trace_at(trace, 1);
}

}  // namespace

size_t attention_smem_bytes(const AttnArgs& a) {
  const bool tq = a.qmax <= 8;
  if (a.hd == 64) return tq ? attention_smem_bytes_hd<64, true>() : attention_smem_bytes_hd<64, false>();
  return tq ? attention_smem_bytes_hd<128, true>() : attention_smem_bytes_hd<128, false>();
}
cudaError_t attention_set_max_smem() {
  for (const void* f : {reinterpret_cast<const void*>(attn_kernel<64, false>),
                        reinterpret_cast<const void*>(attn_kernel<64, true>),
                        reinterpret_cast<const void*>(attn_kernel<128, false>),
                        reinterpret_cast<const void*>(attn_kernel<128, true>)}) {
    const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_attention(const AttnArgs& a, int n_groups, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_splits, a.Hkv * a.row_blocks, n_groups);
  cfg.blockDim = dim3(kAttThreads);
  cfg.dynamicSmemBytes = attention_smem_bytes(a);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  // at most 8 query vectors per CTA: the transposed form (keys as the MMA's M side)
  const bool tq = a.qmax <= 8;
  if (a.hd == 64) return tq ? cudaLaunchKernelEx(&cfg, attn_kernel<64, true>, a)
                            : cudaLaunchKernelEx(&cfg, attn_kernel<64, false>, a);
  if (a.hd == 128) return tq ? cudaLaunchKernelEx(&cfg, attn_kernel<128, true>, a)
                             : cudaLaunchKernelEx(&cfg, attn_kernel<128, false>, a);
  return cudaErrorInvalidValue;
}

}  // namespace memspec
