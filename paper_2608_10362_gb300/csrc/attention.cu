// attention.cu - split-KV flash-decode attention for the verify / draft / prefill
// passes: causal grouped-query attention of a few query positions per request
// against that request's KV cache.
//
// Grid: (key split, kv_head x row_block, request group).  A CTA takes the query
// vectors of one KV head's group of query heads for a block of rows, streams its
// chunk of keys/values once, keeps an online softmax (running max m, sum l,
// unnormalised o) and writes (m, l, o) to a partial buffer.  The last-arriving
// split CTA of each (group, kv head, row block) combines the partials in split
// order (deterministic, no float atomics): o = sum_s e^(m_s - M) o_s /
// sum_s e^(m_s - M) l_s with M = max_s m_s.  Query row i of a group sits at
// position pos0 + i and sees keys 0..pos0+i.
#include "internal.h"
#include "ptx.cuh"

namespace memspec {

namespace {

constexpr int kAttThreads = 256;
constexpr int kKeyTile = 64;

__device__ __forceinline__ float dot8(const float* q, const uint4& raw) {
  const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&raw);
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(b[i]);
    s = fmaf(q[2 * i], f.x, s);
    s = fmaf(q[2 * i + 1], f.y, s);
  }
  return s;
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem_dst)), "l"(gsrc)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

template <int HD>
__global__ void __launch_bounds__(kAttThreads) attn_kernel(const __grid_constant__ AttnArgs a) {
  constexpr int kNvg = kAttThreads / HD;       // PV thread groups
  constexpr int kAcc = 32;                     // max query vectors per PV thread
  constexpr int kSv = 32;                      // max query vectors per score thread
  extern __shared__ __align__(16) uint8_t smem_raw[];
  pdl_launch_dependents();
  pdl_wait();

  const RowPlan* plan = a.plan;
  const int g = blockIdx.z;
  if (g >= plan->n_groups) return;
  const int kvh = blockIdx.y / a.row_blocks, rb = blockIdx.y - kvh * a.row_blocks;
  const int split = blockIdx.x;
  const int R = plan->rows_per_group;
  const int req = plan->req[g], valid = plan->valid[g], pos0 = plan->pos0[g];
  const int r_lo = rb * a.rows_per_block;
  const int r_hi = min(r_lo + a.rows_per_block, valid);
  if (r_lo >= r_hi) return;
  const int nr = r_hi - r_lo;
  const int gs = a.H / a.Hkv;
  const int nq = gs * nr;
  const int kmax = pos0 + r_hi - 1;
  if (pos0 < 0 || kmax >= a.max_seq) {   // out-of-range positions are reported, never read
    if (threadIdx.x == 0 && split == 0) atomicOr(a.status, 0x4u);
    return;
  }
  const int n_active = (kmax + a.chunk) / a.chunk;   // ceil((kmax + 1) / chunk)
  if (split >= n_active) return;
  const int k0 = split * a.chunk;
  const int k1 = min(k0 + a.chunk, kmax + 1);

  float* qs = reinterpret_cast<float*>(smem_raw);                  // [qmax][HD]
  float* sp = qs + a.qmax * HD;                                    // [qmax][kKeyTile]
  float* m_s = sp + a.qmax * kKeyTile;                             // [qmax]
  float* l_s = m_s + a.qmax;
  float* al_s = l_s + a.qmax;
  bf16* vs = reinterpret_cast<bf16*>(al_s + a.qmax + (4 - (3 * a.qmax) % 4) % 4);  // [kKeyTile][HD]

  const int tid = threadIdx.x;
  for (int idx = tid; idx < nq * HD; idx += kAttThreads) {
    const int v = idx / HD, d = idx - v * HD;
    const int hl = v / nr, rr = v - hl * nr;
    const int row = g * R + r_lo + rr;
    const int h = kvh * gs + hl;
    qs[idx] = a.q[(static_cast<size_t>(row) * a.H + h) * HD + d] * a.scale_log2;
  }
  for (int v = tid; v < nq; v += kAttThreads) {
    m_s[v] = -INFINITY;
    l_s[v] = 0.f;
  }
  const size_t kv_base = (static_cast<size_t>(req) * a.Hkv + kvh) * a.max_seq;
  const bf16* kc = a.kcache + kv_base * HD;
  const bf16* vc = a.vcache + kv_base * HD;

  const int pd = tid % HD, pvg = tid / HD;     // PV mapping
  float acc[kAcc];
#pragma unroll
  for (int i = 0; i < kAcc; ++i) acc[i] = 0.f;
  const int sj = tid % kKeyTile, svv = tid / kKeyTile;   // score mapping (4 groups)
  __syncthreads();

  for (int kt0 = k0; kt0 < k1; kt0 += kKeyTile) {
    const int nk = min(kKeyTile, k1 - kt0);
    // V tile -> shared memory (async, overlaps the score computation)
    for (int c = tid; c < nk * (HD / 8); c += kAttThreads) {
      const int j = c / (HD / 8), cc = c - j * (HD / 8);
      cp_async16(vs + j * HD + cc * 8, vc + static_cast<size_t>(kt0 + j) * HD + cc * 8);
    }
    // scores: thread (key sj, query vectors svv, svv+4, ...)
    {
      float s[kSv];
#pragma unroll
      for (int i = 0; i < kSv; ++i) s[i] = 0.f;
      if (sj < nk) {
        const bf16* krow = kc + static_cast<size_t>(kt0 + sj) * HD;
#pragma unroll 4
        for (int dc = 0; dc < HD / 8; ++dc) {
          const uint4 raw = __ldg(reinterpret_cast<const uint4*>(krow) + dc);
#pragma unroll
          for (int i = 0; i < kSv; ++i) {
            const int v = svv + 4 * i;
            if (v < nq) s[i] += dot8(qs + v * HD + dc * 8, raw);
          }
        }
      }
#pragma unroll
      for (int i = 0; i < kSv; ++i) {
        const int v = svv + 4 * i;
        if (v < nq) {
          const int rr = v % nr;
          const int pos = pos0 + r_lo + rr;
          const int key = kt0 + sj;
          sp[v * kKeyTile + sj] = (sj < nk && key <= pos) ? s[i] : -INFINITY;
        }
      }
    }
    __syncthreads();
    // online softmax update, one warp per query vector
    {
      const int w = tid >> 5, lane = tid & 31;
      for (int v = w; v < nq; v += kAttThreads / 32) {
        const float x0 = sp[v * kKeyTile + lane], x1 = sp[v * kKeyTile + lane + 32];
        float mx = fmaxf(x0, x1);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = m_s[v];
        const float m_new = fmaxf(m_old, mx);
        float p0 = 0.f, p1 = 0.f, alpha = 1.f;
        if (m_new != -INFINITY) {
          p0 = exp2f(x0 - m_new);
          p1 = exp2f(x1 - m_new);
          alpha = exp2f(m_old - m_new);
        }
        sp[v * kKeyTile + lane] = p0;
        sp[v * kKeyTile + lane + 32] = p1;
        float sum = p0 + p1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) {
          l_s[v] = l_s[v] * alpha + sum;
          m_s[v] = m_new;
          al_s[v] = alpha;
        }
      }
    }
    cp_async_wait_all();
    __syncthreads();
    // o += p V
#pragma unroll
    for (int i = 0; i < kAcc; ++i) {
      const int v = pvg + kNvg * i;
      if (v < nq) {
        float o = acc[i] * al_s[v];
        const float* pr = sp + v * kKeyTile;
        for (int j = 0; j < nk; ++j) o = fmaf(pr[j], __bfloat162float(vs[j * HD + pd]), o);
        acc[i] = o;
      }
    }
    __syncthreads();
  }

  // partials -> global
  const int unit = (g * a.Hkv + kvh) * a.row_blocks + rb;
  const size_t pbase = (static_cast<size_t>(unit) * a.n_splits + split) * a.qmax;
#pragma unroll
  for (int i = 0; i < kAcc; ++i) {
    const int v = pvg + kNvg * i;
    if (v < nq) a.part_o[(pbase + v) * HD + pd] = acc[i];
  }
  for (int v = tid; v < nq; v += kAttThreads) {
    a.part_ml[(pbase + v) * 2 + 0] = m_s[v];
    a.part_ml[(pbase + v) * 2 + 1] = l_s[v];
  }
  __threadfence();
  __syncthreads();
  __shared__ int last;
  if (tid == 0) last = (atomicAdd(&a.counters[unit], 1) == n_active - 1) ? 1 : 0;
  __syncthreads();
  if (!last) return;
  __threadfence();
  const size_t ubase = static_cast<size_t>(unit) * a.n_splits * a.qmax;
  for (int idx = tid; idx < nq * HD; idx += kAttThreads) {
    const int v = idx / HD, d = idx - v * HD;
    float M = -INFINITY;
    for (int s = 0; s < n_active; ++s) M = fmaxf(M, ld_cg_f(a.part_ml + (ubase + s * a.qmax + v) * 2));
    float L = 0.f, O = 0.f;
    for (int s = 0; s < n_active; ++s) {
      const size_t pv = ubase + s * a.qmax + v;
      const float ms = ld_cg_f(a.part_ml + pv * 2);
      const float w = ms == -INFINITY ? 0.f : exp2f(ms - M);
      L += w * ld_cg_f(a.part_ml + pv * 2 + 1);
      O += w * ld_cg_f(a.part_o + pv * HD + d);
    }
    const int hl = v / nr, rr = v - hl * nr;
    const int row = g * R + r_lo + rr;
    const int h = kvh * gs + hl;
    a.out[(static_cast<size_t>(row) * a.H + h) * HD + d] = __float2bfloat16_rn(O / L);
  }
  if (tid == 0) a.counters[unit] = 0;
}

}  // namespace

size_t attention_smem_bytes(const AttnArgs& a) {
  const size_t f = static_cast<size_t>(a.qmax) * a.hd + static_cast<size_t>(a.qmax) * kKeyTile +
                   3 * a.qmax + 4;
  return f * 4 + static_cast<size_t>(kKeyTile) * a.hd * 2;
}

cudaError_t attention_set_max_smem() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       160 * 1024);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              160 * 1024);
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
  if (a.hd == 64) return cudaLaunchKernelEx(&cfg, attn_kernel<64>, a);
  if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_kernel<128>, a);
  return cudaErrorInvalidValue;
}

}  // namespace memspec
