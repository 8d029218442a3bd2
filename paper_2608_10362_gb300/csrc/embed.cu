// embed.cu - row plan + token-embedding gather that starts every forward pass,
// and the RoPE cos/sin table.
//
// The plan decides, on the device and from the device-resident sequence state,
// which tokens a pass feeds and at which positions, so that a captured CUDA
// graph of the step replays correctly whatever the accepted lengths were:
//   verify       rows [t_{L-1}, x_1..x_K]          at positions L-1 .. L-1+K
//   draft pass 1 the committed tokens the draft has not processed yet
//                (1 token, or 2 after a fully accepted step) from Ld .. L-1
//   draft pass j x_{j-1}                            at position L+j-2
//   prefill      a chunk of committed tokens       from `start`
#include "internal.h"
#include "ptx.cuh"

namespace memspec {

namespace {

__device__ void compute_group(const EmbedArgs& a, int g, int* req, int* valid, int* pos0) {
  if (a.mode == PLAN_PREFILL) {
    *req = a.prefill_req;
    *valid = a.prefill_count;
    *pos0 = a.prefill_start;
    return;
  }
  *req = g;
  const int L = a.seq_state[g * kStateInts + 0];
  if (a.mode == PLAN_VERIFY) {
    *valid = a.R;
    *pos0 = L - 1;
  } else if (a.mode == PLAN_DRAFT_FIRST) {
    const int ld = a.draft_len[g];
    int n = L - ld;
    if (n < 1 || n > a.R) {
      atomicOr(a.status, 0x4u);  // draft cache not caught up with the committed tokens
      n = n < 1 ? 1 : a.R;
    }
    *valid = n;
    *pos0 = L - n;
  } else {  // PLAN_DRAFT_NEXT
    *valid = 1;
    *pos0 = L + a.j - 2;
  }
}

__device__ int row_token(const EmbedArgs& a, int req, int pos, int i) {
  const int L = a.mode == PLAN_PREFILL ? 0 : a.seq_state[req * kStateInts + 0];
  if (a.mode == PLAN_VERIFY) {
    return i == 0 ? a.tokens[static_cast<size_t>(req) * a.max_seq + L - 1]
                  : a.draft_tokens[req * a.max_k + i - 1];
  }
  if (a.mode == PLAN_DRAFT_NEXT) return a.draft_tokens[req * a.max_k + a.j - 2];
  return a.tokens[static_cast<size_t>(req) * a.max_seq + pos];
}

// one CTA per row
__global__ void __launch_bounds__(256) embed_kernel(const __grid_constant__ EmbedArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int r = blockIdx.x;
  const int g = r / a.R, i = r - g * a.R;
  int req, valid, pos0;
  compute_group(a, g, &req, &valid, &pos0);
  if (r == 0 && threadIdx.x < a.n_groups) {
    int rq, vl, p0;
    compute_group(a, threadIdx.x, &rq, &vl, &p0);
    a.plan->req[threadIdx.x] = rq;
    a.plan->valid[threadIdx.x] = vl;
    a.plan->pos0[threadIdx.x] = p0;
  }
  if (r == 0 && threadIdx.x == 0) {
    a.plan->n_groups = a.n_groups;
    a.plan->rows_per_group = a.R;
    a.plan->rows_total = a.n_groups * a.R;
    int mp = 0;
    for (int gg = 0; gg < a.n_groups; ++gg) {
      int rq, vl, p0;
      compute_group(a, gg, &rq, &vl, &p0);
      mp = max(mp, p0 + vl - 1);
    }
    a.plan->max_pos = mp;
  }
  float* hr = a.h + static_cast<size_t>(r) * a.d;
  __shared__ float red[8];
  float sq = 0.f;
  const bool ok = i < valid;
  int tok = 0;
  if (ok) {
    const int pos = pos0 + i;
    if (pos < 0 || pos >= a.max_seq) {
      if (threadIdx.x == 0) atomicOr(a.status, 0x4u);
    } else {
      tok = row_token(a, req, pos, i);
    }
    if (tok < 0 || tok >= a.vocab) {
      if (threadIdx.x == 0) atomicOr(a.status, 0x2u);
      tok = 0;
    }
  }
  const bf16* er = a.emb + static_cast<size_t>(tok) * a.d;
  for (int c = threadIdx.x * 8; c < a.d; c += blockDim.x * 8) {
    float f[8];
    if (ok) {
      const uint4 raw = *reinterpret_cast<const uint4*>(er + c);
      const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
      for (int q = 0; q < 8; ++q) f[q] = __bfloat162float(b[q]);
    } else {
#pragma unroll
      for (int q = 0; q < 8; ++q) f[q] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) sq += f[q] * f[q];
    reinterpret_cast<float4*>(hr + c)[0] = make_float4(f[0], f[1], f[2], f[3]);
    reinterpret_cast<float4*>(hr + c)[1] = make_float4(f[4], f[5], f[6], f[7]);
    // bf16(h * gain): the first projection's input, its RMSNorm scale applied
    // per row in that projection's epilogue
    const uint4 graw = *reinterpret_cast<const uint4*>(a.gain + c);
    const __nv_bfloat16* gb = reinterpret_cast<const __nv_bfloat16*>(&graw);
    __nv_bfloat16 o8[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) o8[q] = __float2bfloat16_rn(f[q] * __bfloat162float(gb[q]));
    *reinterpret_cast<uint4*>(a.xg + static_cast<size_t>(r) * a.d + c) =
        *reinterpret_cast<const uint4*>(o8);
    if (a.xg_lo != nullptr) {   // low-order plane: bf16(x - bf16(x))
      __nv_bfloat16 l8[8];
#pragma unroll
      for (int q = 0; q < 8; ++q)
        l8[q] = __float2bfloat16_rn(f[q] * __bfloat162float(gb[q]) - __bfloat162float(o8[q]));
      *reinterpret_cast<uint4*>(a.xg_lo + static_cast<size_t>(r) * a.d + c) =
          *reinterpret_cast<const uint4*>(l8);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sq;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
    a.ss[r] = s;
  }
}

__global__ void rope_table_kernel(float* cos_t, float* sin_t, int max_seq, int half, float base) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= max_seq * half) return;
  const int pos = idx / half, i = idx - pos * half;
  // angle = pos * base^(-2i/hd), hd = 2*half, evaluated in double
  const double theta = pow(static_cast<double>(base), -2.0 * i / (2.0 * half));
  double s, c;
  sincos(static_cast<double>(pos) * theta, &s, &c);
  cos_t[idx] = static_cast<float>(c);
  sin_t[idx] = static_cast<float>(s);
}

}  // namespace

cudaError_t launch_embed(const EmbedArgs& a, int rows, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(rows);
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, embed_kernel, a);
}

cudaError_t launch_rope_table(float* cos_t, float* sin_t, int max_seq, int half, float base,
                              cudaStream_t s) {
  const int n = max_seq * half;
  rope_table_kernel<<<(n + 255) / 256, 256, 0, s>>>(cos_t, sin_t, max_seq, half, base);
  return cudaGetLastError();
}

}  // namespace memspec
