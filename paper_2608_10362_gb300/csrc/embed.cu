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
#include "embed_body.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace memspec {

namespace {

// one CTA per row
__global__ void __launch_bounds__(256) embed_kernel(const __grid_constant__ EmbedArgs a) {
  __shared__ float red[8];
  pdl_launch_dependents();
  pdl_wait();
  emb::embed_row<256>(a, blockIdx.x, red, threadIdx.x, [] { __syncthreads(); });
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
