// sampling.cu - the draft-token sampler and the acceptance / resample / commit
// kernel (algorithms in sample_body.cuh).
#include "internal.h"
#include "ptx.cuh"
#include "sample_body.cuh"

namespace memspec {

namespace {

using namespace smp;

constexpr int kSThreads = 512;

// one CTA per group
__global__ void __launch_bounds__(kSThreads) sample_kernel(const __grid_constant__ SampleArgs a) {
  __shared__ SampleSmem sm;
  pdl_launch_dependents();
  pdl_wait();
  sample_group<kSThreads>(a, blockIdx.x, sm, threadIdx.x, [] { __syncthreads(); });
}

// grid (2K+1 rows, groups): row statistics per CTA; the last CTA of a group decides
__global__ void __launch_bounds__(kSThreads) accept_kernel(const __grid_constant__ AcceptArgs a) {
  __shared__ SampleSmem sm;
  pdl_launch_dependents();
  pdl_wait();
  accept_row<kSThreads>(a, blockIdx.x, blockIdx.y, sm, threadIdx.x, [] { __syncthreads(); });
}

}  // namespace

cudaError_t launch_sample(const SampleArgs& a, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_groups);
  cfg.blockDim = dim3(kSThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, sample_kernel, a);
}

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * a.K + 1, a.n_groups);
  cfg.blockDim = dim3(kSThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, accept_kernel, a);
}

}  // namespace memspec
