// pack.cu - row-major bf16 weights -> packed tiles (see packed_bytes in internal.h).
//
// The projection GEMM streams its weights with 1-D bulk copies of whole tiles:
// a tile is stored in HBM exactly as the tensor cores read it from shared memory
// (128 rows of 128 bytes, 16-byte chunks permuted by the 128-byte swizzle), and
// tiles follow the GEMM's stream-K order, so each CTA's range is one contiguous
// run of bytes.  Runs once per model when its blob is filled.
#include "internal.h"

namespace memspec {

namespace {

// one CTA per tile; 128 threads x 8 chunks of 16 bytes
__global__ void __launch_bounds__(128) pack_kernel(const bf16* __restrict__ src,
                                                   const bf16* __restrict__ src2, int n, int k,
                                                   int k_tiles, uint8_t* __restrict__ dst) {
  const int tile = blockIdx.x;
  const int rt = tile / k_tiles, kt = tile - rt * k_tiles;
  uint8_t* out = dst + static_cast<size_t>(tile) * kPackTileBytes;
  for (int q = threadIdx.x; q < 1024; q += 128) {
    const int r = q >> 3, c = q & 7;
    const bf16* base;
    int row;
    if (src2 != nullptr) {   // pair: 64 rows of each matrix
      row = rt * 64 + (r & 63);
      base = r < 64 ? src : src2;
    } else {
      row = rt * 128 + r;
      base = src;
    }
    const int col = kt * 64 + c * 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (row < n && col < k) {   // k is a multiple of 8: a chunk is all in or all out
      v = *reinterpret_cast<const uint4*>(base + static_cast<size_t>(row) * k + col);
    }
    *reinterpret_cast<uint4*>(out + r * 128 + ((c ^ (r & 7)) << 4)) = v;
  }
}

}  // namespace

cudaError_t launch_pack(const bf16* src, const bf16* src2, int n, int k, uint8_t* dst,
                        cudaStream_t s) {
  const int rt = src2 != nullptr ? (n + 63) / 64 : (n + 127) / 128;
  const int kt = (k + 63) / 64;
  pack_kernel<<<rt * kt, 128, 0, s>>>(src, src2, n, k, kt, dst);
  return cudaGetLastError();
}

}  // namespace memspec
