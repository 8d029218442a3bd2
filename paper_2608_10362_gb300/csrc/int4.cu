// int4.cu - group-wise INT4 weight-only linear layer for decode-sized row counts
// (the paper's targets are GPTQ INT4 models, Section 4.1).
//
// y[m][r] = sum_c x[m][c] w[r][c],  w[r][c] = (q[r][c] - z[r][g]) s[r][g],  g = c / 128,
// q 4-bit codes, s bf16 scales, z 4-bit zero points (stored one per byte).
//
// Why the tensor pipe.  At 4 bits the weights arrive at ~2 weights per byte of
// HBM traffic, i.e. ~44 weights per clock per SM at the copy bandwidth.  A
// CUDA-core kernel spends ~3 instructions per weight on unpacking plus one FMA
// per weight per activation row, which for the verify pass's K + 1 = 5 rows is
// ~1.7x more issue than an SM has.  So the kernel unpacks the codes straight
// into the A-operand registers of a register-sourced bf16 MMA (m16n8k16; the
// weights are A, 16 rows, the activation rows are the n = 8 side) and lets the
// tensor pipe do the products.  tcgen05 would need the unpacked tile written to
// shared memory or TMEM first (2 extra bytes moved per weight for 0.5 loaded);
// the contraction is far too thin (<= 16 activation rows) to need its rate.
//
// Exactness of the operands.  A code q enters the MMA as the bf16 128 + q
// (exponent of 128, q in the mantissa's low bits: one LOP3 per two codes), the
// zero point is folded out per group:
//   sum_c x (q - z) = sum_c x (128 + q) - (128 + z) sum_c x,
// with sum_c x over the group (sx) formed once per CTA.  Products are exact;
// the MMA's fp32 accumulation of the biased terms is the only rounding beyond
// the epilogue's.
//
// Layout (memspec_int4_pack).  The kernel reads a repacked copy: one record per
// (16-row tile, group) unit, in tile-major order:
//   bytes [0, 512)     rows 0..7 :  lane L = 4 r + t holds 16 bytes = four 32-bit
//   bytes [512, 1024)  rows 8..15:  words, word j = the GPTQ bytes of row r at
//                                   column offsets g*128 + 32 j + 8 t + (0..7)
//   bytes [1024, 1056) eight bf16 pairs (s[r], s[r + 8])
//   bytes [1056, 1072) eight byte pairs (z[r], z[r + 8])
// so a warp reads each record with two fully coalesced 512-byte loads and
// lane L holds exactly its MMA fragment.  Word j's 8 nibbles e = 0..7 become
// the k slots {2t, 2t+1, 2t+8, 2t+9} of two k16 steps as pairs (e, e+4); the
// activation fragments are permuted identically (byte permutes of one 16-byte
// load), so each step contracts matching columns.
//
// Work split.  The U = tiles x groups units are cut into equal contiguous
// ranges, one per CTA (stream-K), and each CTA's range into equal ranges, one
// per warp.  A warp keeps four units' loads in flight.  A tile a warp covers
// whole is stored directly; a tile shared by several warps is summed from
// per-warp shared-memory partials in warp order; a tile shared by several CTAs
// is summed from global partials by the CTA that completes it (a per-tile unit
// counter), in CTA order.  Every sum has a fixed order: results are
// bit-reproducible.  The counters and partials are static device arrays, so
// calls on one device must not overlap.
#include <cuda_bf16.h>

#include "internal.h"

namespace memspec {

constexpr int kI4Warps = 16;
constexpr int kI4Threads = kI4Warps * 32;
constexpr int kI4Depth = 4;            // units in flight per warp
constexpr int kI4MaxCtas = 512;
constexpr int kI4MaxTiles = 65536;     // n <= 1,048,576 rows

__device__ int g_i4_count[kI4MaxTiles];                 // zero between launches
__device__ float g_i4_part[kI4MaxCtas * 2 * 16 * 16];   // [cta][first/last tile][16 rows][16]

namespace {

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

// (w >> sh) nibbles 0 and 4 -> bf16 pair (128 + lo, 128 + hi)
__device__ __forceinline__ uint32_t nib2(uint32_t w) {
  uint32_t d;
  asm("lop3.b32 %0, %1, 0x000F000F, 0x43004300, 0xEA;" : "=r"(d) : "r"(w));   // (a & b) | c
  return d;
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t ld_nc_u32(const void* p) {
  uint32_t v;
  asm volatile("ld.global.nc.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t ld_nc_u16(const void* p) {
  unsigned short v;
  asm volatile("ld.global.nc.u16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}

// largest part index j (of `parts` equal contiguous parts of [0, total)) whose
// range starts at or before v; that part's range is never empty
__device__ __forceinline__ int part_of(long long v, long long total, int parts) {
  return static_cast<int>(((v + 1) * parts + total - 1) / total) - 1;
}
__device__ __forceinline__ long long part_lo(int j, long long total, int parts) {
  return static_cast<long long>(j) * total / parts;
}

template <int NT>
__global__ void __launch_bounds__(kI4Threads, 1) int4_linear_kernel(const __grid_constant__ Int4Args a) {
  constexpr int Mp = 8 * NT;
  extern __shared__ __align__(128) uint8_t dsm[];
  __shared__ int s_last;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rq = lane >> 2, t = lane & 3;
  const int M = a.rows, k = a.k, G = k >> 7, n = a.n;
  const int P = 2 * k + 64;   // bytes per staged activation row (the pad makes the fragment loads conflict-free)
  uint8_t* xs = dsm;                                                     // [Mp][P]
  float* sx = reinterpret_cast<float*>(dsm + static_cast<size_t>(Mp) * P);   // [G][Mp]
  float* part = sx + G * Mp;                                             // [warp][2][16][Mp]

  const long long tiles = (n + 15) / 16;
  const long long U = tiles * G;
  const int NC = gridDim.x, c = blockIdx.x;
  const long long A = part_lo(c, U, NC), B = part_lo(c + 1, U, NC);
  const long long L = B - A;
  const long long aw = A + L * warp / kI4Warps, bw = A + L * (warp + 1) / kI4Warps;

  // ---- start this warp's weight stream before anything else
  const uint8_t* rec = a.packed;
  uint4 qa[kI4Depth], qb[kI4Depth];
  uint32_t sp[kI4Depth], zp[kI4Depth];
#pragma unroll
  for (int i = 0; i < kI4Depth; ++i) {
    if (aw + i < bw) {
      const uint8_t* r = rec + (aw + i) * kInt4RecordBytes;
      qa[i] = ld_stream16(r + lane * 16);
      qb[i] = ld_stream16(r + 512 + lane * 16);
      sp[i] = ld_nc_u32(r + 1024 + rq * 4);
      zp[i] = ld_nc_u16(r + 1056 + rq * 2);
    }
  }

  // ---- activations into shared memory, and their per-group sums sx[g][m]:
  // half a warp covers one group of one row (16 vectors of 8), summed by a
  // fixed xor tree
  {
    const int per_row = k >> 3;
    const int total = M * per_row;
    for (int base = warp * 32; base < total; base += kI4Threads) {
      const int idx = base + lane;
      float s = 0.f;
      if (idx < total) {
        const int m = idx / per_row, v = idx - m * per_row;
        const uint4 xv = reinterpret_cast<const uint4*>(a.x)[idx];
        *reinterpret_cast<uint4*>(xs + static_cast<size_t>(m) * P + v * 16) = xv;
        const uint32_t w4[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) s += __uint_as_float(w4[e] << 16) + __uint_as_float(w4[e] & 0xffff0000u);
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (idx < total && (lane & 15) == 0) {
        const int m = idx / per_row, v = idx - m * per_row;
        sx[(v >> 4) * Mp + m] = s;
      }
    }
    // padding rows M..Mp-1: zero activations and sums
    const int pad16 = (Mp - M) * (P / 16);
    for (int i = tid; i < pad16; i += kI4Threads)
      *reinterpret_cast<uint4*>(xs + static_cast<size_t>(M) * P + i * 16) = make_uint4(0u, 0u, 0u, 0u);
    for (int i = tid; i < (Mp - M) * G; i += kI4Threads) {
      const int g = i / (Mp - M), m = M + i % (Mp - M);
      sx[g * Mp + m] = 0.f;
    }
  }
  __syncthreads();

  // ---- main loop over this warp's units
  float o[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  long long T = aw / G;
  int g = static_cast<int>(aw - T * G);
  const long long T_first = T;
  const uint8_t* xrow[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) xrow[j] = xs + static_cast<size_t>(8 * j + rq) * P + 16 * t;

  for (long long u0 = aw; u0 < bw; u0 += kI4Depth) {
#pragma unroll
    for (int i = 0; i < kI4Depth; ++i) {
      const long long u = u0 + i;
      if (u < bw) {
        float acc[NT][4];
#pragma unroll
        for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
        const uint32_t wa[4] = {qa[i].x, qa[i].y, qa[i].z, qa[i].w};
        const uint32_t wb[4] = {qb[i].x, qb[i].y, qb[i].z, qb[i].w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const uint32_t a0 = nib2(wa[w]), a1 = nib2(wb[w]);
          const uint32_t a2 = nib2(wa[w] >> 4), a3 = nib2(wb[w] >> 4);
          const uint32_t a4 = nib2(wa[w] >> 8), a5 = nib2(wb[w] >> 8);
          const uint32_t a6 = nib2(wa[w] >> 12), a7 = nib2(wb[w] >> 12);
#pragma unroll
          for (int j = 0; j < NT; ++j) {
            const uint4 X = *reinterpret_cast<const uint4*>(xrow[j] + g * 256 + w * 64);
            // k slots (2t, 2t+1) <- columns (e, e + 4); (2t+8, 2t+9) <- (e+1, e+5)
            mma_bf16(acc[j], a0, a1, a2, a3, prmt(X.x, X.z, 0x5410), prmt(X.x, X.z, 0x7632));
            mma_bf16(acc[j], a4, a5, a6, a7, prmt(X.y, X.w, 0x5410), prmt(X.y, X.w, 0x7632));
          }
        }
        // fold the scale and zero point of this group
        const float s0 = __uint_as_float(sp[i] << 16), s1 = __uint_as_float(sp[i] & 0xffff0000u);
        const float z0 = 128.f + static_cast<float>(zp[i] & 0xffu), z1 = 128.f + static_cast<float>(zp[i] >> 8);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
          const float2 sv = *reinterpret_cast<const float2*>(sx + g * Mp + 8 * j + 2 * t);
          o[j][0] = fmaf(s0, fmaf(-z0, sv.x, acc[j][0]), o[j][0]);
          o[j][1] = fmaf(s0, fmaf(-z0, sv.y, acc[j][1]), o[j][1]);
          o[j][2] = fmaf(s1, fmaf(-z1, sv.x, acc[j][2]), o[j][2]);
          o[j][3] = fmaf(s1, fmaf(-z1, sv.y, acc[j][3]), o[j][3]);
        }
        // refill this register slot
        if (u + kI4Depth < bw) {
          const uint8_t* r = rec + (u + kI4Depth) * kInt4RecordBytes;
          qa[i] = ld_stream16(r + lane * 16);
          qb[i] = ld_stream16(r + 512 + lane * 16);
          sp[i] = ld_nc_u32(r + 1024 + rq * 4);
          zp[i] = ld_nc_u16(r + 1056 + rq * 2);
        }
        // end of a tile, or of the warp's range: flush
        ++g;
        if (g == G || u + 1 == bw) {
          const long long lo = T * G > aw ? T * G : aw;
          const long long hi = (T + 1) * G < bw ? (T + 1) * G : bw;
          const int r0 = static_cast<int>(T * 16) + rq, r1 = r0 + 8;
          if (lo == T * G && hi == (T + 1) * G) {
#pragma unroll
            for (int j = 0; j < NT; ++j) {
              const int m = 8 * j + 2 * t;
              if (m < M) {
                if (r0 < n) a.y[static_cast<size_t>(m) * n + r0] = o[j][0];
                if (r1 < n) a.y[static_cast<size_t>(m) * n + r1] = o[j][2];
              }
              if (m + 1 < M) {
                if (r0 < n) a.y[static_cast<size_t>(m + 1) * n + r0] = o[j][1];
                if (r1 < n) a.y[static_cast<size_t>(m + 1) * n + r1] = o[j][3];
              }
            }
          } else {
            float* ps = part + (warp * 2 + (T == T_first ? 0 : 1)) * 16 * Mp;
#pragma unroll
            for (int j = 0; j < NT; ++j) {
              const int m = 8 * j + 2 * t;
              ps[rq * Mp + m] = o[j][0];
              ps[rq * Mp + m + 1] = o[j][1];
              ps[(rq + 8) * Mp + m] = o[j][2];
              ps[(rq + 8) * Mp + m + 1] = o[j][3];
            }
          }
#pragma unroll
          for (int j = 0; j < NT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
          if (g == G) {
            g = 0;
            ++T;
          }
        }
      }
    }
  }
  __syncthreads();
  if (L == 0) return;

  // ---- tiles shared by several warps of this CTA (or by other CTAs): sum the
  // warp partials in warp order
  const long long TA = A / G, TB = (B - 1) / G;
  const int row = tid / Mp, col = tid % Mp;   // one output of the 16 x Mp tile per thread
  for (long long TT = TA; TT <= TB; ++TT) {
    const long long lo = TT * G > A ? TT * G : A;
    const long long hi = (TT + 1) * G < B ? (TT + 1) * G : B;
    const int w_lo = part_of(lo - A, L, kI4Warps), w_hi = part_of(hi - 1 - A, L, kI4Warps);
    const bool cta_full = lo == TT * G && hi == (TT + 1) * G;
    if (w_lo == w_hi && cta_full) continue;   // one warp covered it whole: already stored
    if (tid < 16 * Mp) {
      float v = 0.f;
      for (int w = w_lo; w <= w_hi; ++w) {
        const long long wa = A + part_lo(w, L, kI4Warps), wb = A + part_lo(w + 1, L, kI4Warps);
        if (wa == wb) continue;
        const int slot = (wa / G == TT) ? 0 : 1;
        v += part[(w * 2 + slot) * 16 * Mp + tid];
      }
      const int r = static_cast<int>(TT * 16) + row;
      if (cta_full) {
        if (col < M && r < n) a.y[static_cast<size_t>(col) * n + r] = v;
      } else {
        g_i4_part[(static_cast<size_t>(c) * 2 + (TT == TA ? 0 : 1)) * 256 + row * 16 + col] = v;
      }
    }
  }

  // ---- tiles shared with other CTAs: the CTA that completes a tile's unit
  // count sums every CTA's partial in CTA order
  for (int side = 0; side < 2; ++side) {
    const long long TT = side == 0 ? TA : TB;
    if (side == 1 && TB == TA) break;
    const long long lo = TT * G > A ? TT * G : A;
    const long long hi = (TT + 1) * G < B ? (TT + 1) * G : B;
    if (lo == TT * G && hi == (TT + 1) * G) continue;
    __syncthreads();   // this CTA's partial is written
    if (tid == 0) {
      __threadfence();
      const int covered = static_cast<int>(hi - lo);
      const int before = atomicAdd(&g_i4_count[TT], covered);
      s_last = before + covered == G;
      if (s_last) __threadfence();
    }
    __syncthreads();
    if (s_last) {
      const int c_lo = part_of(TT * G, U, NC), c_hi = part_of((TT + 1) * G - 1, U, NC);
      if (tid < 16 * Mp) {
        float v = 0.f;
        for (int cc = c_lo; cc <= c_hi; ++cc) {
          const long long ca = part_lo(cc, U, NC), cb = part_lo(cc + 1, U, NC);
          if (ca == cb) continue;
          const int slot = (ca / G == TT) ? 0 : 1;
          v += __ldcg(&g_i4_part[(static_cast<size_t>(cc) * 2 + slot) * 256 + row * 16 + col]);
        }
        const int r = static_cast<int>(TT * 16) + row;
        if (col < M && r < n) a.y[static_cast<size_t>(col) * n + r] = v;
      }
      if (tid == 0) g_i4_count[TT] = 0;
    }
  }
}

// One thread per 16-byte code block (64 per unit) plus one per unit tail.
__global__ void int4_pack_kernel(const uint8_t* __restrict__ qweight, const bf16* __restrict__ scales,
                                 const uint8_t* __restrict__ zeros, uint8_t* __restrict__ out, int n, int k,
                                 long long units) {
  const int G = k >> 7;
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= units * 65) return;
  const long long u = i / 65;
  const int b = static_cast<int>(i - u * 65);
  const long long T = u / G;
  const int g = static_cast<int>(u - T * G);
  uint8_t* rec = out + u * kInt4RecordBytes;
  if (b < 64) {
    const int half = b >> 5, lane = b & 31, r = lane >> 2, t = lane & 3;
    const long long row = T * 16 + half * 8 + r;
    uint32_t w4[4] = {0u, 0u, 0u, 0u};
    if (row < n) {
      const uint8_t* src = qweight + row * (k / 2) + g * 64 + 4 * t;
#pragma unroll
      for (int j = 0; j < 4; ++j) w4[j] = *reinterpret_cast<const uint32_t*>(src + 16 * j);
    }
    *reinterpret_cast<uint4*>(rec + half * 512 + lane * 16) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
  } else {
    uint32_t sw[8];
    uint16_t zw[8];
    for (int r = 0; r < 8; ++r) {
      const long long r0 = T * 16 + r, r1 = r0 + 8;
      uint16_t s0 = 0, s1 = 0, z0 = 0, z1 = 0;
      if (r0 < n) {
        s0 = __bfloat16_as_ushort(scales[r0 * G + g]);
        z0 = zeros[r0 * G + g];
      }
      if (r1 < n) {
        s1 = __bfloat16_as_ushort(scales[r1 * G + g]);
        z1 = zeros[r1 * G + g];
      }
      sw[r] = static_cast<uint32_t>(s0) | (static_cast<uint32_t>(s1) << 16);
      zw[r] = static_cast<uint16_t>(z0 | (z1 << 8));
    }
    uint4* d = reinterpret_cast<uint4*>(rec + 1024);
    d[0] = make_uint4(sw[0], sw[1], sw[2], sw[3]);
    d[1] = make_uint4(sw[4], sw[5], sw[6], sw[7]);
    d[2] = make_uint4(zw[0] | (static_cast<uint32_t>(zw[1]) << 16), zw[2] | (static_cast<uint32_t>(zw[3]) << 16),
                      zw[4] | (static_cast<uint32_t>(zw[5]) << 16), zw[6] | (static_cast<uint32_t>(zw[7]) << 16));
  }
}

}  // namespace

size_t int4_packed_bytes(long long n, int k) {
  return static_cast<size_t>((n + 15) / 16) * static_cast<size_t>(k / 128) * kInt4RecordBytes;
}

size_t int4_smem_bytes(int rows, int k) {
  const int Mp = rows <= 8 ? 8 : 16;
  return static_cast<size_t>(Mp) * (2 * k + 64) + static_cast<size_t>(k / 128) * Mp * 4 +
         static_cast<size_t>(kI4Warps) * 2 * 16 * Mp * 4;
}

int int4_max_ctas() { return kI4MaxCtas; }
long long int4_max_rows() { return static_cast<long long>(kI4MaxTiles) * 16; }

cudaError_t int4_set_max_smem() {
  cudaError_t e = cudaFuncSetAttribute(int4_linear_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kInt4MaxSmem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(int4_linear_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kInt4MaxSmem);
}

cudaError_t launch_int4_linear(const Int4Args& a, int grid, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kI4Threads);
  cfg.dynamicSmemBytes = int4_smem_bytes(a.rows, a.k);
  cfg.stream = s;
  cfg.numAttrs = 0;
  if (a.rows <= 8) return cudaLaunchKernelEx(&cfg, int4_linear_kernel<1>, a);
  return cudaLaunchKernelEx(&cfg, int4_linear_kernel<2>, a);
}

cudaError_t launch_int4_pack(const uint8_t* qweight, const bf16* scales, const uint8_t* zeros, uint8_t* out,
                             int n, int k, cudaStream_t s) {
  const long long units = static_cast<long long>((n + 15) / 16) * (k / 128);
  const long long threads = units * 65;
  const int block = 256;
  const long long grid = (threads + block - 1) / block;
  int4_pack_kernel<<<static_cast<unsigned>(grid), block, 0, s>>>(qweight, scales, zeros, out, n, k, units);
  return cudaGetLastError();
}

}  // namespace memspec
