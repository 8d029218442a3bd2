// noalloc.cu - memspec_op_linear_noalloc: the weight-streaming GEMM for callers
// that must not allocate device memory.
//
// memspec_op_linear needs a caller-provided scratch buffer (split-K partial sums,
// per-row-tile arrival counters).  Some callers cannot provide one: plug-ins whose
// host application owns every byte of device memory and hands out none,
// fixed-budget deployments where all allocation happens once at start-up, and
// latency-critical loops that cannot afford cudaMalloc / cudaFree (which may
// synchronise the device).  This entry point keeps that scratch in a file-scope
// device array of fixed size instead, so a call allocates nothing.
//
// Properties a user must know:
//  * the array (kNoAllocScratchBytes, about 2.6 MB) exists on every GPU that
//    loads this library, for as long as the process runs;
//  * rows <= 16, n_out <= 131072 (1024 row tiles), k a multiple of 8; larger
//    sizes are rejected with MEMSPEC_ERR_INVALID_ARG before anything is enqueued;
//  * every call shares the one array: calls whose executions overlap on the GPU
//    (different streams, or different host threads) race and give wrong results;
//    serialise them;
//  * the first call on a device looks up the array's device address (and sets
//    the kernel's shared-memory limit) for that device; make that first call
//    before any stream capture begins.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "../../include/memspec_ops.h"
#include "internal.h"

namespace memspec {
namespace {

constexpr int kNoAllocMaxRows = 16;            // MMA N = 16
constexpr int kNoAllocMaxCtas = 160;           // stream-K grid cap
constexpr int kNoAllocMaxRowTiles = 1024;      // n_out <= 131072
constexpr size_t kPartialBytes =
    static_cast<size_t>(2) * kNoAllocMaxCtas * kNoAllocMaxRows * 128 * 4;
constexpr size_t kCounterBytes = static_cast<size_t>(kNoAllocMaxRowTiles) * 4;
constexpr size_t kNoAllocScratchBytes = kPartialBytes + kCounterBytes + 256;

// split-K partials | arrival counters | status word
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                             const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                             const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                             CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;            // guards everything below
void* g_scratch_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
EncodeFn g_encode_fn = nullptr;      // driver entry point, looked up once

bool encode(EncodeFn fn, CUtensorMap* map, const void* base, int rows, int cols, int box_rows) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Per-device set-up, done once with the device current: the array's device
// address (a host-side reference to the array is not a device address), the SM
// count and the GEMM kernel's shared-memory limit; and, once per process, the
// driver's tensor-map encoder.  All under one mutex, so first calls from
// several host threads are safe.
memspec_status setup_device(int dev, void** scratch, int* n_sm, EncodeFn* encode_fn) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_encode_fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || p == nullptr) {
      set_op_error("cuTensorMapEncodeTiled entry point not found");
      return MEMSPEC_ERR_CUDA;
    }
    g_encode_fn = reinterpret_cast<EncodeFn>(p);
  }
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      set_op_error(std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      return MEMSPEC_ERR_CUDA;
    }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess || sms <= 0) {
      set_op_error(std::string("SM count: ") + cudaGetErrorString(e));
      return MEMSPEC_ERR_CUDA;
    }
    e = gemm_set_max_smem();
    if (e != cudaSuccess) {
      set_op_error(std::string("gemm smem attribute: ") + cudaGetErrorString(e));
      return MEMSPEC_ERR_CUDA;
    }
    g_sm_count[dev] = sms;
    g_scratch_ptr[dev] = p;
  }
  *scratch = g_scratch_ptr[dev];
  *n_sm = g_sm_count[dev];
  *encode_fn = g_encode_fn;
  return MEMSPEC_OK;
}

}  // namespace
}  // namespace memspec

using namespace memspec;

extern "C" memspec_status memspec_op_linear_noalloc(const void* x, const void* w, float* y,
                                                    int32_t rows, int32_t n_out, int32_t k,
                                                    uint32_t* status, void* stream) {
  if (x == nullptr || w == nullptr || y == nullptr) {
    set_op_error("null pointer");
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if (rows < 1 || rows > kNoAllocMaxRows || n_out < 1 || n_out > kNoAllocMaxRowTiles * 128 ||
      k < 8 || k % 8 != 0 || k > (1 << 20)) {
    set_op_error("sizes beyond this entry point's fixed scratch: rows must be in 1..16, "
                      "n_out in 1..131072, k a positive multiple of 8 up to 2^20");
    return MEMSPEC_ERR_INVALID_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(w) & 15)) {
    set_op_error("x and w must be 16-byte aligned");
    return MEMSPEC_ERR_INVALID_ARG;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    set_op_error(std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    return MEMSPEC_ERR_CUDA;
  }
  void* scratch = nullptr;
  int n_sm = 0;
  EncodeFn fn = nullptr;
  memspec_status st = setup_device(dev, &scratch, &n_sm, &fn);
  if (st != MEMSPEC_OK) return st;
  GemmArgs a{};
  const int n_pad = 16;
  if (!encode(fn, &a.map_a, w, n_out, k, 128) || !encode(fn, &a.map_b, x, rows, k, n_pad)) {
    set_op_error("cuTensorMapEncodeTiled failed");
    return MEMSPEC_ERR_CUDA;
  }
  a.n_out = n_out;
  a.k_in = k;
  a.rows_total = rows;
  a.n_pad = n_pad;
  a.row_tiles = (n_out + 127) / 128;
  a.k_tiles = (k + 63) / 64;
  a.stages = gemm_pick_stages(n_pad);
  a.l2_hint = L2_EVICT_FIRST;
  a.epi = EPI_F32;
  a.out = y;
  a.out_ld = n_out;
  uint8_t* sb = static_cast<uint8_t*>(scratch);
  a.partials = reinterpret_cast<float*>(sb);
  a.counters = reinterpret_cast<int*>(sb + kPartialBytes);
  uint32_t* own_status = reinterpret_cast<uint32_t*>(sb + kPartialBytes + kCounterBytes);
  a.status = status != nullptr ? status : own_status;
  a.plan = nullptr;
  // Stream-K grid: at most one CTA per SM and at most four contributors per row
  // tile, capped by the fixed scratch (kNoAllocMaxCtas).  Unlike memspec_op_linear
  // it keeps no SMs spare and reads no tuning variables, so its split-K summation
  // order can differ: results agree with memspec_op_linear within rounding, not
  // bit for bit.
  const int T = a.row_tiles * a.k_tiles;
  const int min_tiles = (a.k_tiles + 3) / 4 > 0 ? (a.k_tiles + 3) / 4 : 1;
  int grid = T;
  if (grid > n_sm) grid = n_sm;
  if (grid > kNoAllocMaxCtas) grid = kNoAllocMaxCtas;
  if (grid > T / min_tiles) grid = T / min_tiles;
  if (grid < 1) grid = 1;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents: counters and status start at zero
  e = cudaMemsetAsync(sb + kPartialBytes, 0, kCounterBytes + 256, s);
  if (e == cudaSuccess) e = launch_gemm(a, grid, gemm_smem_bytes(n_pad, a.stages), s, false);
  if (e != cudaSuccess) {
    set_op_error(std::string("launch: ") + cudaGetErrorString(e));
    return MEMSPEC_ERR_CUDA;
  }
  return MEMSPEC_OK;
}

