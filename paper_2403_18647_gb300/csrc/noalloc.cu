// Skinny GEMM without a context and without device allocations.
//
// Some callers cannot allocate device memory when they want to run a
// projection: code that runs while a CUDA graph is being captured (cudaMalloc
// is not a stream operation and is not allowed there), code inside a host
// framework that owns every byte of device memory through its own allocator,
// or code with a fixed memory budget established at start-up.  For them,
// sdsat_gemm_static computes y = x W^T with the same kernels as
// sdsat_op_gemm, but its scratch (the bf16 hi/lo operand, the split-K partial
// sums and the per-tile counters) lives in the fixed-size device array below,
// which every GPU that loads the library holds until the process exits.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "internal.h"
#include "sdsat.h"

namespace sdsat {
namespace {

// limits of the scratch-free entry point
constexpr int SA_MAX_M = 16;          // activation rows
constexpr int SA_MAX_K = 16384;       // reduction length
constexpr int SA_MAX_N = 65536;       // output features (512 tiles of 128)
constexpr int SA_MAX_SM = 64;         // SMs used
constexpr int SA_MAX_CTAS = GEMM_CTAS_PER_SM * SA_MAX_SM;   // the largest grid launch_gemm builds here
constexpr int SA_TILES = SA_MAX_N / 128;

constexpr size_t SA_X_BYTES = (size_t)SA_MAX_M * SA_MAX_K * 2;          // one of hi / lo: 512 KiB
constexpr size_t SA_PART_BYTES = (size_t)SA_MAX_CTAS * 2 * 16 * 128 * 4;  // 2 MiB
constexpr size_t SA_CNT_BYTES = (size_t)SA_TILES * 4;                    // 2 KiB
constexpr size_t SA_OFF_XLO = SA_X_BYTES;
constexpr size_t SA_OFF_PART = 2 * SA_X_BYTES;
constexpr size_t SA_OFF_CNT = SA_OFF_PART + SA_PART_BYTES;
constexpr size_t SA_BYTES = SA_OFF_CNT + SA_CNT_BYTES;                   // 3 MiB + 2 KiB

// the kernel writes partials [(cta * 2 + slot) * 16 rows][128] for cta < its grid
static_assert(SA_PART_BYTES >= (size_t)SA_MAX_CTAS * 2 * 16 * 128 * sizeof(float), "partials region too small");
static_assert(SA_OFF_CNT % 16 == 0 && SA_OFF_PART % 16 == 0, "scratch regions 16-byte aligned");

}  // namespace
}  // namespace sdsat

// The scratch of sdsat_gemm_static: one copy per device, shared by every call.
static __device__ __align__(256) unsigned char g_gemm_static_scratch[sdsat::SA_BYTES];

namespace sdsat {
namespace {

struct DeviceSetup {
  bool done = false;
  CUcontext cuctx = nullptr;          // the context the set-up was made in
  unsigned char* scratch = nullptr;   // device address of g_gemm_static_scratch in that context
  int sms = 0;
};
constexpr int SA_MAX_DEVICES = 64;
DeviceSetup g_setup[SA_MAX_DEVICES];
std::mutex g_setup_mutex;
PFN_cuTensorMapEncodeTiled_v12000 g_encode_static = nullptr;
PFN_cuCtxGetCurrent_v4000 g_ctx_current = nullptr;

template <typename F>
bool driver_entry(const char* name, int version, F* fn) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, version, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !p)
    return false;
  *fn = reinterpret_cast<F>(p);
  return true;
}

// Per-device set-up, done by the first call on each device (with that device
// current): the device address of the scratch array, the SM count, the kernels'
// shared-memory limits and the tensor-map encoder.  Host code must not use the
// array's name as an address; it is a host-side stand-in for the device symbol.
// The set-up belongs to the device's current context: after a cudaDeviceReset the
// device gets a new primary context, whose scratch address and kernel attributes
// are looked up again on the next call.
sdsat_status setup_device(int dev, DeviceSetup** out) {
  if (dev < 0 || dev >= SA_MAX_DEVICES) return SDSAT_EUNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_ctx_current && !driver_entry("cuCtxGetCurrent", 4000, &g_ctx_current)) return SDSAT_ECUDA;
  CUcontext cur = nullptr;   // null before the runtime has made a context current on this thread
  if (g_ctx_current(&cur) != CUDA_SUCCESS) return SDSAT_ECUDA;
  DeviceSetup& s = g_setup[dev];
  if (!s.done || !cur || s.cuctx != cur) {
    s.done = false;
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_gemm_static_scratch) != cudaSuccess || ptr == nullptr) return SDSAT_ECUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return SDSAT_ECUDA;
    if (gemm_prepare() != cudaSuccess) return SDSAT_ECUDA;
    if (!g_encode_static && !driver_entry("cuTensorMapEncodeTiled", 12000, &g_encode_static)) return SDSAT_ECUDA;
    // the symbol lookup above made the device's context current if none was
    if (g_ctx_current(&cur) != CUDA_SUCCESS || !cur) return SDSAT_ECUDA;
    s.cuctx = cur;
    s.scratch = static_cast<unsigned char*>(ptr);
    s.sms = std::min(sms, SA_MAX_SM);
    s.done = true;
  }
  *out = &s;
  return SDSAT_OK;
}

// bf16 [rows][cols], boxes of box_rows x 64 columns, 128-byte swizzle
bool encode(CUtensorMap* map, const void* ptr, int rows, int cols, int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode_static(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace sdsat

using namespace sdsat;

extern "C" sdsat_status sdsat_gemm_static(const float* x_dev, int M, int K, const void* w_dev, int N, float* y_dev,
                                          void* stream, uint32_t* err_dev) {
  if (!x_dev || !y_dev || !aligned16(x_dev) || !aligned16(w_dev) || M < 1 || K < 8 || K % 8 || N < 1)
    return SDSAT_EINVAL;
  if (M > SA_MAX_M || K > SA_MAX_K || N > SA_MAX_N) return SDSAT_ECAPACITY;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDSAT_ECUDA;
  DeviceSetup* s = nullptr;
  const sdsat_status st = setup_device(dev, &s);
  if (st != SDSAT_OK) return st;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  __nv_bfloat16* xhi = reinterpret_cast<__nv_bfloat16*>(s->scratch);
  __nv_bfloat16* xlo = reinterpret_cast<__nv_bfloat16*>(s->scratch + SA_OFF_XLO);
  float* partials = reinterpret_cast<float*>(s->scratch + SA_OFF_PART);
  int* counters = reinterpret_cast<int*>(s->scratch + SA_OFF_CNT);
  GemmParams g;
  std::memset(&g, 0, sizeof(g));
  // the operand buffers hold SA_MAX_M rows of K columns; the kernel reads 16-row boxes
  if (!encode(&g.tmap[0], w_dev, N, K, 64) || !encode(&g.tmap_x[0], xhi, SA_MAX_M, K, 16) ||
      !encode(&g.tmap_x[1], xlo, SA_MAX_M, K, 16))
    return SDSAT_ECUDA;
  g.map_mode = MAP_PLAIN;
  g.N = N;
  g.K = K;
  g.n_tiles = (N + 127) / 128;
  g.kc = (K + 63) / 64;
  g.M = M;
  g.epi = EPI_STORE;
  g.out = y_dev;
  g.out_ld = N;
  g.partials = partials;
  g.counters = counters;
  g.err = err_dev;   // caller-owned; a bounded wait that runs out ORs SDSAT_DEV_TIMEOUT into it
  // the tile counters must start at zero (the kernel also leaves them at zero)
  if (cudaMemsetAsync(counters, 0, (size_t)g.n_tiles * sizeof(int), cs) != cudaSuccess) return SDSAT_ECUDA;
  if (launch_split(x_dev, M, K, xhi, xlo, cs, false) != cudaSuccess) return SDSAT_ECUDA;
  if (launch_gemm(g, s->sms, cs, false) != cudaSuccess) return SDSAT_ECUDA;
  return SDSAT_OK;
}
