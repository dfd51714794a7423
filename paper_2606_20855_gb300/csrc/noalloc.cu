// Allocation-free row-pointer scan: the scan of scan.cu with its scratch (the
// per-tile partial sums and the small summary block the last tile writes)
// in one fixed array compiled into the library, instead of memory allocated
// per call.
//
// Who needs it: code that must not allocate device memory at the point where
// it builds a CSR row pointer.  Two examples: a caller inside a framework
// that owns all device memory through its own pool and forbids outside
// allocations, and a caller in a latency-critical loop where cudaMalloc or
// cudaFree would block on the whole device.  Such a caller passes only its
// own buffers; this file never calls cudaMalloc, cudaFree or any other
// allocating routine.
//
// Costs of the fixed array: every GPU that loads the library holds it
// (kStaticScanBytes bytes) until the process exits; all calls share it, so
// two calls that overlap on the GPU (different streams, no ordering between
// them) corrupt each other's partial sums.
#include <mutex>

#include "ws_internal.cuh"
#include "ws_spgemm.h"

namespace wsk {
namespace {

constexpr int64_t kStaticScanMaxRows = int64_t{1} << 24;  // 16,777,216 rows
constexpr int64_t kStaticScanTiles = (kStaticScanMaxRows + 4095) / 4096 + 1;
// tile partials, then room for the summary block the scan's last tile writes nnz into
constexpr int64_t kStaticScanWords = kStaticScanTiles + (sizeof(DevSummary) + 7) / 8 + 32;
constexpr int64_t kStaticScanBytes = kStaticScanWords * 8;
static_assert(kStaticScanBytes <= 40 * 1024, "keep the fixed scratch modest (about 33 KB)");

// The fixed scratch.  Host code must not use this name as a device address:
// on the host it only stands for the symbol; the device address comes from
// cudaGetSymbolAddress (see static_scratch below).
static __device__ __align__(256) int64_t g_static_scan_scratch[kStaticScanWords];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
int64_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of the fixed scratch on the current device.  The first call
// on a device looks it up (cudaGetSymbolAddress, with that device current)
// and remembers it for the life of the process.  A cudaDeviceReset destroys
// the module that holds the array, so the remembered address is not valid
// after one; the header says not to call the entry point across a reset.
cudaError_t static_scratch(int dev, int64_t** out) {
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scan_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = static_cast<int64_t*>(p);
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace wsk

extern "C" {

// Declared in include/ws_spgemm.h; see the comment there for the contract.
ws_status_t ws_rowptr_scan_static(int64_t* rowptr, int64_t nrows, ws_stream_t stream) {
  using namespace wsk;
  if (nrows < 0) return WS_ERR_INVALID_ARG;
  if (nrows > kStaticScanMaxRows) return WS_ERR_OVERFLOW;  // beyond the fixed scratch
  if (!rowptr) return WS_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return WS_ERR_CUDA;
  int64_t* scratch = nullptr;
  if (static_scratch(dev, &scratch) != cudaSuccess) return WS_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // Nothing in the scratch has to start at zero: the scan writes every tile
  // partial it reads, and the summary block is written, never read.
  if (cudaMemsetAsync(rowptr, 0, sizeof(int64_t), s) != cudaSuccess) return WS_ERR_CUDA;
  int launches = 0;
  DevSummary* sum = reinterpret_cast<DevSummary*>(scratch + kStaticScanTiles);
  launch_scan(rowptr, nrows, scratch, sum, s, &launches);
  if (cudaGetLastError() != cudaSuccess) return WS_ERR_CUDA;
  return WS_OK;
}

}  // extern "C"
