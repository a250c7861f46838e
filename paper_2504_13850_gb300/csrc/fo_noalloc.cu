// Column sums that allocate nothing.
//
// Some callers cannot allocate device memory at the point where they need
// this reduction: code that runs while its stream is being captured into a
// CUDA graph (an allocation there would break or leak out of the capture),
// processes whose device memory is handed out by an outside allocator
// (a framework's caching allocator, or a fixed arena carved up at start-up,
// where a private cudaMalloc competes for the same memory), and loops that
// must not allocate after initialisation.  For them the partial sums live in
// one fixed device array, declared below, instead of scratch allocated per
// call.  The array holds kScratchFloats floats (1 MiB) on every GPU that
// loads the library, until the process exits.
#include "fo_common.cuh"
#include "fo_kernels.h"
#include "../../include/fedoptima.h"

#include <mutex>
#include <string>

namespace fo {
int report_error(int code, const std::string& msg);
}

namespace {

constexpr int64_t kScratchFloats = 262144;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_colsum_scratch[kScratchFloats];

std::mutex g_mu;
float* g_scratch_addr[kMaxDevices] = {};

// Device address of the array on the current device, looked up once per
// device (host code only sees a host-side stand-in for the symbol).
int scratch_address(float** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fo::report_error(FO_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fo::report_error(FO_ERR_ARG, "device ordinal beyond the supported range");
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev]) {
    float* p = nullptr;
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_colsum_scratch);
    if (e != cudaSuccess)
      return fo::report_error(FO_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return FO_OK;
}

}  // namespace

extern "C" int fo_column_sums_noalloc(const void* x, int dtype, int64_t rows, int cols, float* out, void* stream) {
  if (!x || !out || rows < 1 || cols < 1 || (dtype != FO_DTYPE_F32 && dtype != FO_DTYPE_BF16))
    return fo::report_error(FO_ERR_ARG, "bad column-sum arguments");
  if (rows > fo::kColsumMaxRows)
    return fo::report_error(FO_ERR_ARG, "fo_column_sums_noalloc: " + std::to_string(rows) + " rows exceed " +
                                            std::to_string(fo::kColsumMaxRows) + " (65,535 chunks of 128 rows)");
  const int64_t need = fo::colsum_partial_floats(rows, cols);
  if (need > kScratchFloats)
    return fo::report_error(FO_ERR_ARG, "fo_column_sums_noalloc: ceil(rows / 128) * cols = " + std::to_string(need) +
                                            " partial sums exceed the fixed scratch of " +
                                            std::to_string(kScratchFloats) + " floats");
  float* scratch = nullptr;
  int rc = scratch_address(&scratch);
  if (rc != FO_OK) return rc;
  // Every partial the second kernel reads is written by the first one in
  // the same call, so nothing in the shared array has to start at zero.
  fo::colsum(x, nullptr, rows, cols, dtype == FO_DTYPE_F32 ? fo::kF32 : fo::kBF16, scratch, out,
             static_cast<cudaStream_t>(stream));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fo::report_error(FO_ERR_CUDA, cudaGetErrorString(e));
  return FO_OK;
}
