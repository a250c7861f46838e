// Shared device/host helpers of the FedOptima GB300 library.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>
#include <cstdio>
#include <utility>

namespace fo {

typedef __nv_bfloat16 bf16;

// Element conversions used by the templated kernels.
__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

inline int ceil_div(int64_t a, int64_t b) { return int((a + b - 1) / b); }

// Grid size for grid-stride elementwise kernels: a multiple of the SM count.
int elementwise_blocks(int64_t n_threads_needed, int threads);

// Programmatic dependent launch.  The library's kernels are launched with the
// programmatic-stream-serialization attribute, so that the next kernel of a
// step (or of its CUDA graph) is scheduled while this one drains instead of
// after it.  Every kernel therefore calls pdl_wait() before its first
// global-memory access: it returns once the preceding kernel has completed
// and its writes are visible (and at once without the attribute).  Each
// block calls pdl_trigger() on entry, or, in the tensor-core kernels, once it
// holds its tensor memory: the dependent grid is scheduled only after every
// block has triggered (or exited), so a dependent block that lands on the
// same SM can wait for tensor memory that an earlier kernel frees, but never
// holds any that an earlier kernel still has to allocate.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// False when FO_NO_PDL is set (plain stream order, for comparison).
bool pdl_enabled();

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace fo
