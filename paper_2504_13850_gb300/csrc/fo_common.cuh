// Shared device/host helpers of the FedOptima GB300 library.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>
#include <cstdio>

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

}  // namespace fo
