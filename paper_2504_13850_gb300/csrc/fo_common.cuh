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

// Standard normal distribution function Phi(x) and density phi(x) for the
// GELU, from one exponential and one reciprocal: Abramowitz & Stegun 26.2.17
// (Hastings' rational approximation), for x >= 0
//   1 - Phi(x) = phi(x) (b1 t + b2 t^2 + b3 t^3 + b4 t^4 + b5 t^5),
//   t = 1 / (1 + p x),  p = 0.2316419,
// with an absolute error below 7.5e-8; Phi(-x) = 1 - Phi(x) gives x < 0
// without the cancellation of 1 + erf.  The density's exponential is the
// same one, so the GELU backward gets phi(x) with no further work.
__device__ __forceinline__ void normal_cdf_pdf(float x, float& cdf, float& pdf) {
  float e;   // exp(-x^2 / 2) = 2^(-x^2 log2(e) / 2)
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(x * x * -0.72134752044448170f));
  pdf = 0.39894228040143268f * e;
  const float t = __fdividef(1.f, fmaf(0.2316419f, fabsf(x), 1.f));
  const float poly =
      t * fmaf(t, fmaf(t, fmaf(t, fmaf(t, 1.330274429f, -1.821255978f), 1.781477937f), -0.356563782f), 0.319381530f);
  const float q = pdf * poly;   // 1 - Phi(|x|)
  cdf = x >= 0.f ? 1.f - q : q;
}

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
