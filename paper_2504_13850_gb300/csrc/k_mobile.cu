// Kernels of the MobileNetV3 bottleneck (the MobileNetV3-Large server part
// of Table 4): depthwise convolution, hard swish, hard sigmoid and the
// squeeze-and-excite channel scaling.  Activations are NHWC in fp32 or bf16
// (template parameter T); every arithmetic step runs in fp32.  Channels are
// the fastest index of every thread mapping, so a warp's loads and stores are
// contiguous.  Parameter gradients are written as per-chunk partials that a
// later batched launch sums in chunk order (no atomics: deterministic).
#include "fo_common.cuh"
#include "fo_kernels.h"

#include <algorithm>

namespace fo {

namespace {

#define FO_MB_DISPATCH(dt, T, ...) \
  do {                             \
    if ((dt) == kF32) {            \
      using T = float;             \
      __VA_ARGS__;                 \
    } else {                       \
      using T = bf16;              \
      __VA_ARGS__;                 \
    }                              \
  } while (0)

#define FO_MB_GRID_STRIDE(i, n) \
  for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < (n); i += int64_t(gridDim.x) * blockDim.x)

template <typename T>
__device__ __forceinline__ void store_acc(T* p, int64_t i, float v, bool acc) {
  if (acc) v += to_f(p[i]);
  p[i] = from_f<T>(v);
}

// --------------------------------------------------------- depthwise conv
// KT is the kernel size when known at compile time (3 or 5: the tap loops
// unroll, so a thread's loads are independent), or 0 for a runtime d.k.

// y[n,i,j,c] = b[c] + sum_{r,s} xpad[n, i*st + r, j*st + s, c] * w[c,r,s],
// w [C][k][k] in the activation type (the bf16 path multiplies the bf16
// copy of the weights), zero padding `pad` on each side.
template <typename T, int KT>
__global__ void __launch_bounds__(256) dwconv_fwd_k(const T* __restrict__ x, const T* __restrict__ w,
                                                    const float* __restrict__ bias, T* __restrict__ y,
                                                    DwShape d) {
  pdl_wait();
  pdl_trigger();
  const int K = KT ? KT : d.k;
  const int64_t n_out = int64_t(d.N) * d.Ho * d.Wo * d.C;
  FO_MB_GRID_STRIDE(idx, n_out) {
    const int c = int(idx % d.C);
    const int64_t p = idx / d.C;
    const int j = int(p % d.Wo);
    const int i = int((p / d.Wo) % d.Ho);
    const int64_t n = p / (int64_t(d.Wo) * d.Ho);
    const T* wc = w + int64_t(c) * K * K;
    float acc = bias ? bias[c] : 0.f;
#pragma unroll
    for (int r = 0; r < (KT ? KT : K); ++r) {
      const int h = i * d.stride - d.pad + r;
      if (h < 0 || h >= d.H) continue;
#pragma unroll
      for (int s = 0; s < (KT ? KT : K); ++s) {
        const int ww = j * d.stride - d.pad + s;
        if (ww < 0 || ww >= d.W) continue;
        acc = fmaf(to_f(x[((n * d.H + h) * d.W + ww) * d.C + c]), to_f(wc[r * K + s]), acc);
      }
    }
    y[idx] = from_f<T>(acc);
  }
}

// dx[n,h,w,c] (+)= sum over the taps (r,s) whose output position
// i = (h + pad - r) / st, j = (w + pad - s) / st is whole and in range of
// dy[n,i,j,c] * w[c,r,s].
template <typename T, int KT>
__global__ void __launch_bounds__(256) dwconv_dgrad_k(const T* __restrict__ dy, const T* __restrict__ w,
                                                      T* __restrict__ dx, DwShape d, int acc_flag) {
  pdl_wait();
  pdl_trigger();
  const int K = KT ? KT : d.k;
  const int64_t n_in = int64_t(d.N) * d.H * d.W * d.C;
  FO_MB_GRID_STRIDE(idx, n_in) {
    const int c = int(idx % d.C);
    const int64_t p = idx / d.C;
    const int wx = int(p % d.W);
    const int h = int((p / d.W) % d.H);
    const int64_t n = p / (int64_t(d.W) * d.H);
    const T* wc = w + int64_t(c) * K * K;
    float acc = 0.f;
#pragma unroll
    for (int r = 0; r < (KT ? KT : K); ++r) {
      const int ti = h + d.pad - r;
      if (ti < 0 || ti % d.stride) continue;
      const int i = ti / d.stride;
      if (i >= d.Ho) continue;
#pragma unroll
      for (int s = 0; s < (KT ? KT : K); ++s) {
        const int tj = wx + d.pad - s;
        if (tj < 0 || tj % d.stride) continue;
        const int j = tj / d.stride;
        if (j >= d.Wo) continue;
        acc = fmaf(to_f(dy[((n * d.Ho + i) * d.Wo + j) * d.C + c]), to_f(wc[r * K + s]), acc);
      }
    }
    store_acc(dx, idx, acc, acc_flag != 0);
  }
}

// Weight (and bias) gradient partials: chunk q of the output pixels
// [q * per, min(rows, (q + 1) * per)) gives
//   pw[q][c*k*k + r*k + s] = sum_p dy[p,c] * xpad[p's window at (r,s), c]
//   pb[q][c]               = sum_p dy[p,c]            (when pb is given)
// A block covers 32 channels (lane = channel) of one chunk; its 8 warps take
// every 8th pixel of the chunk with the k*k tap sums in registers, and the
// warps' sums are added in warp order through shared memory.
template <typename T, int KT>
__global__ void __launch_bounds__(256) dwconv_wgrad_k(const T* __restrict__ dy, const T* __restrict__ x,
                                                      float* __restrict__ pw, float* __restrict__ pb, DwShape d,
                                                      int per) {
  pdl_wait();
  pdl_trigger();
  constexpr int KK = KT * KT;
  __shared__ float red[8][KK + 1][33];
  const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
  const int c = blockIdx.x * 32 + lane;
  const int64_t rows = int64_t(d.N) * d.Ho * d.Wo;
  const int64_t p0 = int64_t(blockIdx.y) * per;
  const int64_t p1 = p0 + per < rows ? p0 + per : rows;
  float acc[KK + 1];
#pragma unroll
  for (int t = 0; t <= KK; ++t) acc[t] = 0.f;
  if (c < d.C) {
    for (int64_t p = p0 + warp; p < p1; p += 8) {
      const int j = int(p % d.Wo);
      const int i = int((p / d.Wo) % d.Ho);
      const int64_t n = p / (int64_t(d.Wo) * d.Ho);
      const float g = to_f(dy[p * d.C + c]);
      acc[KK] += g;
#pragma unroll
      for (int r = 0; r < KT; ++r) {
        const int h = i * d.stride - d.pad + r;
        if (h < 0 || h >= d.H) continue;
#pragma unroll
        for (int s = 0; s < KT; ++s) {
          const int ww = j * d.stride - d.pad + s;
          if (ww < 0 || ww >= d.W) continue;
          acc[r * KT + s] = fmaf(g, to_f(x[((n * d.H + h) * d.W + ww) * d.C + c]), acc[r * KT + s]);
        }
      }
    }
  }
#pragma unroll
  for (int t = 0; t <= KK; ++t) red[warp][t][lane] = acc[t];
  __syncthreads();
  const int c0 = blockIdx.x * 32;
  for (int e = threadIdx.x; e < 32 * (KK + 1); e += 256) {
    // e = (channel, tap): consecutive threads write consecutive floats of pw
    const int cl = e / (KK + 1), t = e % (KK + 1);
    if (c0 + cl >= d.C) continue;
    float sum = 0.f;
#pragma unroll
    for (int w8 = 0; w8 < 8; ++w8) sum += red[w8][t][cl];
    if (t < KK) pw[int64_t(blockIdx.y) * d.C * KK + int64_t(c0 + cl) * KK + t] = sum;
    else if (pb) pb[int64_t(blockIdx.y) * d.C + c0 + cl] = sum;
  }
}

// Any kernel size: one thread per (tap, channel) and chunk.
template <typename T>
__global__ void __launch_bounds__(256) dwconv_wgrad_any_k(const T* __restrict__ dy, const T* __restrict__ x,
                                                          float* __restrict__ pw, float* __restrict__ pb, DwShape d,
                                                          int per) {
  pdl_wait();
  pdl_trigger();
  const int kk = d.k * d.k;
  const int taps = kk + (pb ? 1 : 0);
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= taps * d.C) return;
  const int c = t % d.C, tap = t / d.C;
  const int64_t rows = int64_t(d.N) * d.Ho * d.Wo;
  const int64_t p0 = int64_t(blockIdx.y) * per;
  const int64_t p1 = p0 + per < rows ? p0 + per : rows;
  float acc = 0.f;
  if (tap < kk) {
    const int r = tap / d.k, s = tap % d.k;
    for (int64_t p = p0; p < p1; ++p) {
      const int j = int(p % d.Wo);
      const int i = int((p / d.Wo) % d.Ho);
      const int64_t n = p / (int64_t(d.Wo) * d.Ho);
      const int h = i * d.stride - d.pad + r, ww = j * d.stride - d.pad + s;
      if (h < 0 || h >= d.H || ww < 0 || ww >= d.W) continue;
      acc = fmaf(to_f(dy[p * d.C + c]), to_f(x[((n * d.H + h) * d.W + ww) * d.C + c]), acc);
    }
    pw[int64_t(blockIdx.y) * d.C * kk + int64_t(c) * kk + tap] = acc;
  } else {
    for (int64_t p = p0; p < p1; ++p) acc += to_f(dy[p * d.C + c]);
    pb[int64_t(blockIdx.y) * d.C + c] = acc;
  }
}

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

// ------------------------------------------------- hard swish / sigmoid
__device__ __forceinline__ float relu6_p3(float v) { return fminf(fmaxf(v + 3.f, 0.f), 6.f); }

template <typename T>
__global__ void hswish_fwd_k(const T* __restrict__ x, T* __restrict__ y, int64_t n) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(i, n) {
    const float v = to_f(x[i]);
    y[i] = from_f<T>(v * relu6_p3(v) / 6.f);
  }
}
// derivative: 0 below -3, (2x + 3) / 6 on [-3, 3], 1 above 3
template <typename T>
__global__ void hswish_bwd_k(const T* __restrict__ x, const T* __restrict__ dy, T* __restrict__ dx, int64_t n,
                             int acc) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(i, n) {
    const float v = to_f(x[i]);
    const float g = v < -3.f ? 0.f : (v > 3.f ? 1.f : (2.f * v + 3.f) / 6.f);
    store_acc(dx, i, to_f(dy[i]) * g, acc != 0);
  }
}
template <typename T>
__global__ void hsigmoid_fwd_k(const T* __restrict__ x, T* __restrict__ y, int64_t n) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(i, n) y[i] = from_f<T>(relu6_p3(to_f(x[i])) / 6.f);
}
// derivative: 1/6 strictly inside (-3, 3), else 0
template <typename T>
__global__ void hsigmoid_bwd_k(const T* __restrict__ x, const T* __restrict__ dy, T* __restrict__ dx, int64_t n,
                               int acc) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(i, n) {
    const float v = to_f(x[i]);
    store_acc(dx, i, (v > -3.f && v < 3.f) ? to_f(dy[i]) / 6.f : 0.f, acc != 0);
  }
}

// ------------------------------------------------ squeeze-and-excite scale
// y[n,p,c] = x[n,p,c] * s[n,c] over the HW pixels p of image n.
template <typename T>
__global__ void chmul_fwd_k(const T* __restrict__ x, const T* __restrict__ sc, T* __restrict__ y, int N, int HW,
                            int C) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(i, int64_t(N) * HW * C) {
    const int c = int(i % C);
    const int64_t n = i / (int64_t(HW) * C);
    y[i] = from_f<T>(to_f(x[i]) * to_f(sc[n * C + c]));
  }
}
// dx[n,p,c] (+)= dy[n,p,c] s[n,c] (dx may be null);
// ds[n,c] (+)= sum_p dy[n,p,c] x[n,p,c] in pixel order (ds may be null).
template <typename T>
__global__ void chmul_bwd_k(const T* __restrict__ x, const T* __restrict__ sc, const T* __restrict__ dy,
                            T* __restrict__ dx, T* __restrict__ ds, int N, int HW, int C, int acc_dx, int acc_ds) {
  pdl_wait();
  pdl_trigger();
  FO_MB_GRID_STRIDE(o, int64_t(N) * C) {
    const int c = int(o % C);
    const int64_t n = o / C;
    const float s = to_f(sc[o]);
    float sum = 0.f;
    for (int p = 0; p < HW; ++p) {
      const int64_t i = (n * HW + p) * C + c;
      const float g = to_f(dy[i]);
      if (dx) store_acc(dx, i, g * s, acc_dx != 0);
      sum = fmaf(g, to_f(x[i]), sum);
    }
    if (ds) store_acc(ds, o, sum, acc_ds != 0);
  }
}

}  // namespace

void dwconv_fwd(const DwShape& d, const void* x, const void* w, const float* bias, void* y, int dt,
                cudaStream_t st) {
  const int64_t n = int64_t(d.N) * d.Ho * d.Wo * d.C;
  const int blocks = elementwise_blocks(n, 256);
  FO_MB_DISPATCH(dt, T, {
    if (d.k == 3) launch_k(dwconv_fwd_k<T, 3>, blocks, 256, 0, st, (const T*)x, (const T*)w, bias, (T*)y, d);
    else if (d.k == 5) launch_k(dwconv_fwd_k<T, 5>, blocks, 256, 0, st, (const T*)x, (const T*)w, bias, (T*)y, d);
    else launch_k(dwconv_fwd_k<T, 0>, blocks, 256, 0, st, (const T*)x, (const T*)w, bias, (T*)y, d);
  });
}

void dwconv_dgrad(const DwShape& d, const void* dy, const void* w, void* dx, int dt, bool acc, cudaStream_t st) {
  const int64_t n = int64_t(d.N) * d.H * d.W * d.C;
  const int blocks = elementwise_blocks(n, 256);
  const int a = acc ? 1 : 0;
  FO_MB_DISPATCH(dt, T, {
    if (d.k == 3) launch_k(dwconv_dgrad_k<T, 3>, blocks, 256, 0, st, (const T*)dy, (const T*)w, (T*)dx, d, a);
    else if (d.k == 5) launch_k(dwconv_dgrad_k<T, 5>, blocks, 256, 0, st, (const T*)dy, (const T*)w, (T*)dx, d, a);
    else launch_k(dwconv_dgrad_k<T, 0>, blocks, 256, 0, st, (const T*)dy, (const T*)w, (T*)dx, d, a);
  });
}

// Pixel chunks of the weight gradient: for k = 3, 5 about two blocks of 32
// channels per SM, at least 8 pixels (one per warp) per chunk, at most 64
// chunks; for other k, chunks of 32 pixels.
int dwconv_wgrad_chunks(const DwShape& d) {
  const int64_t rows = int64_t(d.N) * d.Ho * d.Wo;
  int64_t q;
  if (d.k == 3 || d.k == 5) {
    const int64_t groups = (d.C + 31) / 32;
    q = (2 * num_sms() + groups - 1) / groups;
    q = std::min<int64_t>(q, (rows + 7) / 8);
  } else {
    q = (rows + 31) / 32;
  }
  q = std::max<int64_t>(1, std::min<int64_t>(q, 64));
  const int64_t per = (rows + q - 1) / q;
  return int((rows + per - 1) / per);
}

void dwconv_wgrad_pass(const DwShape& d, const void* dy, const void* x, int dt, float* pw, float* pb,
                       cudaStream_t st) {
  const int64_t rows = int64_t(d.N) * d.Ho * d.Wo;
  const int chunks = dwconv_wgrad_chunks(d);
  const int per = int((rows + chunks - 1) / chunks);
  if (d.k == 3 || d.k == 5) {
    dim3 grid(ceil_div(d.C, 32), chunks);
    FO_MB_DISPATCH(dt, T, {
      if (d.k == 3) launch_k(dwconv_wgrad_k<T, 3>, grid, 256, 0, st, (const T*)dy, (const T*)x, pw, pb, d, per);
      else launch_k(dwconv_wgrad_k<T, 5>, grid, 256, 0, st, (const T*)dy, (const T*)x, pw, pb, d, per);
    });
    return;
  }
  const int taps = d.k * d.k + (pb ? 1 : 0);
  dim3 grid(ceil_div(int64_t(taps) * d.C, 256), chunks);
  FO_MB_DISPATCH(dt, T, launch_k(dwconv_wgrad_any_k<T>, grid, 256, 0, st, (const T*)dy, (const T*)x, pw, pb, d, per));
}

void hswish_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st) {
  FO_MB_DISPATCH(dt, T, launch_k(hswish_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (T*)y, n));
}
void hswish_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st) {
  FO_MB_DISPATCH(dt, T, launch_k(hswish_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy,
                                                                                      (T*)dx, n, acc ? 1 : 0));
}
void hsigmoid_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st) {
  FO_MB_DISPATCH(dt, T, launch_k(hsigmoid_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (T*)y, n));
}
void hsigmoid_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st) {
  FO_MB_DISPATCH(dt, T, launch_k(hsigmoid_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy,
                                                                                        (T*)dx, n, acc ? 1 : 0));
}

void chmul_fwd(const void* x, const void* s, void* y, int N, int HW, int C, int dt, cudaStream_t st) {
  const int64_t n = int64_t(N) * HW * C;
  FO_MB_DISPATCH(dt, T, launch_k(chmul_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)s, (T*)y,
                                                                                     N, HW, C));
}
void chmul_bwd(const void* x, const void* s, const void* dy, void* dx, bool acc_dx, void* ds, bool acc_ds, int N,
               int HW, int C, int dt, cudaStream_t st) {
  const int64_t n = int64_t(N) * C;
  FO_MB_DISPATCH(dt, T, launch_k(chmul_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)s,
                                                                                     (const T*)dy, (T*)dx, (T*)ds, N,
                                                                                     HW, C, acc_dx ? 1 : 0,
                                                                                     acc_ds ? 1 : 0));
}

}  // namespace fo
