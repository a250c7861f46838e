// Elementwise, pooling, normalisation, loss, optimizer and aggregation
// kernels of the server step.  Activations are NHWC in fp32 or bf16 (the
// template parameter T); every arithmetic step runs in fp32.
#include "fo_common.cuh"
#include "fo_kernels.h"

#include <algorithm>
#include <cmath>
#include <cstdlib>

namespace fo {

static int g_num_sms = 0;

int elementwise_blocks(int64_t n_threads_needed, int threads) {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 1;
  }
  int64_t want = (n_threads_needed + threads - 1) / threads;
  int64_t cap = int64_t(g_num_sms) * 8;
  if (want > cap) want = cap;
  if (want < 1) want = 1;
  return int(want);
}

bool pdl_enabled() {
  static const bool on = getenv("FO_NO_PDL") == nullptr;
  return on;
}

#define FO_DISPATCH(dt, T, ...)   \
  do {                            \
    if ((dt) == kF32) {           \
      using T = float;            \
      __VA_ARGS__;                \
    } else {                      \
      using T = bf16;             \
      __VA_ARGS__;                \
    }                             \
  } while (0)

#define GRID_STRIDE(i, n) \
  for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < (n); i += int64_t(gridDim.x) * blockDim.x)

template <typename T>
__device__ __forceinline__ void store(T* p, int64_t i, float v, bool acc) {
  if (acc) v += to_f(p[i]);
  p[i] = from_f<T>(v);
}

// ------------------------------------------------------------------ relu
template <typename T>
__global__ void relu_fwd_k(const T* x, T* y, int64_t n) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) y[i] = from_f<T>(fmaxf(to_f(x[i]), 0.f));
}
template <typename T>
__global__ void relu_bwd_k(const T* x, const T* dy, T* dx, int64_t n, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) store(dx, i, to_f(x[i]) > 0.f ? to_f(dy[i]) : 0.f, acc);
}
void relu_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st) {
  FO_DISPATCH(dt, T, launch_k(relu_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (T*)y, n));
}
void relu_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st) {
  if (vec8_ok(dt, n)) return relu_bwd_x8(x, dy, dx, n, acc, st);
  FO_DISPATCH(dt, T, launch_k(relu_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy, (T*)dx, n, acc));
}

// --------------------------------------------------------------- maxpool
template <typename T>
__global__ void maxpool2_fwd_k(const T* x, T* y, int N, int H, int W, int C) {
  pdl_wait();
  pdl_trigger();
  const int Ho = H / 2, Wo = W / 2;
  const int64_t n_out = int64_t(N) * Ho * Wo * C;
  GRID_STRIDE(o, n_out) {
    int c = int(o % C);
    int64_t t = o / C;
    int j = int(t % Wo);
    t /= Wo;
    int i = int(t % Ho);
    int n = int(t / Ho);
    const T* base = x + ((int64_t(n) * H + 2 * i) * W + 2 * j) * C + c;
    float m = fmaxf(fmaxf(to_f(base[0]), to_f(base[C])),
                    fmaxf(to_f(base[int64_t(W) * C]), to_f(base[int64_t(W) * C + C])));
    y[o] = from_f<T>(m);
  }
}

// The window's gradient goes to its first maximum in row-major order
// (strict > scan); with relu_mask the routed gradient is also multiplied
// by (x > 0), the derivative of a ReLU that produced x.
template <typename T>
__global__ void maxpool2_bwd_k(const T* x, const T* dy, T* dx, int N, int H, int W, int C,
                               int acc, int relu_mask) {
  pdl_wait();
  pdl_trigger();
  const int Ho = H / 2, Wo = W / 2;
  const int64_t n_out = int64_t(N) * Ho * Wo * C;
  GRID_STRIDE(o, n_out) {
    int c = int(o % C);
    int64_t t = o / C;
    int j = int(t % Wo);
    t /= Wo;
    int i = int(t % Ho);
    int n = int(t / Ho);
    int64_t off[4];
    off[0] = ((int64_t(n) * H + 2 * i) * W + 2 * j) * C + c;
    off[1] = off[0] + C;
    off[2] = off[0] + int64_t(W) * C;
    off[3] = off[2] + C;
    float best = to_f(x[off[0]]);
    int arg = 0;
#pragma unroll
    for (int q = 1; q < 4; ++q) {
      float v = to_f(x[off[q]]);
      if (v > best) { best = v; arg = q; }
    }
    float g = to_f(dy[o]);
    if (relu_mask && !(best > 0.f)) g = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) store(dx, off[q], q == arg ? g : 0.f, acc);
  }
}
// 8 channels per thread with 16-byte loads (bf16, C % 8 == 0).
__global__ void maxpool2_fwd_x8_k(const bf16* __restrict__ x, bf16* __restrict__ y, int N, int H, int W, int C) {
  pdl_wait();
  pdl_trigger();
  const int Ho = H / 2, Wo = W / 2, C8 = C / 8;
  const int64_t n_out = int64_t(N) * Ho * Wo * C8;
  GRID_STRIDE(o, n_out) {
    const int c8 = int(o % C8);
    int64_t t = o / C8;
    const int j = int(t % Wo);
    t /= Wo;
    const int i = int(t % Ho);
    const int n = int(t / Ho);
    const int64_t b0 = ((int64_t(n) * H + 2 * i) * W + 2 * j) * C + 8 * c8;
    const int64_t offs[4] = {b0, b0 + C, b0 + int64_t(W) * C, b0 + int64_t(W) * C + C};
    uint4 u[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) u[q] = *reinterpret_cast<const uint4*>(x + offs[q]);
    uint4 r;
    bf16* rb = reinterpret_cast<bf16*>(&r);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float m = __bfloat162float(reinterpret_cast<const bf16*>(&u[0])[e]);
#pragma unroll
      for (int q = 1; q < 4; ++q) m = fmaxf(m, __bfloat162float(reinterpret_cast<const bf16*>(&u[q])[e]));
      rb[e] = __float2bfloat16_rn(m);
    }
    *reinterpret_cast<uint4*>(y + o * 8) = r;
  }
}

// Backward of the above (optionally fused with the ReLU mask of x): the
// window's gradient goes to its first maximum in row-major order.
__global__ void maxpool2_bwd_x8_k(const bf16* __restrict__ x, const bf16* __restrict__ dy, bf16* __restrict__ dx,
                                  int N, int H, int W, int C, int acc, int relu_mask) {
  pdl_wait();
  pdl_trigger();
  const int Ho = H / 2, Wo = W / 2, C8 = C / 8;
  const int64_t n_out = int64_t(N) * Ho * Wo * C8;
  GRID_STRIDE(o, n_out) {
    const int c8 = int(o % C8);
    int64_t t = o / C8;
    const int j = int(t % Wo);
    t /= Wo;
    const int i = int(t % Ho);
    const int n = int(t / Ho);
    const int64_t b0 = ((int64_t(n) * H + 2 * i) * W + 2 * j) * C + 8 * c8;
    const int64_t offs[4] = {b0, b0 + C, b0 + int64_t(W) * C, b0 + int64_t(W) * C + C};
    uint4 u[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) u[q] = *reinterpret_cast<const uint4*>(x + offs[q]);
    const uint4 g4 = *reinterpret_cast<const uint4*>(dy + o * 8);
    const bf16* gb = reinterpret_cast<const bf16*>(&g4);
    float out[4][8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float best = __bfloat162float(reinterpret_cast<const bf16*>(&u[0])[e]);
      int arg = 0;
#pragma unroll
      for (int q = 1; q < 4; ++q) {
        const float v = __bfloat162float(reinterpret_cast<const bf16*>(&u[q])[e]);
        if (v > best) { best = v; arg = q; }
      }
      float g = __bfloat162float(gb[e]);
      if (relu_mask && !(best > 0.f)) g = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) out[q][e] = q == arg ? g : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4* d = reinterpret_cast<uint4*>(dx + offs[q]);
      if (acc) {
        const uint4 old = *d;
#pragma unroll
        for (int e = 0; e < 8; ++e) out[q][e] += __bfloat162float(reinterpret_cast<const bf16*>(&old)[e]);
      }
      uint4 r;
      bf16* rb = reinterpret_cast<bf16*>(&r);
#pragma unroll
      for (int e = 0; e < 8; ++e) rb[e] = __float2bfloat16_rn(out[q][e]);
      *d = r;
    }
  }
}

// Backward of a 2x2 max-pool (after a ReLU) whose forward ran in the
// producing GEMM's epilogue: that epilogue stored the pooled values and, per
// pooled element and channel, the window position of the first maximum
// (code 0..3, row-major).  The window's gradient goes to that position if the
// pooled value is > 0 (the ReLU mask there), the other three get zero.
__global__ void maxpool2_bwd_codes_x8_k(const bf16* __restrict__ y, const uint8_t* __restrict__ code,
                                        const bf16* __restrict__ dy, bf16* __restrict__ dx, int N, int H, int W,
                                        int C, int acc) {
  pdl_wait();
  pdl_trigger();
  const int Ho = H / 2, Wo = W / 2, C8 = C / 8;
  const int64_t n_out = int64_t(N) * Ho * Wo * C8;
  GRID_STRIDE(o, n_out) {
    const int c8 = int(o % C8);
    int64_t t = o / C8;
    const int j = int(t % Wo);
    t /= Wo;
    const int i = int(t % Ho);
    const int n = int(t / Ho);
    const int64_t b0 = ((int64_t(n) * H + 2 * i) * W + 2 * j) * C + 8 * c8;
    const int64_t offs[4] = {b0, b0 + C, b0 + int64_t(W) * C, b0 + int64_t(W) * C + C};
    const uint4 y4 = *reinterpret_cast<const uint4*>(y + o * 8);
    const uint4 g4 = *reinterpret_cast<const uint4*>(dy + o * 8);
    const uint2 c2 = *reinterpret_cast<const uint2*>(code + o * 8);
    const bf16* yb = reinterpret_cast<const bf16*>(&y4);
    const bf16* gb = reinterpret_cast<const bf16*>(&g4);
    const uint8_t* cb = reinterpret_cast<const uint8_t*>(&c2);
    float out[4][8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float g = __bfloat162float(yb[e]) > 0.f ? __bfloat162float(gb[e]) : 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) out[q][e] = q == int(cb[e]) ? g : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4* d = reinterpret_cast<uint4*>(dx + offs[q]);
      if (acc) {
        const uint4 old = *d;
#pragma unroll
        for (int e = 0; e < 8; ++e) out[q][e] += __bfloat162float(reinterpret_cast<const bf16*>(&old)[e]);
      }
      uint4 r;
      bf16* rb = reinterpret_cast<bf16*>(&r);
#pragma unroll
      for (int e = 0; e < 8; ++e) rb[e] = __float2bfloat16_rn(out[q][e]);
      *d = r;
    }
  }
}

void relu_maxpool2_bwd_codes(const void* y, const uint8_t* code, const void* dy, void* dx, int N, int H, int W,
                             int C, bool acc, cudaStream_t st) {
  const int64_t n = int64_t(N) * (H / 2) * (W / 2) * C;
  launch_k(maxpool2_bwd_codes_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)y, code,
           (const bf16*)dy, (bf16*)dx, N, H, W, C, acc ? 1 : 0);
}

void maxpool2_fwd(const void* x, void* y, int N, int H, int W, int C, int dt, cudaStream_t st) {
  int64_t n = int64_t(N) * (H / 2) * (W / 2) * C;
  if (dt == kBF16 && C % 8 == 0) {
    launch_k(maxpool2_fwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, (bf16*)y, N, H, W, C);
    return;
  }
  FO_DISPATCH(dt, T, launch_k(maxpool2_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (T*)y, N, H, W, C));
}
void maxpool2_bwd(const void* x, const void* dy, void* dx, int N, int H, int W, int C, int dt,
                  bool acc, cudaStream_t st) {
  int64_t n = int64_t(N) * (H / 2) * (W / 2) * C;
  if (dt == kBF16 && C % 8 == 0) {
    launch_k(maxpool2_bwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, (const bf16*)dy, (bf16*)dx, N, H, W, C, acc, 0);
    return;
  }
  FO_DISPATCH(dt, T, launch_k(maxpool2_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy, (T*)dx, N, H, W, C, acc, 0));
}
void relu_maxpool2_bwd(const void* x, const void* dy, void* dx, int N, int H, int W, int C,
                       int dt, bool acc, cudaStream_t st) {
  int64_t n = int64_t(N) * (H / 2) * (W / 2) * C;
  if (dt == kBF16 && C % 8 == 0) {
    launch_k(maxpool2_bwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, (const bf16*)dy, (bf16*)dx, N, H, W, C, acc, 1);
    return;
  }
  FO_DISPATCH(dt, T, launch_k(maxpool2_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy, (T*)dx, N, H, W, C, acc, 1));
}

// ---------------------------------------------------------- affine / add
template <typename T>
__global__ void affine_fwd_k(const T* x, const float* sc, const float* sh, T* y, int64_t n, int C, int relu) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) {
    int c = int(i % C);
    float v = fmaf(to_f(x[i]), sc[c], sh[c]);
    y[i] = from_f<T>(relu ? fmaxf(v, 0.f) : v);
  }
}
template <typename T>
__global__ void affine_dx_k(const T* dy, const float* sc, T* dx, int64_t n, int C, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) store(dx, i, to_f(dy[i]) * sc[int(i % C)], acc);
}
template <typename T>
__global__ void add_fwd_k(const T* a, const T* b, T* y, int64_t n, int relu) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) {
    float v = to_f(a[i]) + to_f(b[i]);
    y[i] = from_f<T>(relu ? fmaxf(v, 0.f) : v);
  }
}
template <typename T>
__global__ void grad_split_k(const T* __restrict__ dy, const T* __restrict__ mask, T* __restrict__ d0, int acc0,
                             T* __restrict__ d1, int acc1, int64_t n) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) {
    const float g = (mask && !(to_f(mask[i]) > 0.f)) ? 0.f : to_f(dy[i]);
    store(d0, i, g, acc0);
    if (d1) store(d1, i, g, acc1);
  }
}
void grad_split(const void* dy, const void* mask, void* d0, bool acc0, void* d1, bool acc1, int64_t n, int dt,
                cudaStream_t st) {
  if (vec8_ok(dt, n)) return grad_split_x8(dy, mask, d0, acc0, d1, acc1, n, st);
  FO_DISPATCH(dt, T, launch_k(grad_split_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)dy, (const T*)mask,
                              (T*)d0, acc0 ? 1 : 0, (T*)d1, acc1 ? 1 : 0, n));
}
void affine_fwd(const void* x, const float* scale, const float* shift, void* y, int64_t rows,
                int C, int dt, bool relu, cudaStream_t st) {
  int64_t n = rows * C;
  if (vec8_ok(dt, n) && C % 8 == 0) return affine_fwd_x8(x, scale, shift, y, n, C, relu, st);
  FO_DISPATCH(dt, T, launch_k(affine_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, scale, shift, (T*)y, n, C, relu));
}
void affine_dx(const void* dy, const float* scale, void* dx, int64_t rows, int C, int dt,
               bool acc, cudaStream_t st) {
  int64_t n = rows * C;
  FO_DISPATCH(dt, T, launch_k(affine_dx_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)dy, scale, (T*)dx, n, C, acc));
}
void add_fwd(const void* a, const void* b, void* y, int64_t n, int dt, bool relu, cudaStream_t st) {
  if (vec8_ok(dt, n)) return add_x8(a, b, y, n, relu, st);
  FO_DISPATCH(dt, T, launch_k(add_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)a, (const T*)b, (T*)y, n, relu));
}

// -------------------------------------------------------------- avgpool
template <typename T>
__global__ void avgpool_fwd_k(const T* x, T* y, int N, int HW, int C) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(o, int64_t(N) * C) {
    int c = int(o % C);
    int64_t n = o / C;
    float s = 0.f;
    for (int p = 0; p < HW; ++p) s += to_f(x[(n * HW + p) * C + c]);
    y[o] = from_f<T>(s / float(HW));
  }
}
template <typename T>
__global__ void avgpool_bwd_k(const T* dy, T* dx, int N, int HW, int C, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, int64_t(N) * HW * C) {
    int c = int(i % C);
    int64_t n = i / (int64_t(HW) * C);
    store(dx, i, to_f(dy[n * C + c]) / float(HW), acc);
  }
}
void avgpool_fwd(const void* x, void* y, int N, int HW, int C, int dt, cudaStream_t st) {
  FO_DISPATCH(dt, T, launch_k(avgpool_fwd_k<T>, elementwise_blocks(int64_t(N) * C, 256), 256, 0, st, (const T*)x, (T*)y, N, HW, C));
}
void avgpool_bwd(const void* dy, void* dx, int N, int HW, int C, int dt, bool acc, cudaStream_t st) {
  FO_DISPATCH(dt, T, launch_k(avgpool_bwd_k<T>, elementwise_blocks(int64_t(N) * HW * C, 256), 256, 0, st, (const T*)dy, (T*)dx, N, HW, C, acc));
}

// ----------------------------------------------------------------- gelu
template <typename T>
__global__ void gelu_fwd_k(const T* x, T* y, int64_t n) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) {
    const float v = to_f(x[i]);
    float cdf, pdf;
    normal_cdf_pdf(v, cdf, pdf);
    y[i] = from_f<T>(v * cdf);
  }
}
template <typename T>
__global__ void gelu_bwd_k(const T* x, const T* dy, T* dx, int64_t n, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) {
    const float v = to_f(x[i]);
    float cdf, pdf;
    normal_cdf_pdf(v, cdf, pdf);
    store(dx, i, to_f(dy[i]) * (cdf + v * pdf), acc);
  }
}
void gelu_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st) {
  if (vec8_ok(dt, n)) return gelu_fwd_x8(x, y, n, st);
  FO_DISPATCH(dt, T, launch_k(gelu_fwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (T*)y, n));
}
void gelu_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st) {
  if (vec8_ok(dt, n)) return gelu_bwd_x8(x, dy, dx, n, acc, st);
  FO_DISPATCH(dt, T, launch_k(gelu_bwd_k<T>, elementwise_blocks(n, 256), 256, 0, st, (const T*)x, (const T*)dy, (T*)dx, n, acc));
}

// ------------------------------------------------------------ layernorm
// One warp per row (C <= 1024, C a multiple of 32).
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T>
__global__ void layernorm_fwd_k(const T* x, const float* gamma, const float* beta, T* y,
                                float* mean_out, float* rstd_out, int64_t rows, int C) {
  pdl_wait();
  pdl_trigger();
  int64_t row = int64_t(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32;
  int lane = threadIdx.x % 32;
  if (row >= rows) return;
  const T* xr = x + row * C;
  float s = 0.f;
  for (int c = lane; c < C; c += 32) s += to_f(xr[c]);
  float mu = warp_sum(s) / float(C);
  float q = 0.f;
  for (int c = lane; c < C; c += 32) {
    float d = to_f(xr[c]) - mu;
    q += d * d;
  }
  float var = warp_sum(q) / float(C);
  float rs = rsqrtf(var + 1e-5f);
  T* yr = y + row * C;
  for (int c = lane; c < C; c += 32) yr[c] = from_f<T>((to_f(xr[c]) - mu) * rs * gamma[c] + beta[c]);
  if (lane == 0) {
    mean_out[row] = mu;
    rstd_out[row] = rs;
  }
}
template <typename T>
__global__ void layernorm_bwd_k(const T* x, const float* gamma, const float* mean,
                                const float* rstd, const T* dy, T* dx, int64_t rows, int C,
                                int acc) {
  pdl_wait();
  pdl_trigger();
  int64_t row = int64_t(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32;
  int lane = threadIdx.x % 32;
  if (row >= rows) return;
  const T* xr = x + row * C;
  const T* dyr = dy + row * C;
  float mu = mean[row], rs = rstd[row];
  float a = 0.f, b = 0.f;
  for (int c = lane; c < C; c += 32) {
    float xh = (to_f(xr[c]) - mu) * rs;
    float dxh = to_f(dyr[c]) * gamma[c];
    a += dxh;
    b += dxh * xh;
  }
  a = warp_sum(a) / float(C);
  b = warp_sum(b) / float(C);
  T* dxr = dx + row * C;
  for (int c = lane; c < C; c += 32) {
    float xh = (to_f(xr[c]) - mu) * rs;
    float dxh = to_f(dyr[c]) * gamma[c];
    store(dxr, c, rs * (dxh - a - xh * b), acc);
  }
}
void layernorm_fwd(const void* x, const float* gamma, const float* beta, void* y, float* mean,
                   float* rstd, int64_t rows, int C, int dt, cudaStream_t st) {
  if (layernorm_fwd8_ok(dt, C)) return layernorm_fwd_x8(x, gamma, beta, y, mean, rstd, rows, C, st);
  int blocks = ceil_div(rows, 8);
  FO_DISPATCH(dt, T, launch_k(layernorm_fwd_k<T>, blocks, 256, 0, st, (const T*)x, gamma, beta, (T*)y, mean, rstd, rows, C));
}
void layernorm_bwd_dx(const void* x, const float* gamma, const float* mean, const float* rstd,
                      const void* dy, void* dx, int64_t rows, int C, int dt, bool acc,
                      cudaStream_t st) {
  int blocks = ceil_div(rows, 8);
  FO_DISPATCH(dt, T, launch_k(layernorm_bwd_k<T>, blocks, 256, 0, st, (const T*)x, gamma, mean, rstd, (const T*)dy, (T*)dx, rows, C, acc));
}

// ---------------------------------------------------- column reductions
// Deterministic two-pass column sums: pass 1 writes one partial per
// (row chunk, column), pass 2 adds the chunks in order.
constexpr int CS_ROWS = 128;   // rows per chunk (generic kernel)
static int colsum_chunks(int64_t rows) { return ceil_div(rows, CS_ROWS); }
int64_t colsum_partial_floats(int64_t rows, int C) { return int64_t(colsum_chunks(rows)) * C; }

// MODE 0: a;  1: a * b;  2: a * (b - mean[r]) * rstd[r]
template <int MODE, typename T>
__global__ void colsum_partial_k(const T* a, const T* b, const float* mean, const float* rstd,
                                 int64_t rows, int C, float* partial) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[8][33];
  int cl = threadIdx.x % 32, rl = threadIdx.x / 32;
  int c = blockIdx.x * 32 + cl;
  int64_t r0 = int64_t(blockIdx.y) * CS_ROWS;
  float s = 0.f;
  if (c < C) {
    for (int64_t r = r0 + rl; r < r0 + CS_ROWS && r < rows; r += 8) {
      float v = to_f(a[r * C + c]);
      if (MODE == 1) v *= to_f(b[r * C + c]);
      if (MODE == 2) v *= (to_f(b[r * C + c]) - mean[r]) * rstd[r];
      s += v;
    }
  }
  red[rl][cl] = s;
  __syncthreads();
  if (rl == 0 && c < C) {
    float t = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) t += red[q][cl];
    partial[int64_t(blockIdx.y) * C + c] = t;
  }
}
// Adds the per-chunk partials of each column: 8 row lanes per column sum
// interleaved chunks, then combine in a fixed order (deterministic).
__global__ void colsum_finish_k(const float* partial, int chunks, int C, float* out) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[8][33];
  const int cl = threadIdx.x % 32, rl = threadIdx.x / 32;
  const int c = blockIdx.x * 32 + cl;
  float s = 0.f;
  if (c < C) {
    int q = rl;
    for (; q + 24 < chunks; q += 32) {   // four independent loads in flight
      const float a0 = partial[int64_t(q) * C + c], a1 = partial[int64_t(q + 8) * C + c];
      const float a2 = partial[int64_t(q + 16) * C + c], a3 = partial[int64_t(q + 24) * C + c];
      s += a0;
      s += a1;
      s += a2;
      s += a3;
    }
    for (; q < chunks; q += 8) s += partial[int64_t(q) * C + c];
  }
  red[rl][cl] = s;
  __syncthreads();
  if (rl == 0 && c < C) {
    float t = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) t += red[q][cl];
    out[c] = t;
  }
}

// Scratch the server's column sums may use: every variant it launches.
int64_t server_colsum_floats(int64_t rows, int C) {
  int64_t a = colsum_partial_floats(rows, C);
  int64_t b = 2 * colsum8_partial_floats(rows, C, true);
  int64_t c = layernorm_bwd8_partial_floats(rows, C);
  return std::max(a, std::max(b, c));
}

void colsum(const void* a, const void* b, int64_t rows, int C, int dt, float* partial, float* out,
            cudaStream_t st, bool adaptive) {
  if (!b && dt == kBF16 && C % 8 == 0) return colsum8(a, rows, C, partial, out, adaptive, st);
  dim3 grid(ceil_div(C, 32), colsum_chunks(rows));
  if (b) {
    FO_DISPATCH(dt, T, launch_k(colsum_partial_k<1, T>, grid, 256, 0, st, (const T*)a, (const T*)b, nullptr, nullptr, rows, C, partial));
  } else {
    FO_DISPATCH(dt, T, launch_k(colsum_partial_k<0, T>, grid, 256, 0, st, (const T*)a, nullptr, nullptr, nullptr, rows, C, partial));
  }
  launch_k(colsum_finish_k, ceil_div(C, 32), 256, 0, st, partial, colsum_chunks(rows), C, out);
}
void colsum_lnx(const void* dy, const void* x, const float* mean, const float* rstd, int64_t rows,
                int C, int dt, float* partial, float* out, cudaStream_t st) {
  dim3 grid(ceil_div(C, 32), colsum_chunks(rows));
  FO_DISPATCH(dt, T, launch_k(colsum_partial_k<2, T>, grid, 256, 0, st, (const T*)dy, (const T*)x, mean, rstd, rows, C, partial));
  launch_k(colsum_finish_k, ceil_div(C, 32), 256, 0, st, partial, colsum_chunks(rows), C, out);
}

// ------------------------------------------------------------- meanpool
template <typename T>
__global__ void meanpool_fwd_k(const T* x, const int32_t* len, T* y, int B, int L, int C) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(o, int64_t(B) * C) {
    int c = int(o % C);
    int b = int(o / C);
    int n = len[b];
    float s = 0.f;
    for (int i = 0; i < n; ++i) s += to_f(x[(int64_t(b) * L + i) * C + c]);
    y[o] = from_f<T>(s / float(n));
  }
}
template <typename T>
__global__ void meanpool_bwd_k(const T* dy, const int32_t* len, T* dx, int B, int L, int C, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, int64_t(B) * L * C) {
    int c = int(i % C);
    int64_t t = i / C;
    int tok = int(t % L);
    int b = int(t / L);
    int n = len[b];
    store(dx, i, tok < n ? to_f(dy[int64_t(b) * C + c]) / float(n) : 0.f, acc);
  }
}
void meanpool_fwd(const void* x, const int32_t* len, void* y, int B, int L, int C, int dt,
                  cudaStream_t st) {
  if (meanpool8_ok(dt, C)) return meanpool_fwd_x8(x, len, y, B, L, C, st);
  FO_DISPATCH(dt, T, launch_k(meanpool_fwd_k<T>, elementwise_blocks(int64_t(B) * C, 256), 256, 0, st, (const T*)x, len, (T*)y, B, L, C));
}
void meanpool_bwd(const void* dy, const int32_t* len, void* dx, int B, int L, int C, int dt,
                  bool acc, cudaStream_t st) {
  if (meanpool8_ok(dt, C)) return meanpool_bwd_x8(dy, len, dx, B, L, C, acc, st);
  FO_DISPATCH(dt, T, launch_k(meanpool_bwd_k<T>, elementwise_blocks(int64_t(B) * L * C, 256), 256, 0, st, (const T*)dy, len, (T*)dx, B, L, C, acc));
}

// ------------------------------------------------------ softmax + CE loss
// One block; warp w handles rows w, w + 8, ...  The batch-mean loss is
// summed in a fixed order.
template <typename T>
__global__ void softmax_ce_k(const float* z, const int32_t* labels, int B, int C, float* losses,
                             const int64_t* step, int64_t mask, T* dz) {
  pdl_wait();
  pdl_trigger();
  __shared__ float row_loss[1024];
  int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int b = warp; b < B; b += blockDim.x / 32) {
    const float* zr = z + int64_t(b) * C;
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, zr[c]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float s = 0.f;
    for (int c = lane; c < C; c += 32) s += expf(zr[c] - m);
    s = warp_sum(s);
    int y = labels[b];
    float lse = m + logf(s);
    for (int c = lane; c < C; c += 32) {
      float p = expf(zr[c] - m) / s;
      dz[int64_t(b) * C + c] = from_f<T>((p - (c == y ? 1.f : 0.f)) / float(B));
    }
    if (lane == 0) row_loss[b] = lse - zr[y];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int b = 0; b < B; ++b) t += row_loss[b];
    losses[*step & mask] = t / float(B);
  }
}
void softmax_ce(const float* logits, const int32_t* labels, int B, int C, float* losses,
                const int64_t* step, int64_t mask, void* dlogits, int dt, cudaStream_t st) {
  FO_DISPATCH(dt, T, launch_k(softmax_ce_k<T>, 1, 256, 0, st, logits, labels, B, C, losses, step, mask, (T*)dlogits));
}

// ------------------------------------------------------ SGD with momentum
// 16-byte vector loads/stores; n is a multiple of 4.  skip64 (may be null)
// marks 64-element blocks updated earlier in the step, which are left alone.
__global__ void sgd_momentum_k(float4* __restrict__ theta, float4* __restrict__ v,
                               const float4* __restrict__ g, uint2* __restrict__ shadow,
                               int64_t n4, float lr, float mu, int64_t* step, const uint8_t* __restrict__ skip64) {
  pdl_wait();
  pdl_trigger();
  if (step && blockIdx.x == 0 && threadIdx.x == 0) *step += 1;
  GRID_STRIDE(i, n4) {
    if (skip64 && skip64[i / 16]) continue;
    float4 t = theta[i], m = v[i];
    const float4 gr = g[i];
    m.x = fmaf(mu, m.x, gr.x);
    m.y = fmaf(mu, m.y, gr.y);
    m.z = fmaf(mu, m.z, gr.z);
    m.w = fmaf(mu, m.w, gr.w);
    t.x = fmaf(-lr, m.x, t.x);
    t.y = fmaf(-lr, m.y, t.y);
    t.z = fmaf(-lr, m.z, t.z);
    t.w = fmaf(-lr, m.w, t.w);
    v[i] = m;
    theta[i] = t;
    if (shadow) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(t.x, t.y), hi = __floats2bfloat162_rn(t.z, t.w);
      uint2 u;
      u.x = *reinterpret_cast<uint32_t*>(&lo);
      u.y = *reinterpret_cast<uint32_t*>(&hi);
      shadow[i] = u;
    }
  }
}
void sgd_momentum(float* theta, float* v, const float* g, void* shadow, int64_t n, float lr,
                  float mu, int64_t* step, cudaStream_t st, const uint8_t* skip64) {
  int64_t n4 = n / 4;
  launch_k(sgd_momentum_k, elementwise_blocks(n4, 256), 256, 0, st,
      (float4*)theta, (float4*)v, (const float4*)g, (uint2*)shadow, n4, lr, mu, step, skip64);
}
// The same update over a list of 64-element blocks (the parameters an
// earlier partial update left): 16 float4 per block.
__global__ void sgd_momentum_blocks_k(float4* __restrict__ theta, float4* __restrict__ v,
                                      const float4* __restrict__ g, uint2* __restrict__ shadow,
                                      const int64_t* __restrict__ blocks, int64_t nb, float lr, float mu,
                                      int64_t* step) {
  pdl_wait();
  pdl_trigger();
  if (step && blockIdx.x == 0 && threadIdx.x == 0) *step += 1;
  GRID_STRIDE(j, nb * 16) {
    const int64_t i = blocks[j / 16] * 16 + j % 16;
    float4 t = theta[i], m = v[i];
    const float4 gr = g[i];
    m.x = fmaf(mu, m.x, gr.x);
    m.y = fmaf(mu, m.y, gr.y);
    m.z = fmaf(mu, m.z, gr.z);
    m.w = fmaf(mu, m.w, gr.w);
    t.x = fmaf(-lr, m.x, t.x);
    t.y = fmaf(-lr, m.y, t.y);
    t.z = fmaf(-lr, m.z, t.z);
    t.w = fmaf(-lr, m.w, t.w);
    v[i] = m;
    theta[i] = t;
    if (shadow) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(t.x, t.y), hi = __floats2bfloat162_rn(t.z, t.w);
      uint2 u;
      u.x = *reinterpret_cast<uint32_t*>(&lo);
      u.y = *reinterpret_cast<uint32_t*>(&hi);
      shadow[i] = u;
    }
  }
}
void sgd_momentum_blocks(float* theta, float* v, const float* g, void* shadow, const int64_t* blocks64, int64_t nb,
                         float lr, float mu, int64_t* step, cudaStream_t st) {
  launch_k(sgd_momentum_blocks_k, elementwise_blocks(nb * 16, 256), 256, 0, st, (float4*)theta, (float4*)v,
           (const float4*)g, (uint2*)shadow, blocks64, nb, lr, mu, step);
}
// The same update over up to kSgdMaxSegs contiguous segments of the
// parameter vector in one launch (weight tensors whose gradients are final),
// so that several small tensors share the launch and its ramp: thread j of the
// concatenated float4 range finds its segment in the prefix table.
__global__ void sgd_momentum_segs_k(float4* __restrict__ theta, float4* __restrict__ v,
                                    const float4* __restrict__ g, uint2* __restrict__ shadow,
                                    const __grid_constant__ SgdSegments sg, float lr, float mu) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(j, sg.pre4[sg.n]) {
    int k = 0;
    while (k + 1 < sg.n && sg.pre4[k + 1] <= j) ++k;
    const int64_t i = sg.off4[k] + (j - sg.pre4[k]);
    float4 t = theta[i], m = v[i];
    const float4 gr = g[i];
    m.x = fmaf(mu, m.x, gr.x);
    m.y = fmaf(mu, m.y, gr.y);
    m.z = fmaf(mu, m.z, gr.z);
    m.w = fmaf(mu, m.w, gr.w);
    t.x = fmaf(-lr, m.x, t.x);
    t.y = fmaf(-lr, m.y, t.y);
    t.z = fmaf(-lr, m.z, t.z);
    t.w = fmaf(-lr, m.w, t.w);
    v[i] = m;
    theta[i] = t;
    if (shadow) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(t.x, t.y), hi = __floats2bfloat162_rn(t.z, t.w);
      uint2 u;
      u.x = *reinterpret_cast<uint32_t*>(&lo);
      u.y = *reinterpret_cast<uint32_t*>(&hi);
      shadow[i] = u;
    }
  }
}
void sgd_momentum_segments(float* theta, float* v, const float* g, void* shadow, const SgdSegments& sg, float lr,
                           float mu, cudaStream_t st) {
  if (sg.n <= 0) return;
  launch_k(sgd_momentum_segs_k, elementwise_blocks(sg.pre4[sg.n], 256), 256, 0, st, (float4*)theta, (float4*)v,
           (const float4*)g, (uint2*)shadow, sg, lr, mu);
}
__global__ void f32_to_bf16_k(const float* x, bf16* y, int64_t n) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) y[i] = __float2bfloat16_rn(x[i]);
}
void f32_to_bf16(const float* x, void* y, int64_t n, cudaStream_t st) {
  launch_k(f32_to_bf16_k, elementwise_blocks(n, 256), 256, 0, st, x, (bf16*)y, n);
}

// ------------------------------------------------------ FedAsync axpby
// g = fmaf(alpha, l - g, g): read g and l, write g (12 bytes per element).
// Two independent 16-byte loads per operand per iteration for memory-level
// parallelism; the scalar head/tail handles n % 8 and unaligned pointers.
__global__ void axpby_vec_k(float4* __restrict__ g, const float4* __restrict__ l, int64_t n8,
                            float alpha) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = int64_t(gridDim.x) * blockDim.x;
  for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < n8; i += stride) {
    float4 a0 = g[2 * i], a1 = g[2 * i + 1];
    const float4 b0 = __ldcs(&l[2 * i]), b1 = __ldcs(&l[2 * i + 1]);
    a0.x = fmaf(alpha, b0.x - a0.x, a0.x);
    a0.y = fmaf(alpha, b0.y - a0.y, a0.y);
    a0.z = fmaf(alpha, b0.z - a0.z, a0.z);
    a0.w = fmaf(alpha, b0.w - a0.w, a0.w);
    a1.x = fmaf(alpha, b1.x - a1.x, a1.x);
    a1.y = fmaf(alpha, b1.y - a1.y, a1.y);
    a1.z = fmaf(alpha, b1.z - a1.z, a1.z);
    a1.w = fmaf(alpha, b1.w - a1.w, a1.w);
    g[2 * i] = a0;
    g[2 * i + 1] = a1;
  }
}
__global__ void axpby_scalar_k(float* g, const float* l, int64_t n, float alpha) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE(i, n) g[i] = fmaf(alpha, l[i] - g[i], g[i]);
}
int axpby_kernels(const float* g, const float* l, int64_t n) {
  if (n <= 0) return 0;
  bool aligned = ((reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(l)) & 15) == 0;
  int64_t n8 = aligned ? n / 8 : 0;
  return (n8 > 0 ? 1 : 0) + (n8 * 8 < n ? 1 : 0);
}

void axpby(float* g, const float* l, int64_t n, float alpha, cudaStream_t st) {
  if (n <= 0) return;
  bool aligned = ((reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(l)) & 15) == 0;
  int64_t n8 = aligned ? n / 8 : 0;
  if (n8 > 0) launch_k(axpby_vec_k, elementwise_blocks(n8, 256), 256, 0, st, (float4*)g, (const float4*)l, n8, alpha);
  int64_t done = n8 * 8;
  if (done < n)
    launch_k(axpby_scalar_k, elementwise_blocks(n - done, 256), 256, 0, st, g + done, l + done, n - done, alpha);
}

}  // namespace fo
