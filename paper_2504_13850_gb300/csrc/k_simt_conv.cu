// CUDA-core implicit-GEMM convolution (forward, input gradient, weight
// gradient) with fp32 accumulation.  This is the fp32 compute path of the
// library (the fp32 tiny workload) and serves layers whose shapes the
// tensor-core kernels do not take (e.g. a classifier with 10 outputs).
//
// All three passes are one tiled GEMM C[M][N] = sum_k A[M][k] B[k][N] whose
// operands are gathered on the fly from NHWC tensors:
//   FWD    M = output pixels, N = Co, k = (r, s, ci):  A = x window, B = w
//   DGRAD  M = input pixels,  N = Ci, k = (r, s, co):  A = dy (strided), B = w
//   WGRAD  M = Co, N = (r, s, ci), k = output pixel:   A = dy^T, B = x window
#include "fo_common.cuh"
#include "fo_kernels.h"

#include <algorithm>

namespace fo {

namespace {

enum Mode { FWD = 0, DGRAD = 1, WGRAD = 2 };

constexpr int BM = 64, BN = 64, BK = 16, NT = 256;

struct Geo {
  int N, H, W, Ci, Co, k, stride, pad, Ho, Wo;
  int64_t M, Ncol, K;
  int64_t kper;   // k-range per blockIdx.z (K split); the output of split z starts at c + z * M * Ncol
};

template <typename T>
__device__ __forceinline__ float ld(const T* p, int64_t i) { return to_f(p[i]); }

// A[m][kk]
template <int MODE, typename TA>
__device__ __forceinline__ float load_a(const Geo& g, const TA* a, int64_t m, int64_t kk) {
  if (m >= g.M || kk >= g.K) return 0.f;
  if (MODE == FWD) {
    int ci = int(kk % g.Ci);
    int rs = int(kk / g.Ci);
    int r = rs / g.k, s = rs % g.k;
    int wo = int(m % g.Wo);
    int64_t t = m / g.Wo;
    int ho = int(t % g.Ho);
    int n = int(t / g.Ho);
    int h = ho * g.stride + r - g.pad, w = wo * g.stride + s - g.pad;
    if (h < 0 || h >= g.H || w < 0 || w >= g.W) return 0.f;
    return ld(a, ((int64_t(n) * g.H + h) * g.W + w) * g.Ci + ci);
  } else if (MODE == DGRAD) {
    int co = int(kk % g.Co);
    int rs = int(kk / g.Co);
    int r = rs / g.k, s = rs % g.k;
    int w = int(m % g.W);
    int64_t t = m / g.W;
    int h = int(t % g.H);
    int n = int(t / g.H);
    int hh = h + g.pad - r, ww = w + g.pad - s;
    if (hh < 0 || ww < 0 || hh % g.stride || ww % g.stride) return 0.f;
    int ho = hh / g.stride, wo = ww / g.stride;
    if (ho >= g.Ho || wo >= g.Wo) return 0.f;
    return ld(a, ((int64_t(n) * g.Ho + ho) * g.Wo + wo) * g.Co + co);
  } else {  // WGRAD: A[co][p] = dy[p][co]
    return ld(a, kk * g.Co + m);
  }
}

// B[kk][ncol]
template <int MODE, typename TB>
__device__ __forceinline__ float load_b(const Geo& g, const TB* b, int64_t kk, int64_t nc) {
  if (kk >= g.K || nc >= g.Ncol) return 0.f;
  if (MODE == FWD) {
    return ld(b, nc * g.K + kk);                  // w[co][(r,s,ci)]
  } else if (MODE == DGRAD) {
    int co = int(kk % g.Co);
    int rs = int(kk / g.Co);                      // w[co][r][s][ci]
    return ld(b, (int64_t(co) * g.k * g.k + rs) * g.Ci + nc);
  } else {  // WGRAD: B[p][(r,s,ci)] = x window
    int ci = int(nc % g.Ci);
    int rs = int(nc / g.Ci);
    int r = rs / g.k, s = rs % g.k;
    int wo = int(kk % g.Wo);
    int64_t t = kk / g.Wo;
    int ho = int(t % g.Ho);
    int n = int(t / g.Ho);
    int h = ho * g.stride + r - g.pad, w = wo * g.stride + s - g.pad;
    if (h < 0 || h >= g.H || w < 0 || w >= g.W) return 0.f;
    return ld(b, ((int64_t(n) * g.H + h) * g.W + w) * g.Ci + ci);
  }
}

template <int MODE, typename TA, typename TB, typename TC>
__global__ void __launch_bounds__(NT) simt_conv_kernel(Geo g, const TA* __restrict__ a,
                                                       const TB* __restrict__ b,
                                                       const float* __restrict__ bias,
                                                       TC* __restrict__ c, int relu, int acc,
                                                       const TC* __restrict__ mask) {
  pdl_wait();
  pdl_trigger();
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int64_t m0 = int64_t(blockIdx.y) * BM, n0 = int64_t(blockIdx.x) * BN;
  const int64_t kb = int64_t(blockIdx.z) * g.kper, ke = min(g.K, kb + g.kper);
  c += int64_t(blockIdx.z) * g.M * g.Ncol;
  float accum[4][4] = {};
  for (int64_t k0 = kb; k0 < ke; k0 += BK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      int e = tid + i * NT;           // 0..1023
      int am = e / BK, ak = e % BK;   // A tile 64 x 16
      As[ak][am] = k0 + ak < ke ? load_a<MODE>(g, a, m0 + am, k0 + ak) : 0.f;
      int bk = e / BN, bn = e % BN;   // B tile 16 x 64
      Bs[bk][bn] = k0 + bk < ke ? load_b<MODE>(g, b, k0 + bk, n0 + bn) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) accum[i][j] = fmaf(av[i], bv[j], accum[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int64_t m = m0 + ty + 16 * i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int64_t n = n0 + tx + 16 * j;
      if (n >= g.Ncol) continue;
      float v = accum[i][j];
      if (bias) v += bias[n];
      if (relu) v = fmaxf(v, 0.f);
      int64_t idx = m * g.Ncol + n;
      if (mask && !(to_f(mask[idx]) > 0.f)) v = 0.f;
      if (acc) v += to_f(c[idx]);
      c[idx] = from_f<TC>(v);
    }
  }
}

Geo make_geo(const ConvShape& s, int mode) {
  Geo g{s.N, s.H, s.W, s.Ci, s.Co, s.k, s.stride, s.pad, s.Ho, s.Wo, 0, 0, 0, 0};
  int64_t pix_out = int64_t(s.N) * s.Ho * s.Wo, pix_in = int64_t(s.N) * s.H * s.W;
  if (mode == FWD) {
    g.M = pix_out; g.Ncol = s.Co; g.K = int64_t(s.k) * s.k * s.Ci;
  } else if (mode == DGRAD) {
    g.M = pix_in; g.Ncol = s.Ci; g.K = int64_t(s.k) * s.k * s.Co;
  } else {
    g.M = s.Co; g.Ncol = int64_t(s.k) * s.k * s.Ci; g.K = pix_out;
  }
  g.kper = g.K;
  return g;
}

// Sums the `splits` partial outputs [splits][n] in order.
__global__ void sum_splits_k(const float* __restrict__ part, int splits, int64_t n, float* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x) {
    float t = 0.f;
    for (int z = 0; z < splits; ++z) t += part[int64_t(z) * n + i];
    out[i] = t;
  }
}

int sm_count() {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 148;
  }
  return sms;
}

template <int MODE, typename TA, typename TB, typename TC>
void launch(const Geo& g, const void* a, const void* b, const float* bias, void* c, bool relu,
            bool acc, cudaStream_t st, const void* mask = nullptr) {
  dim3 grid(ceil_div(g.Ncol, BN), ceil_div(g.M, BM), unsigned(ceil_div(g.K, g.kper)));
  launch_k(simt_conv_kernel<MODE, TA, TB, TC>, grid, NT, 0, st, 
      g, (const TA*)a, (const TB*)b, bias, (TC*)c, relu ? 1 : 0, acc ? 1 : 0, (const TC*)mask);
}

// Instantiate every (A, B, C) dtype combination of one pass.
template <int MODE, typename TA, typename TB>
void launch_c(const Geo& g, const void* a, const void* b, const float* bias, void* c, int dtc,
              bool relu, bool acc, cudaStream_t st, const void* mask) {
  if (dtc == kF32) launch<MODE, TA, TB, float>(g, a, b, bias, c, relu, acc, st, mask);
  else launch<MODE, TA, TB, bf16>(g, a, b, bias, c, relu, acc, st, mask);
}
template <int MODE, typename TA>
void launch_bc(const Geo& g, const void* a, const void* b, int dtb, const float* bias, void* c,
               int dtc, bool relu, bool acc, cudaStream_t st, const void* mask) {
  if (dtb == kF32) launch_c<MODE, TA, float>(g, a, b, bias, c, dtc, relu, acc, st, mask);
  else launch_c<MODE, TA, bf16>(g, a, b, bias, c, dtc, relu, acc, st, mask);
}
template <int MODE>
void launch_any(const Geo& g, const void* a, int dta, const void* b, int dtb, const float* bias,
                void* c, int dtc, bool relu, bool acc, cudaStream_t st, const void* mask = nullptr) {
  if (dta == kF32) launch_bc<MODE, float>(g, a, b, dtb, bias, c, dtc, relu, acc, st, mask);
  else launch_bc<MODE, bf16>(g, a, b, dtb, bias, c, dtc, relu, acc, st, mask);
}

}  // namespace

void conv_fwd_simt(const ConvShape& s, const void* x, int dt_x, const void* w, int dt_w,
                   const float* bias, void* y, int dt_y, bool relu, cudaStream_t st) {
  launch_any<FWD>(make_geo(s, FWD), x, dt_x, w, dt_w, bias, y, dt_y, relu, false, st);
}

void conv_dgrad_simt(const ConvShape& s, const void* dy, int dt_dy, const void* w, int dt_w,
                     void* dx, int dt_dx, bool accumulate, const void* mask, cudaStream_t st) {
  launch_any<DGRAD>(make_geo(s, DGRAD), dy, dt_dy, w, dt_w, nullptr, dx, dt_dx, false, accumulate, st, mask);
}

// The weight gradient's K (output pixels) is long and its output small:
// split K so the grid covers about two blocks per SM, into fp32 partials that
// a second pass sums in split order (deterministic).
int simt_wgrad_splits(const ConvShape& s) {
  const Geo g = make_geo(s, WGRAD);
  const int64_t blocks = ceil_div(g.Ncol, BN) * ceil_div(g.M, BM);
  int64_t sp = (2 * sm_count() + blocks - 1) / blocks;
  sp = std::min<int64_t>(sp, std::max<int64_t>(1, g.K / (8 * BK)));   // at least 8 k-tiles per split
  return int(std::max<int64_t>(1, sp));
}

int64_t simt_wgrad_scratch_floats(const ConvShape& s) {
  const int sp = simt_wgrad_splits(s);
  const Geo g = make_geo(s, WGRAD);
  return sp > 1 ? int64_t(sp) * g.M * g.Ncol : 0;
}

void conv_wgrad_simt(const ConvShape& s, const void* dy, int dt_dy, const void* x, int dt_x,
                     float* dw, float* scratch, cudaStream_t st) {
  Geo g = make_geo(s, WGRAD);
  const int sp = scratch ? simt_wgrad_splits(s) : 1;
  if (sp <= 1) {
    launch_any<WGRAD>(g, dy, dt_dy, x, dt_x, nullptr, dw, kF32, false, false, st);
    return;
  }
  g.kper = (g.K + sp - 1) / sp;
  g.kper = (g.kper + BK - 1) / BK * BK;
  const int real = int(ceil_div(g.K, g.kper));
  launch_any<WGRAD>(g, dy, dt_dy, x, dt_x, nullptr, scratch, kF32, false, false, st);
  const int64_t n = g.M * g.Ncol;
  launch_k(sum_splits_k, int(std::min<int64_t>(ceil_div(n, 256), 4 * sm_count())), 256, 0, st, scratch, real, n, dw);
}

}  // namespace fo
