// Vectorised bf16 elementwise and reduction kernels: 8 elements (16 bytes)
// per thread and per access.  Used when the tensor is bf16 and its element
// count (and, where channels matter, its channel count) is a multiple of 8;
// the scalar kernels of k_elementwise.cu cover the rest.  Column sums are
// taken per (row chunk, 256-column block) and finished in a fixed order, so
// every result is deterministic.
#include "fo_common.cuh"
#include "fo_kernels.h"

#include <algorithm>
#include <vector>

namespace fo {

namespace {

constexpr int kChunk = 128;  // rows per column-sum chunk of the public entry points

struct V8 {
  float v[8];
};

__device__ __forceinline__ V8 ld8(const bf16* p) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const bf16* e = reinterpret_cast<const bf16*>(&u);
  V8 r;
#pragma unroll
  for (int j = 0; j < 8; ++j) r.v[j] = __bfloat162float(e[j]);
  return r;
}
__device__ __forceinline__ void st8(bf16* p, const V8& r) {
  uint4 u;
  bf16* e = reinterpret_cast<bf16*>(&u);
#pragma unroll
  for (int j = 0; j < 8; ++j) e[j] = __float2bfloat16_rn(r.v[j]);
  *reinterpret_cast<uint4*>(p) = u;
}

#define GRID_STRIDE8(i, n8) \
  for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < (n8); i += int64_t(gridDim.x) * blockDim.x)

__global__ void relu_bwd_x8_k(const bf16* __restrict__ y, const bf16* __restrict__ dy, bf16* __restrict__ dx,
                              int64_t n8, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const V8 m = ld8(y + 8 * i), g = ld8(dy + 8 * i);
    V8 o;
#pragma unroll
    for (int j = 0; j < 8; ++j) o.v[j] = m.v[j] > 0.f ? g.v[j] : 0.f;
    if (acc) {
      const V8 p = ld8(dx + 8 * i);
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] += p.v[j];
    }
    st8(dx + 8 * i, o);
  }
}

__global__ void add_x8_k(const bf16* __restrict__ a, const bf16* __restrict__ b, bf16* __restrict__ y, int64_t n8,
                         int relu) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const V8 p = ld8(a + 8 * i), q = ld8(b + 8 * i);
    V8 o;
#pragma unroll
    for (int j = 0; j < 8; ++j) o.v[j] = relu ? fmaxf(p.v[j] + q.v[j], 0.f) : p.v[j] + q.v[j];
    st8(y + 8 * i, o);
  }
}

// Backward of a residual add (optionally with the ReLU that follows it):
// g = dy (times mask > 0 when mask is given) goes to both inputs' gradients,
// d0 (+)= g and d1 (+)= g (d1 may be null), in one pass over dy.
__global__ void grad_split_x8_k(const bf16* __restrict__ dy, const bf16* __restrict__ mask, bf16* __restrict__ d0,
                                int acc0, bf16* __restrict__ d1, int acc1, int64_t n8) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    V8 g = ld8(dy + 8 * i);
    if (mask) {
      const V8 m = ld8(mask + 8 * i);
#pragma unroll
      for (int j = 0; j < 8; ++j) g.v[j] = m.v[j] > 0.f ? g.v[j] : 0.f;
    }
    if (acc0) {
      const V8 q = ld8(d0 + 8 * i);
      V8 o;
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] = g.v[j] + q.v[j];
      st8(d0 + 8 * i, o);
    } else {
      st8(d0 + 8 * i, g);
    }
    if (d1) {
      if (acc1) {
        const V8 q = ld8(d1 + 8 * i);
        V8 o;
#pragma unroll
        for (int j = 0; j < 8; ++j) o.v[j] = g.v[j] + q.v[j];
        st8(d1 + 8 * i, o);
      } else {
        st8(d1 + 8 * i, g);
      }
    }
  }
}

__global__ void affine_fwd_x8_k(const bf16* __restrict__ x, const float* __restrict__ sc,
                                const float* __restrict__ sh, bf16* __restrict__ y, int64_t n8, int C, int relu) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const int c = int((8 * i) % C);
    const V8 p = ld8(x + 8 * i);
    V8 o;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float v = fmaf(p.v[j], sc[c + j], sh[c + j]);
      o.v[j] = relu ? fmaxf(v, 0.f) : v;
    }
    st8(y + 8 * i, o);
  }
}

// Batch-norm affine followed by hard swish, both outputs stored: the affine
// output (the hard swish's input, kept for the backward pass) and the hard
// swish of its stored bf16 value, exactly as the two separate kernels give.
__device__ __forceinline__ float round_bf16(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }
__device__ __forceinline__ float hswish_f(float v) { return v * fminf(fmaxf(v + 3.f, 0.f), 6.f) / 6.f; }
__device__ __forceinline__ float hswish_d(float v) { return v < -3.f ? 0.f : (v > 3.f ? 1.f : (2.f * v + 3.f) / 6.f); }

__global__ void affine_hswish_fwd_x8_k(const bf16* __restrict__ x, const float* __restrict__ sc,
                                       const float* __restrict__ sh, bf16* __restrict__ pre, bf16* __restrict__ post,
                                       int64_t n8, int C) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const int c = int((8 * i) % C);
    const V8 p = ld8(x + 8 * i);
    V8 a, h;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      a.v[j] = fmaf(p.v[j], sc[c + j], sh[c + j]);
      h.v[j] = hswish_f(round_bf16(a.v[j]));
    }
    st8(pre + 8 * i, a);
    st8(post + 8 * i, h);
  }
}

__global__ void gelu_fwd_x8_k(const bf16* __restrict__ x, bf16* __restrict__ y, int64_t n8) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const V8 p = ld8(x + 8 * i);
    V8 o;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      float cdf, pdf;
      normal_cdf_pdf(p.v[j], cdf, pdf);
      o.v[j] = p.v[j] * cdf;
    }
    st8(y + 8 * i, o);
  }
}

__global__ void gelu_bwd_x8_k(const bf16* __restrict__ x, const bf16* __restrict__ dy, bf16* __restrict__ dx,
                              int64_t n8, int acc) {
  pdl_wait();
  pdl_trigger();
  GRID_STRIDE8(i, n8) {
    const V8 p = ld8(x + 8 * i), g = ld8(dy + 8 * i);
    V8 o;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      float cdf, pdf;
      normal_cdf_pdf(p.v[j], cdf, pdf);
      o.v[j] = g.v[j] * (cdf + p.v[j] * pdf);
    }
    if (acc) {
      const V8 q = ld8(dx + 8 * i);
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] += q.v[j];
    }
    st8(dx + 8 * i, o);
  }
}

// Column partial sums over a (128-row chunk, 256-column block): thread
// (g, r) owns columns c0 + 8g .. +7 and rows r, r + 8, ...; the 8 row lanes
// are combined in shared memory in a fixed order.  MODE 0: sums of a;
// MODE 1: affine backward (sums of dy * x and dy, and dx (+)= dy * scale);
// MODE 2: MODE 1 behind a hard swish: `a` is the gradient of the hard
// swish's output and `pre` its input (the affine output), and dy is the
// bf16 value of a * hswish'(pre), as the separate hard swish backward stores.
template <int MODE>
__device__ __forceinline__ void colsum8_block(const bf16* __restrict__ a, const bf16* __restrict__ x,
                                              const float* __restrict__ scale, bf16* __restrict__ dx, int acc,
                                              int64_t rows, int C, int chunk, float* __restrict__ p0,
                                              float* __restrict__ p1, int cb, int ck,
                                              const bf16* __restrict__ pre = nullptr) {
  __shared__ float red0[8][257];
  __shared__ float red1[MODE >= 1 ? 8 : 1][257];
  const int g = threadIdx.x % 32, r = threadIdx.x / 32;
  const int c = cb * 256 + 8 * g;
  const int64_t r0 = int64_t(ck) * chunk;
  float s0[8] = {0, 0, 0, 0, 0, 0, 0, 0}, s1[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (c < C) {
    float sc[8];
    if (MODE >= 1)
#pragma unroll
      for (int j = 0; j < 8; ++j) sc[j] = scale[c + j];
    for (int64_t row = r0 + r; row < r0 + chunk && row < rows; row += 8) {
      V8 d = ld8(a + row * C + c);
      if (MODE == 2) {
        const V8 h = ld8(pre + row * C + c);
#pragma unroll
        for (int j = 0; j < 8; ++j) d.v[j] = round_bf16(d.v[j] * hswish_d(h.v[j]));
      }
      if (MODE == 0) {
#pragma unroll
        for (int j = 0; j < 8; ++j) s0[j] += d.v[j];
      } else {
        const V8 xv = ld8(x + row * C + c);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          s0[j] = fmaf(d.v[j], xv.v[j], s0[j]);
          s1[j] += d.v[j];
        }
        if (dx) {
          V8 o;
#pragma unroll
          for (int j = 0; j < 8; ++j) o.v[j] = d.v[j] * sc[j];
          if (acc) {
            const V8 q = ld8(dx + row * C + c);
#pragma unroll
            for (int j = 0; j < 8; ++j) o.v[j] += q.v[j];
          }
          st8(dx + row * C + c, o);
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    red0[r][8 * g + j] = s0[j];
    if (MODE >= 1) red1[r][8 * g + j] = s1[j];
  }
  __syncthreads();
  const int cc = cb * 256 + threadIdx.x;
  if (cc < C) {
    float t0 = 0.f, t1 = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      t0 += red0[q][threadIdx.x];
      if (MODE >= 1) t1 += red1[q][threadIdx.x];
    }
    p0[int64_t(ck) * C + cc] = t0;
    if (MODE >= 1) p1[int64_t(ck) * C + cc] = t1;
  }
}

template <int MODE>
__global__ void __launch_bounds__(256) colsum8_k(const bf16* __restrict__ a, const bf16* __restrict__ x,
                                                 const float* __restrict__ scale, bf16* __restrict__ dx, int acc,
                                                 int64_t rows, int C, int chunk, float* __restrict__ p0,
                                                 float* __restrict__ p1, const bf16* __restrict__ pre) {
  pdl_wait();
  pdl_trigger();
  colsum8_block<MODE>(a, x, scale, dx, acc, rows, C, chunk, p0, p1, blockIdx.x, blockIdx.y, pre);
}

// Several column sums in one launch: block b belongs to the task t with
// block0[t] <= b < block0[t + 1] and covers (column block, row chunk) of it.
constexpr int kMaxBatch = 40;
struct ColsumBatch {
  int n;
  int block0[kMaxBatch + 1];
  const bf16* a[kMaxBatch];
  float* partial[kMaxBatch];
  int64_t rows[kMaxBatch];
  int C[kMaxBatch];
  int chunk[kMaxBatch];
};
struct FinishBatch {
  int n;
  int block0[kMaxBatch + 1];
  const float* partial[kMaxBatch];
  float* out[kMaxBatch];
  int chunks[kMaxBatch];
  int C[kMaxBatch];
};

__device__ __forceinline__ int batch_task(const int* block0, int n, int b) {
  int t = 0;
  while (t + 1 < n && block0[t + 1] <= b) ++t;
  return t;
}

__global__ void __launch_bounds__(256) colsum8_batch_k(const __grid_constant__ ColsumBatch p) {
  pdl_wait();
  pdl_trigger();
  const int t = batch_task(p.block0, p.n, blockIdx.x);
  const int local = blockIdx.x - p.block0[t];
  const int cbs = (p.C[t] + 255) / 256;
  colsum8_block<0>(p.a[t], nullptr, nullptr, nullptr, 0, p.rows[t], p.C[t], p.chunk[t], p.partial[t], nullptr,
                   local % cbs, local / cbs);
}

// Layernorm forward, rows held in registers (C = 256 NV, NV <= 4, a
// template parameter so that a row takes only the registers it needs): each
// warp takes R consecutive rows and loads all of them before any
// arithmetic; one read of x, mean then biased variance from the registers
// (eps 1e-5), one write of y; the row mean and 1/std are kept for the
// backward pass.  gamma and beta are read as float4 alongside x, so that the
// rows' only dependent global accesses are x.  R = 2 for rows of up to 512
// (the whole 4096-row step in one wave of two blocks per SM).
template <int NV, int R>
__global__ void __launch_bounds__(256, 2) layernorm_fwd_x8_k(const bf16* __restrict__ x, const float* __restrict__ gamma,
                                                          const float* __restrict__ beta, bf16* __restrict__ y,
                                                          float* __restrict__ mean_out, float* __restrict__ rstd_out,
                                                          int64_t rows, int C) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x % 32;
  const int64_t row0 = (int64_t(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32) * R;
  if (row0 >= rows) return;
  uint4 xr[R][NV];
  float4 g4[NV][2], b4[NV][2];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int v = 0; v < NV; ++v)
      xr[r][v] = row0 + r < rows ? *reinterpret_cast<const uint4*>(x + (row0 + r) * C + (v * 32 + lane) * 8)
                                 : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const int c = (v * 32 + lane) * 8;
    g4[v][0] = __ldg(reinterpret_cast<const float4*>(gamma + c));
    g4[v][1] = __ldg(reinterpret_cast<const float4*>(gamma + c) + 1);
    b4[v][0] = __ldg(reinterpret_cast<const float4*>(beta + c));
    b4[v][1] = __ldg(reinterpret_cast<const float4*>(beta + c) + 1);
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int64_t row = row0 + r;
    if (row >= rows) break;
    float sum = 0.f;
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
      for (int j = 0; j < 8; ++j) sum += __bfloat162float(reinterpret_cast<const bf16*>(&xr[r][v])[j]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float mu = sum / float(C);
    float q = 0.f;
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float d = __bfloat162float(reinterpret_cast<const bf16*>(&xr[r][v])[j]) - mu;
        q = fmaf(d, d, q);
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float rs = rsqrtf(q / float(C) + 1e-5f);
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      const int c = (v * 32 + lane) * 8;
      const float gm[8] = {g4[v][0].x, g4[v][0].y, g4[v][0].z, g4[v][0].w, g4[v][1].x, g4[v][1].y, g4[v][1].z, g4[v][1].w};
      const float bt[8] = {b4[v][0].x, b4[v][0].y, b4[v][0].z, b4[v][0].w, b4[v][1].x, b4[v][1].y, b4[v][1].z, b4[v][1].w};
      V8 o;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        o.v[j] = (__bfloat162float(reinterpret_cast<const bf16*>(&xr[r][v])[j]) - mu) * rs * gm[j] + bt[j];
      st8(y + row * C + c, o);
    }
    if (lane == 0) {
      mean_out[row] = mu;
      rstd_out[row] = rs;
    }
  }
}

// Layernorm backward fused with its parameter gradients.  Each warp takes
// kLnRows consecutive rows (a block kLnWarps kLnRows), with all of their operands
// loaded before any arithmetic.  The column partials of dy * xhat (gamma),
// dy (beta) and, with pdx, of the stored dx accumulate in registers over the
// warp's rows and are added over the block's warps, in warp order, through
// shared memory once per block: exchanged row by row, those partials cost
// more than the rest of the pass.  C <= 512, C % 256 == 0; dx may be null (a
// layernorm of the uploaded batch has no input gradient).  dx receives the
// layernorm's input gradient plus the NX extra operands ex0, ex1 (same
// layout): its own old value when accumulating, and the gradient a residual
// connection passes around the layernorm.
constexpr int kLnRows = 4;
constexpr int kLnWarps = 4;   // warps per block: the 4096-row step in 256 blocks
__device__ __forceinline__ float bf_at(const uint4& u, int j) {
  return __bfloat162float(reinterpret_cast<const bf16*>(&u)[j]);
}
template <int NX, int NV, int DXP>   // DXP: 0 no dx, 1 dx, 2 dx and its column partials (pdx)
__global__ void __launch_bounds__(kLnWarps * 32, 1) layernorm_bwd_fused_k(const bf16* __restrict__ x, const float* __restrict__ gamma,
                                                                const float* __restrict__ mean, const float* __restrict__ rstd,
                                                                const bf16* __restrict__ dy, bf16* dx, int64_t rows, int C,
                                                                const bf16* ex0, const bf16* ex1, float* __restrict__ pg,
                                                                float* __restrict__ pb, float* __restrict__ pdx) {
  pdl_wait();
  pdl_trigger();
  constexpr int kMaxV = NV, nv = NV, CC = 256 * NV;   // 8-wide vectors per lane: C = 256 NV
  __shared__ __align__(16) float red[3][kLnWarps][256 * NV];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int64_t row0 = (int64_t(blockIdx.x) * kLnWarps + warp) * kLnRows;
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
  float gm[kMaxV][8];
#pragma unroll
  for (int v = 0; v < kMaxV; ++v) {
    const int c = v < nv ? (v * 32 + lane) * 8 : 0;
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(gamma + c));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(gamma + c) + 1);
    gm[v][0] = g0.x; gm[v][1] = g0.y; gm[v][2] = g0.z; gm[v][3] = g0.w;
    gm[v][4] = g1.x; gm[v][5] = g1.y; gm[v][6] = g1.z; gm[v][7] = g1.w;
  }
  uint4 xr[kLnRows][kMaxV], gr[kLnRows][kMaxV], er[kLnRows][kMaxV][NX > 0 ? NX : 1];
  float mu[kLnRows], rs[kLnRows];
#pragma unroll
  for (int r = 0; r < kLnRows; ++r) {
    const int64_t row = row0 + r;
    const bool live = row < rows;
#pragma unroll
    for (int v = 0; v < kMaxV; ++v) {
      const bool ok = live && v < nv;
      const int64_t off = row * CC + (v * 32 + lane) * 8;
      xr[r][v] = ok ? *reinterpret_cast<const uint4*>(x + off) : z;
      gr[r][v] = ok ? *reinterpret_cast<const uint4*>(dy + off) : z;
      if constexpr (NX > 0) er[r][v][0] = ok ? *reinterpret_cast<const uint4*>(ex0 + off) : z;
      if constexpr (NX > 1) er[r][v][1] = ok ? *reinterpret_cast<const uint4*>(ex1 + off) : z;
    }
    mu[r] = live ? mean[row] : 0.f;
    rs[r] = live ? rstd[row] : 0.f;
  }
  float ag[kMaxV][8] = {}, ab[kMaxV][8] = {}, ax[kMaxV][8] = {};
#pragma unroll
  for (int r = 0; r < kLnRows; ++r) {
    const int64_t row = row0 + r;
    const bool live = row < rows;
    float a = 0.f, b = 0.f;
#pragma unroll
    for (int v = 0; v < kMaxV; ++v)
#pragma unroll
      for (int j = 0; j < 8; ++j) {   // rows past the end and vectors past C hold zeros
        const float xh = (bf_at(xr[r][v], j) - mu[r]) * rs[r];
        const float g = bf_at(gr[r][v], j);
        const float d = g * gm[v][j];
        a += d;
        b += d * xh;
        ag[v][j] += g * xh;
        ab[v][j] += g;
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      a += __shfl_xor_sync(0xffffffffu, a, o);
      b += __shfl_xor_sync(0xffffffffu, b, o);
    }
    a *= 1.f / float(CC);
    b *= 1.f / float(CC);
    if constexpr (DXP > 0) {
#pragma unroll
      for (int v = 0; v < kMaxV; ++v) {
        if (v >= nv) break;
        uint4 o;
        bf16* ob = reinterpret_cast<bf16*>(&o);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float xh = (bf_at(xr[r][v], j) - mu[r]) * rs[r];
          float val = rs[r] * (bf_at(gr[r][v], j) * gm[v][j] - a - xh * b);
          if constexpr (NX > 0) val += bf_at(er[r][v][0], j);
          if constexpr (NX > 1) val += bf_at(er[r][v][1], j);
          ob[j] = __float2bfloat16_rn(val);
          if constexpr (DXP == 2) ax[v][j] += live ? __bfloat162float(ob[j]) : 0.f;   // the stored value
        }
        if (live) *reinterpret_cast<uint4*>(dx + row * CC + (v * 32 + lane) * 8) = o;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < kMaxV; ++v) {
    if (v >= nv) break;
    const int c = (v * 32 + lane) * 8;
    float4* p0 = reinterpret_cast<float4*>(&red[0][warp][c]);
    float4* p1 = reinterpret_cast<float4*>(&red[1][warp][c]);
    float4* p2 = reinterpret_cast<float4*>(&red[2][warp][c]);
    p0[0] = make_float4(ag[v][0], ag[v][1], ag[v][2], ag[v][3]);
    p0[1] = make_float4(ag[v][4], ag[v][5], ag[v][6], ag[v][7]);
    p1[0] = make_float4(ab[v][0], ab[v][1], ab[v][2], ab[v][3]);
    p1[1] = make_float4(ab[v][4], ab[v][5], ab[v][6], ab[v][7]);
    if constexpr (DXP == 2) {
      p2[0] = make_float4(ax[v][0], ax[v][1], ax[v][2], ax[v][3]);
      p2[1] = make_float4(ax[v][4], ax[v][5], ax[v][6], ax[v][7]);
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    float tg = 0.f, tb = 0.f, tx = 0.f;
#pragma unroll
    for (int q = 0; q < kLnWarps; ++q) {
      tg += red[0][q][c];
      tb += red[1][q][c];
      if constexpr (DXP == 2) tx += red[2][q][c];
    }
    pg[int64_t(blockIdx.x) * C + c] = tg;
    pb[int64_t(blockIdx.x) * C + c] = tb;
    if constexpr (DXP == 2) pdx[int64_t(blockIdx.x) * C + c] = tx;
  }
}

// Masked mean over the valid tokens of each sequence: block (b, 256-column
// block), warp w sums tokens w, w + 8, ... of its 8 columns per lane (four
// independent loads in flight), then the 8 warp sums are added in warp order.
__global__ void __launch_bounds__(256) meanpool_fwd_x8_k(const bf16* __restrict__ x, const int32_t* __restrict__ len,
                                                         bf16* __restrict__ y, int L, int C) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[8][257];
  const int b = blockIdx.x, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int c = blockIdx.y * 256 + lane * 8;
  const int n = len[b];
  float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c < C) {
    const bf16* base = x + int64_t(b) * L * C + c;
    int i = warp;
    for (; i + 24 < n; i += 32) {
      const V8 a0 = ld8(base + int64_t(i) * C), a1 = ld8(base + int64_t(i + 8) * C);
      const V8 a2 = ld8(base + int64_t(i + 16) * C), a3 = ld8(base + int64_t(i + 24) * C);
#pragma unroll
      for (int j = 0; j < 8; ++j) s[j] += ((a0.v[j] + a1.v[j]) + (a2.v[j] + a3.v[j]));
    }
    for (; i < n; i += 8) {
      const V8 a = ld8(base + int64_t(i) * C);
#pragma unroll
      for (int j = 0; j < 8; ++j) s[j] += a.v[j];
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) red[warp][lane * 8 + j] = s[j];
  __syncthreads();
  const int cc = blockIdx.y * 256 + threadIdx.x;
  if (cc < C) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += red[w][threadIdx.x];
    y[int64_t(b) * C + cc] = __float2bfloat16_rn(t / float(n));
  }
}

// Its gradient: dx[b, t, :] = dy[b, :] / len[b] for the valid tokens, 0 for
// the padding, 8 columns per thread (plus dx's old value when `acc`).
__global__ void meanpool_bwd_x8_k(const bf16* __restrict__ dy, const int32_t* __restrict__ len,
                                  bf16* __restrict__ dx, int L, int C, int64_t n8, int acc) {
  pdl_wait();
  pdl_trigger();
  const int c8 = C / 8;
  GRID_STRIDE8(i, n8) {
    const int c = int(i % c8) * 8;
    const int64_t bt = i / c8;
    const int b = int(bt / L), t = int(bt % L);
    const int n = len[b];
    V8 o;
    if (t < n) {
      o = ld8(dy + int64_t(b) * C + c);
      const float inv = 1.f / float(n);
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] *= inv;
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] = 0.f;
    }
    if (acc) {
      const V8 q = ld8(dx + 8 * i);
#pragma unroll
      for (int j = 0; j < 8; ++j) o.v[j] += q.v[j];
    }
    st8(dx + 8 * i, o);
  }
}

__global__ void finish_k(const float* __restrict__ partial, int chunks, int C, float* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[8][33];
  const int cl = threadIdx.x % 32, rl = threadIdx.x / 32;
  const int c = blockIdx.x * 32 + cl;
  float s = 0.f;
  if (c < C) {
    int q = rl;
    for (; q + 24 < chunks; q += 32) {
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

// Batched finish: block b covers 32 columns of task t (same fixed summation
// order as finish_k).
__global__ void __launch_bounds__(256) finish_batch_k(const __grid_constant__ FinishBatch p) {
  pdl_wait();
  pdl_trigger();
  const int t = batch_task(p.block0, p.n, blockIdx.x);
  const int local = blockIdx.x - p.block0[t];
  __shared__ float red[8][33];
  const int cl = threadIdx.x % 32, rl = threadIdx.x / 32;
  const int C = p.C[t], chunks = p.chunks[t];
  const float* partial = p.partial[t];
  const int c = local * 32 + cl;
  float s = 0.f;
  if (c < C) {
    int q = rl;
    for (; q + 24 < chunks; q += 32) {
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
    float tot = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) tot += red[q][cl];
    p.out[t][c] = tot;
  }
}

int chunks_of(int64_t rows, int chunk) { return int((rows + chunk - 1) / chunk); }

// Rows per chunk for the server's column sums: about two blocks per SM,
// between 8 and 128 rows, a multiple of 8.
int adaptive_chunk(int64_t rows, int C) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 148;
  }
  const int64_t colblocks = (C + 255) / 256;
  int64_t ch = rows * colblocks / (2 * int64_t(sms));
  ch = (ch + 7) / 8 * 8;
  if (ch < 8) ch = 8;
  if (ch > 128) ch = 128;
  return int(ch);
}

}  // namespace

bool vec8_ok(int dt, int64_t n) { return dt == kBF16 && n % 8 == 0; }

void relu_bwd_x8(const void* y, const void* dy, void* dx, int64_t n, bool acc, cudaStream_t st) {
  launch_k(relu_bwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)y, (const bf16*)dy, (bf16*)dx, n / 8, acc);
}
void add_x8(const void* a, const void* b, void* y, int64_t n, bool relu, cudaStream_t st) {
  launch_k(add_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)a, (const bf16*)b, (bf16*)y, n / 8, relu);
}
void grad_split_x8(const void* dy, const void* mask, void* d0, bool acc0, void* d1, bool acc1, int64_t n,
                   cudaStream_t st) {
  launch_k(grad_split_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)dy, (const bf16*)mask, (bf16*)d0,
           acc0 ? 1 : 0, (bf16*)d1, acc1 ? 1 : 0, n / 8);
}
void affine_fwd_x8(const void* x, const float* sc, const float* sh, void* y, int64_t n, int C, bool relu,
                   cudaStream_t st) {
  launch_k(affine_fwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, sc, sh, (bf16*)y, n / 8, C, relu);
}
void affine_hswish_fwd_x8(const void* x, const float* sc, const float* sh, void* pre, void* post, int64_t n, int C,
                          cudaStream_t st) {
  launch_k(affine_hswish_fwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, sc, sh, (bf16*)pre,
                                                                          (bf16*)post, n / 8, C);
}
void gelu_fwd_x8(const void* x, void* y, int64_t n, cudaStream_t st) {
  launch_k(gelu_fwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, (bf16*)y, n / 8);
}
void gelu_bwd_x8(const void* x, const void* dy, void* dx, int64_t n, bool acc, cudaStream_t st) {
  launch_k(gelu_bwd_x8_k, elementwise_blocks(n / 8, 256), 256, 0, st, (const bf16*)x, (const bf16*)dy, (bf16*)dx, n / 8, acc);
}

int64_t colsum8_partial_floats(int64_t rows, int C, bool adaptive) {
  return int64_t(chunks_of(rows, adaptive ? adaptive_chunk(rows, C) : kChunk)) * C;
}

void colsum8(const void* a, int64_t rows, int C, float* partial, float* out, bool adaptive, cudaStream_t st) {
  const int ch = adaptive ? adaptive_chunk(rows, C) : kChunk;
  dim3 grid(ceil_div(C, 256), chunks_of(rows, ch));
  launch_k(colsum8_k<0>, grid, 256, 0, st, (const bf16*)a, nullptr, nullptr, nullptr, 0, rows, C, ch, partial, nullptr, nullptr);
  launch_k(finish_k, ceil_div(C, 32), 256, 0, st, partial, chunks_of(rows, ch), C, out);
}

int affine_bwd8_chunks(int64_t rows, int C) { return chunks_of(rows, adaptive_chunk(rows, C)); }

void affine_bwd8_pass(const void* dy, const void* x, const float* scale, void* dx, bool acc, int64_t rows, int C,
                      float* p_scale, float* p_shift, cudaStream_t st, const void* hswish_in) {
  const int ch = adaptive_chunk(rows, C);
  dim3 grid(ceil_div(C, 256), chunks_of(rows, ch));
  if (hswish_in)
    launch_k(colsum8_k<2>, grid, 256, 0, st, (const bf16*)dy, (const bf16*)x, scale, (bf16*)dx, acc, rows, C, ch, p_scale,
                                       p_shift, (const bf16*)hswish_in);
  else
    launch_k(colsum8_k<1>, grid, 256, 0, st, (const bf16*)dy, (const bf16*)x, scale, (bf16*)dx, acc, rows, C, ch, p_scale,
                                       p_shift, nullptr);
}

int colsum8_batch_chunks(int64_t rows) { return chunks_of(rows, kChunk); }

void colsum8_batched(const std::vector<ColsumTask>& tasks, cudaStream_t st) {
  for (size_t t0 = 0; t0 < tasks.size(); t0 += kMaxBatch) {
    ColsumBatch p{};
    p.n = int(std::min(tasks.size() - t0, size_t(kMaxBatch)));
    int blocks = 0;
    for (int k = 0; k < p.n; ++k) {
      const ColsumTask& t = tasks[t0 + k];
      p.block0[k] = blocks;
      p.a[k] = static_cast<const bf16*>(t.a);
      p.partial[k] = t.partial;
      p.rows[k] = t.rows;
      p.C[k] = t.C;
      p.chunk[k] = kChunk;
      blocks += ceil_div(t.C, 256) * chunks_of(t.rows, kChunk);
    }
    p.block0[p.n] = blocks;
    if (blocks) launch_k(colsum8_batch_k, blocks, 256, 0, st, p);
  }
}

void finish_batched(const std::vector<FinishTask>& tasks, cudaStream_t st) {
  for (size_t t0 = 0; t0 < tasks.size(); t0 += kMaxBatch) {
    FinishBatch p{};
    p.n = int(std::min(tasks.size() - t0, size_t(kMaxBatch)));
    int blocks = 0;
    for (int k = 0; k < p.n; ++k) {
      const FinishTask& t = tasks[t0 + k];
      p.block0[k] = blocks;
      p.partial[k] = t.partial;
      p.out[k] = t.out;
      p.chunks[k] = t.chunks;
      p.C[k] = t.C;
      blocks += ceil_div(t.C, 32);
    }
    p.block0[p.n] = blocks;
    if (blocks) launch_k(finish_batch_k, blocks, 256, 0, st, p);
  }
}

bool layernorm_bwd8_ok(int dt, int C) { return dt == kBF16 && C % 256 == 0 && C <= 512; }

int layernorm_bwd8_blocks(int64_t rows) { return int((rows + kLnWarps * kLnRows - 1) / (kLnWarps * kLnRows)); }

bool layernorm_fwd8_ok(int dt, int C) { return dt == kBF16 && C % 256 == 0 && C <= 1024; }
void layernorm_fwd_x8(const void* x, const float* gamma, const float* beta, void* y, float* mean, float* rstd,
                      int64_t rows, int C, cudaStream_t st) {
  if (C <= 512) {
    auto k = C <= 256 ? layernorm_fwd_x8_k<1, 2> : layernorm_fwd_x8_k<2, 2>;
    launch_k(k, ceil_div(rows, 16), 256, 0, st, (const bf16*)x, gamma, beta, (bf16*)y, mean, rstd, rows, C);
    return;
  }
  auto k = C <= 768 ? layernorm_fwd_x8_k<3, 1> : layernorm_fwd_x8_k<4, 1>;
  launch_k(k, ceil_div(rows, 8), 256, 0, st, (const bf16*)x, gamma, beta, (bf16*)y, mean, rstd, rows, C);
}

void layernorm_bwd8_pass(const void* x, const float* gamma, const float* mean, const float* rstd, const void* dy,
                         void* dx, int64_t rows, int C, bool acc, float* p_gamma, float* p_beta, cudaStream_t st,
                         const void* addend, float* p_dx) {
  const bf16* ex[2] = {nullptr, nullptr};
  int nx = 0;
  if (dx && acc) ex[nx++] = static_cast<const bf16*>(dx);
  if (dx && addend) ex[nx++] = static_cast<const bf16*>(addend);
  using K = decltype(&layernorm_bwd_fused_k<0, 1, 0>);
  static const K table[2][3][3] = {   // [NV - 1][NX][DXP]; NX > 0 comes with a dx
      {{layernorm_bwd_fused_k<0, 1, 0>, layernorm_bwd_fused_k<0, 1, 1>, layernorm_bwd_fused_k<0, 1, 2>},
       {nullptr, layernorm_bwd_fused_k<1, 1, 1>, layernorm_bwd_fused_k<1, 1, 2>},
       {nullptr, layernorm_bwd_fused_k<2, 1, 1>, layernorm_bwd_fused_k<2, 1, 2>}},
      {{layernorm_bwd_fused_k<0, 2, 0>, layernorm_bwd_fused_k<0, 2, 1>, layernorm_bwd_fused_k<0, 2, 2>},
       {nullptr, layernorm_bwd_fused_k<1, 2, 1>, layernorm_bwd_fused_k<1, 2, 2>},
       {nullptr, layernorm_bwd_fused_k<2, 2, 1>, layernorm_bwd_fused_k<2, 2, 2>}}};
  const int dxp = dx ? (p_dx ? 2 : 1) : 0;
  auto k = table[C <= 256 ? 0 : 1][nx][dxp];
  launch_k(k, layernorm_bwd8_blocks(rows), kLnWarps * 32, 0, st, (const bf16*)x, gamma, mean, rstd, (const bf16*)dy, (bf16*)dx,
           rows, C, ex[0], ex[1], p_gamma, p_beta, dx ? p_dx : nullptr);
}

int64_t layernorm_bwd8_partial_floats(int64_t rows, int C) { return 2 * int64_t(layernorm_bwd8_blocks(rows)) * C; }

bool meanpool8_ok(int dt, int C) { return dt == kBF16 && C % 8 == 0; }
void meanpool_fwd_x8(const void* x, const int32_t* len, void* y, int B, int L, int C, cudaStream_t st) {
  launch_k(meanpool_fwd_x8_k, dim3(B, ceil_div(C, 256)), 256, 0, st, (const bf16*)x, len, (bf16*)y, L, C);
}
void meanpool_bwd_x8(const void* dy, const int32_t* len, void* dx, int B, int L, int C, bool acc, cudaStream_t st) {
  const int64_t n8 = int64_t(B) * L * C / 8;
  launch_k(meanpool_bwd_x8_k, elementwise_blocks(n8, 256), 256, 0, st, (const bf16*)dy, len, (bf16*)dx, L, C, n8,
           acc ? 1 : 0);
}

}  // namespace fo
