// Multi-head scaled dot-product attention with a key-padding mask, forward
// and backward, one CTA per (sequence, head) on CUDA cores.  Input is the
// packed q|k|v projection [B, L, 3C]; keys j >= length[b] are masked out.
// The forward pass saves the softmax probabilities P (fp32 [B, h, L, L]);
// the backward pass uses
//   dV = P^T dO,  dP = dO V^T,  dS = P (dP - rowsum(dO * O)),
//   dQ = dS K / sqrt(dh),  dK = dS^T Q / sqrt(dh).
#include "fo_common.cuh"
#include "fo_kernels.h"

namespace fo {

namespace {

constexpr int kWarps = 8;

template <typename T>
__global__ void __launch_bounds__(256) attn_fwd_k(const T* __restrict__ qkv,
                                                  const int32_t* __restrict__ len,
                                                  T* __restrict__ out, float* __restrict__ probs,
                                                  int L, int C, int heads) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  const int bh = blockIdx.x, b = bh / heads, h = bh % heads;
  const int dh = C / heads, ld = dh + 1;
  float* Ks = sm;
  float* Vs = Ks + L * ld;
  float* qrow = Vs + L * ld;
  float* prow = qrow + kWarps * 64;
  const T* base = qkv + int64_t(b) * L * 3 * C;
  for (int e = threadIdx.x; e < L * dh; e += blockDim.x) {
    int j = e / dh, d = e % dh;
    Ks[j * ld + d] = to_f(base[int64_t(j) * 3 * C + C + h * dh + d]);
    Vs[j * ld + d] = to_f(base[int64_t(j) * 3 * C + 2 * C + h * dh + d]);
  }
  __syncthreads();
  const int n = len[b];
  const float scale = rsqrtf(float(dh));
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  float* q = qrow + warp * 64;
  float* p = prow + warp * L;
  for (int i = warp; i < L; i += kWarps) {
    for (int d = lane; d < dh; d += 32) q[d] = to_f(base[int64_t(i) * 3 * C + h * dh + d]);
    __syncwarp();
    float s[4];
    float m = -INFINITY;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      int j = lane + 32 * t;
      s[t] = -INFINITY;
      if (j < n && j < L) {
        float dot = 0.f;
        for (int d = 0; d < dh; ++d) dot = fmaf(q[d], Ks[j * ld + d], dot);
        s[t] = dot * scale;
        m = fmaxf(m, s[t]);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float sum = 0.f;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      int j = lane + 32 * t;
      if (j < n && j < L) {
        s[t] = expf(s[t] - m);
        sum += s[t];
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    float inv = 1.f / sum;
    float* prow_g = probs + (int64_t(bh) * L + i) * L;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      int j = lane + 32 * t;
      if (j < L) {
        float pj = (j < n) ? s[t] * inv : 0.f;
        p[j] = pj;
        prow_g[j] = pj;
      }
    }
    __syncwarp();
    for (int d = lane; d < dh; d += 32) {
      float o = 0.f;
      for (int j = 0; j < n; ++j) o = fmaf(p[j], Vs[j * ld + d], o);
      out[(int64_t(b) * L + i) * C + h * dh + d] = from_f<T>(o);
    }
    __syncwarp();
  }
}

template <typename T>
__device__ __forceinline__ void st_acc(T* p, int64_t i, float v, int acc) {
  if (acc) v += to_f(p[i]);
  p[i] = from_f<T>(v);
}

template <typename T>
__global__ void __launch_bounds__(256) attn_bwd_k(const T* __restrict__ qkv,
                                                  const float* __restrict__ probs,
                                                  const T* __restrict__ out,
                                                  const T* __restrict__ dout,
                                                  const int32_t* __restrict__ len,
                                                  T* __restrict__ dqkv, int L, int C, int heads,
                                                  int acc) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  const int bh = blockIdx.x, b = bh / heads, h = bh % heads;
  const int dh = C / heads, ld = dh + 1, lds = L + 1;
  float* Qs = sm;
  float* Ks = Qs + L * ld;
  float* Vs = Ks + L * ld;
  float* dOs = Vs + L * ld;
  float* dS = dOs + L * ld;
  const T* base = qkv + int64_t(b) * L * 3 * C;
  for (int e = threadIdx.x; e < L * dh; e += blockDim.x) {
    int j = e / dh, d = e % dh;
    const T* r = base + int64_t(j) * 3 * C + h * dh + d;
    Qs[j * ld + d] = to_f(r[0]);
    Ks[j * ld + d] = to_f(r[C]);
    Vs[j * ld + d] = to_f(r[2 * C]);
    dOs[j * ld + d] = to_f(dout[(int64_t(b) * L + j) * C + h * dh + d]);
  }
  __syncthreads();
  const int n = len[b];
  const float scale = rsqrtf(float(dh));
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  T* dbase = dqkv + int64_t(b) * L * 3 * C;
  for (int i = warp; i < L; i += kWarps) {
    float delta = 0.f;
    for (int d = lane; d < dh; d += 32)
      delta += dOs[i * ld + d] * to_f(out[(int64_t(b) * L + i) * C + h * dh + d]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) delta += __shfl_xor_sync(0xffffffffu, delta, o);
    const float* prow = probs + (int64_t(bh) * L + i) * L;
    for (int j = lane; j < L; j += 32) {
      float ds = 0.f;
      if (j < n) {
        float dp = 0.f;
        for (int d = 0; d < dh; ++d) dp = fmaf(dOs[i * ld + d], Vs[j * ld + d], dp);
        ds = prow[j] * (dp - delta);
      }
      dS[i * lds + j] = ds;
    }
    __syncwarp();
    for (int d = lane; d < dh; d += 32) {
      float a = 0.f;
      for (int j = 0; j < n; ++j) a = fmaf(dS[i * lds + j], Ks[j * ld + d], a);
      st_acc(dbase, int64_t(i) * 3 * C + h * dh + d, a * scale, acc);
    }
  }
  __syncthreads();
  for (int j = warp; j < L; j += kWarps) {
    for (int d = lane; d < dh; d += 32) {
      float dk = 0.f, dv = 0.f;
      if (j < n) {
        for (int i = 0; i < L; ++i) {
          dk = fmaf(dS[i * lds + j], Qs[i * ld + d], dk);
          dv = fmaf(probs[(int64_t(bh) * L + i) * L + j], dOs[i * ld + d], dv);
        }
      }
      st_acc(dbase, int64_t(j) * 3 * C + C + h * dh + d, dk * scale, acc);
      st_acc(dbase, int64_t(j) * 3 * C + 2 * C + h * dh + d, dv, acc);
    }
  }
}

size_t fwd_smem(int L, int dh) { return sizeof(float) * (2 * L * (dh + 1) + kWarps * 64 + kWarps * L); }
size_t bwd_smem(int L, int dh) { return sizeof(float) * (4 * L * (dh + 1) + L * (L + 1)); }

}  // namespace

void attention_prepare(int L, int C, int heads) {
  const int f = int(fwd_smem(L, C / heads)), b = int(bwd_smem(L, C / heads));
  cudaFuncSetAttribute(attn_fwd_k<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, f);
  cudaFuncSetAttribute(attn_fwd_k<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, f);
  cudaFuncSetAttribute(attn_bwd_k<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, b);
  cudaFuncSetAttribute(attn_bwd_k<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, b);
}

void attention_fwd(const void* qkv, const int32_t* len, void* out, float* probs, int B, int L,
                   int C, int heads, int dt, cudaStream_t st) {
  size_t sm = fwd_smem(L, C / heads);
  if (dt == kF32) {
    launch_k(attn_fwd_k<float>, B * heads, 256, sm, st, (const float*)qkv, len, (float*)out, probs, L, C, heads);
  } else {
    launch_k(attn_fwd_k<bf16>, B * heads, 256, sm, st, (const bf16*)qkv, len, (bf16*)out, probs, L, C, heads);
  }
}

void attention_bwd(const void* qkv, const int32_t* len, const float* probs, const void* out,
                   const void* dout, void* dqkv, int B, int L, int C, int heads, int dt, bool acc,
                   cudaStream_t st) {
  size_t sm = bwd_smem(L, C / heads);
  if (dt == kF32) {
    launch_k(attn_bwd_k<float>, B * heads, 256, sm, st, (const float*)qkv, probs, (const float*)out,
                                                   (const float*)dout, len, (float*)dqkv, L, C,
                                                   heads, acc ? 1 : 0);
  } else {
    launch_k(attn_bwd_k<bf16>, B * heads, 256, sm, st, (const bf16*)qkv, probs, (const bf16*)out,
                                                  (const bf16*)dout, len, (bf16*)dqkv, L, C,
                                                  heads, acc ? 1 : 0);
  }
}

}  // namespace fo
