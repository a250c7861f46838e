// Classifier head of the server network: the last linear layer (few
// outputs) fused with the server loss f_s (softmax cross-entropy averaged
// over the batch) and its backward pass.
//   head_fwd_ce : logits z = x W^T + b, per-row CE, dz = (softmax(z) - onehot)/B,
//                 and (optionally, in the same blocks) dx (+)= dz W, times a
//                 ReLU mask (mask > 0) when one is given
//   head_wgrad  : dW = dz^T x, db = sum_b dz, loss = mean of the row losses
//                 (summed in row order, deterministic)
// W and b are the fp32 master weights; dz and the gradients are fp32.
#include "fo_common.cuh"
#include "fo_kernels.h"

namespace fo {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// One block per batch row; warps split the classes.  smem: x row (K floats)
// and the logits (C floats).
// With `dx` given, the same block then forms its row's input gradient
// dx[b][k] (+)= (sum_c dz[b][c] W[c][k]) * (mask[b][k] > 0): a row's input
// gradient needs only that row's dz, so the backward needs no second launch.
template <typename T>
__global__ void head_fwd_ce_k(const T* __restrict__ x, const float* __restrict__ W,
                              const float* __restrict__ bias, const int32_t* __restrict__ labels, int B,
                              int K, int C, float* __restrict__ logits, float* __restrict__ dz,
                              float* __restrict__ row_loss, const T* __restrict__ mask, T* __restrict__ dx,
                              int acc) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  float* xr = sm;
  float* z = sm + K;
  float* zd = z + C;
  const int b = blockIdx.x;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, nw = blockDim.x / 32;
  for (int k = threadIdx.x; k < K; k += blockDim.x) xr[k] = to_f(x[int64_t(b) * K + k]);
  __syncthreads();
  for (int c = warp; c < C; c += nw) {
    const float* w = W + int64_t(c) * K;
    float s = 0.f;
    for (int k = lane; k < K; k += 32) s = fmaf(xr[k], w[k], s);
    s = warp_sum(s);
    if (lane == 0) z[c] = s + (bias ? bias[c] : 0.f);
  }
  __syncthreads();
  if (warp == 0) {
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, z[c]);
    m = warp_max(m);
    float se = 0.f;
    for (int c = lane; c < C; c += 32) se += expf(z[c] - m);
    se = warp_sum(se);
    const int y = labels[b];
    for (int c = lane; c < C; c += 32) {
      const float p = expf(z[c] - m) / se;
      const float d = (p - (c == y ? 1.f : 0.f)) / float(B);
      dz[int64_t(b) * C + c] = d;
      zd[c] = d;
      logits[int64_t(b) * C + c] = z[c];
    }
    if (lane == 0) row_loss[b] = m + logf(se) - z[y];
  }
  if (!dx) return;
  __syncthreads();
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    float s = 0.f;
    for (int c = 0; c < C; ++c) s = fmaf(zd[c], W[int64_t(c) * K + k], s);
    const int64_t i = int64_t(b) * K + k;
    if (mask && !(to_f(mask[i]) > 0.f)) s = 0.f;
    if (acc) s += to_f(dx[i]);
    dx[i] = from_f<T>(s);
  }
}

// dW[c][k] = sum_b dz[b][c] x[b][k]: block = 32 columns k x 8 classes c,
// rows staged through shared memory 64 at a time; grid (ceil(K/32),
// ceil(C/8)).  Block (0, y) also writes db for its classes; block (0, 0)
// the batch-mean loss (row order).
template <typename T>
__global__ void head_wgrad_k(const float* __restrict__ dz, const T* __restrict__ x, int B, int K, int C,
                             float* __restrict__ dW, float* __restrict__ db, const float* __restrict__ row_loss,
                             float* __restrict__ losses, const int64_t* __restrict__ step, int64_t mask) {
  pdl_wait();
  pdl_trigger();
  __shared__ float xs[64][33];
  __shared__ float ds[64][8];
  const int kk = threadIdx.x % 32, cc = threadIdx.x / 32;
  const int k = blockIdx.x * 32 + kk, c = blockIdx.y * 8 + cc;
  float acc = 0.f;
  for (int b0 = 0; b0 < B; b0 += 64) {
    for (int e = threadIdx.x; e < 64 * 32; e += blockDim.x) {
      const int b = b0 + e / 32, kx = blockIdx.x * 32 + e % 32;
      xs[e / 32][e % 32] = (b < B && kx < K) ? to_f(x[int64_t(b) * K + kx]) : 0.f;
    }
    for (int e = threadIdx.x; e < 64 * 8; e += blockDim.x) {
      const int b = b0 + e / 8, cx = blockIdx.y * 8 + e % 8;
      ds[e / 8][e % 8] = (b < B && cx < C) ? dz[int64_t(b) * C + cx] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int b = 0; b < 64; ++b) acc = fmaf(ds[b][cc], xs[b][kk], acc);
    __syncthreads();
  }
  if (k < K && c < C) dW[int64_t(c) * K + k] = acc;
  if (blockIdx.x == 0 && kk == 0 && c < C) {
    if (db) {
      float s = 0.f;
      for (int b = 0; b < B; ++b) s += dz[int64_t(b) * C + c];
      db[c] = s;
    }
    if (c == 0) {
      float t = 0.f;
      for (int b = 0; b < B; ++b) t += row_loss[b];
      losses[*step & mask] = t / float(B);
    }
  }
}

}  // namespace

void head_forward_loss(const void* x, int dt, const float* W, const float* bias, const int32_t* labels, int B,
                       int K, int C, float* logits, float* dz, float* row_loss, cudaStream_t st, const void* mask,
                       void* dx, bool acc) {
  size_t sm = sizeof(float) * (K + 2 * C);
  if (dt == kF32)
    launch_k(head_fwd_ce_k<float>, B, 256, sm, st, (const float*)x, W, bias, labels, B, K, C, logits, dz, row_loss,
             (const float*)mask, (float*)dx, acc ? 1 : 0);
  else
    launch_k(head_fwd_ce_k<bf16>, B, 256, sm, st, (const bf16*)x, W, bias, labels, B, K, C, logits, dz, row_loss,
             (const bf16*)mask, (bf16*)dx, acc ? 1 : 0);
}

void head_weight_grad(const float* dz, const void* x, int dt, int B, int K, int C, float* dW, float* db,
                      const float* row_loss, float* losses, const int64_t* step, int64_t mask,
                      cudaStream_t st) {
  dim3 grid(ceil_div(K, 32), ceil_div(C, 8));
  if (dt == kF32)
    launch_k(head_wgrad_k<float>, grid, 256, 0, st, dz, (const float*)x, B, K, C, dW, db, row_loss, losses, step, mask);
  else
    launch_k(head_wgrad_k<bf16>, grid, 256, 0, st, dz, (const bf16*)x, B, K, C, dW, db, row_loss, losses, step, mask);
}

}  // namespace fo
