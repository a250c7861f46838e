// Host launchers of the library's CUDA kernels (internal interface).
#pragma once
#include <vector>
#include <cuda_runtime.h>
#include <cstdint>

namespace fo {

enum DType { kF32 = 0, kBF16 = 1 };

// ---- CUDA-core implicit-GEMM convolution / linear (fp32 accumulate) ----
// A linear layer over rows is a 1x1 convolution of N = rows 1x1 images.
struct ConvShape {
  int N, H, W, Ci, Co, k, stride, pad, Ho, Wo;
};
// y = conv(x, w) + bias, optional ReLU.  x NHWC, w [Co][k][k][Ci], bias fp32
// or null, y NHWC; each operand's dtype is given (kF32 / kBF16).
void conv_fwd_simt(const ConvShape& s, const void* x, int dt_x, const void* w, int dt_w,
                   const float* bias, void* y, int dt_y, bool relu, cudaStream_t st);
// dx (+)= conv^T(dy, w), times (mask > 0) when mask (same layout as dx) is given.
void conv_dgrad_simt(const ConvShape& s, const void* dy, int dt_dy, const void* w, int dt_w,
                     void* dx, int dt_dx, bool accumulate, const void* mask, cudaStream_t st);
// dw[Co][k][k][Ci] = sum over output pixels of dy (x) x-window (fp32 out).
// Weight gradient; K is split over blocks into `scratch` (simt_wgrad_scratch_floats
// floats, or null for one pass) and summed in split order.
int simt_wgrad_splits(const ConvShape& s);
int64_t simt_wgrad_scratch_floats(const ConvShape& s);
void conv_wgrad_simt(const ConvShape& s, const void* dy, int dt_dy, const void* x, int dt_x,
                     float* dw, float* scratch, cudaStream_t st);

// ---- elementwise / reductions (templated on the activation dtype) ----
void relu_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st);
// dx (+)= dy * (x > 0)
void relu_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc,
              cudaStream_t st);
void maxpool2_fwd(const void* x, void* y, int N, int H, int W, int C, int dt, cudaStream_t st);
void maxpool2_bwd(const void* x, const void* dy, void* dx, int N, int H, int W, int C,
                  int dt, bool acc, cudaStream_t st);
// Fused backward of relu(x) followed by maxpool2: dx (+)= route(dy) * (x > 0)
// ReLU + 2x2 max-pool backward from the pooled values y and the window codes
// (first-maximum position 0..3 per pooled element) that a GEMM epilogue
// stored in the forward pass (bf16, C % 8 == 0).
void relu_maxpool2_bwd_codes(const void* y, const uint8_t* code, const void* dy, void* dx, int N, int H, int W,
                             int C, bool acc, cudaStream_t st);
void relu_maxpool2_bwd(const void* x, const void* dy, void* dx, int N, int H, int W, int C,
                       int dt, bool acc, cudaStream_t st);
void affine_fwd(const void* x, const float* scale, const float* shift, void* y, int64_t rows,
                int C, int dt, bool relu, cudaStream_t st);
// dx (+)= dy * scale (dx may be null)
void affine_dx(const void* dy, const float* scale, void* dx, int64_t rows, int C, int dt,
               bool acc, cudaStream_t st);
void add_fwd(const void* a, const void* b, void* y, int64_t n, int dt, bool relu, cudaStream_t st);
// Backward of a residual add, optionally through the ReLU after it:
// g = dy * (mask > 0) (mask may be null); d0 (+)= g; d1 (+)= g (d1 may be null).
void grad_split(const void* dy, const void* mask, void* d0, bool acc0, void* d1, bool acc1, int64_t n, int dt,
                cudaStream_t st);
void avgpool_fwd(const void* x, void* y, int N, int HW, int C, int dt, cudaStream_t st);
void avgpool_bwd(const void* dy, void* dx, int N, int HW, int C, int dt, bool acc,
                 cudaStream_t st);
void gelu_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st);
void gelu_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc,
              cudaStream_t st);
void layernorm_fwd(const void* x, const float* gamma, const float* beta, void* y,
                   float* mean, float* rstd, int64_t rows, int C, int dt, cudaStream_t st);
// dx (+)= layernorm input gradient (gamma/beta gradients come from colsum / colsum_lnx)
void layernorm_bwd_dx(const void* x, const float* gamma, const float* mean, const float* rstd,
                      const void* dy, void* dx, int64_t rows, int C, int dt, bool acc,
                      cudaStream_t st);
// out[c] = sum_r a[r][c] * f(r, c) where f = 1, b[r][c], or the layernorm xhat.
// `partial` is scratch of at least colsum_partial_floats(rows, C) floats
// (128-row chunks); the server passes adaptive = true (chunks sized to the
// GPU, scratch from server_colsum_floats).
int64_t colsum_partial_floats(int64_t rows, int C);
// Most rows the public column sums take: their row chunks (128 rows each)
// are one grid dimension, at most 65,535 blocks.
constexpr int64_t kColsumMaxRows = int64_t(65535) * 128;
int64_t server_colsum_floats(int64_t rows, int C);
void colsum(const void* a, const void* b, int64_t rows, int C, int dt, float* partial,
            float* out, cudaStream_t st, bool adaptive = false);
void colsum_lnx(const void* dy, const void* x, const float* mean, const float* rstd,
                int64_t rows, int C, int dt, float* partial, float* out, cudaStream_t st);
void meanpool_fwd(const void* x, const int32_t* len, void* y, int B, int L, int C, int dt,
                  cudaStream_t st);
void meanpool_bwd(const void* dy, const int32_t* len, void* dx, int B, int L, int C, int dt,
                  bool acc, cudaStream_t st);
// Attention over packed qkv [B, L, 3C], heads h (C/h <= 64); probs fp32 [B,h,L,L] saved.
// attention_prepare sets the kernels' shared-memory limits (call before use / capture).
void attention_prepare(int L, int C, int heads);
void attention_fwd(const void* qkv, const int32_t* len, void* out, float* probs, int B, int L,
                   int C, int heads, int dt, cudaStream_t st);
void attention_bwd(const void* qkv, const int32_t* len, const float* probs, const void* out,
                   const void* dout, void* dqkv, int B, int L, int C, int heads, int dt, bool acc,
                   cudaStream_t st);

// Classifier head (last linear layer + softmax cross-entropy), fp32 weights.
// With dx given, also the input gradient dx (+)= dz W (times mask > 0 when
// mask is given), formed by the same blocks (no second launch).
void head_forward_loss(const void* x, int dt, const float* W, const float* bias, const int32_t* labels,
                       int B, int K, int C, float* logits, float* dz, float* row_loss, cudaStream_t st,
                       const void* mask = nullptr, void* dx = nullptr, bool acc = false);
// The batch loss goes to losses[*step & mask].
void head_weight_grad(const float* dz, const void* x, int dt, int B, int K, int C, float* dW, float* db,
                      const float* row_loss, float* losses, const int64_t* step, int64_t mask,
                      cudaStream_t st);

// Softmax cross-entropy: losses[*step & mask] <- mean_b CE; dlogits = (softmax - onehot)/B.
void softmax_ce(const float* logits, const int32_t* labels, int B, int C, float* losses,
                const int64_t* step, int64_t mask, void* dlogits, int dt, cudaStream_t st);

// SGD with momentum over a flat vector (n a multiple of 4, 16-byte aligned):
// v = mu v + g; theta -= lr v; shadow (bf16, may be null) = bf16(theta).
// The step counter (may be null) is incremented once.  skip64 (device, may
// be null): one flag per 64 elements; flagged blocks are not touched.
void sgd_momentum(float* theta, float* v, const float* g, void* shadow, int64_t n, float lr,
                  float mu, int64_t* step, cudaStream_t st, const uint8_t* skip64 = nullptr);
// The update restricted to the 64-element blocks listed in blocks64 (device,
// nb entries: block b covers elements 64b .. 64b + 63).
// Contiguous segments of the parameter vector updated by one launch:
// segment k is float4 elements [off4[k], off4[k] + pre4[k+1] - pre4[k]).
constexpr int kSgdMaxSegs = 32;
struct SgdSegments {
  int n;
  int64_t off4[kSgdMaxSegs];
  int64_t pre4[kSgdMaxSegs + 1];
};
void sgd_momentum_segments(float* theta, float* v, const float* g, void* shadow, const SgdSegments& sg, float lr,
                           float mu, cudaStream_t st);
void sgd_momentum_blocks(float* theta, float* v, const float* g, void* shadow, const int64_t* blocks64, int64_t nb,
                         float lr, float mu, int64_t* step, cudaStream_t st);
void f32_to_bf16(const float* x, void* y, int64_t n, cudaStream_t st);

// ---- vectorised bf16 kernels (k_vec.cu): 8 elements per 16-byte access ----
bool vec8_ok(int dt, int64_t n);
void relu_bwd_x8(const void* y, const void* dy, void* dx, int64_t n, bool acc, cudaStream_t st);
void add_x8(const void* a, const void* b, void* y, int64_t n, bool relu, cudaStream_t st);
void grad_split_x8(const void* dy, const void* mask, void* d0, bool acc0, void* d1, bool acc1, int64_t n,
                   cudaStream_t st);
void affine_fwd_x8(const void* x, const float* sc, const float* sh, void* y, int64_t n, int C, bool relu,
                   cudaStream_t st);
void gelu_fwd_x8(const void* x, void* y, int64_t n, cudaStream_t st);
void gelu_bwd_x8(const void* x, const void* dy, void* dx, int64_t n, bool acc, cudaStream_t st);
// Column sums (C % 8 == 0) with a (column block, row chunk) grid; chunks of
// 128 rows, or sized to the GPU (about two blocks per SM) when `adaptive`.
int64_t colsum8_partial_floats(int64_t rows, int C, bool adaptive);
void colsum8(const void* a, int64_t rows, int C, float* partial, float* out, bool adaptive, cudaStream_t st);
// Deferred parameter-gradient reductions, batched into one launch each (at
// most a few dozen launches' worth of work per call; fixed summation order).
// ColsumTask: column sums of a bf16 [rows, C] matrix (C % 8 == 0) into
// `partial` ([colsum8_batch_chunks(rows), C] floats).  FinishTask: out[c] =
// sum over the `chunks` rows of partial [chunks, C].
struct ColsumTask {
  const void* a;
  float* partial;
  int64_t rows;
  int C;
};
struct FinishTask {
  const float* partial;
  float* out;
  int chunks;
  int C;
};
int colsum8_batch_chunks(int64_t rows);
void colsum8_batched(const std::vector<ColsumTask>& tasks, cudaStream_t st);
void finish_batched(const std::vector<FinishTask>& tasks, cudaStream_t st);
// Affine backward pass without its finish: partials of dscale and dshift
// ([affine_bwd8_chunks(rows, C), C] each) and dx (+)= dy * scale.  With
// `hswish_in` (the affine output feeding a hard swish) dy is the gradient of
// the hard swish's output and the pass applies hswish'(hswish_in) first.
int affine_bwd8_chunks(int64_t rows, int C);
void affine_bwd8_pass(const void* dy, const void* x, const float* scale, void* dx, bool acc, int64_t rows, int C,
                      float* p_scale, float* p_shift, cudaStream_t st, const void* hswish_in = nullptr);
// Affine then hard swish in one pass: pre = x * scale + shift, post = hswish(pre).
void affine_hswish_fwd_x8(const void* x, const float* sc, const float* sh, void* pre, void* post, int64_t n, int C,
                          cudaStream_t st);
// Layernorm forward with the row in registers (bf16, C % 256 == 0, C <= 1024).
bool layernorm_fwd8_ok(int dt, int C);
void layernorm_fwd_x8(const void* x, const float* gamma, const float* beta, void* y, float* mean, float* rstd,
                      int64_t rows, int C, cudaStream_t st);
// Layernorm backward fused with dgamma / dbeta (C % 256 == 0, C <= 512).
// Masked mean-pool over tokens and its gradient, 8 bf16 columns per access.
bool meanpool8_ok(int dt, int C);
void meanpool_fwd_x8(const void* x, const int32_t* len, void* y, int B, int L, int C, cudaStream_t st);
void meanpool_bwd_x8(const void* dy, const int32_t* len, void* dx, int B, int L, int C, bool acc, cudaStream_t st);
bool layernorm_bwd8_ok(int dt, int C);
int64_t layernorm_bwd8_partial_floats(int64_t rows, int C);
// The same pass without its finish: partials [layernorm_bwd8_blocks(rows), C]
// of dgamma and dbeta.
int layernorm_bwd8_blocks(int64_t rows);
// dx = (dx if acc) + input gradient + (addend if given, dx's layout).
// With p_dx, also the column partial sums of the stored dx per block
// ([layernorm_bwd8_blocks(rows)][C]): the bias gradient of the layer whose
// output gradient dx is.
void layernorm_bwd8_pass(const void* x, const float* gamma, const float* mean, const float* rstd, const void* dy,
                         void* dx, int64_t rows, int C, bool acc, float* p_gamma, float* p_beta, cudaStream_t st,
                         const void* addend = nullptr, float* p_dx = nullptr);


// ---- MobileNetV3 bottleneck (k_mobile.cu) ----
// Depthwise k x k convolution, NHWC, weights [C][k][k] in the activation
// dtype `dt`, bias fp32 or null, padding `pad`.
struct DwShape {
  int N, H, W, C, k, stride, pad, Ho, Wo;
};
void dwconv_fwd(const DwShape& d, const void* x, const void* w, const float* bias, void* y, int dt,
                cudaStream_t st);
// dx (+)= transposed depthwise convolution of dy.
void dwconv_dgrad(const DwShape& d, const void* dy, const void* w, void* dx, int dt, bool acc, cudaStream_t st);
// Per-chunk partials of dW ([chunks][C*k*k]) and, when pb is given, of the
// bias gradient ([chunks][C]); chunks = dwconv_wgrad_chunks(d).
int dwconv_wgrad_chunks(const DwShape& d);
void dwconv_wgrad_pass(const DwShape& d, const void* dy, const void* x, int dt, float* pw, float* pb,
                       cudaStream_t st);
// Hard swish x * relu6(x + 3) / 6 and hard sigmoid relu6(x + 3) / 6; the
// backward kernels take the forward input x: dx (+)= dy * f'(x).
void hswish_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st);
void hswish_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st);
void hsigmoid_fwd(const void* x, void* y, int64_t n, int dt, cudaStream_t st);
void hsigmoid_bwd(const void* x, const void* dy, void* dx, int64_t n, int dt, bool acc, cudaStream_t st);
// Squeeze-and-excite scaling y[n,p,c] = x[n,p,c] s[n,c] (s is [N, C]);
// backward dx (+)= dy s and ds (+)= sum_p dy x (either output may be null).
void chmul_fwd(const void* x, const void* s, void* y, int N, int HW, int C, int dt, cudaStream_t st);
void chmul_bwd(const void* x, const void* s, const void* dy, void* dx, bool acc_dx, void* ds, bool acc_ds, int N,
               int HW, int C, int dt, cudaStream_t st);

// FedAsync update: g = fmaf(alpha, l - g, g).
void axpby(float* g, const float* l, int64_t n, float alpha, cudaStream_t st);
// Number of kernels axpby launches for these arguments (vector body, tail).
int axpby_kernels(const float* g, const float* l, int64_t n);

}  // namespace fo
