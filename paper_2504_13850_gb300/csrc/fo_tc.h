// Tensor-core (tcgen05 / TMEM / TMA) GEMM and implicit-GEMM convolution
// planner for the bf16 compute path.  The plan functions return nullptr for
// shapes the tensor-core kernels do not take; the caller then uses the
// CUDA-core kernels.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <vector>

struct fo_server;

namespace fo {

struct TcContext;
struct TcGemm;

int tc_create(TcContext** out, fo_server* s);
void tc_destroy(TcContext* c);
// Selects the tensor maps of batch slot `slot` for the first layer.
void tc_set_input(TcContext* c, int slot);
// Extra epilogue work of a GEMM with a bf16 output (all fields optional).
struct TcEpilogue {
  // out = result + addend: a residual add in the forward pass, or the
  // gradient a residual connection passes around a layer in the backward
  // pass (bf16, out's layout)
  const void* addend = nullptr;
  bool addend_is_input = false;   // the addend is the uploaded batch of the step's slot
  // forward with ReLU: a 2x2 max-pool of the output (output width <= 16):
  // the pooled values [N][H/2][W/2][C] and the window code of each pooled
  // element (first maximum, 0..3 row-major) instead of the full output
  void* pool_out = nullptr;
  uint8_t* pool_code = nullptr;
  // forward of a linear layer whose output feeds only a GELU: `out` gets the
  // bias-added result and gelu_out the GELU of it (bf16, the same layout)
  void* gelu_out = nullptr;
};
// Forward of conv/linear op `op` into `out` (bf16, the op's output layout),
// applying a ReLU when `relu`.
TcGemm* tc_plan_forward(TcContext* c, fo_server* s, int op, void* out, bool relu, const TcEpilogue* ex = nullptr);
// Input gradient of op `op` into `dx` (accumulating when `accumulate`),
// multiplied by (mask > 0) when `mask` (same layout as dx) is given.  A
// strided convolution gives one GEMM per output-parity class; when some
// class has no taps and this is the first contribution, *zero_first asks
// the caller to clear dx before the GEMMs (which then accumulate).
// Returns false when the tensor cores do not take the shape.
// An `ex` (plain GEMMs only: linear layers and 1x1 convolutions) adds an
// addend (then `accumulate` must be 0).
bool tc_plan_dgrad(TcContext* c, fo_server* s, int op, int accumulate, void* dx, const void* mask,
                   std::vector<TcGemm*>* out, bool* zero_first, const TcEpilogue* ex = nullptr);
// True when the tensor cores take op `op` as one plain GEMM (a linear layer
// or a 1x1 stride-1 convolution on the bf16 path), so that its forward and
// input-gradient epilogues can take a TcEpilogue.
bool tc_plain_ok(TcContext* c, const fo_server* s, int op);
TcGemm* tc_plan_wgrad(TcContext* c, fo_server* s, int op);
// Launches the GEMM kernel; a split-K plan runs as clusters of tc_splits(g)
// CTAs that reduce their partial tiles through an L2-resident workspace.
void tc_run(TcGemm* g, const void* input, cudaStream_t st);
int tc_splits(const TcGemm* g);
double tc_flops(const TcGemm* g);
const char* tc_name(const TcGemm* g);
// Allocates the split-K workspace after every plan is known.
int tc_finalize(TcContext* c);
// Stream lane of a plan's GEMM (0 compute stream, 1 side stream): GEMMs of
// different lanes may run concurrently, so each lane has its own split-K
// workspace.  Set before tc_finalize.
void tc_set_lane(TcGemm* g, int lane);
// Device word the tensor-core kernels set on a timed-out wait (0 = none).
int* tc_error_word(TcContext* c);
// Tensor map of a row-major bf16 matrix [rows][cols] with 128-byte-swizzled
// boxes of 64 columns x box_rows rows.
bool tc_encode_2d(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows);

// Tensor-core attention (k_attention_tc.cu): sequences of at most 128 tokens,
// head width 64, bf16.  A plan holds the tensor maps of the packed q|k|v
// input [B*L, 3C] and of dO [B*L, C], and the address of the output O
// [B*L, C] (the backward reads its rows directly).
struct AttnTcPlan;
bool attention_tc_ok(int L, int C, int heads);
AttnTcPlan* attention_tc_plan(const void* qkv, const void* out, const void* dout, int B, int L, int C, int heads,
                              int* err);
void attention_tc_destroy(AttnTcPlan* a);
// O and the per-row log-sum-exp of the scaled scores (lse: [B * heads * L]).
void attention_tc_fwd(const AttnTcPlan* a, const int32_t* len, void* out, float* lse, int B, cudaStream_t st);
// d(q|k|v) [B*L, 3C] from dO, the saved lse and the forward output.
void attention_tc_bwd(const AttnTcPlan* a, const int32_t* len, const float* lse, void* dqkv, int B, bool acc,
                      cudaStream_t st);

}  // namespace fo
