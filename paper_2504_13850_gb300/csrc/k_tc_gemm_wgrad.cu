// Instantiations of the tensor-core GEMM kernels for the wgrad kinds
// (LIN_WGRAD, CONV_WGRAD) and the epilogue variants the planner uses; kept
// in a translation unit of their own so that the kind groups compile in
// parallel.
#include "tc_gemm_kernels.cuh"

namespace fo {
namespace tcg {

KernelFn pick_wgrad(int kind, int bn, bool cluster, int epi, size_t* smem) {
  if (kind == LIN_WGRAD && epi == (E_F32)) return kernel_bn<LIN_WGRAD, E_F32>(bn, cluster, smem);
  if (kind == CONV_WGRAD && epi == (E_F32)) return kernel_bn<CONV_WGRAD, E_F32>(bn, cluster, smem);
  return nullptr;
}

}  // namespace tcg
}  // namespace fo
