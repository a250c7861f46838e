// Instantiations of the tensor-core GEMM kernels for the fwd kinds
// (LIN_FWD, CONV_FPROP) and the epilogue variants the planner uses; kept
// in a translation unit of their own so that the kind groups compile in
// parallel.
#include "tc_gemm_kernels.cuh"

namespace fo {
namespace tcg {

KernelFn pick_fwd(int kind, int bn, bool cluster, int epi, size_t* smem) {
  if (kind == LIN_FWD && epi == (0)) return kernel_bn<LIN_FWD, 0>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_RELU)) return kernel_bn<LIN_FWD, E_RELU>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_ACC)) return kernel_bn<LIN_FWD, E_ACC>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_RELU | E_POOL)) return kernel_bn<LIN_FWD, E_RELU | E_POOL>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_TMA)) return kernel_bn<LIN_FWD, E_TMA>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_RELU | E_TMA)) return kernel_bn<LIN_FWD, E_RELU | E_TMA>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_ACC | E_TMA)) return kernel_bn<LIN_FWD, E_ACC | E_TMA>(bn, cluster, smem);
  if (kind == LIN_FWD && epi == (E_GELU | E_TMA)) return kernel_bn<LIN_FWD, E_GELU | E_TMA>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (0)) return kernel_bn<CONV_FPROP, 0>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_RELU)) return kernel_bn<CONV_FPROP, E_RELU>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_ACC)) return kernel_bn<CONV_FPROP, E_ACC>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_RELU | E_POOL)) return kernel_bn<CONV_FPROP, E_RELU | E_POOL>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_TMA)) return kernel_bn<CONV_FPROP, E_TMA>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_RELU | E_TMA)) return kernel_bn<CONV_FPROP, E_RELU | E_TMA>(bn, cluster, smem);
  if (kind == CONV_FPROP && epi == (E_ACC | E_TMA)) return kernel_bn<CONV_FPROP, E_ACC | E_TMA>(bn, cluster, smem);
  return nullptr;
}

}  // namespace tcg
}  // namespace fo
