// Instantiations of the tensor-core GEMM kernels for the dgrad kinds
// (LIN_DGRAD, CONV_DGRAD) and the epilogue variants the planner uses; kept
// in a translation unit of their own so that the kind groups compile in
// parallel.
#include "tc_gemm_kernels.cuh"

namespace fo {
namespace tcg {

KernelFn pick_dgrad(int kind, int bn, bool cluster, int epi, size_t* smem) {
  if (kind == LIN_DGRAD && epi == (0)) return kernel_bn<LIN_DGRAD, 0>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_MASK)) return kernel_bn<LIN_DGRAD, E_MASK>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_ACC)) return kernel_bn<LIN_DGRAD, E_ACC>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_MASK | E_ACC)) return kernel_bn<LIN_DGRAD, E_MASK | E_ACC>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (0)) return kernel_bn<CONV_DGRAD, 0>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_MASK)) return kernel_bn<CONV_DGRAD, E_MASK>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_ACC)) return kernel_bn<CONV_DGRAD, E_ACC>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_MASK | E_ACC)) return kernel_bn<CONV_DGRAD, E_MASK | E_ACC>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_TMA)) return kernel_bn<LIN_DGRAD, E_TMA>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_MASK | E_TMA)) return kernel_bn<LIN_DGRAD, E_MASK | E_TMA>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_ACC | E_TMA)) return kernel_bn<LIN_DGRAD, E_ACC | E_TMA>(bn, cluster, smem);
  if (kind == LIN_DGRAD && epi == (E_MASK | E_ACC | E_TMA)) return kernel_bn<LIN_DGRAD, E_MASK | E_ACC | E_TMA>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_TMA)) return kernel_bn<CONV_DGRAD, E_TMA>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_MASK | E_TMA)) return kernel_bn<CONV_DGRAD, E_MASK | E_TMA>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_ACC | E_TMA)) return kernel_bn<CONV_DGRAD, E_ACC | E_TMA>(bn, cluster, smem);
  if (kind == CONV_DGRAD && epi == (E_MASK | E_ACC | E_TMA)) return kernel_bn<CONV_DGRAD, E_MASK | E_ACC | E_TMA>(bn, cluster, smem);
  return nullptr;
}

}  // namespace tcg
}  // namespace fo
