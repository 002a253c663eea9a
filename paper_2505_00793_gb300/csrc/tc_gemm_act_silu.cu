// Activation-epilogue instances of the tcgen05 dual GEMM for ACT_SILU (forward: bias + phi,
// phi' z'; backward: phi' da, phi'' z' da + phi' da'), one translation unit per activation so
// that the instances compile in parallel.
#include "tc_gemm_impl.cuh"

namespace mf {

cudaError_t tc_gemm_act_silu(const GemmArgs& a, cudaStream_t s, const char** why, int bn,
                              int pair) {
  if (a.epi.mode == EPI_ACT_FWD) return launch_bn<EPI_ACT_FWD, ACT_SILU>(a, s, why, bn, pair);
  return launch_bn<EPI_ACT_BWD, ACT_SILU>(a, s, why, bn, pair);
}

}  // namespace mf
