// Activation-epilogue instances of the tcgen05 dual GEMM (forward: bias + phi, phi' z';
// backward: phi' da, phi'' z' da + phi' da').  Kept in their own translation unit so that the
// instances compile in parallel with the plain-store ones.
#include "tc_gemm_impl.cuh"

namespace mf {

cudaError_t tc_gemm_act(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair) {
  const int act = a.epi.act;
  if (a.epi.mode == EPI_ACT_FWD) {
    switch (act) {
      case ACT_IDENT: return launch_bn<EPI_ACT_FWD, ACT_IDENT>(a, s, why, bn, pair);
      case ACT_TANH: return launch_bn<EPI_ACT_FWD, ACT_TANH>(a, s, why, bn, pair);
      case ACT_GELU: return launch_bn<EPI_ACT_FWD, ACT_GELU>(a, s, why, bn, pair);
      case ACT_SILU: return launch_bn<EPI_ACT_FWD, ACT_SILU>(a, s, why, bn, pair);
    }
  } else if (a.epi.mode == EPI_ACT_BWD) {
    switch (act) {
      case ACT_IDENT: return launch_bn<EPI_ACT_BWD, ACT_IDENT>(a, s, why, bn, pair);
      case ACT_TANH: return launch_bn<EPI_ACT_BWD, ACT_TANH>(a, s, why, bn, pair);
      case ACT_GELU: return launch_bn<EPI_ACT_BWD, ACT_GELU>(a, s, why, bn, pair);
      case ACT_SILU: return launch_bn<EPI_ACT_BWD, ACT_SILU>(a, s, why, bn, pair);
    }
  }
  *why = "unknown epilogue mode or activation";
  return cudaErrorInvalidValue;
}

}  // namespace mf
