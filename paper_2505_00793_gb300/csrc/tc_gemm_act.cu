// Activation-epilogue instances of the tcgen05 dual GEMM (forward: bias + phi, phi' z';
// backward: phi' da, phi'' z' da + phi' da').  The instances of each activation live in a
// translation unit of their own (tc_gemm_act_<activation>.cu) so that they compile in
// parallel; this file dispatches on the epilogue mode and the activation.
#include "internal.h"

namespace mf {

cudaError_t tc_gemm_act(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair) {
  if (a.epi.mode != EPI_ACT_FWD && a.epi.mode != EPI_ACT_BWD) {
    *why = "unknown epilogue mode or activation";
    return cudaErrorInvalidValue;
  }
  switch (a.epi.act) {
    case ACT_IDENT: return tc_gemm_act_ident(a, s, why, bn, pair);
    case ACT_TANH: return tc_gemm_act_tanh(a, s, why, bn, pair);
    case ACT_GELU: return tc_gemm_act_gelu(a, s, why, bn, pair);
    case ACT_SILU: return tc_gemm_act_silu(a, s, why, bn, pair);
  }
  *why = "unknown epilogue mode or activation";
  return cudaErrorInvalidValue;
}

}  // namespace mf
