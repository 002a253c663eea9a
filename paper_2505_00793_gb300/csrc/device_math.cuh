// Device helpers shared by the GEMM epilogues and the elementwise kernels.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace mf {

template <typename T> __device__ __forceinline__ T to_t(float x);
template <> __device__ __forceinline__ float to_t<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 to_t<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// phi, phi', phi'' of the hidden activations.
//   tanh:  phi' = 1 - t^2,                     phi'' = -2 t (1 - t^2)
//   GELU:  phi = x Phi(x), phi' = Phi + x pdf,  phi'' = pdf (2 - x^2)
//   SiLU:  phi = x s(x),  phi' = s (1 + x (1 - s)),  phi'' = s (1 - s) (2 + x (1 - 2 s))
__device__ __forceinline__ void act_eval(int act, float z, float& f, float& d1, float& d2) {
  switch (act) {
    case ACT_TANH: {
      const float t = tanhf(z);
      f = t; d1 = 1.f - t * t; d2 = -2.f * t * d1;
      break;
    }
    case ACT_GELU: {
      const float cdf = 0.5f * (1.f + erff(z * 0.70710678118654752f));
      const float pdf = 0.39894228040143268f * expf(-0.5f * z * z);
      f = z * cdf; d1 = cdf + z * pdf; d2 = pdf * (2.f - z * z);
      break;
    }
    case ACT_SILU: {
      const float sg = 1.f / (1.f + expf(-z));
      f = z * sg; d1 = sg * (1.f + z * (1.f - sg));
      d2 = sg * (1.f - sg) * (2.f + z * (1.f - 2.f * sg));
      break;
    }
    default:
      f = z; d1 = 1.f; d2 = 0.f;
  }
}

// Per-element epilogue of a dual GEMM (shared by the tensor-core and SIMT kernels).
//  EPI_STORE:   C0 = acc0 + bias0, C1 = acc1 + bias1.
//  EPI_ACT_FWD: z = acc0 + bias0, z' = acc1 + bias1 -> C0 = z, C1 = z' (float32),
//               a = phi(z), a' = phi'(z) z'  -> A, Ad (row-major).
//  EPI_ACT_BWD: da = acc0, da' = acc1, z, z' read from Z, Zd ->
//               dz = phi'(z) da, dz' = phi''(z) z' da + phi'(z) da'  -> A, Ad.
struct EpiOut {
  float c0, c1;     // float32 outputs for C0 / C1
  float o0, o1;     // values for A / Ad
};

__device__ __forceinline__ EpiOut epi_eval(const EpiParams& e, int m, int n, float acc0,
                                           float acc1, const float* bias0, const float* bias1,
                                           bool dual) {
  EpiOut r;
  if (e.mode == EPI_ACT_BWD) {
    const float z = e.Z[static_cast<int64_t>(m) * e.ldz + n];
    float f, d1, d2;
    act_eval(e.act, z, f, d1, d2);
    r.c0 = acc0; r.c1 = acc1;
    r.o0 = d1 * acc0;
    r.o1 = dual ? d2 * e.Zd[static_cast<int64_t>(m) * e.ldz + n] * acc0 + d1 * acc1 : 0.f;
    return r;
  }
  const float z = acc0 + (bias0 ? bias0[n] : 0.f);
  const float zd = acc1 + (bias1 ? bias1[n] : 0.f);
  r.c0 = z; r.c1 = zd;
  if (e.mode == EPI_ACT_FWD) {
    float f, d1, d2;
    act_eval(e.act, z, f, d1, d2);
    r.o0 = f;
    r.o1 = dual ? d1 * zd : 0.f;
  } else {
    r.o0 = r.o1 = 0.f;
  }
  return r;
}

// Compile-time specialisations of act_eval / epi_eval (one activation, one epilogue mode per
// kernel instance: the per-element code stays small).
template <int ACT>
__device__ __forceinline__ void act_eval_t(float z, float& f, float& d1, float& d2) {
  if constexpr (ACT == ACT_TANH) {
    const float t = tanhf(z);
    f = t; d1 = 1.f - t * t; d2 = -2.f * t * d1;
  } else if constexpr (ACT == ACT_GELU) {
    const float cdf = 0.5f * (1.f + erff(z * 0.70710678118654752f));
    const float pdf = 0.39894228040143268f * expf(-0.5f * z * z);
    f = z * cdf; d1 = cdf + z * pdf; d2 = pdf * (2.f - z * z);
  } else if constexpr (ACT == ACT_SILU) {
    const float sg = 1.f / (1.f + expf(-z));
    f = z * sg; d1 = sg * (1.f + z * (1.f - sg));
    d2 = sg * (1.f - sg) * (2.f + z * (1.f - 2.f * sg));
  } else {
    f = z; d1 = 1.f; d2 = 0.f;
  }
}

// The per-element arithmetic of epi_eval_t on values already loaded: z, zd the stored
// pre-activation and its tangent (EPI_ACT_BWD), b0, b1 the biases (0 when absent).
template <int MODE, int ACT>
__device__ __forceinline__ EpiOut epi_core_t(float acc0, float acc1, float z_in, float zd_in,
                                             float b0, float b1, bool dual) {
  EpiOut r;
  if constexpr (MODE == EPI_ACT_BWD) {
    float f, d1, d2;
    act_eval_t<ACT>(z_in, f, d1, d2);
    r.c0 = acc0; r.c1 = acc1;
    r.o0 = d1 * acc0;
    r.o1 = dual ? d2 * zd_in * acc0 + d1 * acc1 : 0.f;
  } else {
    const float z = acc0 + b0;
    const float zd = acc1 + b1;
    r.c0 = z; r.c1 = zd;
    if constexpr (MODE == EPI_ACT_FWD) {
      float f, d1, d2;
      act_eval_t<ACT>(z, f, d1, d2);
      r.o0 = f;
      r.o1 = dual ? d1 * zd : 0.f;
    } else {
      r.o0 = r.o1 = 0.f;
    }
  }
  return r;
}

template <int MODE, int ACT>
__device__ __forceinline__ EpiOut epi_eval_t(const EpiParams& e, int m, int n, float acc0,
                                             float acc1, const float* bias0,
                                             const float* bias1, bool dual) {
  if constexpr (MODE == EPI_ACT_BWD) {
    const float z = e.Z[static_cast<int64_t>(m) * e.ldz + n];
    const float zd = dual ? e.Zd[static_cast<int64_t>(m) * e.ldz + n] : 0.f;
    return epi_core_t<MODE, ACT>(acc0, acc1, z, zd, 0.f, 0.f, dual);
  } else {
    return epi_core_t<MODE, ACT>(acc0, acc1, 0.f, 0.f, bias0 ? bias0[n] : 0.f,
                                 bias1 ? bias1[n] : 0.f, dual);
  }
}

}  // namespace mf
