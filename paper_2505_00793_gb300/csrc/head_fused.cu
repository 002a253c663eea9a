// Fused narrow head of an MLP (opt-in: MF_OPT_FUSED_HEAD).
//
// For an output layer with at most 16 units (the 10-class head of the wide workload, the
// scalar head of the toy regression) the three steps around the loss are tiny: the head's
// dual forward product (K = the hidden width, N <= 16), the per-example loss with its
// seeds and mixed term (the Eq. 7 tangent per-example loss), and the head's dual data
// product (K <= 16) with the activation backward of the layer below.  As separate launches
// each costs a kernel's latency on the sweep's critical path.  Here one block per example
// row does all three:
//   1. z = a W + b and, dual, z' = a' W + a U + u_b (a' W only above the input layer), with
//      float32 accumulation of the operand copies (T), reduced across the block in a fixed
//      order;
//   2. the loss of the row (squared: 1/2 mean (z - y)^2; softmax CE), its seeds
//      w/B dl/dz and, dual, w/B (d2l/dz2) z', the per-example loss l, the tangent loss
//      l' = dl/dz . z' and d eta = sigmoid'(eta) l' / B, as the separate loss kernel
//      computes them; the seeds are stored in T (the head's weight product reads them);
//   3. da = dz W^T and, dual, da' = dz' W^T + dz U^T from the T-rounded seeds, then the
//      activation backward of the layer below (dz_prev = phi'(z) da,
//      dz'_prev = phi''(z) z' da + phi'(z) da') through the same element rule as the GEMM
//      epilogue, stored in T.
// The head's weight product stays a GEMM (it reduces over the batch).
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "device_math.cuh"
#include "internal.h"
#include "launch.cuh"

namespace mf {
namespace {

constexpr int HEAD_THREADS = 256;
constexpr int HEAD_WARPS = HEAD_THREADS / 32;

__device__ __forceinline__ float hsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float hmax(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

// LOSS: 0 squared, 1 softmax CE.  DUAL: tangent pass along u.
template <typename T, int ACT, bool DUAL, int LOSS>
__global__ void __launch_bounds__(HEAD_THREADS) head_fused_kernel(const HeadArgs a) {
  pdl_entry();
  __shared__ float red[HEAD_WARPS][2 * kHeadMaxOut];
  __shared__ float seed[2][kHeadMaxOut];
  __shared__ int skip;
  const int row = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int C = a.C, D = a.D;
  const T* A = static_cast<const T*>(a.A) + static_cast<int64_t>(row) * a.lda;
  const T* Ad = a.Ad ? static_cast<const T*>(a.Ad) + static_cast<int64_t>(row) * a.lda : nullptr;
  const T* W = static_cast<const T*>(a.W);
  const T* U = static_cast<const T*>(a.U);

  // ---- 1. head forward: per-thread partial dot products over k = tid, tid + 256, ... -----
  float z[kHeadMaxOut], zd[kHeadMaxOut];
#pragma unroll
  for (int j = 0; j < kHeadMaxOut; ++j) z[j] = zd[j] = 0.f;
  for (int k = tid; k < D; k += HEAD_THREADS) {
    const float ak = to_f<T>(A[k]);
    const float adk = (DUAL && Ad) ? to_f<T>(Ad[k]) : 0.f;
    const T* w = W + static_cast<int64_t>(k) * a.ldw;
    const T* u = U + static_cast<int64_t>(k) * a.ldw;
#pragma unroll
    for (int j = 0; j < kHeadMaxOut; ++j) {
      if (j < C) {
        const float wj = to_f<T>(w[j]);
        z[j] = fmaf(ak, wj, z[j]);
        if (DUAL) zd[j] = fmaf(adk, wj, fmaf(ak, to_f<T>(u[j]), zd[j]));
      }
    }
  }
#pragma unroll
  for (int j = 0; j < kHeadMaxOut; ++j) {
    if (j < C) {
      const float s0 = hsum(z[j]);
      const float s1 = DUAL ? hsum(zd[j]) : 0.f;
      if (lane == 0) { red[wid][j] = s0; red[wid][kHeadMaxOut + j] = s1; }
    }
  }
  if (tid == 0) skip = 0;
  __syncthreads();

  // ---- 2. loss, seeds and mixed term of the row (warp 0, lane c holds output c) ----------
  if (wid == 0) {
    const LossArgs& L = a.loss;
    const bool on = lane < C;
    float f = 0.f, fd = 0.f;
    if (on) {
      for (int w = 0; w < HEAD_WARPS; ++w) {
        f += red[w][lane];
        if (DUAL) fd += red[w][kHeadMaxOut + lane];
      }
      if (a.bias) f += a.bias[lane];
      if (DUAL && a.ubias) fd += a.ubias[lane];
    }
    float wgt = 1.f, sg = 0.f;
    if (L.ex_w) wgt = L.ex_w[row];
    else if (L.eta_w) { sg = 1.f / (1.f + expf(-L.eta_w[row])); wgt = sg; }
    const float scale = wgt * L.inv_norm;
    T* dF = static_cast<T*>(L.dF);
    T* dFd = static_cast<T*>(L.dFd);
    const int64_t orow = static_cast<int64_t>(row) * L.ldo;
    float l = 0.f, ld = 0.f, s0 = 0.f, s1 = 0.f;
    bool bad = false;
    if (LOSS == 0) {
      const float invC = 1.f / static_cast<float>(C);
      const float r = on ? f - L.Yf[static_cast<int64_t>(row) * C + lane] : 0.f;
      l = 0.5f * hsum(r * r) * invC;
      ld = DUAL ? hsum(r * fd) * invC : 0.f;
      s0 = scale * r * invC;
      s1 = DUAL ? scale * fd * invC : 0.f;
    } else {
      const int y = L.Yi[row];
      if (y < 0 || y >= C) {
        bad = true;
      } else {
        const float mx = hmax(on ? f : -INFINITY);
        const float se = hsum(on ? expf(f - mx) : 0.f);
        const float lse = mx + logf(se);
        const float pc = on ? expf(f - lse) : 0.f;
        const float pf = DUAL ? hsum(pc * fd) : 0.f;
        const float fy = __shfl_sync(0xffffffffu, f, y);
        const float fdy = __shfl_sync(0xffffffffu, fd, y);
        l = lse - fy;
        ld = DUAL ? pf - fdy : 0.f;
        s0 = scale * (pc - (lane == y ? 1.f : 0.f));
        s1 = DUAL ? scale * pc * (fd - pf) : 0.f;
      }
    }
    if (bad) {
      if (lane == 0) {
        skip = 1;
        if (L.status) atomicMax(L.status, 1);
      }
    } else {
      if (on) {
        const T t0 = to_t<T>(s0);
        if (dF) dF[orow + lane] = t0;
        seed[0][lane] = to_f<T>(t0);
        if (DUAL) {
          const T t1 = to_t<T>(s1);
          if (dFd) dFd[orow + lane] = t1;
          seed[1][lane] = to_f<T>(t1);
        }
      }
      if (lane == 0) {
        if (L.l) L.l[row] = l;
        if (L.ld) L.ld[row] = ld;
        if (L.d_eta && L.eta_w) L.d_eta[row] = sg * (1.f - sg) * ld * L.inv_norm;
      }
    }
  }
  __syncthreads();
  if (skip || !a.dz_prev) return;

  // ---- 3. head data product and the activation backward of the layer below ------------
  EpiParams e;
  e.mode = EPI_ACT_BWD;
  e.act = ACT;
  e.Z = a.Z; e.Zd = a.Zd; e.ldz = a.ldz;
  T* dzp = static_cast<T*>(a.dz_prev) + static_cast<int64_t>(row) * a.ld_prev;
  T* dzdp = DUAL ? static_cast<T*>(a.dzd_prev) + static_cast<int64_t>(row) * a.ld_prev : nullptr;
  for (int k = tid; k < D; k += HEAD_THREADS) {
    const T* w = W + static_cast<int64_t>(k) * a.ldw;
    const T* u = U + static_cast<int64_t>(k) * a.ldw;
    float da = 0.f, dad = 0.f;
#pragma unroll
    for (int j = 0; j < kHeadMaxOut; ++j) {
      if (j < C) {
        const float wj = to_f<T>(w[j]);
        da = fmaf(seed[0][j], wj, da);
        if (DUAL) dad = fmaf(seed[1][j], wj, fmaf(seed[0][j], to_f<T>(u[j]), dad));
      }
    }
    const EpiOut o = epi_eval_t<EPI_ACT_BWD, ACT>(e, row, k, da, dad, nullptr, nullptr, DUAL);
    dzp[k] = to_t<T>(o.o0);
    if (DUAL) dzdp[k] = to_t<T>(o.o1);
  }
}

template <typename T, int ACT>
cudaError_t launch_act(const HeadArgs& a, cudaStream_t s) {
  const dim3 grid(a.rows), block(HEAD_THREADS);
  const int lk = a.loss.loss;
  if (a.dual) {
    if (lk == 0) return launch_k(head_fused_kernel<T, ACT, true, 0>, grid, block, 0, s, a);
    return launch_k(head_fused_kernel<T, ACT, true, 1>, grid, block, 0, s, a);
  }
  if (lk == 0) return launch_k(head_fused_kernel<T, ACT, false, 0>, grid, block, 0, s, a);
  return launch_k(head_fused_kernel<T, ACT, false, 1>, grid, block, 0, s, a);
}

}  // namespace

int g_fused_head = 0;

template <typename T>
cudaError_t head_fused(const HeadArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  if (a.C < 1 || a.C > kHeadMaxOut || a.D < 1 || (a.loss.loss != 0 && a.loss.loss != 1) ||
      (a.loss.loss == 0 && !a.loss.Yf) || (a.loss.loss == 1 && !a.loss.Yi))
    return cudaErrorInvalidValue;
  switch (a.act) {
    case ACT_IDENT: return launch_act<T, ACT_IDENT>(a, s);
    case ACT_TANH: return launch_act<T, ACT_TANH>(a, s);
    case ACT_GELU: return launch_act<T, ACT_GELU>(a, s);
    case ACT_SILU: return launch_act<T, ACT_SILU>(a, s);
  }
  return cudaErrorInvalidValue;
}

template cudaError_t head_fused<float>(const HeadArgs&, cudaStream_t);
template cudaError_t head_fused<__nv_bfloat16>(const HeadArgs&, cudaStream_t);

}  // namespace mf
