// Float32 dual GEMM on the CUDA cores, for the float32-precision path (small models whose
// meta-gradient is checked at 1e-4 relative error, below what bf16/tf32 operands allow).
// Same term semantics and fused epilogues as the tensor-core kernel: C_j = sum of selected
// X Y^T products (both operands K-major), then the per-element epilogue of device_math.cuh.
// 64x64 output tile per block, 256 threads, 4x4 outputs per thread and accumulator.
#include <cuda_runtime.h>
#include <stdint.h>

#include "device_math.cuh"
#include "internal.h"
#include "launch.cuh"

namespace mf {
namespace {

constexpr int TM = 64, TN = 64, TK = 16;

struct SimtParams {
  int M, N, K;
  unsigned terms;
  const float* A[2]; int lda[2];
  const float* B[2]; int ldb[2];
  int a_mn, b_mn;                  // MN-major operands: X[row][k] at k * ld + row
  float* C[2]; int ldc[2]; const float* bias[2];
  EpiParams epi;
  int64_t bsA[2], bsB[2], bsC[2];   // batch strides (blockIdx.z = batch index)
};

__global__ void __launch_bounds__(256) simt_dual_gemm_kernel(SimtParams p) {
  pdl_entry();
  const int64_t bz = blockIdx.z;
  for (int i = 0; i < 2; ++i) {
    if (p.A[i]) p.A[i] += bz * p.bsA[i];
    if (p.B[i]) p.B[i] += bz * p.bsB[i];
    if (p.C[i]) p.C[i] += bz * p.bsC[i];
  }
  __shared__ float As[TK][TM + 1];
  __shared__ float Bs[TK][TN + 1];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  const int tacc[6] = {0, 0, 0, 1, 1, 0};
  const int ta[6] = {0, 1, 0, 1, 0, 1};
  const int tb[6] = {0, 0, 1, 0, 1, 1};
  float c[2][4][4] = {};
  for (int t = 0; t < 6; ++t) {
    if (!(p.terms & (1u << t))) continue;
    const int acc = tacc[t];
    const float* A = p.A[ta[t]];
    const float* B = p.B[tb[t]];
    const int lda = p.lda[ta[t]], ldb = p.ldb[tb[t]];
    for (int k0 = 0; k0 < p.K; k0 += TK) {
      for (int i = threadIdx.x; i < TM * TK; i += 256) {
        const int r = i / TK, kk = i % TK;
        const int gm = m0 + r, gk = k0 + kk;
        As[kk][r] = (gm < p.M && gk < p.K)
                        ? A[p.a_mn ? static_cast<int64_t>(gk) * lda + gm : static_cast<int64_t>(gm) * lda + gk]
                        : 0.f;
        const int gn = n0 + r;
        Bs[kk][r] = (gn < p.N && gk < p.K)
                        ? B[p.b_mn ? static_cast<int64_t>(gk) * ldb + gn : static_cast<int64_t>(gn) * ldb + gk]
                        : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < TK; ++kk) {
        float a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
        for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
        if (acc == 0) {
#pragma unroll
          for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) c[0][i][j] = fmaf(a[i], b[j], c[0][i][j]);
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) c[1][i][j] = fmaf(a[i], b[j], c[1][i][j]);
        }
      }
      __syncthreads();
    }
  }
  const bool dual = (p.terms & (T_C1_A1B0 | T_C1_A0B1)) != 0;
  const EpiParams& e = p.epi;
  float* A = static_cast<float*>(e.A);
  float* Ad = static_cast<float*>(e.Ad);
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= p.M) continue;
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx * 4 + j;
      if (gn >= p.N) continue;
      const EpiOut o = epi_eval(e, gm, gn, c[0][i][j], c[1][i][j], p.bias[0], p.bias[1], dual);
      if (p.C[0]) p.C[0][static_cast<int64_t>(gm) * p.ldc[0] + gn] = o.c0;
      if (p.C[1] && dual) p.C[1][static_cast<int64_t>(gm) * p.ldc[1] + gn] = o.c1;
      if (e.mode != EPI_STORE) {
        if (A) A[static_cast<int64_t>(gm) * e.lda + gn] = o.o0;
        if (dual && Ad) Ad[static_cast<int64_t>(gm) * e.lda + gn] = o.o1;
      }
    }
  }
}

}  // namespace

cudaError_t simt_gemm(const GemmArgs& a, cudaStream_t s) {
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  SimtParams p;
  p.M = a.M; p.N = a.N; p.K = a.K; p.terms = a.terms;
  p.A[0] = static_cast<const float*>(a.A0); p.lda[0] = a.lda0;
  p.A[1] = static_cast<const float*>(a.A1); p.lda[1] = a.lda1;
  p.B[0] = static_cast<const float*>(a.B0); p.ldb[0] = a.ldb0;
  p.B[1] = static_cast<const float*>(a.B1); p.ldb[1] = a.ldb1;
  p.C[0] = a.C0; p.ldc[0] = a.ldc0; p.bias[0] = a.bias0;
  p.C[1] = a.C1; p.ldc[1] = a.ldc1; p.bias[1] = a.bias1;
  p.epi = a.epi;
  p.a_mn = a.a_mn ? 1 : 0;
  p.b_mn = a.b_mn ? 1 : 0;
  p.bsA[0] = a.bsA0; p.bsA[1] = a.bsA1; p.bsB[0] = a.bsB0; p.bsB[1] = a.bsB1;
  p.bsC[0] = a.bsC0; p.bsC[1] = a.bsC1;
  if (a.batch > 1 && a.epi.mode != EPI_STORE) return cudaErrorInvalidValue;
  dim3 grid((a.N + TN - 1) / TN, (a.M + TM - 1) / TM, a.batch < 1 ? 1 : a.batch);
  launch_k(simt_dual_gemm_kernel, dim3(grid), dim3(256), 0, s, p);
  return cudaGetLastError();
}

}  // namespace mf
