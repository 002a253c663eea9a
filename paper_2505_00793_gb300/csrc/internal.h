// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace mf {

// Device status word values (also the mf_status codes they map to).
enum : int { DEV_OK = 0, DEV_NONFINITE = 5, DEV_TIMEOUT = 6 };

// GEMM product terms (same bit meaning as mf_dual_gemm_bf16's `terms`).
enum : unsigned {
  T_C0_A0B0 = 1u, T_C0_A1B0 = 2u, T_C0_A0B1 = 4u, T_C1_A1B0 = 8u, T_C1_A0B1 = 16u
};

inline int term_count(unsigned t) { return __builtin_popcount(t & 31u); }

// C[m][n] (+)= sum over selected terms of X[m][k] * Y[n][k]   (both operands K-major).
struct GemmArgs {
  int M = 0, N = 0, K = 0;
  const void* A0 = nullptr; int lda0 = 0;
  const void* A1 = nullptr; int lda1 = 0;
  const void* B0 = nullptr; int ldb0 = 0;
  const void* B1 = nullptr; int ldb1 = 0;
  float* C0 = nullptr; int ldc0 = 0; const float* bias0 = nullptr;
  float* C1 = nullptr; int ldc1 = 0; const float* bias1 = nullptr;
  unsigned terms = 0;
  int* status = nullptr;   // device status word (timeouts), may be null
};

// tcgen05 bf16 GEMM (tc_gemm.cu).  Returns cudaSuccess or the launch error; sets *why on a
// host-side rejection (bad alignment/ld) and returns cudaErrorInvalidValue.
cudaError_t tc_gemm(const GemmArgs& a, cudaStream_t s, const char** why);
// SIMT float32 GEMM with the same semantics (simt_gemm.cu).
cudaError_t simt_gemm(const GemmArgs& a, cudaStream_t s);

// ---- elementwise / row kernels (kernels.cu); T is float or __nv_bfloat16 -------------
enum Act : int { ACT_IDENT = 0, ACT_TANH = 1, ACT_GELU = 2, ACT_SILU = 3 };

// W [rows][cols] float32 (ld = cols) -> Wo [rows][ldo] (T), WoT [cols][ldoT] (T).
template <typename T>
void cast_transpose(const float* W, int rows, int cols, T* Wo, int ldo, T* WoT, int ldoT,
                    cudaStream_t s);
// X [rows][ld] (T) -> XT [cols][ldT] (T)
template <typename T>
void transpose(const T* X, int rows, int cols, int ld, T* XT, int ldT, cudaStream_t s);

// Dual activation forward: a = phi(z), a_dot = phi'(z) z_dot (when Zd != null).
template <typename T>
void act_fwd(int act, const float* Z, const float* Zd, int rows, int cols, T* A, T* Ad,
             int ld, T* AT, T* AdT, int ldT, cudaStream_t s);
// Dual activation backward: dz = phi'(z) da ; dz_dot = phi''(z) z_dot da + phi'(z) da_dot.
// Writes T copies (normal + transposed) and float32 copies (for bias reductions).
template <typename T>
void act_bwd(int act, const float* Z, const float* Zd, const float* dA, const float* dAd,
             int rows, int cols, T* dZ, T* dZd, int ld, T* dZT, T* dZdT, int ldT,
             float* dZ32, float* dZd32, cudaStream_t s);

struct LossArgs {
  int loss = 0;            // 0 squared, 1 softmax CE
  int rows = 0, cols = 0;
  const float* F = nullptr;  const float* Fd = nullptr;  // logits [rows][cols], tangent
  const float* Yf = nullptr; const int* Yi = nullptr;    // targets
  const float* eta_w = nullptr;   // example weight logits [rows] (weights = sigmoid), or
  const float* ex_w = nullptr;    // explicit weights [rows]; both null = 1
  float inv_norm = 1.f;    // 1/B
  float* l = nullptr;      // per-example loss [rows] (nullable)
  float* ld = nullptr;     // per-example tangent loss [rows] (nullable)
  float* d_eta = nullptr;  // += sigmoid'(eta_w) * ld * inv_norm  [rows] (nullable)
  float* dF32 = nullptr; float* dFd32 = nullptr;   // seeds float32 [rows][cols]
  void* dF = nullptr; void* dFd = nullptr; int ldo = 0; // seeds in T [rows][ldo]
  int* status = nullptr;
};
template <typename T>
void loss_seed(const LossArgs& a, cudaStream_t s);

// out[n] = sum_{r<rows} X[r][n]  (deterministic, float32)
void colsum(const float* X, int rows, int cols, float* out, cudaStream_t s);
// out[0] = scale * sum_i x[i] (deterministic, one block)
void sum_scaled(const float* x, int n, float scale, float* out, cudaStream_t s);

struct LrArgs {
  float alpha = 0.f;
  const float* plr = nullptr;   // per-parameter log-lr [P]
  const float* slr = nullptr;   // scalar log-lr [1]
};

// Rollout update (K4):  m' = mu m + g ;  theta' = theta - lr m'   (m may be null = 0)
void rollout_update(int64_t P, const float* theta, const float* m, const float* g, float mu,
                    LrArgs lr, float* theta_out, float* m_out, int* status, cudaStream_t s);

// Adjoint update (K5):  theta_bar += Hu (Hu nullable);
//   if m != null: d_plr += -lr m theta_bar  (per parameter)  or partial[blk] = sum(-lr m theta_bar)
//   u = mu u - lr theta_bar   (u_in nullable = 0)
void adjoint_update(int64_t P, float* theta_bar, const float* Hu, const float* m,
                    const float* u_in, float* u_out, float mu, LrArgs lr, float* d_plr,
                    float* partials, int n_partials, int* status, cudaStream_t s);
int adjoint_partials_blocks(int64_t P);

void fill(float* p, int64_t n, float v, cudaStream_t s);
void copy_f32(float* dst, const float* src, int64_t n, cudaStream_t s);

}  // namespace mf
