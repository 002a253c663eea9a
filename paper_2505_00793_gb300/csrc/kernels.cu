// Elementwise, row and update kernels of the mixed-mode sweep (HBM-bound work).
//
//  * dual activation forward / backward (the tangent rules of a = phi(z) and of its VJP),
//    writing both the row-major operand and its transpose for the next tensor-core GEMM;
//  * per-example loss seeds with the tangent per-example loss (the mixed term of Eq. 7 for
//    per-example weights) and d eta_{t,b} = sigmoid'(eta_{t,b}) * l'_b / B;
//  * the inner-step update (Eq. 2) and the adjoint update of the reverse sweep (Eq. 5 with
//    the Hessian product supplied by the forward-over-reverse pass).
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace mf {
namespace {

template <typename T> __device__ __forceinline__ T to_t(float x);
template <> __device__ __forceinline__ float to_t<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 to_t<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// phi, phi', phi'' of the hidden activations.
__device__ __forceinline__ void act_eval(int act, float z, float& f, float& d1, float& d2) {
  switch (act) {
    case ACT_TANH: {
      const float t = tanhf(z);
      f = t; d1 = 1.f - t * t; d2 = -2.f * t * d1;
      break;
    }
    case ACT_GELU: {   // x * Phi(x): phi' = Phi + x pdf, phi'' = pdf (2 - x^2)
      const float cdf = 0.5f * (1.f + erff(z * 0.70710678118654752f));
      const float pdf = 0.39894228040143268f * expf(-0.5f * z * z);
      f = z * cdf; d1 = cdf + z * pdf; d2 = pdf * (2.f - z * z);
      break;
    }
    case ACT_SILU: {   // x * s(x): phi' = s (1 + x (1 - s)), phi'' = s (1 - s) (2 + x (1 - 2 s))
      const float sg = 1.f / (1.f + expf(-z));
      f = z * sg; d1 = sg * (1.f + z * (1.f - sg));
      d2 = sg * (1.f - sg) * (2.f + z * (1.f - 2.f * sg));
      break;
    }
    default:
      f = z; d1 = 1.f; d2 = 0.f;
  }
}

constexpr int TILE = 32, TROWS = 8;

template <typename T>
__global__ void cast_transpose_kernel(const float* __restrict__ W, int rows, int cols,
                                      T* __restrict__ Wo, int ldo, T* __restrict__ WoT, int ldoT) {
  __shared__ float tile[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float v = 0.f;
    if (r < rows && c < cols) {
      v = W[static_cast<int64_t>(r) * cols + c];
      if (Wo) Wo[static_cast<int64_t>(r) * ldo + c] = to_t<T>(v);
    }
    tile[i][tx] = v;
  }
  if (!WoT) return;
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (c < cols && r < rows) WoT[static_cast<int64_t>(c) * ldoT + r] = to_t<T>(tile[tx][i]);
  }
}

template <typename T>
__global__ void transpose_kernel(const T* __restrict__ X, int rows, int cols, int ld,
                                 T* __restrict__ XT, int ldT) {
  __shared__ T tile[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    if (r < rows && c < cols) tile[i][tx] = X[static_cast<int64_t>(r) * ld + c];
  }
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (c < cols && r < rows) XT[static_cast<int64_t>(c) * ldT + r] = tile[tx][i];
  }
}

template <typename T>
__global__ void act_fwd_kernel(int act, const float* __restrict__ Z, const float* __restrict__ Zd,
                               int rows, int cols, T* __restrict__ A, T* __restrict__ Ad, int ld,
                               T* __restrict__ AT, T* __restrict__ AdT, int ldT) {
  __shared__ float ta[TILE][TILE + 1];
  __shared__ float tad[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const bool dual = Zd != nullptr;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float a = 0.f, ad = 0.f;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float d1, d2;
      act_eval(act, Z[o], a, d1, d2);
      A[static_cast<int64_t>(r) * ld + c] = to_t<T>(a);
      if (dual) {
        ad = d1 * Zd[o];
        Ad[static_cast<int64_t>(r) * ld + c] = to_t<T>(ad);
      }
    }
    ta[i][tx] = a;
    tad[i][tx] = ad;
  }
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (c < cols && r < rows) {
      const int64_t o = static_cast<int64_t>(c) * ldT + r;
      AT[o] = to_t<T>(ta[tx][i]);
      if (dual) AdT[o] = to_t<T>(tad[tx][i]);
    }
  }
}

template <typename T>
__global__ void act_bwd_kernel(int act, const float* __restrict__ Z, const float* __restrict__ Zd,
                               const float* __restrict__ dA, const float* __restrict__ dAd,
                               int rows, int cols, T* __restrict__ dZ, T* __restrict__ dZd, int ld,
                               T* __restrict__ dZT, T* __restrict__ dZdT, int ldT,
                               float* __restrict__ dZ32, float* __restrict__ dZd32) {
  __shared__ float t0[TILE][TILE + 1];
  __shared__ float t1[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const bool dual = dAd != nullptr;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float g = 0.f, gd = 0.f;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float f, d1, d2;
      act_eval(act, Z[o], f, d1, d2);
      const float da = dA[o];
      g = d1 * da;
      const int64_t on = static_cast<int64_t>(r) * ld + c;
      dZ[on] = to_t<T>(g);
      if (dZ32) dZ32[o] = g;
      if (dual) {
        gd = d2 * Zd[o] * da + d1 * dAd[o];
        dZd[on] = to_t<T>(gd);
        if (dZd32) dZd32[o] = gd;
      }
    }
    t0[i][tx] = g;
    t1[i][tx] = gd;
  }
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (c < cols && r < rows) {
      const int64_t o = static_cast<int64_t>(c) * ldT + r;
      dZT[o] = to_t<T>(t0[tx][i]);
      if (dual) dZdT[o] = to_t<T>(t1[tx][i]);
    }
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// One warp per example row.  Squared loss l = 1/2 mean_o (f - y)^2; softmax CE
// l = logsumexp(f) - f_y.  Seeds scaled by w_b / B.
template <typename T>
__global__ void loss_seed_kernel(const LossArgs a) {
  const int warps = blockDim.x >> 5;
  const int row = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= a.rows) return;
  const int C = a.cols;
  const float* f = a.F + static_cast<int64_t>(row) * C;
  const float* fd = a.Fd ? a.Fd + static_cast<int64_t>(row) * C : nullptr;
  float w = 1.f, sg = 0.f;
  if (a.ex_w) w = a.ex_w[row];
  else if (a.eta_w) { sg = 1.f / (1.f + expf(-a.eta_w[row])); w = sg; }
  const float scale = w * a.inv_norm;
  T* dF = static_cast<T*>(a.dF);
  T* dFd = static_cast<T*>(a.dFd);
  const int64_t orow = static_cast<int64_t>(row) * a.ldo;
  const int64_t frow = static_cast<int64_t>(row) * C;
  float l = 0.f, ld = 0.f;
  if (a.loss == 0) {
    const float* y = a.Yf + static_cast<int64_t>(row) * C;
    const float invC = 1.f / static_cast<float>(C);
    float s2 = 0.f, s1 = 0.f;
    for (int c = lane; c < C; c += 32) {
      const float r = f[c] - y[c];
      s2 += r * r;
      if (fd) s1 += r * fd[c];
      const float g = scale * r * invC;
      if (dF) dF[orow + c] = to_t<T>(g);
      if (a.dF32) a.dF32[frow + c] = g;
      if (fd) {
        const float gd = scale * fd[c] * invC;
        if (dFd) dFd[orow + c] = to_t<T>(gd);
        if (a.dFd32) a.dFd32[frow + c] = gd;
      }
    }
    l = 0.5f * warp_sum(s2) * invC;
    ld = warp_sum(s1) * invC;
  } else {
    const int y = a.Yi[row];
    if (y < 0 || y >= C) {
      if (lane == 0 && a.status) atomicExch(a.status, 1);
      return;
    }
    float mx = -INFINITY;
    for (int c = lane; c < C; c += 32) mx = fmaxf(mx, f[c]);
    mx = warp_max(mx);
    float se = 0.f;
    for (int c = lane; c < C; c += 32) se += expf(f[c] - mx);
    se = warp_sum(se);
    const float lse = mx + logf(se);
    float pf = 0.f;
    if (fd) {
      for (int c = lane; c < C; c += 32) pf += expf(f[c] - lse) * fd[c];
      pf = warp_sum(pf);
    }
    for (int c = lane; c < C; c += 32) {
      const float pc = expf(f[c] - lse);
      const float g = scale * (pc - (c == y ? 1.f : 0.f));
      if (dF) dF[orow + c] = to_t<T>(g);
      if (a.dF32) a.dF32[frow + c] = g;
      if (fd) {
        const float gd = scale * pc * (fd[c] - pf);
        if (dFd) dFd[orow + c] = to_t<T>(gd);
        if (a.dFd32) a.dFd32[frow + c] = gd;
      }
    }
    l = lse - f[y];
    if (fd) ld = pf - fd[y];
  }
  if (lane == 0) {
    if (a.l) a.l[row] = l;
    if (a.ld) a.ld[row] = ld;
    if (a.d_eta && a.eta_w) a.d_eta[row] = sg * (1.f - sg) * ld * a.inv_norm;
  }
}

__global__ void colsum_kernel(const float* __restrict__ X, int rows, int cols,
                              float* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float s = 0.f;
  for (int r = 0; r < rows; ++r) s += X[static_cast<int64_t>(r) * cols + c];
  out[c] = s;
}

__global__ void sum_scaled_kernel(const float* __restrict__ x, int n, float scale,
                                  float* __restrict__ out) {
  __shared__ float red[32];
  float s = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += x[i];
  s = warp_sum(s);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    v = warp_sum(v);
    if (threadIdx.x == 0) out[0] = v * scale;
  }
}

__device__ __forceinline__ float lr_at(const LrArgs& lr, int64_t i) {
  if (lr.plr) return expf(lr.plr[i]);
  if (lr.slr) return expf(lr.slr[0]);
  return lr.alpha;
}

__global__ void rollout_update_kernel(int64_t P, const float* __restrict__ theta,
                                      const float* __restrict__ m, const float* __restrict__ g,
                                      float mu, LrArgs lr, float* __restrict__ theta_out,
                                      float* __restrict__ m_out, int* status) {
  bool bad = false;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < P;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float mn = (m ? mu * m[i] : 0.f) + g[i];
    const float tn = theta[i] - lr_at(lr, i) * mn;
    if (m_out) m_out[i] = mn;
    theta_out[i] = tn;
    bad |= !isfinite(tn);
  }
  if (bad && status) atomicExch(status, DEV_NONFINITE);
}

__global__ void adjoint_update_kernel(int64_t P, float* __restrict__ theta_bar,
                                      const float* __restrict__ Hu, const float* __restrict__ m,
                                      const float* __restrict__ u_in, float* __restrict__ u_out,
                                      float mu, LrArgs lr, float* __restrict__ d_plr,
                                      float* __restrict__ partials, int* status) {
  __shared__ float red[32];
  bool bad = false;
  float acc = 0.f;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < P;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float tb = theta_bar[i] + (Hu ? Hu[i] : 0.f);
    theta_bar[i] = tb;
    bad |= !isfinite(tb);
    const float r = lr_at(lr, i);
    if (m) {
      const float contrib = -r * m[i] * tb;
      if (d_plr) d_plr[i] += contrib;
      else acc += contrib;
    }
    if (u_out) u_out[i] = (u_in ? mu * u_in[i] : 0.f) - r * tb;
  }
  if (bad && status) atomicExch(status, DEV_NONFINITE);
  if (partials) {
    acc = warp_sum(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x < 32) {
      float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
      v = warp_sum(v);
      if (threadIdx.x == 0) partials[blockIdx.x] = v;
    }
  }
}

__global__ void fill_kernel(float* p, int64_t n, float v) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    p[i] = v;
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  const int64_t cap = 152 * 16;
  if (b > cap) b = cap;
  if (b < 1) b = 1;
  return static_cast<int>(b);
}

}  // namespace

template <typename T>
void cast_transpose(const float* W, int rows, int cols, T* Wo, int ldo, T* WoT, int ldoT,
                    cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  cast_transpose_kernel<T><<<grid, dim3(TILE, TROWS), 0, s>>>(W, rows, cols, Wo, ldo, WoT, ldoT);
}

template <typename T>
void transpose(const T* X, int rows, int cols, int ld, T* XT, int ldT, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  transpose_kernel<T><<<grid, dim3(TILE, TROWS), 0, s>>>(X, rows, cols, ld, XT, ldT);
}

template <typename T>
void act_fwd(int act, const float* Z, const float* Zd, int rows, int cols, T* A, T* Ad, int ld,
             T* AT, T* AdT, int ldT, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  act_fwd_kernel<T><<<grid, dim3(TILE, TROWS), 0, s>>>(act, Z, Zd, rows, cols, A, Ad, ld, AT,
                                                        AdT, ldT);
}

template <typename T>
void act_bwd(int act, const float* Z, const float* Zd, const float* dA, const float* dAd,
             int rows, int cols, T* dZ, T* dZd, int ld, T* dZT, T* dZdT, int ldT, float* dZ32,
             float* dZd32, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  act_bwd_kernel<T><<<grid, dim3(TILE, TROWS), 0, s>>>(act, Z, Zd, dA, dAd, rows, cols, dZ, dZd,
                                                        ld, dZT, dZdT, ldT, dZ32, dZd32);
}

template <typename T>
void loss_seed(const LossArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return;
  const int warps = 8;
  loss_seed_kernel<T><<<(a.rows + warps - 1) / warps, warps * 32, 0, s>>>(a);
}

void colsum(const float* X, int rows, int cols, float* out, cudaStream_t s) {
  if (cols <= 0) return;
  colsum_kernel<<<(cols + 255) / 256, 256, 0, s>>>(X, rows, cols, out);
}

void sum_scaled(const float* x, int n, float scale, float* out, cudaStream_t s) {
  sum_scaled_kernel<<<1, 1024, 0, s>>>(x, n, scale, out);
}

void rollout_update(int64_t P, const float* theta, const float* m, const float* g, float mu,
                    LrArgs lr, float* theta_out, float* m_out, int* status, cudaStream_t s) {
  rollout_update_kernel<<<grid_for(P, 256), 256, 0, s>>>(P, theta, m, g, mu, lr, theta_out, m_out,
                                                         status);
}

int adjoint_partials_blocks(int64_t P) { return grid_for(P, 256); }

void adjoint_update(int64_t P, float* theta_bar, const float* Hu, const float* m,
                    const float* u_in, float* u_out, float mu, LrArgs lr, float* d_plr,
                    float* partials, int n_partials, int* status, cudaStream_t s) {
  const int g = grid_for(P, 256);
  (void)n_partials;
  adjoint_update_kernel<<<g, 256, 0, s>>>(P, theta_bar, Hu, m, u_in, u_out, mu, lr, d_plr,
                                          partials, status);
}

void fill(float* p, int64_t n, float v, cudaStream_t s) {
  if (n <= 0) return;
  fill_kernel<<<grid_for(n, 256), 256, 0, s>>>(p, n, v);
}

void copy_f32(float* dst, const float* src, int64_t n, cudaStream_t s) {
  if (n > 0) cudaMemcpyAsync(dst, src, n * sizeof(float), cudaMemcpyDeviceToDevice, s);
}

#define MF_INST(T)                                                                           \
  template void cast_transpose<T>(const float*, int, int, T*, int, T*, int, cudaStream_t);  \
  template void transpose<T>(const T*, int, int, int, T*, int, cudaStream_t);               \
  template void act_fwd<T>(int, const float*, const float*, int, int, T*, T*, int, T*, T*,  \
                           int, cudaStream_t);                                              \
  template void act_bwd<T>(int, const float*, const float*, const float*, const float*, int, \
                           int, T*, T*, int, T*, T*, int, float*, float*, cudaStream_t);     \
  template void loss_seed<T>(const LossArgs&, cudaStream_t);
MF_INST(float)
MF_INST(__nv_bfloat16)
#undef MF_INST

}  // namespace mf
