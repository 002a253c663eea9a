// Elementwise, row and update kernels of the mixed-mode sweep (HBM-bound work).
//
//  * per-example loss seeds with the tangent per-example loss (the mixed term of Eq. 7 for
//    per-example weights) and d eta_{t,b} = sigmoid'(eta_{t,b}) * l'_b / B;
//  * the fused per-layer update kernel: the inner-step update of Eq. 2 (rollout) or the
//    adjoint update of the reverse sweep (Eq. 5 with the Hessian product supplied by the
//    forward-over-reverse pass), each fused with the cast of the next step's parameters /
//    tangent into the row-major and transposed GEMM operand copies;
//  * transposes, row fills and a deterministic sum.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "device_math.cuh"
#include "internal.h"
#include "launch.cuh"

namespace mf {

int g_pdl = 1;
namespace {

constexpr int TILE = 32, TROWS = 8;

template <typename T>
__global__ void transpose_kernel(const T* __restrict__ X, int rows, int cols, int ld,
                                 T* __restrict__ XT, int ldT) {
  pdl_entry();
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
__global__ void fill_rows_kernel(const RowFill f, int cols) {
  pdl_entry();
  const int k = blockIdx.y;
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= f.n || c >= cols) return;
  T* dst = static_cast<T*>(f.dst[k]);
  dst[static_cast<int64_t>(f.row[k]) * f.ld[k] + c] = to_t<T>(f.value[k]);
}

template <typename T>
__global__ void fill_cols_kernel(const ColFill f, int rows) {
  pdl_entry();
  const int n = blockIdx.y;
  T* dst = static_cast<T*>(f.dst[n]);
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += gridDim.x * blockDim.x)
    dst[static_cast<int64_t>(r) * f.ld[n] + f.col[n]] = to_t<T>(f.value[n]);
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
  pdl_entry();
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
  float l = 0.f, ld = 0.f;
  if (a.loss == 0) {
    const float* y = a.Yf + static_cast<int64_t>(row) * C;
    const float invC = 1.f / static_cast<float>(C);
    float s2 = 0.f, s1 = 0.f;
    for (int c = lane; c < C; c += 32) {
      const float r = f[c] - y[c];
      s2 += r * r;
      if (fd) s1 += r * fd[c];
      if (dF) dF[orow + c] = to_t<T>(scale * r * invC);
      if (fd && dFd) dFd[orow + c] = to_t<T>(scale * fd[c] * invC);
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
      if (dF) dF[orow + c] = to_t<T>(scale * (pc - (c == y ? 1.f : 0.f)));
      if (fd && dFd) dFd[orow + c] = to_t<T>(scale * pc * (fd[c] - pf));
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

// Motivating example of Section 3 (Eq. 8): the model output is f = x theta followed by the
// elementwise recursion y_0 = f, y_i = i (2 + sin y_{i-1})^cos y_{i-1}, i = 1..M, and
// l_b = mean_o (y_M - t)^2.  Per element the recursion is carried with its first and second
// derivatives in f (y', y''), so the loss seed 2/C r y' and its tangent 2/C (y'^2 + r y'') f'
// come out of one pass; nothing of the recursion is stored.  One block per example.
__device__ __forceinline__ void chain_eval(float f, int M, float& y, float& d1, float& d2) {
  y = f; d1 = 1.f; d2 = 0.f;
  for (int i = 1; i <= M; ++i) {
    float sn, cs;
    sincosf(y, &sn, &cs);
    const float b = 2.f + sn;                 // >= 1
    const float lb = logf(b);
    const float g1 = -sn * lb + cs * cs / b;  // d/dy [cos y log(2 + sin y)]
    const float g2 = -cs * lb - 3.f * sn * cs / b - cs * cs * cs / (b * b);
    const float yi = static_cast<float>(i) * expf(cs * lb);
    const float f1 = yi * g1, f2 = yi * (g1 * g1 + g2);
    d2 = f2 * d1 * d1 + f1 * d2;
    d1 = f1 * d1;
    y = yi;
  }
}

template <typename T>
__global__ void chain_loss_kernel(const LossArgs a) {
  pdl_entry();
  __shared__ float red[2][8];
  const int row = blockIdx.x;
  const int C = a.cols;
  const float* f = a.F + static_cast<int64_t>(row) * C;
  const float* fd = a.Fd ? a.Fd + static_cast<int64_t>(row) * C : nullptr;
  const float* t = a.Yf + static_cast<int64_t>(row) * C;
  float w = 1.f, sg = 0.f;
  if (a.ex_w) w = a.ex_w[row];
  else if (a.eta_w) { sg = 1.f / (1.f + expf(-a.eta_w[row])); w = sg; }
  const float invC = 1.f / static_cast<float>(C);
  const float scale = w * a.inv_norm;
  T* dF = static_cast<T*>(a.dF);
  T* dFd = static_cast<T*>(a.dFd);
  const int64_t orow = static_cast<int64_t>(row) * a.ldo;
  float s2 = 0.f, s1 = 0.f;
  bool bad = false;
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    float y, d1, d2;
    chain_eval(f[c], a.chain, y, d1, d2);
    const float r = y - t[c];
    bad |= !isfinite(y) || !isfinite(d1);
    s2 += r * r;
    if (dF) dF[orow + c] = to_t<T>(scale * 2.f * invC * r * d1);
    if (fd) {
      const float ad = d1 * fd[c];
      s1 += r * ad;
      if (dFd) dFd[orow + c] = to_t<T>(scale * 2.f * invC * (d1 * ad + r * d2 * fd[c]));
    }
  }
  if (bad && a.status) atomicExch(a.status, DEV_NONFINITE);
  s2 = warp_sum(s2);
  s1 = warp_sum(s1);
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { red[0][wid] = s2; red[1][wid] = s1; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f, ld = 0.f;
    for (int k = 0; k < static_cast<int>(blockDim.x >> 5); ++k) { l += red[0][k]; ld += red[1][k]; }
    l *= invC;
    ld *= 2.f * invC;
    if (a.l) a.l[row] = l;
    if (a.ld) a.ld[row] = ld;
    if (a.d_eta && a.eta_w) a.d_eta[row] = sg * (1.f - sg) * ld * a.inv_norm;
  }
}

// The same loss by reverse-over-reverse (Algorithm 1's schedule applied inside the chain).
// ror = 1, primal: forward y_i = phi_i(y_{i-1}) recording y_0..y_{M-1}, then the backward
// ybar_M = c r, ybar_{i-1} = ybar_i phi_i'(y_{i-1}) recording ybar_1..ybar_M, with
// c = 2 w / (B C) and phi_i' = y_i (d/dy)[cos y log(2 + sin y)]; dF = ybar_0.
// ror = 2, adjoint of that backward along a_0 = Fd (the incoming adjoint of ybar_0): forward
// a_i = a_{i-1} phi_i'(y_{i-1}) leaving yhat_{i-1} = a_{i-1} ybar_i phi_i''(y_{i-1}) in
// ybar_i's slot, then yhat_M = c a_M and back yhat_{i-1} += yhat_i phi_i'(y_{i-1});
// dFd = yhat_0, and ld = 2/C sum r a_M.  Both phases read the tape back instead of carrying
// derivatives, so the tape (2 M floats per element) is what this mode holds beyond the
// mixed mode.  Tape slot k of element e = row * C + c is at tape[k * rows * C + e].
__device__ __forceinline__ float chain_step(int i, float y, float& g1, float& g2) {
  float sn, cs;
  sincosf(y, &sn, &cs);
  const float b = 2.f + sn;
  const float lb = logf(b);
  g1 = -sn * lb + cs * cs / b;
  g2 = -cs * lb - 3.f * sn * cs / b - cs * cs * cs / (b * b);
  return static_cast<float>(i) * expf(cs * lb);
}

template <typename T>
__global__ void chain_ror_kernel(const LossArgs a) {
  pdl_entry();
  __shared__ float red[2][8];
  const int row = blockIdx.x;
  const int C = a.cols, M = a.chain;
  const int64_t E = static_cast<int64_t>(a.rows) * C;
  const float* f = a.F + static_cast<int64_t>(row) * C;
  const float* t = a.Yf + static_cast<int64_t>(row) * C;
  float w = 1.f, sg = 0.f;
  if (a.ex_w) w = a.ex_w[row];
  else if (a.eta_w) { sg = 1.f / (1.f + expf(-a.eta_w[row])); w = sg; }
  const float invC = 1.f / static_cast<float>(C);
  const float cw = w * a.inv_norm * 2.f * invC;
  const int64_t orow = static_cast<int64_t>(row) * a.ldo;
  float s2 = 0.f, s1 = 0.f;
  bool bad = false;
  float g1, g2;
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    float* tp = a.tape + static_cast<int64_t>(row) * C + c;   // slot k at tp[k * E]
    if (a.ror == 1) {
      float y = f[c];
      for (int i = 1; i <= M; ++i) {
        tp[(i - 1) * E] = y;
        y = chain_step(i, y, g1, g2);
      }
      const float yM = y;
      const float r = yM - t[c];
      s2 += r * r;
      float yb = cw * r;
      for (int i = M; i >= 1; --i) {
        tp[(M + i - 1) * E] = yb;
        const float yi = i == M ? yM : tp[i * E];
        chain_step(i, tp[(i - 1) * E], g1, g2);
        yb *= yi * g1;
      }
      bad |= !isfinite(yM) || !isfinite(yb);
      if (a.dF) static_cast<T*>(a.dF)[orow + c] = to_t<T>(yb);
    } else {
      float ad = a.Fd[static_cast<int64_t>(row) * C + c];
      const float yM = chain_step(M, tp[(M - 1) * E], g1, g2);
      for (int i = 1; i <= M; ++i) {
        const float yi = i == M ? yM : tp[i * E];
        chain_step(i, tp[(i - 1) * E], g1, g2);
        float* slot = tp + (M + i - 1) * E;
        *slot = ad * *slot * yi * (g1 * g1 + g2);
        ad *= yi * g1;
      }
      const float r = yM - t[c];
      s1 += r * ad;
      float yh = cw * ad;
      for (int i = M; i >= 1; --i) {
        const float yi = i == M ? yM : tp[i * E];
        chain_step(i, tp[(i - 1) * E], g1, g2);
        yh = tp[(M + i - 1) * E] + yh * yi * g1;
      }
      bad |= !isfinite(yh);
      if (a.dFd) static_cast<T*>(a.dFd)[orow + c] = to_t<T>(yh);
    }
  }
  if (bad && a.status) atomicExch(a.status, DEV_NONFINITE);
  s2 = warp_sum(s2);
  s1 = warp_sum(s1);
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { red[0][wid] = s2; red[1][wid] = s1; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f, ld = 0.f;
    for (int k = 0; k < static_cast<int>(blockDim.x >> 5); ++k) { l += red[0][k]; ld += red[1][k]; }
    if (a.ror == 1) {
      if (a.l) a.l[row] = l * invC;
    } else {
      ld *= 2.f * invC;
      if (a.ld) a.ld[row] = ld;
      if (a.d_eta && a.eta_w) a.d_eta[row] = sg * (1.f - sg) * ld * a.inv_norm;
    }
  }
}

__global__ void sum_scaled_kernel(const float* __restrict__ x, int n, float scale,
                                  float* __restrict__ out) {
  pdl_entry();
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

// One 32 x 32 tile of one layer's [rows][dout] slice of the flat parameter vector per block.
template <typename T>
__global__ void __launch_bounds__(TILE * TROWS) layer_update_kernel(const LayerTable tab,
                                                                    const LayerUpdArgs a) {
  pdl_entry();
  __shared__ float tw[TILE][TILE + 1];   // values cast into W / WT
  __shared__ float tu[TILE][TILE + 1];   // values cast into U / UT
  __shared__ float red[TILE * TROWS / 32];
  int l = 0;
  while (l + 1 < tab.n && static_cast<int>(blockIdx.x) >= tab.tile0[l + 1]) ++l;
  const int t = blockIdx.x - tab.tile0[l];
  const int dout = tab.dout[l], rows = tab.rows[l], din = tab.din[l];
  const int tiles_c = (dout + TILE - 1) / TILE;
  const int r0 = (t / tiles_c) * TILE, c0 = (t % tiles_c) * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const bool cast_w = (a.mode == LU_ROLLOUT) || (a.mode == LU_CAST && !a.cast_src_to_u) ||
                      (a.mode == LU_ADJOINT && a.cast_src);
  const bool cast_u = (a.mode == LU_CAST && a.cast_src_to_u) || (a.mode == LU_ADJOINT && a.u_out);
  bool bad = false;
  float acc = 0.f;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float vw = 0.f, vu = 0.f;
    if (r < rows && c < dout) {
      const int64_t k = tab.off[l] + static_cast<int64_t>(r) * dout + c;
      if (a.mode == LU_ROLLOUT && a.adam) {
        const float g = a.g[k];
        const float mn = (a.m ? a.b1 * a.m[k] : 0.f) + (1.f - a.b1) * g;
        const float vn = (a.v ? a.b2 * a.v[k] : 0.f) + (1.f - a.b2) * g * g;
        const float tn = a.theta[k] - lr_at(a.lr, k) * (mn / a.c1) / (sqrtf(vn / a.c2) + a.eps);
        a.theta_out[k] = tn;
        if (a.m_out) a.m_out[k] = mn;
        if (a.v_out) a.v_out[k] = vn;
        bad |= !isfinite(tn);
        vw = tn;
      } else if (a.mode == LU_ROLLOUT) {
        const float mn = (a.m ? a.mu * a.m[k] : 0.f) + a.g[k];
        const float tn = a.theta[k] - lr_at(a.lr, k) * mn;
        a.theta_out[k] = tn;
        if (a.m_out) a.m_out[k] = mn;
        bad |= !isfinite(tn);
        vw = tn;
      } else if (a.mode == LU_ADJOINT && a.adam) {
        const float tb = a.theta_bar[k] + (a.Hu ? a.Hu[k] : 0.f);
        a.theta_bar[k] = tb;
        bad |= !isfinite(tb);
        if (a.adam_pre) {
          // theta_{j+1} = theta_j - lr (m/c1) / (s + eps), s = sqrt(v/c2), m = m_{j+1}, v = v_{j+1}
          const float lr = lr_at(a.lr, k);
          const float m1 = a.m_adj[k], v1 = a.v_adj[k];
          const float s = sqrtf(v1 / a.c2);
          const float den = s + a.eps;
          const float q = -lr * tb;
          // cotangents of m_{j+1} and v_{j+1} (at v = 0, where m = g = 0, the sqrt term is 0)
          const float Mb = (a.bar_in ? a.mbar[k] : 0.f) + q / (a.c1 * den);
          const float Vb = (a.bar_in ? a.vbar[k] : 0.f) -
                           (s > 0.f ? q * m1 / (a.c1 * den * den * 2.f * s * a.c2) : 0.f);
          const float g = (m1 - (a.m_prev ? a.b1 * a.m_prev[k] : 0.f)) / (1.f - a.b1);
          vu = (1.f - a.b1) * Mb + 2.f * (1.f - a.b2) * g * Vb;
          a.u_out[k] = vu;
          a.mbar[k] = a.b1 * Mb;
          a.vbar[k] = a.b2 * Vb;
          const float contrib = -lr * (m1 / a.c1) / den * tb;
          if (a.d_plr) a.d_plr[k] += contrib;
          else acc += contrib;
          bad |= !isfinite(vu);
        }
        if (a.cast_src) vw = a.cast_src[k];
      } else if (a.mode == LU_ADJOINT) {
        const float tb = a.theta_bar[k] + (a.Hu ? a.Hu[k] : 0.f);
        a.theta_bar[k] = tb;
        bad |= !isfinite(tb);
        const float lr = lr_at(a.lr, k);
        if (a.m_adj) {
          const float contrib = -lr * a.m_adj[k] * tb;
          if (a.d_plr) a.d_plr[k] += contrib;
          else acc += contrib;
        }
        if (a.u_out) {
          vu = (a.u_in ? a.mu * a.u_in[k] : 0.f) - lr * tb;
          a.u_out[k] = vu;
        }
        if (a.cast_src) vw = a.cast_src[k];
      } else {
        const float v = a.cast_src[k];
        vw = v;
        vu = v;
      }
    }
    tw[i][tx] = vw;
    tu[i][tx] = vu;
    // row-major operand copies (only the din weight rows; the bias row stays float32)
    if (r < din && c < dout) {
      const int64_t o = static_cast<int64_t>(r) * tab.ldw[l] + c;
      if (cast_w) static_cast<T*>(tab.W[l])[o] = to_t<T>(vw);
      if (cast_u) static_cast<T*>(tab.U[l])[o] = to_t<T>(vu);
    }
  }
  if (bad && a.status) atomicExch(a.status, DEV_NONFINITE);
  if (a.partials) {
    acc = warp_sum(acc);
    const int lin = ty * TILE + tx;
    if ((lin & 31) == 0) red[lin >> 5] = acc;
  }
  __syncthreads();
  if (a.partials && ty == 0) {
    float v = tx < (TILE * TROWS / 32) ? red[tx] : 0.f;
    v = warp_sum(v);
    if (tx == 0) a.partials[blockIdx.x] = v;
  }
  // transposed operand copies [dout][ldwt]
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (c < dout && r < din) {
      const int64_t o = static_cast<int64_t>(c) * tab.ldwt[l] + r;
      if (cast_w && tab.WT[l]) static_cast<T*>(tab.WT[l])[o] = to_t<T>(tw[tx][i]);
      if (cast_u && tab.UT[l]) static_cast<T*>(tab.UT[l])[o] = to_t<T>(tu[tx][i]);
    }
  }
}

// Reverse-over-reverse, forward layer order: from dzbar (the adjoint of the backward's dz):
//   dabar = dzbar phi'(z)  (T, row-major and transposed),  zpart = dzbar phi''(z) da.
template <typename T>
__global__ void ror_fwd_elem_kernel(int act, const float* __restrict__ dzbar,
                                    const float* __restrict__ Z, const float* __restrict__ dA,
                                    int rows, int cols, T* __restrict__ dab, int ld,
                                    T* __restrict__ dabT, int ldT, float* __restrict__ zpart) {
  pdl_entry();
  __shared__ float tile[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float v = 0.f;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float f, d1, d2;
      act_eval(act, Z[o], f, d1, d2);
      v = dzbar[o] * d1;
      zpart[o] = dzbar[o] * d2 * dA[o];
      dab[static_cast<int64_t>(r) * ld + c] = to_t<T>(v);
    }
    tile[i][tx] = v;
  }
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (dabT && c < cols && r < rows) dabT[static_cast<int64_t>(c) * ldT + r] = to_t<T>(tile[tx][i]);
  }
}

// Reverse-over-reverse, reverse layer order:  zbar = zpart + abar phi'(z)  (T, both layouts).
template <typename T>
__global__ void ror_bwd_elem_kernel(int act, const float* __restrict__ zpart,
                                    const float* __restrict__ abar, const float* __restrict__ Z,
                                    int rows, int cols, T* __restrict__ zb, int ld,
                                    T* __restrict__ zbT, int ldT) {
  pdl_entry();
  __shared__ float tile[TILE][TILE + 1];
  const int c0 = blockIdx.x * TILE, r0 = blockIdx.y * TILE;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int i = ty; i < TILE; i += TROWS) {
    const int r = r0 + i, c = c0 + tx;
    float v = 0.f;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float f, d1, d2;
      act_eval(act, Z[o], f, d1, d2);
      v = zpart[o] + abar[o] * d1;
      zb[static_cast<int64_t>(r) * ld + c] = to_t<T>(v);
    }
    tile[i][tx] = v;
  }
  __syncthreads();
  for (int i = ty; i < TILE; i += TROWS) {
    const int c = c0 + i, r = r0 + tx;
    if (zbT && c < cols && r < rows) zbT[static_cast<int64_t>(c) * ldT + r] = to_t<T>(tile[tx][i]);
  }
}

__global__ void fill_kernel(float* p, int64_t n, float v) {
  pdl_entry();
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    p[i] = v;
}

}  // namespace

template <typename T>
void transpose(const T* X, int rows, int cols, int ld, T* XT, int ldT, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  launch_k(transpose_kernel<T>, dim3(grid), dim3(TILE, TROWS), 0, s, X, rows, cols, ld, XT, ldT);
}

template <typename T>
void fill_rows(const RowFill& f, int cols, cudaStream_t s) {
  if (f.n <= 0 || cols <= 0) return;
  dim3 grid((cols + 255) / 256, f.n);
  launch_k(fill_rows_kernel<T>, dim3(grid), dim3(256), 0, s, f, cols);
}

template <typename T>
void fill_cols(const ColFill& f, int rows, cudaStream_t s) {
  if (f.n == 0 || rows <= 0) return;
  launch_k(fill_cols_kernel<T>, dim3((rows + 255) / 256, f.n), dim3(256), 0, s, f, rows);
}

template <typename T>
void loss_seed(const LossArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return;
  if ((a.loss == 1 && !a.Yi) || (a.loss != 1 && !a.Yf) || !a.F) return;   // no targets: nothing read
  if (a.loss == 2) {
    if (a.ror && a.tape && a.chain > 0 && (a.ror == 1 || a.Fd))
      launch_k(chain_ror_kernel<T>, dim3(a.rows), dim3(256), 0, s, a);
    else
      launch_k(chain_loss_kernel<T>, dim3(a.rows), dim3(256), 0, s, a);
    return;
  }
  const int warps = 8;
  launch_k(loss_seed_kernel<T>, dim3((a.rows + warps - 1) / warps), dim3(warps * 32), 0, s, a);
}

void sum_scaled(const float* x, int n, float scale, float* out, cudaStream_t s) {
  launch_k(sum_scaled_kernel, dim3(1), dim3(1024), 0, s, x, n, scale, out);
}

template <typename T>
void layer_update(const LayerTable& tab, const LayerUpdArgs& a, cudaStream_t s) {
  const int blocks = tab.tile0[tab.n];
  if (blocks <= 0) return;
  launch_k(layer_update_kernel<T>, dim3(blocks), dim3(TILE, TROWS), 0, s, tab, a);
}

template <typename T>
void ror_fwd_elem(int act, const float* dzbar, const float* Z, const float* dA, int rows, int cols,
                  T* dab, int ld, T* dabT, int ldT, float* zpart, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  launch_k(ror_fwd_elem_kernel<T>, dim3(grid), dim3(TILE, TROWS), 0, s, act, dzbar, Z, dA, rows, cols, dab, ld,
                                                             dabT, ldT, zpart);
}

template <typename T>
void ror_bwd_elem(int act, const float* zpart, const float* abar, const float* Z, int rows,
                  int cols, T* zb, int ld, T* zbT, int ldT, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  launch_k(ror_bwd_elem_kernel<T>, dim3(grid), dim3(TILE, TROWS), 0, s, act, zpart, abar, Z, rows, cols, zb, ld,
                                                             zbT, ldT);
}

void fill(float* p, int64_t n, float v, cudaStream_t s) {
  if (n <= 0) return;
  int64_t b = (n + 255) / 256;
  if (b > 152 * 16) b = 152 * 16;
  launch_k(fill_kernel, dim3(static_cast<int>(b)), dim3(256), 0, s, p, n, v);
}

#define MF_INST(T)                                                                 \
  template void transpose<T>(const T*, int, int, int, T*, int, cudaStream_t);     \
  template void fill_rows<T>(const RowFill&, int, cudaStream_t);                  \
  template void fill_cols<T>(const ColFill&, int, cudaStream_t);                  \
  template void loss_seed<T>(const LossArgs&, cudaStream_t);                      \
  template void layer_update<T>(const LayerTable&, const LayerUpdArgs&, cudaStream_t);        \
  template void ror_fwd_elem<T>(int, const float*, const float*, const float*, int, int, T*, int, \
                                T*, int, float*, cudaStream_t);                                   \
  template void ror_bwd_elem<T>(int, const float*, const float*, const float*, int, int, T*, int,  \
                                T*, int, cudaStream_t);
MF_INST(float)
MF_INST(__nv_bfloat16)
#undef MF_INST

}  // namespace mf
