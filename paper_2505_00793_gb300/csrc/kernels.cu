// Elementwise, row and update kernels of the mixed-mode sweep (HBM-bound work).
//
//  * per-example loss seeds with the tangent per-example loss (the mixed term of Eq. 7 for
//    per-example weights) and d eta_{t,b} = sigmoid'(eta_{t,b}) * l'_b / B;
//  * the fused per-layer update kernel: the inner-step update of Eq. 2 (rollout, SGD,
//    heavy ball or Adam) or the adjoint update of the reverse sweep (Eq. 5 with the Hessian
//    product supplied by the forward-over-reverse pass, and the elementwise reverse of the
//    optimiser step), each fused with the cast of the next step's parameters / tangent into
//    the bf16 GEMM operand copies;
//  * the chain loss of the motivating example, in both HVP modes;
//  * the reverse-over-reverse element kernels, column fills and a deterministic sum.
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
      if (lane == 0 && a.status) atomicMax(a.status, 1);
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
  if (bad && a.status) atomicMax(a.status, DEV_NONFINITE);
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
  if (bad && a.status) atomicMax(a.status, DEV_NONFINITE);
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

// Four consecutive parameters per thread, UPD_ELEMS per block, blocks assigned to layers by
// tab.tile0.  A layer whose offset and width are multiples of 4 moves them as float4 (and
// its operand copies as four-element stores in one row); others go element by element.
__device__ __forceinline__ void ld4(float (&x)[4], const float* p, int64_t k, bool vec, int cnt) {
  if (vec) {
    const float4 t = *reinterpret_cast<const float4*>(p + k);
    x[0] = t.x; x[1] = t.y; x[2] = t.z; x[3] = t.w;
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) x[j] = j < cnt ? p[k + j] : 0.f;
  }
}

__device__ __forceinline__ void st4(float* p, int64_t k, const float (&x)[4], bool vec, int cnt) {
  if (vec) {
    *reinterpret_cast<float4*>(p + k) = make_float4(x[0], x[1], x[2], x[3]);
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < cnt) p[k + j] = x[j];
  }
}

template <typename T>
__device__ __forceinline__ void st_copy(T* W, int64_t e0, int dout, int din, int ldw,
                                        const float (&x)[4], bool vec, int cnt) {
  if (vec) {   // four elements of one row
    const int r = static_cast<int>(e0 / dout), c = static_cast<int>(e0 % dout);
    if (r >= din) return;
    T* q = W + static_cast<int64_t>(r) * ldw + c;
    if constexpr (sizeof(T) == 2) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(x[0], x[1]);
      __nv_bfloat162 hi = __floats2bfloat162_rn(x[2], x[3]);
      uint2 v;
      v.x = *reinterpret_cast<uint32_t*>(&lo);
      v.y = *reinterpret_cast<uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(q) = v;
    } else {
      *reinterpret_cast<float4*>(q) = make_float4(x[0], x[1], x[2], x[3]);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (j >= cnt) break;
      const int64_t e = e0 + j;
      const int r = static_cast<int>(e / dout), c = static_cast<int>(e % dout);
      if (r < din) W[static_cast<int64_t>(r) * ldw + c] = to_t<T>(x[j]);
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(UPD_THREADS) layer_update_kernel(const LayerTable tab,
                                                                   const LayerUpdArgs a) {
  pdl_entry();
  __shared__ float red[UPD_THREADS / 32];
  // the layer of this block: the last l with tile0[l] <= blockIdx.x (binary search)
  int l = 0;
  {
    int hi = tab.n - 1;
    while (l < hi) {
      const int mid = (l + hi + 1) >> 1;
      if (static_cast<int>(blockIdx.x) >= tab.tile0[mid]) l = mid;
      else hi = mid - 1;
    }
  }
  const int dout = tab.dout[l], din = tab.din[l];
  const int64_t n = static_cast<int64_t>(tab.rows[l]) * dout;
  const int64_t e0 = (static_cast<int64_t>(blockIdx.x - tab.tile0[l]) * UPD_THREADS + threadIdx.x) * 4;
  const bool cast_w = (a.mode == LU_ROLLOUT) || (a.mode == LU_CAST && !a.cast_src_to_u) ||
                      (a.mode == LU_ADJOINT && a.cast_src);
  const bool cast_u = (a.mode == LU_CAST && a.cast_src_to_u) || (a.mode == LU_ADJOINT && a.u_out);
  bool bad = false;
  float acc = 0.f;
  if (e0 < n) {
    const int cnt = static_cast<int>(n - e0 < 4 ? n - e0 : 4);
    const bool vec = a.vec_ok && cnt == 4 && (tab.off[l] & 3) == 0 && (dout & 3) == 0;
    const int64_t k = tab.off[l] + e0;
    float vw[4] = {0.f, 0.f, 0.f, 0.f}, vu[4] = {0.f, 0.f, 0.f, 0.f};
    float lr[4];
    const bool need_lr = a.mode == LU_ROLLOUT ||
                         (a.mode == LU_ADJOINT && (a.adam_pre || a.m_adj || a.u_out));
    if (a.lr.plr && need_lr) {
      ld4(lr, a.lr.plr, k, vec, cnt);
#pragma unroll
      for (int j = 0; j < 4; ++j) lr[j] = expf(lr[j]);
    } else {
      const float l0 = a.lr.slr ? expf(a.lr.slr[0]) : a.lr.alpha;
#pragma unroll
      for (int j = 0; j < 4; ++j) lr[j] = l0;
    }
    if (a.mode == LU_ROLLOUT) {
      float th[4], g[4], m[4] = {0.f, 0.f, 0.f, 0.f}, v[4] = {0.f, 0.f, 0.f, 0.f};
      ld4(th, a.theta, k, vec, cnt);
      ld4(g, a.g, k, vec, cnt);
      if (a.m) ld4(m, a.m, k, vec, cnt);
      if (a.adam && a.v) ld4(v, a.v, k, vec, cnt);
      float mn[4], vn[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (a.adam) {
          mn[j] = a.b1 * m[j] + (1.f - a.b1) * g[j];
          vn[j] = a.b2 * v[j] + (1.f - a.b2) * g[j] * g[j];
          vw[j] = th[j] - lr[j] * (mn[j] / a.c1) / (sqrtf(vn[j] / a.c2) + a.eps);
        } else {
          mn[j] = a.mu * m[j] + g[j];
          vn[j] = 0.f;
          vw[j] = th[j] - lr[j] * mn[j];
        }
        bad |= j < cnt && !isfinite(vw[j]);
      }
      st4(a.theta_out, k, vw, vec, cnt);
      if (a.m_out) st4(a.m_out, k, mn, vec, cnt);
      if (a.adam && a.v_out) st4(a.v_out, k, vn, vec, cnt);
    } else if (a.mode == LU_ADJOINT) {
      float tb[4], hu[4] = {0.f, 0.f, 0.f, 0.f};
      ld4(tb, a.theta_bar, k, vec, cnt);
      if (a.Hu) ld4(hu, a.Hu, k, vec, cnt);
      // every other input of the plain (non-Adam) adjoint is loaded before the first store,
      // so that a thread's loads are in flight together (the pointers may alias in place)
      float ma[4] = {0.f, 0.f, 0.f, 0.f}, ui[4] = {0.f, 0.f, 0.f, 0.f};
      float dp[4] = {0.f, 0.f, 0.f, 0.f};
      const bool plain = !a.adam;
      if (plain && a.m_adj) ld4(ma, a.m_adj, k, vec, cnt);
      if (plain && a.u_out && a.u_in) ld4(ui, a.u_in, k, vec, cnt);
      if (plain && a.m_adj && a.d_plr) ld4(dp, a.d_plr, k, vec, cnt);
      if (plain && a.cast_src) ld4(vw, a.cast_src, k, vec, cnt);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        tb[j] += hu[j];
        bad |= j < cnt && !isfinite(tb[j]);
      }
      st4(a.theta_bar, k, tb, vec, cnt);
      float contrib[4] = {0.f, 0.f, 0.f, 0.f};
      bool have_contrib = false;
      if (a.adam && a.adam_pre) {
        // reverse of Adam step j from its outputs m1 = m_{j+1}, v1 = v_{j+1} (see LayerUpdArgs)
        float m1[4], v1[4], mp[4] = {0.f, 0.f, 0.f, 0.f};
        float mb[4] = {0.f, 0.f, 0.f, 0.f}, vb[4] = {0.f, 0.f, 0.f, 0.f};
        ld4(m1, a.m_adj, k, vec, cnt);
        ld4(v1, a.v_adj, k, vec, cnt);
        if (a.m_prev) ld4(mp, a.m_prev, k, vec, cnt);
        if (a.bar_in) {
          ld4(mb, a.mbar, k, vec, cnt);
          ld4(vb, a.vbar, k, vec, cnt);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float sq = sqrtf(v1[j] / a.c2);
          const float den = sq + a.eps;
          const float q = -lr[j] * tb[j];
          // at v = 0 (where m = g = 0) the sqrt term is 0
          const float Mb = mb[j] + q / (a.c1 * den);
          const float Vb = vb[j] - (sq > 0.f ? q * m1[j] / (a.c1 * den * den * 2.f * sq * a.c2) : 0.f);
          const float g = (m1[j] - a.b1 * mp[j]) / (1.f - a.b1);
          vu[j] = (1.f - a.b1) * Mb + 2.f * (1.f - a.b2) * g * Vb;
          mb[j] = a.b1 * Mb;
          vb[j] = a.b2 * Vb;
          contrib[j] = -lr[j] * (m1[j] / a.c1) / den * tb[j];
          bad |= j < cnt && !isfinite(vu[j]);
        }
        st4(a.u_out, k, vu, vec, cnt);
        st4(a.mbar, k, mb, vec, cnt);
        st4(a.vbar, k, vb, vec, cnt);
        have_contrib = true;
      } else if (plain) {
        if (a.m_adj) {
#pragma unroll
          for (int j = 0; j < 4; ++j) contrib[j] = -lr[j] * ma[j] * tb[j];
          have_contrib = true;
        }
        if (a.u_out) {
#pragma unroll
          for (int j = 0; j < 4; ++j) vu[j] = a.mu * ui[j] - lr[j] * tb[j];
          st4(a.u_out, k, vu, vec, cnt);
        }
      }
      if (have_contrib) {
        if (a.d_plr) {
          if (!plain) ld4(dp, a.d_plr, k, vec, cnt);
#pragma unroll
          for (int j = 0; j < 4; ++j) dp[j] += contrib[j];
          st4(a.d_plr, k, dp, vec, cnt);
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) acc += j < cnt ? contrib[j] : 0.f;
        }
      }
      if (!plain && a.cast_src) ld4(vw, a.cast_src, k, vec, cnt);
    } else {
      ld4(vw, a.cast_src, k, vec, cnt);
#pragma unroll
      for (int j = 0; j < 4; ++j) vu[j] = vw[j];
    }
    if (cast_w && tab.W[l]) st_copy<T>(static_cast<T*>(tab.W[l]), e0, dout, din, tab.ldw[l], vw, vec, cnt);
    if (cast_u && tab.U[l]) st_copy<T>(static_cast<T*>(tab.U[l]), e0, dout, din, tab.ldw[l], vu, vec, cnt);
  }
  if (bad && a.status) atomicMax(a.status, DEV_NONFINITE);
  if (a.partials) {   // one deterministic partial sum per block (scalar log-lr)
    acc = warp_sum(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x < 32) {
      float v = threadIdx.x < UPD_THREADS / 32 ? red[threadIdx.x] : 0.f;
      v = warp_sum(v);
      if (threadIdx.x == 0) a.partials[blockIdx.x] = v;
    }
  }
}

// Reverse-over-reverse, forward layer order: from dzbar (the adjoint of the backward's dz):
//   dabar = dzbar phi'(z)  (T, row-major [rows][ld]),  zpart = dzbar phi''(z) da.
template <typename T>
__global__ void ror_fwd_elem_kernel(int act, const float* __restrict__ dzbar,
                                    const float* __restrict__ Z, const float* __restrict__ dA,
                                    int rows, int cols, T* __restrict__ dab, int ld,
                                    float* __restrict__ zpart) {
  pdl_entry();
  const int c = blockIdx.x * TILE + threadIdx.x;
  for (int i = threadIdx.y; i < TILE; i += TROWS) {
    const int r = blockIdx.y * TILE + i;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float f, d1, d2;
      act_eval(act, Z[o], f, d1, d2);
      zpart[o] = dzbar[o] * d2 * dA[o];
      dab[static_cast<int64_t>(r) * ld + c] = to_t<T>(dzbar[o] * d1);
    }
  }
}

// Reverse-over-reverse, reverse layer order:  zbar = zpart + abar phi'(z)  (T, [rows][ld]).
template <typename T>
__global__ void ror_bwd_elem_kernel(int act, const float* __restrict__ zpart,
                                    const float* __restrict__ abar, const float* __restrict__ Z,
                                    int rows, int cols, T* __restrict__ zb, int ld) {
  pdl_entry();
  const int c = blockIdx.x * TILE + threadIdx.x;
  for (int i = threadIdx.y; i < TILE; i += TROWS) {
    const int r = blockIdx.y * TILE + i;
    if (r < rows && c < cols) {
      const int64_t o = static_cast<int64_t>(r) * cols + c;
      float f, d1, d2;
      act_eval(act, Z[o], f, d1, d2);
      zb[static_cast<int64_t>(r) * ld + c] = to_t<T>(zpart[o] + abar[o] * d1);
    }
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
void layer_update(const LayerTable& tab, const LayerUpdArgs& args, cudaStream_t s) {
  const int blocks = tab.tile0[tab.n];
  if (blocks <= 0) return;
  // float4 access only when every vector the call touches is 16-byte aligned (caller
  // pointers such as theta or eta + offset need not be)
  LayerUpdArgs a = args;
  uintptr_t any = 0;
  for (const void* p : {static_cast<const void*>(a.cast_src), static_cast<const void*>(a.theta),
                        static_cast<const void*>(a.m), static_cast<const void*>(a.g),
                        static_cast<const void*>(a.theta_out), static_cast<const void*>(a.m_out),
                        static_cast<const void*>(a.theta_bar), static_cast<const void*>(a.Hu),
                        static_cast<const void*>(a.m_adj), static_cast<const void*>(a.u_in),
                        static_cast<const void*>(a.u_out), static_cast<const void*>(a.d_plr),
                        static_cast<const void*>(a.lr.plr), static_cast<const void*>(a.v),
                        static_cast<const void*>(a.v_out), static_cast<const void*>(a.v_adj),
                        static_cast<const void*>(a.m_prev), static_cast<const void*>(a.mbar),
                        static_cast<const void*>(a.vbar)})
    any |= reinterpret_cast<uintptr_t>(p);
  a.vec_ok = (any & 15) == 0;
  launch_k(layer_update_kernel<T>, dim3(blocks), dim3(UPD_THREADS), 0, s, tab, a);
}

template <typename T>
void ror_fwd_elem(int act, const float* dzbar, const float* Z, const float* dA, int rows, int cols,
                  T* dab, int ld, float* zpart, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  launch_k(ror_fwd_elem_kernel<T>, dim3(grid), dim3(TILE, TROWS), 0, s, act, dzbar, Z, dA, rows,
           cols, dab, ld, zpart);
}

template <typename T>
void ror_bwd_elem(int act, const float* zpart, const float* abar, const float* Z, int rows,
                  int cols, T* zb, int ld, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return;
  dim3 grid((cols + TILE - 1) / TILE, (rows + TILE - 1) / TILE);
  launch_k(ror_bwd_elem_kernel<T>, dim3(grid), dim3(TILE, TROWS), 0, s, act, zpart, abar, Z, rows,
           cols, zb, ld);
}

void fill(float* p, int64_t n, float v, cudaStream_t s) {
  if (n <= 0) return;
  int64_t b = (n + 255) / 256;
  if (b > 152 * 16) b = 152 * 16;
  launch_k(fill_kernel, dim3(static_cast<int>(b)), dim3(256), 0, s, p, n, v);
}

#define MF_INST(T)                                                                 \
  template void fill_cols<T>(const ColFill&, int, cudaStream_t);                  \
  template void loss_seed<T>(const LossArgs&, cudaStream_t);                      \
  template void layer_update<T>(const LayerTable&, const LayerUpdArgs&, cudaStream_t);        \
  template void ror_fwd_elem<T>(int, const float*, const float*, const float*, int, int, T*, int, \
                                float*, cudaStream_t);                                            \
  template void ror_bwd_elem<T>(int, const float*, const float*, const float*, int, int, T*, int,  \
                                cudaStream_t);
MF_INST(float)
MF_INST(__nv_bfloat16)
#undef MF_INST

}  // namespace mf
