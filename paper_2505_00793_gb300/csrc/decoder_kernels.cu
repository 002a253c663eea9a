// Row and elementwise kernels of the dual (primal + tangent) decoder-only transformer:
// embedding gather and deterministic scatter-add, fused residual + RMSNorm forward and its
// dual backward, RoPE with the head split (and its transpose for the backward), causal
// softmax with its tangent, the softmax backward with its tangent, next-token
// cross-entropy with per-sequence weights (the mixed term of Eq. 7 per sequence), and
// deterministic column reductions for the RMSNorm gains.
//
// Notation (per token row): n = x r, r = (mean x^2 + eps)^-1/2, h = g n;
// tangents carry a dot: r' = -r^3 mean(x x'), n' = x' r + x r', h' = g' n + g n'.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "device_math.cuh"
#include "internal.h"
#include "launch.cuh"

namespace mf {
namespace {

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

// SMs of a GB300 (152): sets the grid size of the grid-stride row kernels (a performance
// choice; every kernel is correct for any grid).
constexpr int ROW_SMS = 152;

// Block-wide sum of two values (fixed reduction order), blockDim.x a multiple of 32, <= 1024.
__device__ __forceinline__ float2 block_sum2(float a, float b) {
  __shared__ float2 red[32];
  a = warp_sum(a);
  b = warp_sum(b);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = make_float2(a, b);
  __syncthreads();
  float2 r = make_float2(0.f, 0.f);
  const int nw = blockDim.x >> 5;
  if (w == 0) {
    float2 v = l < nw ? red[l] : make_float2(0.f, 0.f);
    v.x = warp_sum(v.x);
    v.y = warp_sum(v.y);
    if (l == 0) red[0] = v;
  }
  __syncthreads();
  r = red[0];
  return r;
}

__device__ __forceinline__ float ld_t(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ld_t(const __nv_bfloat16* p, int64_t i) { return __bfloat162float(p[i]); }

// x[r] = E[id(r)], x'[r] = U_E[id(r)]  (ids [B][S+1]; row r = b S + s uses ids[b][s])
__global__ void embed_fwd_kernel(const int* __restrict__ ids, int S, int d, int V,
                                 const float* __restrict__ E, const float* __restrict__ UE,
                                 float* __restrict__ x, float* __restrict__ xd, int* status) {
  pdl_entry();
  const int r = blockIdx.x;
  const int b = r / S, s = r % S;
  int id = ids[static_cast<int64_t>(b) * (S + 1) + s];
  if (id < 0 || id >= V) {
    if (threadIdx.x == 0 && status) atomicMax(status, 1);
    id = 0;
  }
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    x[static_cast<int64_t>(r) * d + j] = E[static_cast<int64_t>(id) * d + j];
    if (xd) xd[static_cast<int64_t>(r) * d + j] = UE[static_cast<int64_t>(id) * d + j];
  }
}

// Fused residual add + RMSNorm (dual).  x = x_in (+ y); stores x (float32), r, r', and
// h = g x r (and h') in T, row-major [N][ldh].
template <typename T>
__global__ void rmsnorm_fwd_kernel(int d, float eps, const float* __restrict__ x_in,
                                   const float* __restrict__ y, const float* __restrict__ xd_in,
                                   const float* __restrict__ yd, const float* __restrict__ g,
                                   const float* __restrict__ gd, float* __restrict__ x_out,
                                   float* __restrict__ xd_out, float* __restrict__ rr,
                                   float* __restrict__ rrd, T* __restrict__ h, T* __restrict__ hd,
                                   int ldh) {
  pdl_entry();
  const int r = blockIdx.x;
  const int64_t o = static_cast<int64_t>(r) * d;
  const bool dual = xd_in != nullptr;
  float s2 = 0.f, s1 = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    float v = x_in[o + j] + (y ? y[o + j] : 0.f);
    x_out[o + j] = v;
    s2 += v * v;
    if (dual) {
      const float vd = xd_in[o + j] + (yd ? yd[o + j] : 0.f);
      xd_out[o + j] = vd;
      s1 += v * vd;
    }
  }
  const float2 sums = block_sum2(s2, s1);
  const float inv_d = 1.f / static_cast<float>(d);
  const float rs = rsqrtf(sums.x * inv_d + eps);
  const float rsd = -rs * rs * rs * sums.y * inv_d;
  if (threadIdx.x == 0) {
    rr[r] = rs;
    if (dual) rrd[r] = rsd;
  }
  const int64_t oh = static_cast<int64_t>(r) * ldh;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float v = x_out[o + j];
    const float n = v * rs;
    h[oh + j] = to_t<T>(g[j] * n);
    if (dual) {
      const float nd = xd_out[o + j] * rs + v * rsd;
      hd[oh + j] = to_t<T>(gd[j] * n + g[j] * nd);
    }
  }
}

// Dual RMSNorm backward, accumulated into the residual gradient:
//   dx += r (dn - n c),  c = mean(dn n),  dn = dy g
//   dx' += r' (dn - n c) + r (dn' - n' c - n c'),  dn' = dy' g + dy g',  c' = mean(dn' n + dn n')
// Warp-per-row versions of the RMSNorm forward and backward (eight rows per block, float4
// access, shuffle reductions), used when every vector is 16-byte aligned and d is a multiple
// of 4; same arithmetic as the block-per-row kernels above and below.
__device__ __forceinline__ float warp_sum_all(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T>
__device__ __forceinline__ void st_t4(T* p, float a, float b, float c, float d) {
  if constexpr (sizeof(T) == 2) {
    __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
    uint2 v;
    v.x = *reinterpret_cast<uint32_t*>(&lo);
    v.y = *reinterpret_cast<uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(p) = v;
  } else {
    *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
  }
}

__device__ __forceinline__ float4 ld4f(const float* p) { return *reinterpret_cast<const float4*>(p); }

template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_fwd_warp_kernel(
    int N, int d, float eps, const float* __restrict__ x_in, const float* __restrict__ y,
    const float* __restrict__ xd_in, const float* __restrict__ yd, const float* __restrict__ g,
    const float* __restrict__ gd, float* __restrict__ x_out, float* __restrict__ xd_out,
    float* __restrict__ rr, float* __restrict__ rrd, T* __restrict__ h, T* __restrict__ hd,
    int ldh) {
  pdl_entry();
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= N) return;
  const int64_t o = static_cast<int64_t>(r) * d;
  const bool dual = xd_in != nullptr;
  float s2 = 0.f, s1 = 0.f;
  for (int c = lane * 4; c < d; c += 128) {
    float4 v = ld4f(x_in + o + c);
    if (y) { const float4 t = ld4f(y + o + c); v.x += t.x; v.y += t.y; v.z += t.z; v.w += t.w; }
    *reinterpret_cast<float4*>(x_out + o + c) = v;
    s2 += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    if (dual) {
      float4 vd = ld4f(xd_in + o + c);
      if (yd) { const float4 t = ld4f(yd + o + c); vd.x += t.x; vd.y += t.y; vd.z += t.z; vd.w += t.w; }
      *reinterpret_cast<float4*>(xd_out + o + c) = vd;
      s1 += v.x * vd.x + v.y * vd.y + v.z * vd.z + v.w * vd.w;
    }
  }
  s2 = warp_sum_all(s2);
  s1 = warp_sum_all(s1);
  const float inv_d = 1.f / static_cast<float>(d);
  const float rs = rsqrtf(s2 * inv_d + eps);
  const float rsd = -rs * rs * rs * s1 * inv_d;
  if (lane == 0) {
    rr[r] = rs;
    if (dual) rrd[r] = rsd;
  }
  const int64_t oh = static_cast<int64_t>(r) * ldh;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 v = ld4f(x_out + o + c), gg = ld4f(g + c);
    const float n0 = v.x * rs, n1 = v.y * rs, n2 = v.z * rs, n3 = v.w * rs;
    st_t4<T>(h + oh + c, gg.x * n0, gg.y * n1, gg.z * n2, gg.w * n3);
    if (dual) {
      const float4 vd = ld4f(xd_out + o + c), ggd = ld4f(gd + c);
      const float m0 = vd.x * rs + v.x * rsd, m1 = vd.y * rs + v.y * rsd;
      const float m2 = vd.z * rs + v.z * rsd, m3 = vd.w * rs + v.w * rsd;
      st_t4<T>(hd + oh + c, ggd.x * n0 + gg.x * m0, ggd.y * n1 + gg.y * m1,
               ggd.z * n2 + gg.z * m2, ggd.w * n3 + gg.w * m3);
    }
  }
}

// Row r of the warp-per-row RMSNorm backward (this lane's columns lane*4 + 128 k).
template <typename T>
__device__ __forceinline__ void rmsnorm_bwd_row(
    int r, int lane, int d, const float* __restrict__ x, const float* __restrict__ xd,
    const float* __restrict__ rr, const float* __restrict__ rrd, const float* __restrict__ g,
    const float* __restrict__ gd, const float* __restrict__ dy, const float* __restrict__ dyd,
    float* __restrict__ dx, float* __restrict__ dxd, T* __restrict__ dxb, T* __restrict__ dxdb) {
  const int64_t o = static_cast<int64_t>(r) * d;
  const bool dual = dyd != nullptr;
  const float rs = rr[r];
  const float rsd = dual ? rrd[r] : 0.f;
  float sc = 0.f, scd = 0.f;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 xv = ld4f(x + o + c), dv = ld4f(dy + o + c), gg = ld4f(g + c);
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w}, ds[4] = {dv.x, dv.y, dv.z, dv.w};
    const float gs[4] = {gg.x, gg.y, gg.z, gg.w};
    float xds[4] = {0.f, 0.f, 0.f, 0.f}, dds[4] = {0.f, 0.f, 0.f, 0.f}, gds[4] = {0.f, 0.f, 0.f, 0.f};
    if (dual) {
      const float4 a = ld4f(xd + o + c), b = ld4f(dyd + o + c), e = ld4f(gd + c);
      xds[0] = a.x; xds[1] = a.y; xds[2] = a.z; xds[3] = a.w;
      dds[0] = b.x; dds[1] = b.y; dds[2] = b.z; dds[3] = b.w;
      gds[0] = e.x; gds[1] = e.y; gds[2] = e.z; gds[3] = e.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float n = xs[j] * rs;
      const float dn = ds[j] * gs[j];
      sc += dn * n;
      if (dual) {
        const float nd = xds[j] * rs + xs[j] * rsd;
        const float dnd = dds[j] * gs[j] + ds[j] * gds[j];
        scd += dnd * n + dn * nd;
      }
    }
  }
  sc = warp_sum_all(sc);
  scd = warp_sum_all(scd);
  const float inv_d = 1.f / static_cast<float>(d);
  const float cc = sc * inv_d, ccd = scd * inv_d;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 xv = ld4f(x + o + c), dv = ld4f(dy + o + c), gg = ld4f(g + c), ov = ld4f(dx + o + c);
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w}, ds[4] = {dv.x, dv.y, dv.z, dv.w};
    const float gs[4] = {gg.x, gg.y, gg.z, gg.w}, os[4] = {ov.x, ov.y, ov.z, ov.w};
    float out[4], outd[4] = {0.f, 0.f, 0.f, 0.f};
    float xds[4] = {0.f, 0.f, 0.f, 0.f}, dds[4] = {0.f, 0.f, 0.f, 0.f}, gds[4] = {0.f, 0.f, 0.f, 0.f};
    float ods[4] = {0.f, 0.f, 0.f, 0.f};
    if (dual) {
      const float4 a = ld4f(xd + o + c), b = ld4f(dyd + o + c), e = ld4f(gd + c), f = ld4f(dxd + o + c);
      xds[0] = a.x; xds[1] = a.y; xds[2] = a.z; xds[3] = a.w;
      dds[0] = b.x; dds[1] = b.y; dds[2] = b.z; dds[3] = b.w;
      gds[0] = e.x; gds[1] = e.y; gds[2] = e.z; gds[3] = e.w;
      ods[0] = f.x; ods[1] = f.y; ods[2] = f.z; ods[3] = f.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float n = xs[j] * rs;
      const float dn = ds[j] * gs[j];
      out[j] = os[j] + rs * (dn - n * cc);
      if (dual) {
        const float nd = xds[j] * rs + xs[j] * rsd;
        const float dnd = dds[j] * gs[j] + ds[j] * gds[j];
        outd[j] = ods[j] + rsd * (dn - n * cc) + rs * (dnd - nd * cc - n * ccd);
      }
    }
    *reinterpret_cast<float4*>(dx + o + c) = make_float4(out[0], out[1], out[2], out[3]);
    if (dxb) st_t4<T>(dxb + o + c, out[0], out[1], out[2], out[3]);
    if (dual) {
      *reinterpret_cast<float4*>(dxd + o + c) = make_float4(outd[0], outd[1], outd[2], outd[3]);
      if (dxdb) st_t4<T>(dxdb + o + c, outd[0], outd[1], outd[2], outd[3]);
    }
  }
}

// The warp-per-row RMSNorm backward, and with part set the gain gradient's partial sums over
// the block's eight rows (data the row passes have just read, so the rows come from L2):
// warp w takes 128-column chunks w, w + 8, ..., adds the rows in order and writes partial
// row blockIdx.x of part (and of partd for the tangent).  The formulas per element are those
// of gain_grad_partial_kernel.
template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_bwd_warp_kernel(
    int N, int d, const float* __restrict__ x, const float* __restrict__ xd,
    const float* __restrict__ rr, const float* __restrict__ rrd, const float* __restrict__ g,
    const float* __restrict__ gd, const float* __restrict__ dy, const float* __restrict__ dyd,
    float* __restrict__ dx, float* __restrict__ dxd, T* __restrict__ dxb, T* __restrict__ dxdb,
    float* __restrict__ part, float* __restrict__ partd) {
  pdl_entry();
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + w;
  if (r < N) rmsnorm_bwd_row<T>(r, lane, d, x, xd, rr, rrd, g, gd, dy, dyd, dx, dxd, dxb, dxdb);
  if (!part) return;
  const bool dual = partd != nullptr;
  const int q0 = blockIdx.x * 8, q1 = min(N, q0 + 8);
  for (int c = w * 128 + lane * 4; c < d; c += 1024) {
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), ad = a;
#pragma unroll 4
    for (int q = q0; q < q1; ++q) {
      const int64_t o = static_cast<int64_t>(q) * d + c;
      const float rs = rr[q];
      const float4 xv = ld4f(x + o), dv = ld4f(dy + o);
      const float n0 = xv.x * rs, n1 = xv.y * rs, n2 = xv.z * rs, n3 = xv.w * rs;
      a.x += dv.x * n0; a.y += dv.y * n1; a.z += dv.z * n2; a.w += dv.w * n3;
      if (dual) {
        const float rsd = rrd[q];
        const float4 xdv = ld4f(xd + o), ddv = ld4f(dyd + o);
        ad.x += ddv.x * n0 + dv.x * (xdv.x * rs + xv.x * rsd);
        ad.y += ddv.y * n1 + dv.y * (xdv.y * rs + xv.y * rsd);
        ad.z += ddv.z * n2 + dv.z * (xdv.z * rs + xv.z * rsd);
        ad.w += ddv.w * n3 + dv.w * (xdv.w * rs + xv.w * rsd);
      }
    }
    const int64_t po = static_cast<int64_t>(blockIdx.x) * d + c;
    *reinterpret_cast<float4*>(part + po) = a;
    if (dual) *reinterpret_cast<float4*>(partd + po) = ad;
  }
}

template <typename T>
__global__ void rmsnorm_bwd_kernel(int d, const float* __restrict__ x, const float* __restrict__ xd,
                                   const float* __restrict__ rr, const float* __restrict__ rrd,
                                   const float* __restrict__ g, const float* __restrict__ gd,
                                   const float* __restrict__ dy, const float* __restrict__ dyd,
                                   float* __restrict__ dx, float* __restrict__ dxd,
                                   T* __restrict__ dxb, T* __restrict__ dxdb) {
  pdl_entry();
  const int r = blockIdx.x;
  const int64_t o = static_cast<int64_t>(r) * d;
  const bool dual = dyd != nullptr;
  const float rs = rr[r];
  const float rsd = dual ? rrd[r] : 0.f;
  float sc = 0.f, scd = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float n = x[o + j] * rs;
    const float dn = dy[o + j] * g[j];
    sc += dn * n;
    if (dual) {
      const float nd = xd[o + j] * rs + x[o + j] * rsd;
      const float dnd = dyd[o + j] * g[j] + dy[o + j] * gd[j];
      scd += dnd * n + dn * nd;
    }
  }
  const float2 sums = block_sum2(sc, scd);
  const float inv_d = 1.f / static_cast<float>(d);
  const float c = sums.x * inv_d, cd = sums.y * inv_d;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float n = x[o + j] * rs;
    const float dn = dy[o + j] * g[j];
    const float v = dx[o + j] + rs * (dn - n * c);
    dx[o + j] = v;
    if (dxb) dxb[o + j] = to_t<T>(v);
    if (dual) {
      const float nd = xd[o + j] * rs + x[o + j] * rsd;
      const float dnd = dyd[o + j] * g[j] + dy[o + j] * gd[j];
      const float vd = dxd[o + j] + rsd * (dn - n * c) + rs * (dnd - nd * c - n * cd);
      dxd[o + j] = vd;
      if (dxdb) dxdb[o + j] = to_t<T>(vd);
    }
  }
}

// RMSNorm gain gradient: dg[j] = sum_r dy[r][j] x[r][j] r_r (and its tangent), as a
// fixed-order two-stage reduction: stage 1 sums 256-row chunks (one partial row per chunk),
// stage 2 sums the chunk partials in chunk order.
constexpr int GG_ROWS = 256;

__global__ void gain_grad_partial_kernel(int N, int d, const float* __restrict__ x,
                                         const float* __restrict__ xd, const float* __restrict__ rr,
                                         const float* __restrict__ rrd, const float* __restrict__ dy,
                                         const float* __restrict__ dyd, float* __restrict__ part,
                                         float* __restrict__ partd) {
  pdl_entry();
  __shared__ float sp[8][33];
  __shared__ float spd[8][33];
  const int j = blockIdx.x * 32 + threadIdx.x;
  const int r0 = blockIdx.y * GG_ROWS;
  const int r1 = min(N, r0 + GG_ROWS);
  const bool dual = dyd != nullptr;
  float a = 0.f, ad = 0.f;
  if (j < d) {
    for (int r = r0 + threadIdx.y; r < r1; r += 8) {
      const int64_t o = static_cast<int64_t>(r) * d + j;
      const float n = x[o] * rr[r];
      a += dy[o] * n;
      if (dual) {
        const float nd = xd[o] * rr[r] + x[o] * rrd[r];
        ad += dyd[o] * n + dy[o] * nd;
      }
    }
  }
  sp[threadIdx.y][threadIdx.x] = a;
  spd[threadIdx.y][threadIdx.x] = ad;
  __syncthreads();
  if (threadIdx.y == 0 && j < d) {
    float t = 0.f, td = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) { t += sp[k][threadIdx.x]; td += spd[k][threadIdx.x]; }
    part[static_cast<int64_t>(blockIdx.y) * d + j] = t;
    if (dual) partd[static_cast<int64_t>(blockIdx.y) * d + j] = td;
  }
}

// Stage 2: the nchunk partial rows summed per column in a fixed order.  Block (32, 32) owns 32
// columns; thread (x, y) adds partial rows y, y + 32, ... in order, then the 32 sums of a
// column are added in y order.
constexpr int GF_Y = 32;

__global__ void __launch_bounds__(32 * GF_Y) gain_grad_final_kernel(
    int nchunk, int d, const float* __restrict__ part, const float* __restrict__ partd,
    float* __restrict__ dg, float* __restrict__ dgd) {
  pdl_entry();
  __shared__ float sp[GF_Y][33];
  __shared__ float spd[GF_Y][33];
  const int j = blockIdx.x * 32 + threadIdx.x;
  float t = 0.f, td = 0.f;
  if (j < d) {
#pragma unroll 8
    for (int c = threadIdx.y; c < nchunk; c += GF_Y) {
      t += part[static_cast<int64_t>(c) * d + j];
      if (partd) td += partd[static_cast<int64_t>(c) * d + j];
    }
  }
  sp[threadIdx.y][threadIdx.x] = t;
  spd[threadIdx.y][threadIdx.x] = td;
  __syncthreads();
  if (threadIdx.y == 0 && j < d) {
    float u = 0.f, ud = 0.f;
#pragma unroll
    for (int k = 0; k < GF_Y; ++k) {
      u += sp[k][threadIdx.x];
      ud += spd[k][threadIdx.x];
    }
    if (dg) dg[j] = u;
    if (partd && dgd) dgd[j] = ud;
  }
}

// RoPE angle table: (cos, sin) of s * base^(-2 j / dh) for positions s < S and pairs
// j < dh/2, interleaved, computed once per call in double precision.
__global__ void rope_table_kernel(int S, int half, int dh, double base, float* __restrict__ tab) {
  pdl_entry();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= S * half) return;
  const int s = i / half, j = i % half;
  const double ang = static_cast<double>(s) * pow(base, -2.0 * j / dh);
  tab[2 * i] = static_cast<float>(cos(ang));
  tab[2 * i + 1] = static_cast<float>(sin(ang));
}

// RoPE (rotate-half) on q and k, q scaled by 1/sqrt(dh), head split.  qkv [N][3d] float32
// (token-major) -> Q, K, V [B*H][S][dh] in T.  cos / sin of the angle of pair j at position
// s come from the table of rope_table_kernel.
// Four consecutive values stored as T (one 16-byte or 8-byte store).
template <typename T>
__device__ __forceinline__ void store4(T* p, float a, float b, float c, float d);
template <>
__device__ __forceinline__ void store4<float>(float* p, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
}
template <>
__device__ __forceinline__ void store4<__nv_bfloat16>(__nv_bfloat16* p, float a, float b, float c,
                                                      float d) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  uint2 v;
  v.x = *reinterpret_cast<const uint32_t*>(&lo);
  v.y = *reinterpret_cast<const uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(p) = v;
}

// Each thread takes four consecutive dimensions e..e+3 of one head (dh a multiple of 8, so
// the rotate-half partners e +- dh/2 are four consecutive values too): 16-byte loads of q, k,
// v, their partners and two (cos, sin) pairs of the table; 8-byte (bf16) stores.
template <typename T>
__global__ void rope_split_kernel(int S, int H, int dh, const float* __restrict__ rtab, float qscale,
                                  const float* __restrict__ qkv, T* __restrict__ Q,
                                  T* __restrict__ K, T* __restrict__ Vv) {
  pdl_entry();
  const int r = blockIdx.x;                 // token row
  const int b = r / S, s = r % S;
  const int d = H * dh, half = dh / 2;
  const float* row = qkv + static_cast<int64_t>(r) * 3 * d;
  for (int c = 4 * threadIdx.x; c < d; c += 4 * blockDim.x) {
    const int h = c / dh, e = c % dh;
    const bool lo = e < half;
    const int j = lo ? e : e - half;
    const int po = lo ? c + half : c - half;            // partner columns
    const float sg = lo ? -1.f : 1.f;                   // rot(x) = [-x2, x1]
    const float4 t01 = *reinterpret_cast<const float4*>(rtab + 2 * (s * half + j));
    const float4 t23 = *reinterpret_cast<const float4*>(rtab + 2 * (s * half + j + 2));
    const float cs[4] = {t01.x, t01.z, t23.x, t23.z}, sn[4] = {t01.y, t01.w, t23.y, t23.w};
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    const float4 qp = *reinterpret_cast<const float4*>(row + po);
    const float4 k = *reinterpret_cast<const float4*>(row + d + c);
    const float4 kp = *reinterpret_cast<const float4*>(row + d + po);
    const float4 v = *reinterpret_cast<const float4*>(row + 2 * d + c);
    const float qa[4] = {q.x, q.y, q.z, q.w}, qb[4] = {qp.x, qp.y, qp.z, qp.w};
    const float ka[4] = {k.x, k.y, k.z, k.w}, kb[4] = {kp.x, kp.y, kp.z, kp.w};
    float qo[4], ko[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      qo[i] = (qa[i] * cs[i] + sg * qb[i] * sn[i]) * qscale;
      ko[i] = ka[i] * cs[i] + sg * kb[i] * sn[i];
    }
    const int64_t o = ((static_cast<int64_t>(b) * H + h) * S + s) * dh + e;
    store4<T>(Q + o, qo[0], qo[1], qo[2], qo[3]);
    store4<T>(K + o, ko[0], ko[1], ko[2], ko[3]);
    store4<T>(Vv + o, v.x, v.y, v.z, v.w);
  }
}

// Transpose of the RoPE/split map for the backward: dQ, dK, dV [B*H][S][dh] (float32) ->
// dqkv [N][3d] row-major (T):  dq = R^T(dQ) qscale, dk = R^T(dK), dv = dV, with
// R^T(y) = y cos + [y2, -y1] sin.  Four consecutive dimensions per thread, as above.
template <typename T>
__global__ void rope_merge_kernel(int S, int H, int dh, const float* __restrict__ rtab, float qscale,
                                  const float* __restrict__ dQ, const float* __restrict__ dK,
                                  const float* __restrict__ dV, T* __restrict__ out, int ldo) {
  pdl_entry();
  const int r = blockIdx.x;
  const int b = r / S, s = r % S;
  const int d = H * dh, half = dh / 2;
  T* row = out + static_cast<int64_t>(r) * ldo;
  for (int c = 4 * threadIdx.x; c < d; c += 4 * blockDim.x) {
    const int h = c / dh, e = c % dh;
    const bool lo = e < half;
    const int j = lo ? e : e - half;
    const int pe = lo ? e + half : e - half;
    const float sg = lo ? 1.f : -1.f;                   // R^T: [y2, -y1]
    const float4 t01 = *reinterpret_cast<const float4*>(rtab + 2 * (s * half + j));
    const float4 t23 = *reinterpret_cast<const float4*>(rtab + 2 * (s * half + j + 2));
    const float cs[4] = {t01.x, t01.z, t23.x, t23.z}, sn[4] = {t01.y, t01.w, t23.y, t23.w};
    const int64_t o = ((static_cast<int64_t>(b) * H + h) * S + s) * dh;
    const float4 q = *reinterpret_cast<const float4*>(dQ + o + e);
    const float4 qp = *reinterpret_cast<const float4*>(dQ + o + pe);
    const float4 k = *reinterpret_cast<const float4*>(dK + o + e);
    const float4 kp = *reinterpret_cast<const float4*>(dK + o + pe);
    const float4 v = *reinterpret_cast<const float4*>(dV + o + e);
    const float qa[4] = {q.x, q.y, q.z, q.w}, qb[4] = {qp.x, qp.y, qp.z, qp.w};
    const float ka[4] = {k.x, k.y, k.z, k.w}, kb[4] = {kp.x, kp.y, kp.z, kp.w};
    float qo[4], ko[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      qo[i] = (qa[i] * cs[i] + sg * qb[i] * sn[i]) * qscale;
      ko[i] = ka[i] * cs[i] + sg * kb[i] * sn[i];
    }
    store4<T>(row + c, qo[0], qo[1], qo[2], qo[3]);
    store4<T>(row + d + c, ko[0], ko[1], ko[2], ko[3]);
    store4<T>(row + 2 * d + c, v.x, v.y, v.z, v.w);
  }
}

// Head merge: O [B*H][S][dh] (float32) -> [N][ldo] (T) token-major, column h*dh + e.
template <typename T>
__global__ void head_merge_kernel(int S, int H, int dh, const float* __restrict__ O,
                                  T* __restrict__ out, int ldo) {
  pdl_entry();
  const int r = blockIdx.x;
  const int b = r / S, s = r % S;
  const int d = H * dh;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const int h = c / dh, e = c % dh;
    out[static_cast<int64_t>(r) * ldo + c] =
        to_t<T>(O[((static_cast<int64_t>(b) * H + h) * S + s) * dh + e]);
  }
}

// Head split of a token-major float32 gradient [N][d] -> [B*H][S][dh] (T).
template <typename T>
__global__ void head_split_kernel(int S, int H, int dh, const float* __restrict__ X,
                                  T* __restrict__ out) {
  pdl_entry();
  const int r = blockIdx.x;
  const int b = r / S, s = r % S;
  const int d = H * dh;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const int h = c / dh, e = c % dh;
    out[((static_cast<int64_t>(b) * H + h) * S + s) * dh + e] =
        to_t<T>(X[static_cast<int64_t>(r) * d + c]);
  }
}

// Causal softmax with tangent, one warp per score row (q): P = softmax(S), keys k > q masked;
// P' = P (S' - sum_k P S').
template <typename T>
__global__ void softmax_fwd_kernel(int S, int rows, const float* __restrict__ Sc,
                                   const float* __restrict__ Scd, T* __restrict__ P,
                                   T* __restrict__ Pd) {
  pdl_entry();
  const int warps = blockDim.x >> 5;
  const int row = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const int q = row % S;
  const int64_t o = static_cast<int64_t>(row) * S;
  float mx = -INFINITY;
  for (int k = lane; k <= q; k += 32) mx = fmaxf(mx, Sc[o + k]);
  mx = warp_max(mx);
  float se = 0.f;
  for (int k = lane; k <= q; k += 32) se += expf(Sc[o + k] - mx);
  se = warp_sum(se);
  const float inv = 1.f / se;
  float ps = 0.f;
  if (Scd) {
    for (int k = lane; k <= q; k += 32) ps += expf(Sc[o + k] - mx) * inv * Scd[o + k];
    ps = warp_sum(ps);
  }
  for (int k = lane; k < S; k += 32) {
    float p = 0.f, pd = 0.f;
    if (k <= q) {
      p = expf(Sc[o + k] - mx) * inv;
      if (Scd) pd = p * (Scd[o + k] - ps);
    }
    P[o + k] = to_t<T>(p);
    if (Pd) Pd[o + k] = to_t<T>(pd);
  }
}

// Softmax backward with tangent, one warp per row:
//   D = sum_k P dP,  D' = sum_k (P' dP + P dP'),
//   dS = P (dP - D),  dS' = P' (dP - D) + P (dP' - D').
template <typename T>
__global__ void softmax_bwd_kernel(int S, int rows, const T* __restrict__ P,
                                   const T* __restrict__ Pd, const float* __restrict__ dP,
                                   const float* __restrict__ dPd, T* __restrict__ dS,
                                   T* __restrict__ dSd) {
  pdl_entry();
  const int warps = blockDim.x >> 5;
  const int row = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const int64_t o = static_cast<int64_t>(row) * S;
  const bool dual = dPd != nullptr;
  float D = 0.f, Dd = 0.f;
  for (int k = lane; k < S; k += 32) {
    const float p = ld_t(P, o + k);
    D += p * dP[o + k];
    if (dual) Dd += ld_t(Pd, o + k) * dP[o + k] + p * dPd[o + k];
  }
  D = warp_sum(D);
  if (dual) Dd = warp_sum(Dd);
  for (int k = lane; k < S; k += 32) {
    const float p = ld_t(P, o + k);
    const float g = dP[o + k] - D;
    dS[o + k] = to_t<T>(p * g);
    if (dual) dSd[o + k] = to_t<T>(ld_t(Pd, o + k) * g + p * (dPd[o + k] - Dd));
  }
}

// Next-token cross-entropy row statistics, one block per token row r = b S + s, target
// ids[b][s+1]:  lse, l = lse - f_y, l' = p.f' - f'_y (with p = softmax(f)).
// Running softmax statistics (max m, sum of exp(f - m), sum of exp(f - m) f'), merged
// exactly: rescale both sums to the larger max.
struct SoftStat {
  float m, s, t;
};
__device__ __forceinline__ SoftStat soft_merge(SoftStat a, SoftStat b) {
  const float M = fmaxf(a.m, b.m);
  if (M == -INFINITY) return a;
  const float ea = expf(a.m - M), eb = expf(b.m - M);
  return {M, a.s * ea + b.s * eb, a.t * ea + b.t * eb};
}

// Next-token CE statistics of one token row in one pass over the logits (and their
// tangent): lse = m + log s, pf = sum_c p_c f'_c = t / s, then l = lse - f_y and
// l' = pf - f'_y.  Fixed reduction order (lanes, then warps), so results are deterministic.
__global__ void ce_stats_kernel(int S, int V, const int* __restrict__ ids,
                                const float* __restrict__ F, const float* __restrict__ Fd,
                                float* __restrict__ lse, float* __restrict__ l,
                                float* __restrict__ pf, float* __restrict__ ld, int* status) {
  pdl_entry();
  const int r = blockIdx.x;
  const int b = r / S, s = r % S;
  int y = ids[static_cast<int64_t>(b) * (S + 1) + s + 1];
  if (y < 0 || y >= V) {
    if (threadIdx.x == 0 && status) atomicMax(status, 1);
    y = 0;
  }
  const float* f = F + static_cast<int64_t>(r) * V;
  const float* fd = Fd ? Fd + static_cast<int64_t>(r) * V : nullptr;
  SoftStat st{-INFINITY, 0.f, 0.f};
  auto add = [&](float x, float xd) {
    if (x > st.m) {
      const float sc = expf(st.m - x);
      st.s *= sc;
      st.t *= sc;
      st.m = x;
    }
    const float e = expf(x - st.m);
    st.s += e;
    st.t += e * xd;
  };
  // rows are V floats with V a multiple of 8 (validated), so float4 loads stay aligned
  for (int c = threadIdx.x * 4; c < V; c += blockDim.x * 4) {
    const float4 x = *reinterpret_cast<const float4*>(f + c);
    float4 xd = make_float4(0.f, 0.f, 0.f, 0.f);
    if (fd) xd = *reinterpret_cast<const float4*>(fd + c);
    add(x.x, xd.x); add(x.y, xd.y); add(x.z, xd.z); add(x.w, xd.w);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const SoftStat q{__shfl_xor_sync(0xffffffffu, st.m, o), __shfl_xor_sync(0xffffffffu, st.s, o),
                     __shfl_xor_sync(0xffffffffu, st.t, o)};
    st = soft_merge(st, q);
  }
  __shared__ SoftStat red[32];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  if (lane == 0) red[w] = st;
  __syncthreads();
  if (threadIdx.x == 0) {
    SoftStat tot = red[0];
    for (int k = 1; k < nw; ++k) tot = soft_merge(tot, red[k]);
    const float lz = tot.m + logf(tot.s);
    lse[r] = lz;
    l[r] = lz - f[y];
    if (fd) {
      const float p_f = tot.t / tot.s;
      pf[r] = p_f;
      ld[r] = p_f - fd[y];
    }
  }
}

// Cross-entropy seeds over a [rows x V] tile grid: dF = c (p - onehot), dF' = c p (f' - p.f'),
// with c = w_b / (B S).  Writes row-major [N][ldo].
template <typename T>
__global__ void ce_seed_kernel(int S, int V, const int* __restrict__ ids,
                               const float* __restrict__ F, const float* __restrict__ Fd,
                               const float* __restrict__ lse, const float* __restrict__ pf,
                               const float* __restrict__ eta_w, const float* __restrict__ ex_w,
                               float inv_norm, T* __restrict__ dF, T* __restrict__ dFd, int ldo) {
  // four consecutive logits per thread (V and ldo multiples of 8): 16-byte loads
  pdl_entry();
  const int r = blockIdx.y;
  const int b = r / S, s = r % S;
  const int y = ids[static_cast<int64_t>(b) * (S + 1) + s + 1];
  float w = 1.f;
  if (ex_w) w = ex_w[b];
  else if (eta_w) w = 1.f / (1.f + expf(-eta_w[b]));
  const float c = w * inv_norm;
  const float lz = lse[r];
  const float pfr = Fd ? pf[r] : 0.f;
  const int64_t orow = static_cast<int64_t>(r) * V, drow = static_cast<int64_t>(r) * ldo;
  for (int col = 4 * (blockIdx.x * blockDim.x + threadIdx.x); col < V;
       col += 4 * gridDim.x * blockDim.x) {
    const float4 f = *reinterpret_cast<const float4*>(F + orow + col);
    const float p0 = expf(f.x - lz), p1 = expf(f.y - lz), p2 = expf(f.z - lz), p3 = expf(f.w - lz);
    store4<T>(dF + drow + col, c * (p0 - (col == y ? 1.f : 0.f)),
              c * (p1 - (col + 1 == y ? 1.f : 0.f)), c * (p2 - (col + 2 == y ? 1.f : 0.f)),
              c * (p3 - (col + 3 == y ? 1.f : 0.f)));
    if (Fd) {
      const float4 fd = *reinterpret_cast<const float4*>(Fd + orow + col);
      store4<T>(dFd + drow + col, c * p0 * (fd.x - pfr), c * p1 * (fd.y - pfr),
                c * p2 * (fd.z - pfr), c * p3 * (fd.w - pfr));
    }
  }
}

// Per-sequence reductions, one warp per sequence: l_b = mean_s l_bs, l'_b = mean_s l'_bs;
// d eta_b = sigmoid'(eta_b) l'_b / B; optional outputs.
__global__ void seq_reduce_kernel(int B, int S, const float* __restrict__ l,
                                  const float* __restrict__ ld, const float* __restrict__ eta_w,
                                  float invB, float* __restrict__ l_seq, float* __restrict__ ld_seq,
                                  float* __restrict__ d_eta) {
  pdl_entry();
  const int warps = blockDim.x >> 5;
  const int b = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= B) return;
  float a = 0.f, ad = 0.f;
  for (int s = lane; s < S; s += 32) {
    a += l[static_cast<int64_t>(b) * S + s];
    if (ld) ad += ld[static_cast<int64_t>(b) * S + s];
  }
  a = warp_sum(a) / static_cast<float>(S);
  ad = warp_sum(ad) / static_cast<float>(S);
  if (lane == 0) {
    if (l_seq) l_seq[b] = a;
    if (ld_seq) ld_seq[b] = ad;
    if (d_eta && eta_w) {
      const float sg = 1.f / (1.f + expf(-eta_w[b]));
      d_eta[b] = sg * (1.f - sg) * ad * invB;
    }
  }
}

// ---- deterministic embedding scatter-add --------------------------------------------------
__global__ void token_count_kernel(int N, int S, int V, const int* __restrict__ ids,
                                   int* __restrict__ count) {
  pdl_entry();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= N) return;
  int id = ids[static_cast<int64_t>(r / S) * (S + 1) + r % S];
  if (id < 0 || id >= V) id = 0;
  atomicAdd(&count[id], 1);
}

// Exclusive scan of count[0..V) into start[0..V] (one block of SCAN_THREADS).  Thread t owns
// the run [t per, (t + 1) per): it adds the run (eight independent loads at a time), the block
// scans the run totals with warp shuffles, and the thread writes its run's starts.
constexpr int SCAN_THREADS = 1024;

__device__ __forceinline__ int warp_incl_scan(int v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  return v;
}

__global__ void __launch_bounds__(SCAN_THREADS) scan_kernel(int V, const int* __restrict__ count,
                                                            int* __restrict__ start) {
  pdl_entry();
  __shared__ int wtot[SCAN_THREADS / 32];
  const int per = (V + SCAN_THREADS - 1) / SCAN_THREADS;
  const int b0 = threadIdx.x * per, b1 = min(V, b0 + per);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int run = 0;
  for (int i0 = b0; i0 < b1; i0 += 8) {
    int v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = i0 + k < b1 ? count[i0 + k] : 0;
#pragma unroll
    for (int k = 0; k < 8; ++k) run += v[k];
  }
  const int inc = warp_incl_scan(run, lane);
  if (lane == 31) wtot[w] = inc;
  __syncthreads();
  if (w == 0) wtot[lane] = warp_incl_scan(wtot[lane], lane);   // 32 warps
  __syncthreads();
  int acc = inc - run + (w > 0 ? wtot[w - 1] : 0);
  if (threadIdx.x == 0) start[V] = wtot[SCAN_THREADS / 32 - 1];
  for (int i0 = b0; i0 < b1; i0 += 8) {
    int v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = i0 + k < b1 ? count[i0 + k] : 0;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (i0 + k < b1) start[i0 + k] = acc;
      acc += v[k];
    }
  }
}

// Placement in two steps: every token takes a free slot of its id's segment (atomic, any
// order), then each segment is put in position order (stable, deterministic): an entry's
// rank is the number of entries of the segment at earlier positions.
__global__ void token_scatter_kernel(int N, int S, int V, const int* __restrict__ ids,
                                     const int* __restrict__ start, int* __restrict__ count,
                                     int* __restrict__ tmp) {
  pdl_entry();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= N) return;
  int id = ids[static_cast<int64_t>(r / S) * (S + 1) + r % S];
  if (id < 0 || id >= V) id = 0;
  const int slot = atomicSub(&count[id], 1) - 1;
  tmp[start[id] + slot] = r;
}

// Ids are dealt to blocks with a stride of gridDim.x (block b takes ids b, b + G, b + 2G, ...),
// so that the most frequent ids (the smallest, under a Zipf law) land in different blocks,
// and a block stages the segment bounds of ID_BATCH of its ids at a time.
constexpr int ID_BATCH = 256;

__device__ __forceinline__ int stage_bounds(const int* __restrict__ start, int b, int G, int k0,
                                            int nb, int* s_a, int* s_n) {
  __syncthreads();   // the previous batch's bounds are no longer read
  if (threadIdx.x < nb) {
    const int v = b + (k0 + static_cast<int>(threadIdx.x)) * G;
    const int a = start[v];
    s_a[threadIdx.x] = a;
    s_n[threadIdx.x] = start[v + 1] - a;
  }
  __syncthreads();
  return nb;
}

// Each segment of the scattered positions is put in position order: an entry's rank is the
// number of entries of the segment at earlier positions.  Segments of up to 32 entries take
// one warp (ranks by shuffles); longer ones the block, through a bitmap of the positions
// (rank = set bits below the position) when the batch has at most 32 ORD_BM_WORDS tokens, by
// direct counting otherwise.
constexpr int ORD_BM_WORDS = 2048;

__global__ void __launch_bounds__(256) token_order_kernel(int V, int N, const int* __restrict__ start,
                                                          const int* __restrict__ tmp,
                                                          int* __restrict__ order) {
  pdl_entry();
  __shared__ int s_a[ID_BATCH], s_n[ID_BATCH];
  __shared__ unsigned bm[ORD_BM_WORDS];
  __shared__ int wpre[ORD_BM_WORDS];
  __shared__ int wtot[8];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, b = blockIdx.x;
  const int nmine = (V - b + G - 1) / G;
  const bool use_bm = N <= 32 * ORD_BM_WORDS;
  const int nw = (N + 31) >> 5;
  const int per = (nw + 255) / 256;   // bitmap words per thread in the prefix count
  for (int k0 = 0; k0 < nmine; k0 += ID_BATCH) {
    const int nb = stage_bounds(start, b, G, k0, min(ID_BATCH, nmine - k0), s_a, s_n);
    for (int i = w; i < nb; i += 8) {
      const int L = s_n[i];
      if (L == 0 || L > 32) continue;
      const int a = s_a[i];
      const int pi = lane < L ? tmp[a + lane] : 0;
      int rank = 0;
      for (int k = 0; k < L; ++k) rank += __shfl_sync(0xffffffffu, pi, k) < pi ? 1 : 0;
      if (lane < L) order[a + rank] = pi;
    }
    for (int i = 0; i < nb; ++i) {
      const int L = s_n[i];   // uniform across the block
      if (L <= 32) continue;
      const int a = s_a[i];
      if (!use_bm) {
        for (int j = threadIdx.x; j < L; j += blockDim.x) {
          const int pi = tmp[a + j];
          int rank = 0;
          for (int k = 0; k < L; ++k) rank += tmp[a + k] < pi ? 1 : 0;
          order[a + rank] = pi;
        }
        continue;
      }
      for (int j = threadIdx.x; j < nw; j += blockDim.x) bm[j] = 0u;
      __syncthreads();
      for (int j = threadIdx.x; j < L; j += blockDim.x) {
        const int pi = tmp[a + j];
        atomicOr(&bm[pi >> 5], 1u << (pi & 31));
      }
      __syncthreads();
      // exclusive prefix of the words' bit counts: thread t owns words [t per, (t + 1) per)
      const int j0 = threadIdx.x * per, j1 = min(nw, j0 + per);
      int run = 0;
      for (int j = j0; j < j1; ++j) run += __popc(bm[j]);
      const int inc = warp_incl_scan(run, lane);
      if (lane == 31) wtot[w] = inc;
      __syncthreads();
      int acc = inc - run;
      for (int k = 0; k < w; ++k) acc += wtot[k];
      for (int j = j0; j < j1; ++j) {
        wpre[j] = acc;
        acc += __popc(bm[j]);
      }
      __syncthreads();
      for (int j = threadIdx.x; j < L; j += blockDim.x) {
        const int pi = tmp[a + j];
        const int wd = pi >> 5;
        order[a + wpre[wd] + __popc(bm[wd] & ((1u << (pi & 31)) - 1u))] = pi;
      }
      __syncthreads();   // bm, wpre and wtot are reused by the next segment
    }
  }
}

// Embedding gradient: row v of dE is the sum of dx over the tokens with id v, in token order
// (start/order from the counting sort).  blockIdx.y picks a slice of EB_SLICE columns (one
// float4 per lane); ids are dealt to blocks with a stride (as in token_order_kernel).  A
// segment of more than EB_WARP tokens is split by the block's eight warps into contiguous
// parts, each summed in order, and the parts are added in warp order; a shorter segment (and
// the zero row of an id absent from the batch) takes one warp, which adds its rows in order,
// the same sums since each of the eight parts would hold at most one row.  Deterministic.
constexpr int EB_SLICE = 128;
constexpr int EB_WARP = 8;

__device__ __forceinline__ void add4(float4& a, const float4& b) {
  a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
}

__device__ __forceinline__ void put_row4(float* out, int64_t off, const float4& v, bool vec_out) {
  if (vec_out) {
    *reinterpret_cast<float4*>(out + off) = v;
  } else {   // the caller's gradient buffer need not be 16-byte aligned
    out[off] = v.x; out[off + 1] = v.y; out[off + 2] = v.z; out[off + 3] = v.w;
  }
}

__global__ void __launch_bounds__(256) embed_bwd_kernel(int V, int d, const int* __restrict__ start,
                                                        const int* __restrict__ order,
                                                        const float* __restrict__ dx,
                                                        const float* __restrict__ dxd,
                                                        float* __restrict__ dE,
                                                        float* __restrict__ dEd, bool vec_out) {
  pdl_entry();
  __shared__ float4 part[2][8][32];
  __shared__ int s_a[ID_BATCH], s_n[ID_BATCH];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.y * EB_SLICE + lane * 4;
  const bool col = c < d;
  const int G = gridDim.x, b = blockIdx.x;
  const int nmine = (V - b + G - 1) / G;
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int k0 = 0; k0 < nmine; k0 += ID_BATCH) {
    const int nb = stage_bounds(start, b, G, k0, min(ID_BATCH, nmine - k0), s_a, s_n);
    for (int i = w; i < nb; i += 8) {
      const int cnt = s_n[i];
      if (cnt > EB_WARP) continue;
      const int a = s_a[i];
      const int mine = lane < cnt ? order[a + lane] : 0;
      float4 acc = zero, dacc = zero;
      for (int t = 0; t < cnt; ++t) {
        const int64_t ro = static_cast<int64_t>(__shfl_sync(0xffffffffu, mine, t)) * d + c;
        if (col) {
          add4(acc, ld4f(dx + ro));
          if (dxd) add4(dacc, ld4f(dxd + ro));
        }
      }
      if (col) {
        const int64_t off = static_cast<int64_t>(b + (k0 + i) * G) * d + c;
        if (dE) put_row4(dE, off, acc, vec_out);
        if (dEd) put_row4(dEd, off, dacc, vec_out);
      }
    }
    for (int i = 0; i < nb; ++i) {
      const int cnt = s_n[i];   // uniform across the block
      if (cnt <= EB_WARP) continue;
      const int a = s_a[i];
      const int r0 = a + (w * cnt) / 8, r1 = a + ((w + 1) * cnt) / 8;
      float4 acc = zero, dacc = zero;
      // the row indices of 32 rows at a time, one per lane, broadcast by shuffles, so a row's
      // loads do not wait on its index load
      for (int kb = r0; kb < r1; kb += 32) {
        const int mine = kb + lane < r1 ? order[kb + lane] : 0;
        const int nr = r1 - kb < 32 ? r1 - kb : 32;
#pragma unroll 4
        for (int t = 0; t < nr; ++t) {
          const int64_t ro = static_cast<int64_t>(__shfl_sync(0xffffffffu, mine, t)) * d + c;
          if (col) {
            add4(acc, ld4f(dx + ro));
            if (dxd) add4(dacc, ld4f(dxd + ro));
          }
        }
      }
      part[0][w][lane] = acc;
      part[1][w][lane] = dacc;
      __syncthreads();
      if (threadIdx.x < 64) {
        const int which = threadIdx.x >> 5, l = threadIdx.x & 31;
        const int cc = blockIdx.y * EB_SLICE + l * 4;
        float4 t = part[which][0][l];
        for (int r = 1; r < 8; ++r) add4(t, part[which][r][l]);
        float* out = which == 0 ? dE : dEd;
        if (out && cc < d) put_row4(out, static_cast<int64_t>(b + (k0 + i) * G) * d + cc, t, vec_out);
      }
      __syncthreads();
    }
  }
}

// Row-major cast (with a leading dimension) float32 -> T.
template <typename T>
__global__ void cast_rows_kernel(const float* __restrict__ X, int rows, int cols, T* __restrict__ Y,
                                 int ldy) {
  pdl_entry();
  const int64_t n = static_cast<int64_t>(rows) * cols;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / cols, c = i % cols;
    Y[r * ldy + c] = to_t<T>(X[i]);
  }
}

int blocks_for(int64_t n) {
  int64_t b = (n + 255) / 256;
  if (b > ROW_SMS * 16) b = ROW_SMS * 16;
  return static_cast<int>(b < 1 ? 1 : b);
}

}  // namespace

// ---- launchers -------------------------------------------------------------------------------
void dec_embed_fwd(int N, int S, int d, int V, const int* ids, const float* E, const float* UE,
                   float* x, float* xd, int* status, cudaStream_t s) {
  launch_k(embed_fwd_kernel, dim3(N), dim3(256), 0, s, ids, S, d, V, E, UE, x, xd, status);
}

template <typename T>
void dec_rmsnorm_fwd(int N, int d, float eps, const float* x_in, const float* y, const float* xd_in,
                     const float* yd, const float* g, const float* gd, float* x_out, float* xd_out,
                     float* r, float* rd, T* h, T* hd, int ldh, cudaStream_t s) {
  uintptr_t any = reinterpret_cast<uintptr_t>(x_in) | reinterpret_cast<uintptr_t>(y) |
                  reinterpret_cast<uintptr_t>(xd_in) | reinterpret_cast<uintptr_t>(yd) |
                  reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(gd) |
                  reinterpret_cast<uintptr_t>(x_out) | reinterpret_cast<uintptr_t>(xd_out) |
                  reinterpret_cast<uintptr_t>(h) | reinterpret_cast<uintptr_t>(hd);
  if ((any & 15) == 0 && (d & 3) == 0 && (ldh & 7) == 0) {
    launch_k(rmsnorm_fwd_warp_kernel<T>, dim3((N + 7) / 8), dim3(256), 0, s, N, d, eps, x_in, y,
             xd_in, yd, g, gd, x_out, xd_out, r, rd, h, hd, ldh);
    return;
  }
  launch_k(rmsnorm_fwd_kernel<T>, dim3(N), dim3(256), 0, s, d, eps, x_in, y, xd_in, yd, g, gd, x_out, xd_out, r, rd,
                                          h, hd, ldh);
}

// RMSNorm backward (dx += ...) and, when dg or dg' is wanted, the gain gradient; returns the
// number of kernels launched.  The warp-per-row kernel writes the gain's partial sums of
// eight rows per block itself; the block-per-row fallback takes the separate column pass.
int dec_gain_chunks(int N) { return (N + 7) / 8; }

template <typename T>
int dec_rmsnorm_bwd(int N, int d, const float* x, const float* xd, const float* r, const float* rd,
                    const float* g, const float* gd, const float* dy, const float* dyd, float* dx,
                    float* dxd, float* dg, float* dgd, float* part, cudaStream_t s, T* dxb,
                    T* dxdb) {
  const bool gain = dg || (dyd && dgd);
  uintptr_t any = reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(xd) |
                  reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(gd) |
                  reinterpret_cast<uintptr_t>(dy) | reinterpret_cast<uintptr_t>(dyd) |
                  reinterpret_cast<uintptr_t>(dx) | reinterpret_cast<uintptr_t>(dxd) |
                  reinterpret_cast<uintptr_t>(dxb) | reinterpret_cast<uintptr_t>(dxdb) |
                  reinterpret_cast<uintptr_t>(part);
  const dim3 fin_grid((d + 31) / 32), fin_block(32, GF_Y);
  if ((any & 15) == 0 && (d & 3) == 0) {
    const int nblk = (N + 7) / 8;
    float* pp = gain ? part : nullptr;
    float* ppd = gain && dyd ? part + static_cast<int64_t>(nblk) * d : nullptr;
    launch_k(rmsnorm_bwd_warp_kernel<T>, dim3(nblk), dim3(256), 0, s, N, d, x, xd, r, rd, g, gd,
             dy, dyd, dx, dxd, dxb, dxdb, pp, ppd);
    if (!gain) return 1;
    launch_k(gain_grad_final_kernel, fin_grid, fin_block, 0, s, nblk, d,
             static_cast<const float*>(pp), static_cast<const float*>(ppd), dg, dgd);
    return 2;
  }
  launch_k(rmsnorm_bwd_kernel<T>, dim3(N), dim3(256), 0, s, d, x, xd, r, rd, g, gd, dy, dyd, dx, dxd,
           dxb, dxdb);
  if (!gain) return 1;
  const int nchunk = (N + GG_ROWS - 1) / GG_ROWS;
  float* partd = dyd ? part + static_cast<int64_t>(nchunk) * d : nullptr;
  launch_k(gain_grad_partial_kernel, dim3((d + 31) / 32, nchunk), dim3(32, 8), 0, s, N, d, x, xd,
           r, rd, dy, dyd, part, partd);
  launch_k(gain_grad_final_kernel, fin_grid, fin_block, 0, s, nchunk, d,
           static_cast<const float*>(part), static_cast<const float*>(partd), dg, dgd);
  return 3;
}

void dec_rope_table(int S, int dh, float base, float* tab, cudaStream_t s) {
  const int n = S * (dh / 2);
  launch_k(rope_table_kernel, dim3((n + 255) / 256), dim3(256), 0, s, S, dh / 2, dh,
           static_cast<double>(base), tab);
}

template <typename T>
void dec_rope_split(int N, int S, int H, int dh, const float* rtab, float qscale, const float* qkv,
                    T* Q, T* K, T* V, cudaStream_t s) {
  launch_k(rope_split_kernel<T>, dim3(N), dim3(256), 0, s, S, H, dh, rtab, qscale, qkv, Q, K, V);
}

template <typename T>
void dec_rope_merge(int N, int S, int H, int dh, const float* rtab, float qscale, const float* dQ,
                    const float* dK, const float* dV, T* out, int ldo, cudaStream_t s) {
  launch_k(rope_merge_kernel<T>, dim3(N), dim3(256), 0, s, S, H, dh, rtab, qscale, dQ, dK, dV, out, ldo);
}

template <typename T>
void dec_head_merge(int N, int S, int H, int dh, const float* O, T* out, int ldo, cudaStream_t s) {
  launch_k(head_merge_kernel<T>, dim3(N), dim3(256), 0, s, S, H, dh, O, out, ldo);
}

template <typename T>
void dec_head_split(int N, int S, int H, int dh, const float* X, T* out, cudaStream_t s) {
  launch_k(head_split_kernel<T>, dim3(N), dim3(256), 0, s, S, H, dh, X, out);
}

template <typename T>
void dec_softmax_fwd(int S, int rows, const float* Sc, const float* Scd, T* P, T* Pd,
                     cudaStream_t s) {
  launch_k(softmax_fwd_kernel<T>, dim3((rows + 7) / 8), dim3(256), 0, s, S, rows, Sc, Scd, P, Pd);
}

template <typename T>
void dec_softmax_bwd(int S, int rows, const T* P, const T* Pd, const float* dP, const float* dPd,
                     T* dS, T* dSd, cudaStream_t s) {
  launch_k(softmax_bwd_kernel<T>, dim3((rows + 7) / 8), dim3(256), 0, s, S, rows, P, Pd, dP, dPd, dS, dSd);
}

void dec_ce_stats(int N, int S, int V, const int* ids, const float* F, const float* Fd, float* lse,
                  float* l, float* pf, float* ld, int* status, cudaStream_t s) {
  launch_k(ce_stats_kernel, dim3(N), dim3(512), 0, s, S, V, ids, F, Fd, lse, l, pf, ld, status);
}

template <typename T>
void dec_ce_seed(int N, int S, int V, const int* ids, const float* F, const float* Fd,
                 const float* lse, const float* pf, const float* eta_w, const float* ex_w,
                 float inv_norm, T* dF, T* dFd, int ldo, cudaStream_t s) {
  dim3 grid((V + 1023) / 1024 > 8 ? 8 : (V + 1023) / 1024, N);
  launch_k(ce_seed_kernel<T>, dim3(grid), dim3(256), 0, s, S, V, ids, F, Fd, lse, pf, eta_w, ex_w, inv_norm, dF, dFd,
                                         ldo);
}

void dec_seq_reduce(int B, int S, const float* l, const float* ld, const float* eta_w, float invB,
                    float* l_seq, float* ld_seq, float* d_eta, cudaStream_t s) {
  launch_k(seq_reduce_kernel, dim3((B + 7) / 8), dim3(256), 0, s, B, S, l, ld, eta_w, invB, l_seq, ld_seq, d_eta);
}

void dec_token_csr(int N, int S, int V, const int* ids, int* count, int* start, int* order,
                   int* tmp, cudaStream_t s) {
  cudaMemsetAsync(count, 0, sizeof(int) * V, s);
  launch_k(token_count_kernel, dim3((N + 255) / 256), dim3(256), 0, s, N, S, V, ids, count);
  launch_k(scan_kernel, dim3(1), dim3(SCAN_THREADS), 0, s, V, count, start);
  launch_k(token_scatter_kernel, dim3((N + 255) / 256), dim3(256), 0, s, N, S, V, ids, start,
           count, tmp);
  // two blocks per SM, each over V / grid ids
  launch_k(token_order_kernel, dim3(V < 2 * ROW_SMS ? V : 2 * ROW_SMS), dim3(256), 0, s, V, N,
           start, static_cast<const int*>(tmp), order);
}

void dec_embed_bwd(int V, int d, const int* start, const int* order, const float* dx,
                   const float* dxd, float* dE, float* dEd, cudaStream_t s) {
  const bool vec_out = ((reinterpret_cast<uintptr_t>(dE) | reinterpret_cast<uintptr_t>(dEd)) & 15) == 0;
  // about eight blocks per SM over all column slices
  const int slices = (d + EB_SLICE - 1) / EB_SLICE;
  int gx = 8 * ROW_SMS / slices;
  gx = gx < 1 ? 1 : gx > V ? V : gx;
  launch_k(embed_bwd_kernel, dim3(gx, slices), dim3(256), 0, s, V, d, start, order, dx, dxd, dE,
           dEd, vec_out);
}

template <typename T>
void cast_rows(const float* X, int rows, int cols, T* Y, int ldy, cudaStream_t s) {
  launch_k(cast_rows_kernel<T>, dim3(blocks_for(static_cast<int64_t>(rows) * cols)), dim3(256), 0, s, X, rows, cols, Y, ldy);
}

#define MF_DEC_INST(T)                                                                            \
  template void dec_rmsnorm_fwd<T>(int, int, float, const float*, const float*, const float*,      \
                                   const float*, const float*, const float*, float*, float*,       \
                                   float*, float*, T*, T*, int, cudaStream_t);                     \
  template int dec_rmsnorm_bwd<T>(int, int, const float*, const float*, const float*,              \
                                  const float*, const float*, const float*, const float*,          \
                                  const float*, float*, float*, float*, float*, float*,            \
                                  cudaStream_t, T*, T*);                                           \
  template void dec_rope_split<T>(int, int, int, int, const float*, float, const float*, T*, T*, T*,      \
                                  cudaStream_t);                                                   \
  template void dec_rope_merge<T>(int, int, int, int, const float*, float, const float*, const float*,    \
                                  const float*, T*, int, cudaStream_t);                            \
  template void dec_head_merge<T>(int, int, int, int, const float*, T*, int, cudaStream_t);       \
  template void dec_head_split<T>(int, int, int, int, const float*, T*, cudaStream_t);            \
  template void dec_softmax_fwd<T>(int, int, const float*, const float*, T*, T*, cudaStream_t);   \
  template void dec_softmax_bwd<T>(int, int, const T*, const T*, const float*, const float*, T*,  \
                                   T*, cudaStream_t);                                              \
  template void dec_ce_seed<T>(int, int, int, const int*, const float*, const float*,              \
                               const float*, const float*, const float*, const float*, float, T*,  \
                               T*, int, cudaStream_t);                                             \
  template void cast_rows<T>(const float*, int, int, T*, int, cudaStream_t);
MF_DEC_INST(float)
MF_DEC_INST(__nv_bfloat16)
#undef MF_DEC_INST

}  // namespace mf
