// Fused causal attention with its forward tangent and the tangent of its backward (the
// dual attention of the transformer HVP), without materialising the S x S probabilities.
//
// Per head, with q pre-scaled by 1/sqrt(d_head):
//   S = Q K^T, P = softmax(S) (causal), O = P V
//   tangent: S' = Q' K^T + Q K'^T, P' = P (*) (S' - rbar), rbar = rowsum(P (*) S'),
//            O' = P' V + P V'
//   backward: dP = dO V^T, D = rowsum(dO (*) O), dS = P (*) (dP - D),
//             dQ = dS K, dK = dS^T Q, dV = P^T dO
//   its tangent: dP' = dO' V^T + dO V'^T, D' = rowsum(dO' (*) O + dO (*) O'),
//             dS' = P' (*) (dP - D) + P (*) (dP' - D'),
//             dQ' = dS' K + dS K', dK' = dS'^T Q + dS^T Q', dV' = P'^T dO + P^T dO'.
// The forward keeps per query row only lse = m + log l and rbar; the backward rebuilds P and
// P' tile by tile from them.  O' comes out of the online softmax as A/l - rbar O + B/l with
// A = sum (P (*) S') V and B = sum P V' accumulated next to O.
//
// Tiles: 64 queries x 64 keys, head dimension 64, one CTA of four warps per (head, tile);
// each warp owns 16 rows.  Operands are staged in shared memory by cp.async (rows padded to
// 72 elements so ldmatrix is conflict free) and multiplied with warp-level mma.sync
// m16n8k16 (bf16 in, float32 accumulate).  The backward runs as two kernels, one per key tile
// (dK, dV and tangents) and one per query tile (dQ and tangent), so every sum has a fixed
// order and results are deterministic.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "internal.h"
#include "launch.cuh"

namespace mf {
namespace {

constexpr int FT = 64;        // tile rows (queries or keys)
constexpr int FDH = 64;       // head dimension
constexpr int LDS = 72;       // shared-memory row stride (elements)
constexpr int TILE_ELEMS = FT * LDS;
constexpr int FTHREADS = 128;
using bf16 = __nv_bfloat16;

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void ldsm4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}

__device__ __forceinline__ void ldsm4t(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}

__device__ __forceinline__ void mma(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                    uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// A fragment (16 rows x 16 k) of a row-major tile: rows r0.., columns k0..
__device__ __forceinline__ void frag_a(uint32_t (&a)[4], const bf16* t, int r0, int k0) {
  const int l = threadIdx.x & 31;
  ldsm4(a, su32(t + (r0 + (l & 7) + ((l >> 3) & 1) * 8) * LDS + k0 + (l >> 4) * 8));
}

// B fragments of two 8-wide n tiles (n0.., n0+8..) x 16 k, from a tile stored [n][k]
__device__ __forceinline__ void frag_b_nk(uint32_t (&b)[4], const bf16* t, int n0, int k0) {
  const int l = threadIdx.x & 31;
  ldsm4(b, su32(t + (n0 + (l & 7) + (l >> 4) * 8) * LDS + k0 + ((l >> 3) & 1) * 8));
}

// the same from a tile stored [k][n]
__device__ __forceinline__ void frag_b_kn(uint32_t (&b)[4], const bf16* t, int k0, int n0) {
  const int l = threadIdx.x & 31;
  ldsm4t(b, su32(t + (k0 + (l & 7) + ((l >> 3) & 1) * 8) * LDS + n0 + (l >> 4) * 8));
}

// Accumulator pair (two 8-wide n tiles of 16 rows) as an A fragment with k = those 16 columns.
__device__ __forceinline__ void c_to_a(uint32_t (&a)[4], const float (&c0)[4], const float (&c1)[4]) {
  a[0] = pack(c0[0], c0[1]);
  a[1] = pack(c0[2], c0[3]);
  a[2] = pack(c1[0], c1[1]);
  a[3] = pack(c1[2], c1[3]);
}

// Stage a 64 x 64 bf16 tile (rows row0.. of a [S][64] head) into shared memory.
__device__ __forceinline__ void load_tile(bf16* t, const bf16* g, int row0) {
  const bf16* src = g + static_cast<int64_t>(row0) * FDH;
  for (int i = threadIdx.x; i < FT * (FDH / 8); i += FTHREADS) {
    const int r = i >> 3, c = (i & 7) * 8;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n"
                 :: "r"(su32(t + r * LDS + c)), "l"(src + r * FDH + c));
  }
}

__device__ __forceinline__ void cp_wait_all() {
  asm volatile("cp.async.commit_group;\n" ::);
  asm volatile("cp.async.wait_group 0;\n" ::);
}

__device__ __forceinline__ float quad_max(float v) {
  v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
  return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}

__device__ __forceinline__ float quad_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

// ---- forward ------------------------------------------------------------------------------
template <bool DUAL>
__global__ void __launch_bounds__(FTHREADS) flash_fwd_kernel(const FlashArgs a) {
  pdl_entry();
  extern __shared__ __align__(16) unsigned char fsm[];
  bf16* Qs = reinterpret_cast<bf16*>(fsm);
  bf16* Ks = Qs + TILE_ELEMS;
  bf16* Vs = Ks + TILE_ELEMS;
  bf16* Qds = Vs + TILE_ELEMS;     // dual only
  bf16* Kds = Qds + TILE_ELEMS;
  bf16* Vds = Kds + TILE_ELEMS;
  const int nq = a.S / FT;
  // grid (heads, tiles): blocks dispatch heads fastest, so every head's longest query tile
  // goes first and the shortest ones fill the tail of the launch
  const int qt = nq - 1 - static_cast<int>(blockIdx.y);
  const int bh = blockIdx.x;
  const int64_t hoff = static_cast<int64_t>(bh) * a.S * FDH;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r0 = w * 16;
  load_tile(Qs, a.Q + hoff, qt * FT);
  if (DUAL) load_tile(Qds, a.Qd + hoff, qt * FT);
  cp_wait_all();
  __syncthreads();
  uint32_t qf[4][4], qdf[4][4];
#pragma unroll
  for (int ks = 0; ks < 4; ++ks) {
    frag_a(qf[ks], Qs, r0, ks * 16);
    if (DUAL) frag_a(qdf[ks], Qds, r0, ks * 16);
  }
  float m[2] = {-INFINITY, -INFINITY}, lsum[2] = {0.f, 0.f}, rsum[2] = {0.f, 0.f};
  float o[8][4], oa[8][4], ob[8][4];
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) { o[n][e] = 0.f; oa[n][e] = 0.f; ob[n][e] = 0.f; }
  const int qrow0 = qt * FT + r0 + (lane >> 2);   // this thread's rows: qrow0, qrow0 + 8
  for (int kt = 0; kt <= qt; ++kt) {
    __syncthreads();
    load_tile(Ks, a.K + hoff, kt * FT);
    load_tile(Vs, a.V + hoff, kt * FT);
    if (DUAL) {
      load_tile(Kds, a.Kd + hoff, kt * FT);
      load_tile(Vds, a.Vd + hoff, kt * FT);
    }
    cp_wait_all();
    __syncthreads();
    float s[8][4], sd[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) { s[n][e] = 0.f; sd[n][e] = 0.f; }
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b[4];
        frag_b_nk(b, Ks, np * 16, ks * 16);
        mma(s[2 * np], qf[ks], b[0], b[1]);
        mma(s[2 * np + 1], qf[ks], b[2], b[3]);
        if (DUAL) {
          mma(sd[2 * np], qdf[ks], b[0], b[1]);
          mma(sd[2 * np + 1], qdf[ks], b[2], b[3]);
          uint32_t bd[4];
          frag_b_nk(bd, Kds, np * 16, ks * 16);
          mma(sd[2 * np], qf[ks], bd[0], bd[1]);
          mma(sd[2 * np + 1], qf[ks], bd[2], bd[3]);
        }
      }
    }
    // causal mask on the diagonal tile, then the online softmax of both rows
    if (kt == qt) {
#pragma unroll
      for (int n = 0; n < 8; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kt * FT + n * 8 + (lane & 3) * 2 + (e & 1);
          const int q = qrow0 + (e >> 1) * 8;
          if (key > q) s[n][e] = -INFINITY;
        }
    }
    float scale[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float mx = -INFINITY;
#pragma unroll
      for (int n = 0; n < 8; ++n) mx = fmaxf(mx, fmaxf(s[n][2 * h], s[n][2 * h + 1]));
      mx = quad_max(mx);
      const float mn = fmaxf(m[h], mx);
      scale[h] = __expf(m[h] - mn);
      m[h] = mn;
    }
    float ls[2] = {0.f, 0.f}, rs[2] = {0.f, 0.f};
#pragma unroll
    for (int n = 0; n < 8; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int h = e >> 1;
        const float p = __expf(s[n][e] - m[h]);
        s[n][e] = p;
        ls[h] += p;
        if (DUAL) {
          sd[n][e] *= p;     // P (*) S' (unnormalised)
          rs[h] += sd[n][e];
        }
      }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      lsum[h] = lsum[h] * scale[h] + quad_sum(ls[h]);
      if (DUAL) rsum[h] = rsum[h] * scale[h] + quad_sum(rs[h]);
    }
#pragma unroll
    for (int n = 0; n < 8; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        o[n][e] *= scale[e >> 1];
        if (DUAL) { oa[n][e] *= scale[e >> 1]; ob[n][e] *= scale[e >> 1]; }
      }
    // O += P V ; A += (P (*) S') V ; B += P V'
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t pa[4], psa[4];
      c_to_a(pa, s[2 * kk], s[2 * kk + 1]);
      if (DUAL) c_to_a(psa, sd[2 * kk], sd[2 * kk + 1]);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b[4];
        frag_b_kn(b, Vs, kk * 16, np * 16);
        mma(o[2 * np], pa, b[0], b[1]);
        mma(o[2 * np + 1], pa, b[2], b[3]);
        if (DUAL) {
          mma(oa[2 * np], psa, b[0], b[1]);
          mma(oa[2 * np + 1], psa, b[2], b[3]);
          uint32_t bd[4];
          frag_b_kn(bd, Vds, kk * 16, np * 16);
          mma(ob[2 * np], pa, bd[0], bd[1]);
          mma(ob[2 * np + 1], pa, bd[2], bd[3]);
        }
      }
    }
  }
  // O = o / l ; rbar = r / l ; O' = A / l - rbar O + B / l
  float inv[2], rb[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    inv[h] = 1.f / lsum[h];
    rb[h] = DUAL ? rsum[h] * inv[h] : 0.f;
  }
  // head-merged bf16 rows: token b*S + q, column hh*64 + e (see FlashArgs::Om)
  const int hb = a.H > 0 ? bh / a.H : 0, hh = a.H > 0 ? bh % a.H : 0;
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int col = n * 8 + (lane & 3) * 2;
      const int64_t off = hoff + static_cast<int64_t>(qrow0 + h * 8) * FDH + col;
      const int64_t moff = (static_cast<int64_t>(hb) * a.S + qrow0 + h * 8) * a.ldo + hh * FDH + col;
      const float o0 = o[n][2 * h] * inv[h], o1 = o[n][2 * h + 1] * inv[h];
      if (a.Om) *reinterpret_cast<uint32_t*>(a.Om + moff) = pack(o0, o1);
      else *reinterpret_cast<float2*>(a.O + off) = make_float2(o0, o1);
      if (DUAL) {
        const float d0 = (oa[n][2 * h] + ob[n][2 * h]) * inv[h] - rb[h] * o0;
        const float d1 = (oa[n][2 * h + 1] + ob[n][2 * h + 1]) * inv[h] - rb[h] * o1;
        if (a.Om) *reinterpret_cast<uint32_t*>(a.Omd + moff) = pack(d0, d1);
        else *reinterpret_cast<float2*>(a.Od + off) = make_float2(d0, d1);
      }
    }
  if ((lane & 3) == 0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t i = static_cast<int64_t>(bh) * a.S + qrow0 + h * 8;
      a.lse[i] = m[h] + __logf(lsum[h]);
      if (DUAL) a.rbar[i] = rb[h];
    }
  }
}

// ---- backward: dK, dV (and tangents), one CTA per key tile ----------------------------------
template <bool DUAL>
__global__ void __launch_bounds__(FTHREADS) flash_bwd_kv_kernel(const FlashArgs a) {
  pdl_entry();
  extern __shared__ __align__(16) unsigned char fsm[];
  bf16* Ks = reinterpret_cast<bf16*>(fsm);
  bf16* Vs = Ks + TILE_ELEMS;
  bf16* Qs = Vs + TILE_ELEMS;
  bf16* dOs = Qs + TILE_ELEMS;
  bf16* Kds = dOs + TILE_ELEMS;    // dual only
  bf16* Vds = Kds + TILE_ELEMS;
  bf16* Qds = Vds + TILE_ELEMS;
  bf16* dOds = Qds + TILE_ELEMS;
  float* st = reinterpret_cast<float*>(fsm + (DUAL ? 8 : 4) * TILE_ELEMS * sizeof(bf16));
  float* s_lse = st;               // [64] per query tile
  float* s_rb = st + FT;
  float* s_D = st + 2 * FT;
  float* s_Dd = st + 3 * FT;
  const int nt_ = a.S / FT;
  const int kt = static_cast<int>(blockIdx.y);     // grid (heads, tiles): longest first
  const int bh = blockIdx.x;
  const int64_t hoff = static_cast<int64_t>(bh) * a.S * FDH;
  const int64_t soff = static_cast<int64_t>(bh) * a.S;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kr0 = w * 16;                                 // this warp's 16 keys in the tile
  const int key0 = kt * FT + kr0 + (lane >> 2);           // thread's keys: key0, key0 + 8
  load_tile(Ks, a.K + hoff, kt * FT);
  load_tile(Vs, a.V + hoff, kt * FT);
  if (DUAL) {
    load_tile(Kds, a.Kd + hoff, kt * FT);
    load_tile(Vds, a.Vd + hoff, kt * FT);
  }
  float dv[8][4], dk[8][4], dvd[8][4], dkd[8][4];
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) { dv[n][e] = dk[n][e] = dvd[n][e] = dkd[n][e] = 0.f; }
  for (int qt = kt; qt < nt_; ++qt) {
    __syncthreads();
    load_tile(Qs, a.Q + hoff, qt * FT);
    load_tile(dOs, a.dO + hoff, qt * FT);
    if (DUAL) {
      load_tile(Qds, a.Qd + hoff, qt * FT);
      load_tile(dOds, a.dOd + hoff, qt * FT);
    }
    if (threadIdx.x < FT) {
      const int64_t i = soff + qt * FT + threadIdx.x;
      s_lse[threadIdx.x] = a.lse[i];
      s_D[threadIdx.x] = a.D[i];
      if (DUAL) { s_rb[threadIdx.x] = a.rbar[i]; s_Dd[threadIdx.x] = a.Dd[i]; }
    }
    cp_wait_all();
    __syncthreads();
#pragma unroll 1
    for (int c = 0; c < 4; ++c) {            // 16-query chunks
      const int q0 = c * 16;                 // within the query tile
      if (qt == kt && q0 + 15 < kr0) continue;   // every query of the chunk precedes every key
      // S^T (16 keys x 16 queries) and its tangent
      float sT[2][4] = {}, sdT[2][4] = {}, dpT[2][4] = {}, dpdT[2][4] = {};
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        uint32_t ka[4], b[4];
        frag_a(ka, Ks, kr0, ks * 16);
        frag_b_nk(b, Qs, q0, ks * 16);
        mma(sT[0], ka, b[0], b[1]);
        mma(sT[1], ka, b[2], b[3]);
        uint32_t va[4], bo[4];
        frag_a(va, Vs, kr0, ks * 16);
        frag_b_nk(bo, dOs, q0, ks * 16);
        mma(dpT[0], va, bo[0], bo[1]);
        mma(dpT[1], va, bo[2], bo[3]);
        if (DUAL) {
          uint32_t kda[4], bq[4];
          frag_a(kda, Kds, kr0, ks * 16);
          mma(sdT[0], kda, b[0], b[1]);
          mma(sdT[1], kda, b[2], b[3]);
          frag_b_nk(bq, Qds, q0, ks * 16);
          mma(sdT[0], ka, bq[0], bq[1]);
          mma(sdT[1], ka, bq[2], bq[3]);
          uint32_t vda[4], bod[4];
          frag_a(vda, Vds, kr0, ks * 16);
          mma(dpdT[0], vda, bo[0], bo[1]);
          mma(dpdT[1], vda, bo[2], bo[3]);
          frag_b_nk(bod, dOds, q0, ks * 16);
          mma(dpdT[0], va, bod[0], bod[1]);
          mma(dpdT[1], va, bod[2], bod[3]);
        }
      }
      // P^T, P'^T, dS^T, dS'^T (element: key = key0 + 8 (e >> 1), query = q0 + 8 n + ...)
      float pT[2][4], pdT[2][4], dsT[2][4], dsdT[2][4];
#pragma unroll
      for (int n = 0; n < 2; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int ql = q0 + n * 8 + (lane & 3) * 2 + (e & 1);
          const int key = key0 + (e >> 1) * 8;
          const int q = qt * FT + ql;
          const float p = q >= key ? __expf(sT[n][e] - s_lse[ql]) : 0.f;
          const float dpm = dpT[n][e] - s_D[ql];
          pT[n][e] = p;
          dsT[n][e] = p * dpm;
          if (DUAL) {
            const float pd = p * (sdT[n][e] - s_rb[ql]);
            pdT[n][e] = pd;
            dsdT[n][e] = pd * dpm + p * (dpdT[n][e] - s_Dd[ql]);
          }
        }
      uint32_t pa[4], dsa[4], pda[4], dsda[4];
      c_to_a(pa, pT[0], pT[1]);
      c_to_a(dsa, dsT[0], dsT[1]);
      if (DUAL) {
        c_to_a(pda, pdT[0], pdT[1]);
        c_to_a(dsda, dsdT[0], dsdT[1]);
      }
      // dV += P^T dO, dV' += P'^T dO + P^T dO', dK += dS^T Q, dK' += dS'^T Q + dS^T Q'
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bo[4], bq[4];
        frag_b_kn(bo, dOs, q0, np * 16);
        frag_b_kn(bq, Qs, q0, np * 16);
        mma(dv[2 * np], pa, bo[0], bo[1]);
        mma(dv[2 * np + 1], pa, bo[2], bo[3]);
        mma(dk[2 * np], dsa, bq[0], bq[1]);
        mma(dk[2 * np + 1], dsa, bq[2], bq[3]);
        if (DUAL) {
          mma(dvd[2 * np], pda, bo[0], bo[1]);
          mma(dvd[2 * np + 1], pda, bo[2], bo[3]);
          mma(dkd[2 * np], dsda, bq[0], bq[1]);
          mma(dkd[2 * np + 1], dsda, bq[2], bq[3]);
          uint32_t bod[4], bqd[4];
          frag_b_kn(bod, dOds, q0, np * 16);
          frag_b_kn(bqd, Qds, q0, np * 16);
          mma(dvd[2 * np], pa, bod[0], bod[1]);
          mma(dvd[2 * np + 1], pa, bod[2], bod[3]);
          mma(dkd[2 * np], dsa, bqd[0], bqd[1]);
          mma(dkd[2 * np + 1], dsa, bqd[2], bqd[3]);
        }
      }
    }
  }
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t off = hoff + static_cast<int64_t>(key0 + h * 8) * FDH + n * 8 + (lane & 3) * 2;
      *reinterpret_cast<float2*>(a.dV + off) = make_float2(dv[n][2 * h], dv[n][2 * h + 1]);
      *reinterpret_cast<float2*>(a.dK + off) = make_float2(dk[n][2 * h], dk[n][2 * h + 1]);
      if (DUAL) {
        *reinterpret_cast<float2*>(a.dVd + off) = make_float2(dvd[n][2 * h], dvd[n][2 * h + 1]);
        *reinterpret_cast<float2*>(a.dKd + off) = make_float2(dkd[n][2 * h], dkd[n][2 * h + 1]);
      }
    }
}

// ---- backward: dQ (and tangent), one CTA per query tile -------------------------------------
template <bool DUAL>
__global__ void __launch_bounds__(FTHREADS) flash_bwd_q_kernel(const FlashArgs a) {
  pdl_entry();
  extern __shared__ __align__(16) unsigned char fsm[];
  bf16* Qs = reinterpret_cast<bf16*>(fsm);
  bf16* dOs = Qs + TILE_ELEMS;
  bf16* Ks = dOs + TILE_ELEMS;
  bf16* Vs = Ks + TILE_ELEMS;
  bf16* Qds = Vs + TILE_ELEMS;     // dual only
  bf16* dOds = Qds + TILE_ELEMS;
  bf16* Kds = dOds + TILE_ELEMS;
  bf16* Vds = Kds + TILE_ELEMS;
  const int nq = a.S / FT;
  const int qt = nq - 1 - static_cast<int>(blockIdx.y);   // grid (heads, tiles): longest first
  const int bh = blockIdx.x;
  const int64_t hoff = static_cast<int64_t>(bh) * a.S * FDH;
  const int64_t soff = static_cast<int64_t>(bh) * a.S;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r0 = w * 16;
  const int qrow0 = qt * FT + r0 + (lane >> 2);
  float lse[2], rb[2], Dv[2], Ddv[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int64_t i = soff + qrow0 + h * 8;
    lse[h] = a.lse[i];
    Dv[h] = a.D[i];
    rb[h] = DUAL ? a.rbar[i] : 0.f;
    Ddv[h] = DUAL ? a.Dd[i] : 0.f;
  }
  load_tile(Qs, a.Q + hoff, qt * FT);
  load_tile(dOs, a.dO + hoff, qt * FT);
  if (DUAL) {
    load_tile(Qds, a.Qd + hoff, qt * FT);
    load_tile(dOds, a.dOd + hoff, qt * FT);
  }
  float dq[8][4], dqd[8][4];
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) { dq[n][e] = 0.f; dqd[n][e] = 0.f; }
  for (int kt = 0; kt <= qt; ++kt) {
    __syncthreads();
    load_tile(Ks, a.K + hoff, kt * FT);
    load_tile(Vs, a.V + hoff, kt * FT);
    if (DUAL) {
      load_tile(Kds, a.Kd + hoff, kt * FT);
      load_tile(Vds, a.Vd + hoff, kt * FT);
    }
    cp_wait_all();
    __syncthreads();
#pragma unroll 1
    for (int c = 0; c < 4; ++c) {            // 16-key chunks
      const int k0 = c * 16;
      if (kt == qt && k0 > r0 + 15) continue;    // every key of the chunk follows every query
      float s[2][4] = {}, sd[2][4] = {}, dp[2][4] = {}, dpd[2][4] = {};
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        uint32_t qa[4], b[4];
        frag_a(qa, Qs, r0, ks * 16);
        frag_b_nk(b, Ks, k0, ks * 16);
        mma(s[0], qa, b[0], b[1]);
        mma(s[1], qa, b[2], b[3]);
        uint32_t oa[4], bv[4];
        frag_a(oa, dOs, r0, ks * 16);
        frag_b_nk(bv, Vs, k0, ks * 16);
        mma(dp[0], oa, bv[0], bv[1]);
        mma(dp[1], oa, bv[2], bv[3]);
        if (DUAL) {
          uint32_t qda[4], bk[4];
          frag_a(qda, Qds, r0, ks * 16);
          mma(sd[0], qda, b[0], b[1]);
          mma(sd[1], qda, b[2], b[3]);
          frag_b_nk(bk, Kds, k0, ks * 16);
          mma(sd[0], qa, bk[0], bk[1]);
          mma(sd[1], qa, bk[2], bk[3]);
          uint32_t oda[4], bvd[4];
          frag_a(oda, dOds, r0, ks * 16);
          mma(dpd[0], oda, bv[0], bv[1]);
          mma(dpd[1], oda, bv[2], bv[3]);
          frag_b_nk(bvd, Vds, k0, ks * 16);
          mma(dpd[0], oa, bvd[0], bvd[1]);
          mma(dpd[1], oa, bvd[2], bvd[3]);
        }
      }
      float ds[2][4], dsd[2][4];
#pragma unroll
      for (int n = 0; n < 2; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int h = e >> 1;
          const int key = kt * FT + k0 + n * 8 + (lane & 3) * 2 + (e & 1);
          const int q = qrow0 + h * 8;
          const float p = key <= q ? __expf(s[n][e] - lse[h]) : 0.f;
          const float dpm = dp[n][e] - Dv[h];
          ds[n][e] = p * dpm;
          if (DUAL) {
            const float pd = p * (sd[n][e] - rb[h]);
            dsd[n][e] = pd * dpm + p * (dpd[n][e] - Ddv[h]);
          }
        }
      uint32_t dsa[4], dsda[4];
      c_to_a(dsa, ds[0], ds[1]);
      if (DUAL) c_to_a(dsda, dsd[0], dsd[1]);
      // dQ += dS K ; dQ' += dS' K + dS K'
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bk[4];
        frag_b_kn(bk, Ks, k0, np * 16);
        mma(dq[2 * np], dsa, bk[0], bk[1]);
        mma(dq[2 * np + 1], dsa, bk[2], bk[3]);
        if (DUAL) {
          mma(dqd[2 * np], dsda, bk[0], bk[1]);
          mma(dqd[2 * np + 1], dsda, bk[2], bk[3]);
          uint32_t bkd[4];
          frag_b_kn(bkd, Kds, k0, np * 16);
          mma(dqd[2 * np], dsa, bkd[0], bkd[1]);
          mma(dqd[2 * np + 1], dsa, bkd[2], bkd[3]);
        }
      }
    }
  }
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t off = hoff + static_cast<int64_t>(qrow0 + h * 8) * FDH + n * 8 + (lane & 3) * 2;
      *reinterpret_cast<float2*>(a.dQ + off) = make_float2(dq[n][2 * h], dq[n][2 * h + 1]);
      if (DUAL)
        *reinterpret_cast<float2*>(a.dQd + off) = make_float2(dqd[n][2 * h], dqd[n][2 * h + 1]);
    }
}

// D = rowsum(dO (*) O) and D' = rowsum(dO' (*) O + dO (*) O') per (token, head), from the
// float32 head-merged output gradients [N][ld] and the bf16 merged attention outputs; the
// same pass writes dO (dO') as bf16 per head ([B*H][S][64]) for the backward kernels.  Two
// (token, head) rows per warp, four adjacent columns per lane (16-byte loads of dO).
__global__ void flash_prep_kernel(int N, int S, int H, const float* __restrict__ dO,
                                  const float* __restrict__ dOd, const bf16* __restrict__ O,
                                  const bf16* __restrict__ Od, int ld, float* __restrict__ D,
                                  float* __restrict__ Dd, bf16* __restrict__ dOh,
                                  bf16* __restrict__ dOhd) {
  pdl_entry();
  // two (token, head) rows per warp, 16 lanes of four columns each
  const int lane = threadIdx.x & 31;
  const int row = ((blockIdx.x * blockDim.x + threadIdx.x) >> 5) * 2 + (lane >> 4);
  const int c = (lane & 15) * 4;
  const bool ok = row < N * H;
  const int n = ok ? row / H : 0, hh = ok ? row % H : 0;
  const int64_t base = static_cast<int64_t>(n) * ld + hh * FDH + c;
  const int b = n / S, sidx = n % S;
  const int64_t i = (static_cast<int64_t>(b) * H + hh) * S + sidx;
  float d = 0.f, dd = 0.f;
  if (ok) {
    const float4 g = *reinterpret_cast<const float4*>(dO + base);
    const uint2 ob = *reinterpret_cast<const uint2*>(O + base);
    const float2 o01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ob.x));
    const float2 o23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ob.y));
    d = g.x * o01.x + g.y * o01.y + g.z * o23.x + g.w * o23.y;
    if (dOh) *reinterpret_cast<uint2*>(dOh + i * FDH + c) = make_uint2(pack(g.x, g.y), pack(g.z, g.w));
    if (Dd) {
      const float4 gd = *reinterpret_cast<const float4*>(dOd + base);
      const uint2 odb = *reinterpret_cast<const uint2*>(Od + base);
      const float2 od01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&odb.x));
      const float2 od23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&odb.y));
      dd = gd.x * o01.x + gd.y * o01.y + gd.z * o23.x + gd.w * o23.y + g.x * od01.x +
           g.y * od01.y + g.z * od23.x + g.w * od23.y;
      if (dOhd)
        *reinterpret_cast<uint2*>(dOhd + i * FDH + c) = make_uint2(pack(gd.x, gd.y), pack(gd.z, gd.w));
    }
  }
#pragma unroll
  for (int s = 8; s > 0; s >>= 1) {
    d += __shfl_xor_sync(0xffffffffu, d, s);
    dd += __shfl_xor_sync(0xffffffffu, dd, s);
  }
  if (ok && (lane & 15) == 0) {
    D[i] = d;
    if (Dd) Dd[i] = dd;
  }
}

constexpr int SMEM_FWD1 = 6 * TILE_ELEMS * 2, SMEM_FWD0 = 3 * TILE_ELEMS * 2;
constexpr int SMEM_KV1 = 8 * TILE_ELEMS * 2 + 4 * FT * 4, SMEM_KV0 = 4 * TILE_ELEMS * 2 + 4 * FT * 4;
constexpr int SMEM_Q1 = 8 * TILE_ELEMS * 2, SMEM_Q0 = 4 * TILE_ELEMS * 2;

// Dynamic shared-memory limits of all six kernels, once per device (before any capture:
// the first call of a captured sequence runs eagerly).
void init_attributes() {
  static PerDeviceOnce once;
  once.run([](int&) {
    const auto a = cudaFuncAttributeMaxDynamicSharedMemorySize;
    cudaFuncSetAttribute(flash_fwd_kernel<true>, a, SMEM_FWD1);
    cudaFuncSetAttribute(flash_fwd_kernel<false>, a, SMEM_FWD0);
    cudaFuncSetAttribute(flash_bwd_kv_kernel<true>, a, SMEM_KV1);
    cudaFuncSetAttribute(flash_bwd_kv_kernel<false>, a, SMEM_KV0);
    cudaFuncSetAttribute(flash_bwd_q_kernel<true>, a, SMEM_Q1);
    return cudaFuncSetAttribute(flash_bwd_q_kernel<false>, a, SMEM_Q0);
  });
}

}  // namespace

bool flash_supported(int S, int dh) { return dh == FDH && S > 0 && S % FT == 0; }

void flash_fwd(const FlashArgs& a, bool dual, cudaStream_t s) {
  // tcgen05 forward: the dual kernel at tc >= 1, the primal one too at tc = 2 (launch errors
  // surface at the caller's check)
  if (a.tc >= (dual ? 1 : 2) && flash_tc_supported(a.S, FDH)) {
    flash_tc_fwd(a, dual, s);
    return;
  }
  init_attributes();
  const dim3 grid(a.BH, a.S / FT);
  if (dual)
    launch_k(flash_fwd_kernel<true>, grid, dim3(FTHREADS), SMEM_FWD1, s, a);
  else
    launch_k(flash_fwd_kernel<false>, grid, dim3(FTHREADS), SMEM_FWD0, s, a);
}

bool flash_bwd_merges(const FlashArgs& a, bool dual) {
  return a.tc_bwd && flash_tc_bwd_supported(a, dual);
}

void flash_bwd(const FlashArgs& a, bool dual, cudaStream_t s) {
  // tcgen05 backward (launch errors surface at the caller's check)
  if (a.tc_bwd && flash_tc_bwd_supported(a, dual)) {
    flash_tc_bwd(a, dual, s);
    return;
  }
  init_attributes();
  const dim3 grid(a.BH, a.S / FT);
  if (dual) {
    launch_k(flash_bwd_kv_kernel<true>, grid, dim3(FTHREADS), SMEM_KV1, s, a);
    launch_k(flash_bwd_q_kernel<true>, grid, dim3(FTHREADS), SMEM_Q1, s, a);
  } else {
    launch_k(flash_bwd_kv_kernel<false>, grid, dim3(FTHREADS), SMEM_KV0, s, a);
    launch_k(flash_bwd_q_kernel<false>, grid, dim3(FTHREADS), SMEM_Q0, s, a);
  }
}

void flash_prep(int N, int S, int H, const float* dO, const float* dOd, const void* O,
                const void* Od, int ld, float* D, float* Dd, void* dOh, void* dOhd,
                cudaStream_t s) {
  const int warps = (N * H + 1) / 2;
  const int threads = 256;
  const int blocks = (warps * 32 + threads - 1) / threads;
  launch_k(flash_prep_kernel, dim3(blocks), dim3(threads), 0, s, N, S, H, dO, dOd,
           static_cast<const bf16*>(O), static_cast<const bf16*>(Od), ld, D, Dd,
           static_cast<bf16*>(dOh), static_cast<bf16*>(dOhd));
}

}  // namespace mf
