// Fused causal attention and its forward tangent on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA): the forward kernel of the dual attention for sequences of whole
// 128-token tiles (flash_attn.cu holds the formulas, the backward and the warp-level kernels
// used for other lengths).
//
// One CTA per (head, 128-query tile), walking 64-key tiles up to the diagonal:
//   warp 0      TMA producer: Q (and Q') once, then K, V (and K', V') per key tile into a
//               ring of shared-memory stages (128-byte swizzle, K-major rows of 64 dims);
//   warp 1      owns TMEM; one thread issues the MMAs:
//                 S  = Q K^T,  S' = Q' K^T + Q K'^T            (M 128, N 64 keys, K 64)
//                 O += P V,  T += (P (*) S') V + P V'          (M 128, N 64, K 64 keys; V
//                                                               and V' read MN-major in place)
//   warps 2..5  softmax: thread r owns query row r (TMEM lane r).  It reads its row of S
//               (and S') from TMEM, updates the running maximum, writes P = exp(S - m) and
//               P (*) S' as bf16 into shared memory (the A operands of the next products) and
//               keeps l = sum P and r = sum P (*) S'.
// The tangent's two products share one accumulator T, since O' needs only their sum:
// O' = T / l - rbar O.  TMEM columns: S 0..63, S' 64..127, O 128..191, T 192..255 (the
// primal kernel: S 0..63, O 64..127), so two CTAs share an SM and one
// CTA's softmax overlaps another's products.
//
// The reference maximum m of a row moves only when a tile's maximum exceeds it by more than
// TAU = 8 (then O, T, l and r of the row are rescaled in place); between moves P may reach
// e^8.  Every quantity of the row uses the same m, so O = o / l, the log-sum-exp
// lse = m + log l, rbar = r / l and O' are exact for any m; only overflow needs the bound.
//
// Every wait is bounded (2 s); a role that gives up records the timeout in the status word
// and raises a CTA-local abort flag; the MMA thread then waits for its own last commit and
// the producer for the loads it issued, so no asynchronous copy or MMA outlives the CTA.
#include "tc_gemm_impl.cuh"

namespace mf {
namespace {

constexpr int TQ = 128;            // queries per CTA (MMA M)
constexpr int TK = 64;             // keys per tile (MMA N of S, K of the P products)
constexpr int HD = 64;             // head dimension (one 128-byte swizzle atom)
constexpr int Q_TILE_B = TQ * HD * 2;          // 16 KB: [128][64] bf16
constexpr int K_TILE_B = TK * HD * 2;          // 8 KB: [64][64] bf16
constexpr int P_ATOM = TQ * TK * 2;            // 16 KB: P of one key tile, [128][64] bf16
constexpr int FTC_THREADS = 192;               // producer, MMA, four softmax warps
constexpr float TAU = 8.f;
constexpr long long FTC_WAIT_NS = 2000000000LL;

template <bool DUAL>
struct FtcCfg {
  static constexpr int STAGES = DUAL ? 1 : 2;
  static constexpr int STAGE_B = (DUAL ? 4 : 2) * K_TILE_B;  // K, V (K', V')
  static constexpr int Q_B = (DUAL ? 2 : 1) * Q_TILE_B;      // Q (Q')
  static constexpr int P_B = (DUAL ? 2 : 1) * P_ATOM;        // P (P (*) S')
  static constexpr int SMEM = Q_B + STAGES * STAGE_B + P_B + 1024;
  static constexpr int CTAS = 2;                             // per SM
  static constexpr uint32_t TMEM_COLS = DUAL ? 256 : 128;
  // TMEM column offsets
  static constexpr uint32_t C_S = 0, C_SD = 64, C_O = DUAL ? 128 : 64, C_T = 192;
};

struct FtcParams {
  int BH, S;
  float *O, *Od, *lse, *rbar;
  int H, ldo;                        // head-merged bf16 outputs when Om is set
  __nv_bfloat16 *Om, *Omd;
  int* status;
};

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 32 consecutive TMEM columns of this thread's lane, without waiting (tmem_wait_ld after a
// batch of loads).
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_local(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bounded wait that gives up at once when another role of the CTA has given up.
__device__ __forceinline__ bool fwait(uint64_t* bar, uint32_t parity, int* status,
                                      volatile int* abort) {
  if (*abort) return false;
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = global_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (global_ns() - t0 > FTC_WAIT_NS) {
      if (status) atomicMax(status, DEV_TIMEOUT);
      *abort = 1;
      return false;
    }
  }
}

// Byte offset of (row r, 16-byte chunk ch) in a K-major [128][64] bf16 atom, 128-byte swizzle.
__device__ __forceinline__ uint32_t swz(int r, int ch) {
  return static_cast<uint32_t>(r * 128 + ((ch ^ (r & 7)) << 4));
}


// Warp-uniform bounded wait: every lane polls, and the warp proceeds only if all lanes saw
// the phase complete (the TMEM loads after it are warp-collective).
__device__ __forceinline__ bool wwait(uint64_t* bar, uint32_t parity, int* status,
                                      volatile int* abort) {
  const bool ok = fwait(bar, parity, status, abort);
  return __all_sync(0xffffffffu, ok);
}

template <bool DUAL>
__global__ void __launch_bounds__(FTC_THREADS, FtcCfg<DUAL>::CTAS)
    flash_tc_fwd_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV,
                        const __grid_constant__ CUtensorMap tmQd,
                        const __grid_constant__ CUtensorMap tmKd,
                        const __grid_constant__ CUtensorMap tmVd, const FtcParams prm) {
  using C = FtcCfg<DUAL>;
  const FtcParams p = prm;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t q_full, s_full, s_free, p_full, o_done, drain;
  __shared__ __align__(8) uint64_t kv_full[C::STAGES], kv_empty[C::STAGES];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;                       // Q, then Q'
  uint8_t* sKV = smem + C::Q_B;             // stage st: K, V, K', V' (8 KB each)
  uint8_t* sP = sKV + C::STAGES * C::STAGE_B;   // P, then P (*) S' (16 KB each)
  const int nq = p.S / TQ;
  // grid (heads, tiles): heads dispatch fastest, so every head's longest query tile goes
  // first and the shortest ones fill the tail of the launch
  const int qt = nq - 1 - static_cast<int>(blockIdx.y);
  const int bh = static_cast<int>(blockIdx.x);
  const int row0 = bh * p.S;                // the head's first row in the [BH*S][64] maps
  const int nkt = (qt + 1) * (TQ / TK);     // key tiles up to the diagonal
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&q_full, 1);
    mbar_init(&s_full, 1);
    mbar_init(&s_free, 4);
    mbar_init(&p_full, 4);
    mbar_init(&o_done, 1);
    mbar_init(&drain, 1);
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    if (DUAL) {
      prefetch_tmap(&tmQd);
      prefetch_tmap(&tmKd);
      prefetch_tmap(&tmVd);
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_slot)),
                 "r"(C::TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tb = tmem_slot;
  volatile int* abort = &abort_flag;
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer ---------------------------------------------------------------
      mbar_expect_tx(&q_full, C::Q_B);
      tma_load_3d(sQ, &tmQ, &q_full, 0, row0 + qt * TQ, 0);
      if (DUAL) tma_load_3d(sQ + Q_TILE_B, &tmQd, &q_full, 0, row0 + qt * TQ, 0);
      int issued = 0;
      for (int j = 0; j < nkt; ++j, ++issued) {
        const int st = j % C::STAGES;
        const uint32_t ph = (j / C::STAGES) & 1;
        if (!fwait(&kv_empty[st], ph ^ 1, p.status, abort)) break;
        mbar_expect_tx(&kv_full[st], C::STAGE_B);
        uint8_t* b = sKV + st * C::STAGE_B;
        const int kr = row0 + j * TK;
        tma_load_3d(b, &tmK, &kv_full[st], 0, kr, 0);
        tma_load_3d(b + K_TILE_B, &tmV, &kv_full[st], 0, kr, 0);
        if (DUAL) {
          tma_load_3d(b + 2 * K_TILE_B, &tmKd, &kv_full[st], 0, kr, 0);
          tma_load_3d(b + 3 * K_TILE_B, &tmVd, &kv_full[st], 0, kr, 0);
        }
      }
      // every load issued has landed before the CTA can end
      mbar_wait(&q_full, 0, p.status, FTC_WAIT_NS);
      drain_loads(kv_full, issued, C::STAGES, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer -------------------------------------------------------------------
      const uint32_t idS = idesc_bf16(TQ, TK);
      const uint32_t idO = idesc_bf16(TQ, HD) | (1u << 16);   // B (V) read MN-major
      const uint32_t aQ = smem_u32(sQ), aP = smem_u32(sP);
      bool ok = fwait(&q_full, 0, p.status, abort);
      for (int j = 0; ok && j < nkt; ++j) {
        const int st = j % C::STAGES;
        const uint32_t ph = (j / C::STAGES) & 1;
        if (!fwait(&kv_full[st], ph, p.status, abort)) break;
        if (j > 0 && !fwait(&s_free, (j - 1) & 1, p.status, abort)) break;
        tc_fence_after();
        const uint32_t aK = smem_u32(sKV + st * C::STAGE_B);
        const uint32_t aV = aK + K_TILE_B;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_bf16(tb + C::C_S, sdesc_sw128(aQ) + 2 * kk, sdesc_sw128(aK) + 2 * kk, idS, kk > 0);
        if (DUAL) {
          const uint32_t aQd = aQ + Q_TILE_B, aKd = aK + 2 * K_TILE_B;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_SD, sdesc_sw128(aQd) + 2 * kk, sdesc_sw128(aK) + 2 * kk, idS, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_SD, sdesc_sw128(aQ) + 2 * kk, sdesc_sw128(aKd) + 2 * kk, idS, 1);
        }
        mma_commit(&s_full);
        if (!fwait(&p_full, j & 1, p.status, abort)) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < TK / 16; ++kk) {
          const uint64_t pa = sdesc_sw128(aP) + 2 * kk;
          const uint64_t vb = sdesc_mn_sw128(aV) + 128 * kk;
          const uint32_t acc = (j > 0 || kk > 0) ? 1u : 0u;
          mma_bf16(tb + C::C_O, pa, vb, idO, acc);
          if (DUAL) {
            const uint64_t psa = sdesc_sw128(aP + P_ATOM) + 2 * kk;
            const uint64_t vdb = sdesc_mn_sw128(aK + 3 * K_TILE_B) + 128 * kk;
            mma_bf16(tb + C::C_T, psa, vb, idO, acc);
            mma_bf16(tb + C::C_T, pa, vdb, idO, 1);
          }
        }
        mma_commit(&kv_empty[st]);
        mma_commit(&o_done);
      }
      // every MMA issued here has completed before TMEM is released
      mma_commit(&drain);
      mbar_wait(&drain, 0, p.status, FTC_WAIT_NS);
    }
    __syncwarp();
  } else {
    // ---- softmax: thread r owns query row r of the tile (TMEM lane r) -------------------
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const uint32_t lo = static_cast<uint32_t>(q4 * 32) << 16;
    float m = -INFINITY, l = 0.f, rs = 0.f;
    bool ok = true;
    for (int j = 0; j < nkt; ++j) {
      if (!wwait(&s_full, j & 1, p.status, abort)) { ok = false; break; }
      tc_fence_after();
      // key c of this tile is masked for this row when kbase + c > r (the causal diagonal)
      const int kbase = j * TK - qt * TQ;
      float sv[TK], sd[TK];
      tmem_ld32_nowait(tb + lo + C::C_S, sv);
      tmem_ld32_nowait(tb + lo + C::C_S + 32, sv + 32);
      if (DUAL) {
        tmem_ld32_nowait(tb + lo + C::C_SD, sd);
        tmem_ld32_nowait(tb + lo + C::C_SD + 32, sd + 32);
      }
      tmem_wait_ld();
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int i = 0; i < TK; i += 2) {
        if (kbase + i <= r) mx0 = fmaxf(mx0, sv[i]);
        if (kbase + i + 1 <= r) mx1 = fmaxf(mx1, sv[i + 1]);
      }
      const float mx = fmaxf(mx0, mx1);
      float scale = 1.f;
      if (mx > m + TAU) {
        scale = __expf(m - mx);
        m = mx;
      }
      // P and P (*) S' of this tile, in registers
      uint32_t pk[TK / 2], psk[TK / 2];
      float l0 = 0.f, l1 = 0.f, r0s = 0.f, r1s = 0.f;
#pragma unroll
      for (int i = 0; i < TK; i += 2) {
        const float p0 = kbase + i > r ? 0.f : __expf(sv[i] - m);
        const float p1 = kbase + i + 1 > r ? 0.f : __expf(sv[i + 1] - m);
        l0 += p0;
        l1 += p1;
        pk[i / 2] = pack_bf16x2(p0, p1);
        if (DUAL) {
          const float s0 = p0 * sd[i], s1 = p1 * sd[i + 1];
          r0s += s0;
          r1s += s1;
          psk[i / 2] = pack_bf16x2(s0, s1);
        }
      }
      l = l * scale + (l0 + l1);
      rs = rs * scale + (r0s + r1s);
      if (j > 0) {
        // the products of tile j - 1 are done: O, T may be rescaled and P rewritten
        if (!wwait(&o_done, (j - 1) & 1, p.status, abort)) { ok = false; break; }
        tc_fence_after();
        if (__any_sync(0xffffffffu, scale != 1.f)) {
#pragma unroll 1
          for (int c0 = 0; c0 < HD; c0 += 16) {
            float v[16];
            tmem_ld16(tb + lo + C::C_O + c0, v);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] *= scale;
            tmem_st16(tb + lo + C::C_O + c0, v);
            if (DUAL) {
              tmem_ld16(tb + lo + C::C_T + c0, v);
#pragma unroll
              for (int i = 0; i < 16; ++i) v[i] *= scale;
              tmem_st16(tb + lo + C::C_T + c0, v);
            }
          }
        }
      }
#pragma unroll
      for (int ch = 0; ch < TK / 8; ++ch) {
        *reinterpret_cast<uint4*>(sP + swz(r, ch)) =
            make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]);
        if (DUAL)
          *reinterpret_cast<uint4*>(sP + P_ATOM + swz(r, ch)) =
              make_uint4(psk[4 * ch], psk[4 * ch + 1], psk[4 * ch + 2], psk[4 * ch + 3]);
      }
      tc_fence_before();
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive_local(&s_free);
        mbar_arrive_local(&p_full);
      }
    }
    // ---- outputs: O = o / l, lse, and O' = T / l - rbar O, rbar = r / l -----------------
    if (ok && wwait(&o_done, (nkt - 1) & 1, p.status, abort)) {
      tc_fence_after();
      const float inv = 1.f / l;
      const float rb = DUAL ? rs * inv : 0.f;
      const int64_t grow = static_cast<int64_t>(row0) + qt * TQ + r;
      // head-merged bf16 row: token b*S + q, columns hh*64 .. hh*64 + 63
      const int hb = p.H > 0 ? bh / p.H : 0, hh = p.H > 0 ? bh % p.H : 0;
      const int64_t mrow = (static_cast<int64_t>(hb) * p.S + qt * TQ + r) * p.ldo + hh * HD;
#pragma unroll 1
      for (int c0 = 0; c0 < HD; c0 += 16) {
        float o[16];
        tmem_ld16(tb + lo + C::C_O + c0, o);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] *= inv;
        if (p.Om) {
          uint4* dst = reinterpret_cast<uint4*>(p.Om + mrow + c0);
          dst[0] = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                              pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
          dst[1] = make_uint4(pack_bf16x2(o[8], o[9]), pack_bf16x2(o[10], o[11]),
                              pack_bf16x2(o[12], o[13]), pack_bf16x2(o[14], o[15]));
        } else {
          float* orow = p.O + grow * HD;
#pragma unroll
          for (int i = 0; i < 16; i += 4)
            *reinterpret_cast<float4*>(orow + c0 + i) =
                make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
        }
        if (DUAL) {
          float t[16];
          tmem_ld16(tb + lo + C::C_T + c0, t);
#pragma unroll
          for (int i = 0; i < 16; ++i) t[i] = t[i] * inv - rb * o[i];
          if (p.Om) {
            uint4* dst = reinterpret_cast<uint4*>(p.Omd + mrow + c0);
            dst[0] = make_uint4(pack_bf16x2(t[0], t[1]), pack_bf16x2(t[2], t[3]),
                                pack_bf16x2(t[4], t[5]), pack_bf16x2(t[6], t[7]));
            dst[1] = make_uint4(pack_bf16x2(t[8], t[9]), pack_bf16x2(t[10], t[11]),
                                pack_bf16x2(t[12], t[13]), pack_bf16x2(t[14], t[15]));
          } else {
            float* drow = p.Od + grow * HD;
#pragma unroll
            for (int i = 0; i < 16; i += 4)
              *reinterpret_cast<float4*>(drow + c0 + i) =
                  make_float4(t[i], t[i + 1], t[i + 2], t[i + 3]);
          }
        }
      }
      p.lse[grow] = m + __logf(l);
      if (DUAL) p.rbar[grow] = rb;
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tb),
                 "r"(C::TMEM_COLS));
  }
}

template <bool DUAL>
cudaError_t launch_ftc_fwd(const FlashArgs& a, cudaStream_t s) {
  using C = FtcCfg<DUAL>;
  const int rows = a.BH * a.S;
  CUtensorMap mQ, mK, mV, mQd, mKd, mVd;
  memset(&mQd, 0, sizeof(mQd)); memset(&mKd, 0, sizeof(mKd)); memset(&mVd, 0, sizeof(mVd));
  if (!make_map(&mQ, a.Q, HD, rows, HD, TQ) || !make_map(&mK, a.K, HD, rows, HD, TK) ||
      !make_map(&mV, a.V, HD, rows, HD, TK))
    return cudaErrorInvalidValue;
  if (DUAL && (!make_map(&mQd, a.Qd, HD, rows, HD, TQ) || !make_map(&mKd, a.Kd, HD, rows, HD, TK) ||
               !make_map(&mVd, a.Vd, HD, rows, HD, TK)))
    return cudaErrorInvalidValue;
  static PerDeviceOnce attr_once;
  cudaError_t e = attr_once.run([](int&) {
    return cudaFuncSetAttribute(flash_tc_fwd_kernel<DUAL>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  });
  if (e != cudaSuccess) return e;
  FtcParams p;
  p.BH = a.BH;
  p.S = a.S;
  p.O = a.O;
  p.Od = a.Od;
  p.lse = a.lse;
  p.rbar = a.rbar;
  p.H = a.H;
  p.ldo = a.ldo;
  p.Om = a.Om;
  p.Omd = a.Omd;
  p.status = a.status;
  return launch_k(flash_tc_fwd_kernel<DUAL>, dim3(a.BH, a.S / TQ), dim3(FTC_THREADS),
                  C::SMEM, s, mQ, mK, mV, mQd, mKd, mVd, p);
}

}  // namespace
}  // namespace mf

namespace mf {

bool flash_tc_supported(int S, int dh) { return dh == HD && S > 0 && S % TQ == 0; }

cudaError_t flash_tc_fwd(const FlashArgs& a, bool dual, cudaStream_t s) {
  if (!flash_tc_supported(a.S, HD) || a.BH < 1) return cudaErrorInvalidValue;
  return dual ? launch_ftc_fwd<true>(a, s) : launch_ftc_fwd<false>(a, s);
}

}  // namespace mf
