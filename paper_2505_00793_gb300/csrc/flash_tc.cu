// Fused causal attention and its forward tangent on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA) for sequences of whole 128-token tiles: the forward kernel of the
// dual (and primal) attention, and below it the two backward kernels (flash_attn.cu holds
// the formulas, the D / D' prep and the warp-level kernels used for other lengths).
//
// Forward: one CTA per (head, 128-query tile), walking 64-key tiles up to the diagonal:
//   warp 0      TMA producer: Q (and Q') once, then K, V (and K', V') per key tile into a
//               ring of shared-memory stages (128-byte swizzle, K-major rows of 64 dims);
//   warp 1      owns TMEM; one thread issues the MMAs:
//                 S  = Q K^T,  S' = Q' K^T + Q K'^T            (M 128, N 64 keys, K 64)
//                 O += P V,  T += (P (*) S') V + P V'          (M 128, N 64, K 64 keys; V
//                                                               and V' read MN-major in place)
//               with the products that share an A operand as one N = 128 MMA over adjacent
//               B tiles and accumulators: Q [K | K']^T -> [S | Q K'^T], P [V | V'] -> [O | P V']
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
constexpr int BT_Q = 64;           // backward: queries (key-tile kernel) or keys (query-tile
                                   // kernel) per streamed tile

template <bool DUAL>
struct FtcCfg {
  static constexpr int STAGES = DUAL ? 1 : 2;
  static constexpr int STAGE_B = (DUAL ? 4 : 2) * K_TILE_B;  // K, (K',) V (, V')
  static constexpr int OFF_V = (DUAL ? 2 : 1) * K_TILE_B;     // K' follows K, V' follows V
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
  uint8_t* sKV = smem + C::Q_B;             // stage st: K, K', V, V' (8 KB each)
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
        tma_load_3d(b + C::OFF_V, &tmV, &kv_full[st], 0, kr, 0);
        if (DUAL) {
          tma_load_3d(b + K_TILE_B, &tmKd, &kv_full[st], 0, kr, 0);
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
      const uint32_t idS2 = idesc_bf16(TQ, 2 * TK);
      const uint32_t idO2 = idesc_bf16(TQ, 2 * HD) | (1u << 16);
      // operand descriptors, built once: a byte offset moves a descriptor by offset >> 4
      const uint64_t dQ = sdesc_sw128(smem_u32(sQ)), dQd = dQ + (Q_TILE_B >> 4);
      const uint64_t dP = sdesc_sw128(smem_u32(sP)), dPS = dP + (P_ATOM >> 4);
      const uint64_t dKV = sdesc_sw128(smem_u32(sKV)), mKV = sdesc_mn_sw128(smem_u32(sKV));
      constexpr uint64_t ST_STEP = C::STAGE_B >> 4, V_STEP = C::OFF_V >> 4;
      bool ok = fwait(&q_full, 0, p.status, abort);
      for (int j = 0; ok && j < nkt; ++j) {
        const int st = j % C::STAGES;
        const uint32_t ph = (j / C::STAGES) & 1;
        if (!fwait(&kv_full[st], ph, p.status, abort)) break;
        if (j > 0 && !fwait(&s_free, (j - 1) & 1, p.status, abort)) break;
        tc_fence_after();
        const uint64_t dK = dKV + st * ST_STEP, mV = mKV + st * ST_STEP + V_STEP;
        if (DUAL) {
          // Q [K | K']^T -> [S | Q K'^T] in one N = 128 MMA (K' follows K), then Q' K^T into S'
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dQ + 2 * kk, dK + 2 * kk, idS2, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_SD, dQd + 2 * kk, dK + 2 * kk, idS, 1);
        } else {
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dQ + 2 * kk, dK + 2 * kk, idS, kk > 0);
        }
        mma_commit(&s_full);
        if (!fwait(&p_full, j & 1, p.status, abort)) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < TK / 16; ++kk) {
          const uint64_t vb = mV + 128 * kk;
          const uint32_t acc = (j > 0 || kk > 0) ? 1u : 0u;
          if (DUAL) {
            // P [V | V'] -> [O | P V'] in one N = 128 MMA (T follows O), then (P (*) S') V into T
            mma_bf16(tb + C::C_O, dP + 2 * kk, vb, idO2, acc);
            mma_bf16(tb + C::C_T, dPS + 2 * kk, vb, idO, 1);
          } else {
            mma_bf16(tb + C::C_O, dP + 2 * kk, vb, idO, acc);
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

// ---- backward on tcgen05 --------------------------------------------------------------
// Two kernels, as the warp-level backward: one CTA per (head, 128-key tile) for dK, dV and
// their tangents, one per (head, 128-query tile) for dQ and its tangent, so every sum keeps
// a fixed order.  The key-tile kernel walks 64-query tiles from the diagonal on:
//   warp 0      TMA producer: K, V (K', V') once; per query tile Q, dO (Q', dO') and the
//               row statistics lse, D (rbar, D') into a two-stage ring;
//   warp 1      one thread issues the MMAs (M 128 keys, N 64, K 64):
//                 S^T = K Q^T,  S'^T = K' Q^T + K Q'^T,  dP^T = V dO^T,
//                 dP'^T = V' dO^T + V dO'^T                          (scores, TMEM)
//                 dV += P^T dO,  dV' += P'^T dO + P^T dO',
//                 dK += dS^T Q,  dK' += dS'^T Q + dS^T Q'            (Q, dO read MN-major)
//               and issues the next tile's scores as soon as the elementwise warps have read
//               this tile's, before this tile's accumulating products, so the tensor pipe
//               computes them while the elementwise warps work on the next tile;
//   warps 2..9  two threads per key row r (TMEM lane r), each on 32 of the 64 query
//               columns: P^T = exp(S^T - lse) (causal),
//               dS^T = P^T (*) (dP^T - D), P'^T = P^T (*) (S'^T - rbar),
//               dS'^T = P'^T (*) (dP^T - D) + P^T (*) (dP'^T - D'), kept as bf16 in
//               registers, then written to shared memory (the A operands) once the previous
//               tile's accumulating products have read it.
// The query-tile kernel is the same with the roles of queries and keys exchanged: Q, dO
// (Q', dO') stay resident, K, V (K', V') stream per 64-key tile, and dQ += dS K,
// dQ' += dS' K + dS K' (K read MN-major).
constexpr int BW_EW = 8;                       // elementwise warps: two per TMEM lane quadrant,
                                               // each on half of the tile's 64 columns
constexpr int BW_THREADS = 64 + 32 * BW_EW;
constexpr int ROWS128_B = 128 * HD * 2;        // 16 KB: [128][64] bf16
constexpr int ROWS64_B = 64 * HD * 2;          // 8 KB: [64][64] bf16
constexpr int OPND_B = 128 * 64 * 2;           // 16 KB: [128][64] bf16 A operand

template <bool DUAL>
struct KvCfg {
  static constexpr int NRES = DUAL ? 4 : 2;    // K, V (K', V'): 128 rows each
  static constexpr int NT = DUAL ? 4 : 2;      // Q, (Q',) dO (, dO') per query tile: 64 rows
  static constexpr int OFF_DO = DUAL ? 2 * ROWS64_B : ROWS64_B;   // Q' right after Q, dO' after dO
  static constexpr int NSTAT = DUAL ? 4 : 2;   // lse, D (rbar, D'): 64 floats each
  static constexpr int STAGES = 2;
  static constexpr int STAT_OFF = NT * ROWS64_B;
  static constexpr int STAGE_B = STAT_OFF + 1024;
  static constexpr int NOP = DUAL ? 4 : 2;     // P^T, dS^T (P'^T, dS'^T)
  static constexpr int SMEM = NRES * ROWS128_B + STAGES * STAGE_B + NOP * OPND_B + 1024;
  static constexpr int CTAS = DUAL ? 1 : 2;
  static constexpr uint32_t TMEM_COLS = DUAL ? 512 : 256;
  static constexpr uint32_t C_S = 0, C_SD = 64, C_DP = DUAL ? 128 : 64, C_DPD = 192;
  static constexpr uint32_t C_DV = DUAL ? 256 : 128, C_DVD = 320, C_DK = DUAL ? 384 : 192,
                            C_DKD = 448;
};

template <bool DUAL>
struct QCfg {
  static constexpr int NRES = DUAL ? 4 : 2;    // Q, dO (Q', dO'): 128 rows each
  static constexpr int NT = DUAL ? 4 : 2;      // K, (K',) V (, V') per key tile: 64 rows
  static constexpr int OFF_V = DUAL ? 2 * ROWS64_B : ROWS64_B;    // K' right after K, V' after V
  static constexpr int STAGES = 2;
  static constexpr int STAGE_B = NT * ROWS64_B;
  static constexpr int NOP = DUAL ? 2 : 1;     // dS (dS')
  static constexpr int SMEM = NRES * ROWS128_B + STAGES * STAGE_B + NOP * OPND_B + 1024;
  static constexpr int CTAS = DUAL ? 1 : 2;
  static constexpr uint32_t TMEM_COLS = DUAL ? 512 : 256;
  static constexpr uint32_t C_S = 0, C_SD = 64, C_DP = DUAL ? 128 : 64, C_DPD = 192;
  static constexpr uint32_t C_DQ = DUAL ? 256 : 128, C_DQD = 320;
};

struct FtbParams {
  int BH, S;
  const float *lse, *rbar, *D, *Dd;
  float *dQ, *dQd, *dK, *dKd, *dV, *dVd;
  int* status;
  // merged bf16 outputs (FlashArgs::dqkv): heads H, row stride ldq, RoPE table, q scale
  __nv_bfloat16 *dqkv, *dqkvd;
  int H, ldq;
  const float* rope;
  float qscale;
};

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Four 16-column TMEM loads in flight, then one wait.
__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Columns cb .. cb + 31 of a 128 x 64 float32 accumulator row (this thread's TMEM lane) to
// global memory.
__device__ __forceinline__ void store_acc_row(uint32_t taddr, float* dst, int cb) {
#pragma unroll 1
  for (int c0 = cb; c0 < cb + 32; c0 += 16) {
    float v[16];
    tmem_ld16(taddr + c0, v);
#pragma unroll
    for (int i = 0; i < 16; i += 4)
      *reinterpret_cast<float4*>(dst + c0 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
  }
}

// Columns cb .. cb + 31 of a 64-wide accumulator row (this thread's TMEM lane, row r of
// the tile) as bf16 into a [128][64] staging tile (128-byte rows, 16-byte chunk c of row r at
// position c ^ (r & 7)), with the inverse RoPE rotation of position pos when rot is set: the
// first half's element j becomes (x_j cos_j + x_{j+32} sin_j) scale, the second half's
// (x_{j+32} cos_j - x_j sin_j) scale (the partner half is read from the same TMEM lane).
__device__ __forceinline__ void stage_merged_row(uint32_t taddr, int cb, bool rot, int pos,
                                                 const float* rtab, float scale, uint8_t* buf,
                                                 int r) {
  const int pb = cb ^ 32;
  const float sg = cb == 0 ? 1.f : -1.f;
#pragma unroll 1
  for (int c0 = 0; c0 < 32; c0 += 16) {
    float x[16], y[16];
    tmem_ld16_nowait(taddr + cb + c0, x);
    if (rot) tmem_ld16_nowait(taddr + pb + c0, y);
    tmem_wait_ld();
    uint32_t pk[8];
#pragma unroll
    for (int e = 0; e < 16; e += 2) {
      float o0 = x[e], o1 = x[e + 1];
      if (rot) {
        const float4 t = *reinterpret_cast<const float4*>(rtab + 2 * (pos * 32 + c0 + e));
        o0 = (x[e] * t.x + sg * y[e] * t.y) * scale;
        o1 = (x[e + 1] * t.z + sg * y[e + 1] * t.w) * scale;
      }
      pk[e / 2] = pack_bf16x2(o0, o1);
    }
    const int ch = (cb + c0) >> 3;
    *reinterpret_cast<uint4*>(buf + r * 128 + (((ch) ^ (r & 7)) << 4)) =
        make_uint4(pk[0], pk[1], pk[2], pk[3]);
    *reinterpret_cast<uint4*>(buf + r * 128 + (((ch + 1) ^ (r & 7)) << 4)) =
        make_uint4(pk[4], pk[5], pk[6], pk[7]);
  }
}

// The elementwise warps' barrier (named barrier 1, BW_EW warps).
__device__ __forceinline__ void ew_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(BW_EW * 32) : "memory");
}

// A staged [128][64] bf16 tile to 128 rows of global memory (row i at row_base(i)), by the
// elementwise threads (et = 0 .. BW_EW*32 - 1): eight consecutive threads write one row's
// 128 bytes.
template <class RowBase>
__device__ __forceinline__ void staged_rows_out(const uint8_t* buf, int et, RowBase row_base) {
#pragma unroll 1
  for (int i = et; i < 128 * 8; i += BW_EW * 32) {
    const int row = i >> 3, c = i & 7;
    const uint4 v = *reinterpret_cast<const uint4*>(buf + row * 128 + ((c ^ (row & 7)) << 4));
    *reinterpret_cast<uint4*>(row_base(row) + c * 8) = v;
  }
}

template <bool DUAL>
__global__ void __launch_bounds__(BW_THREADS, KvCfg<DUAL>::CTAS)
    flash_tc_bwd_kv_kernel(const __grid_constant__ CUtensorMap tmK,
                           const __grid_constant__ CUtensorMap tmV,
                           const __grid_constant__ CUtensorMap tmKd,
                           const __grid_constant__ CUtensorMap tmVd,
                           const __grid_constant__ CUtensorMap tmQ,
                           const __grid_constant__ CUtensorMap tmdO,
                           const __grid_constant__ CUtensorMap tmQd,
                           const __grid_constant__ CUtensorMap tmdOd, const FtbParams prm) {
  using C = KvCfg<DUAL>;
  const FtbParams p = prm;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t res_full, s_full, s_free, p_full, o_done, drain;
  __shared__ __align__(8) uint64_t st_full[C::STAGES], st_empty[C::STAGES];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sRes = smem;                                  // K, V, K', V'
  uint8_t* sSt = smem + C::NRES * ROWS128_B;             // stage: Q, dO, Q', dO', statistics
  uint8_t* sOp = sSt + C::STAGES * C::STAGE_B;           // P^T, dS^T, P'^T, dS'^T
  // grid (heads, key tiles): heads fastest, and key tile 0 meets the most query tiles
  const int kt = static_cast<int>(blockIdx.y);
  const int bh = static_cast<int>(blockIdx.x);
  const int row0 = bh * p.S;
  const int key0 = kt * 128;
  const int j0 = key0 / BT_Q;                            // first query tile on the diagonal
  const int ntile = p.S / BT_Q - j0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&res_full, 1);
    mbar_init(&s_full, 1);
    mbar_init(&s_free, BW_EW);
    mbar_init(&p_full, BW_EW);
    mbar_init(&o_done, 1);
    mbar_init(&drain, 1);
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(&st_full[i], 1);
      mbar_init(&st_empty[i], 1);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmdO);
    if (DUAL) {
      prefetch_tmap(&tmKd);
      prefetch_tmap(&tmVd);
      prefetch_tmap(&tmQd);
      prefetch_tmap(&tmdOd);
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
      mbar_expect_tx(&res_full, C::NRES * ROWS128_B);
      tma_load_3d(sRes, &tmK, &res_full, 0, row0 + key0, 0);
      tma_load_3d(sRes + ROWS128_B, &tmV, &res_full, 0, row0 + key0, 0);
      if (DUAL) {
        tma_load_3d(sRes + 2 * ROWS128_B, &tmKd, &res_full, 0, row0 + key0, 0);
        tma_load_3d(sRes + 3 * ROWS128_B, &tmVd, &res_full, 0, row0 + key0, 0);
      }
      int issued = 0;
      for (int i = 0; i < ntile; ++i, ++issued) {
        const int st = i % C::STAGES;
        const uint32_t ph = (i / C::STAGES) & 1;
        if (!fwait(&st_empty[st], ph ^ 1, p.status, abort)) break;
        mbar_expect_tx(&st_full[st], C::NT * ROWS64_B + C::NSTAT * BT_Q * 4);
        uint8_t* b = sSt + st * C::STAGE_B;
        const int qr = row0 + (j0 + i) * BT_Q;
        tma_load_3d(b, &tmQ, &st_full[st], 0, qr, 0);
        tma_load_3d(b + C::OFF_DO, &tmdO, &st_full[st], 0, qr, 0);
        bulk_load(b + C::STAT_OFF, p.lse + qr, BT_Q * 4, &st_full[st]);
        bulk_load(b + C::STAT_OFF + 256, p.D + qr, BT_Q * 4, &st_full[st]);
        if (DUAL) {
          tma_load_3d(b + ROWS64_B, &tmQd, &st_full[st], 0, qr, 0);
          tma_load_3d(b + 3 * ROWS64_B, &tmdOd, &st_full[st], 0, qr, 0);
          bulk_load(b + C::STAT_OFF + 512, p.rbar + qr, BT_Q * 4, &st_full[st]);
          bulk_load(b + C::STAT_OFF + 768, p.Dd + qr, BT_Q * 4, &st_full[st]);
        }
      }
      // every load issued has landed before the CTA can end
      mbar_wait(&res_full, 0, p.status, FTC_WAIT_NS);
      drain_loads(st_full, issued, C::STAGES, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer -------------------------------------------------------------------
      const uint32_t idS = idesc_bf16(128, BT_Q);
      const uint32_t idA = idesc_bf16(128, HD) | (1u << 16);   // B (Q, dO) read MN-major
      const uint32_t aK = smem_u32(sRes), aV = aK + ROWS128_B;
      const uint32_t aKd = aK + 2 * ROWS128_B, aVd = aK + 3 * ROWS128_B;
      const uint32_t aP = smem_u32(sOp), adS = aP + OPND_B;
      const uint32_t aPd = aP + 2 * OPND_B, adSd = aP + 3 * OPND_B;
      // operand descriptors, built once: a byte offset moves a descriptor by offset >> 4
      const uint64_t dK = sdesc_sw128(aK), dV = sdesc_sw128(aV);
      const uint64_t dKd = sdesc_sw128(aKd), dVd = sdesc_sw128(aVd);
      const uint64_t dP = sdesc_sw128(aP), ddS = sdesc_sw128(adS);
      const uint64_t dPd = sdesc_sw128(aPd), ddSd = sdesc_sw128(adSd);
      const uint64_t dSt = sdesc_sw128(smem_u32(sSt)), mSt = sdesc_mn_sw128(smem_u32(sSt));
      constexpr uint64_t ST_STEP = C::STAGE_B >> 4, DO_STEP = C::OFF_DO >> 4;
      // scores of query tile i (waits for its stage).  Dual: the products that share an A
      // operand run as one N = 128 MMA over the adjacent B tiles and TMEM accumulators,
      // K [Q | Q']^T -> [S^T | S'^T] and V [dO | dO']^T -> [dP^T | dP'^T], then the
      // remaining terms K' Q^T, V' dO^T accumulate into the tangents.
      const uint32_t idS2 = idesc_bf16(128, 2 * BT_Q);
      auto scores = [&](int i) -> bool {
        const int st = i % C::STAGES;
        if (!fwait(&st_full[st], (i / C::STAGES) & 1, p.status, abort)) return false;
        tc_fence_after();
        const uint64_t dQ = dSt + st * ST_STEP, ddO = dQ + DO_STEP;
        if (DUAL) {
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dK + 2 * kk, dQ + 2 * kk, idS2, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DP, dV + 2 * kk, ddO + 2 * kk, idS2, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_SD, dKd + 2 * kk, dQ + 2 * kk, idS, 1);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DPD, dVd + 2 * kk, ddO + 2 * kk, idS, 1);
        } else {
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dK + 2 * kk, dQ + 2 * kk, idS, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DP, dV + 2 * kk, ddO + 2 * kk, idS, kk > 0);
        }
        mma_commit(&s_full);
        return true;
      };
      bool ok = fwait(&res_full, 0, p.status, abort) && scores(0);
      for (int i = 0; ok && i < ntile; ++i) {
        // the elementwise warps have read the scores of tile i: the next tile's may overwrite
        if (!fwait(&s_free, i & 1, p.status, abort)) break;
        if (i + 1 < ntile && !scores(i + 1)) break;
        if (!fwait(&p_full, i & 1, p.status, abort)) break;
        tc_fence_after();
        const int st = i % C::STAGES;
        const uint64_t mQ = mSt + st * ST_STEP, mdO = mQ + DO_STEP;
        // dual: P^T [dO | dO'] -> [dV | dV'] and dS^T [Q | Q'] -> [dK | dK'] as N = 128
        // MMAs (the tangent tiles sit one 64-column MN box after the primal ones), then
        // P'^T dO into dV' and dS'^T Q into dK'
        const uint32_t idA2 = idesc_bf16(128, 2 * HD) | (1u << 16);
#pragma unroll
        for (int kk = 0; kk < BT_Q / 16; ++kk) {
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          const uint64_t bO = mdO + 128 * kk, bQ = mQ + 128 * kk;
          if (DUAL) {
            mma_bf16(tb + C::C_DV, dP + 2 * kk, bO, idA2, acc);
            mma_bf16(tb + C::C_DK, ddS + 2 * kk, bQ, idA2, acc);
            mma_bf16(tb + C::C_DVD, dPd + 2 * kk, bO, idA, 1);
            mma_bf16(tb + C::C_DKD, ddSd + 2 * kk, bQ, idA, 1);
          } else {
            mma_bf16(tb + C::C_DV, dP + 2 * kk, bO, idA, acc);
            mma_bf16(tb + C::C_DK, ddS + 2 * kk, bQ, idA, acc);
          }
        }
        mma_commit(&st_empty[st]);
        mma_commit(&o_done);
      }
      // every MMA issued here has completed before TMEM is released
      mma_commit(&drain);
      mbar_wait(&drain, 0, p.status, FTC_WAIT_NS);
    }
    __syncwarp();
  } else {
    // ---- elementwise: key row r (TMEM lane r), query columns cb .. cb + 31 -----------------
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const int cb = ((warp - 2) >> 2) * 32;
    const uint32_t lo = static_cast<uint32_t>(q4 * 32) << 16;
    const int key = key0 + r;
    bool ok = true;
    for (int i = 0; i < ntile; ++i) {
      if (!wwait(&s_full, i & 1, p.status, abort)) { ok = false; break; }
      tc_fence_after();
      const float4* stat = reinterpret_cast<const float4*>(
          sSt + (i % C::STAGES) * C::STAGE_B + C::STAT_OFF);   // lse, D, rbar, D' (16 float4 each)
      const int qbase = (j0 + i) * BT_Q;
      uint32_t pk[16], dsk[16], pdk[DUAL ? 16 : 1], dsdk[DUAL ? 16 : 1];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int c0 = cb + 16 * h;
        float sv[16], dp[16], sd[16], dpd[16];
        tmem_ld16_nowait(tb + lo + C::C_S + c0, sv);
        tmem_ld16_nowait(tb + lo + C::C_DP + c0, dp);
        if (DUAL) {
          tmem_ld16_nowait(tb + lo + C::C_SD + c0, sd);
          tmem_ld16_nowait(tb + lo + C::C_DPD + c0, dpd);
        }
        tmem_wait_ld();
        if (h == 1) {
          // this tile's scores are read: the next tile's may be computed meanwhile
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_local(&s_free);
        }
#pragma unroll
        for (int e = 0; e < 16; e += 4) {
          const int c = c0 + e;
          const float4 l4 = stat[c / 4], d4 = stat[16 + c / 4];
          float4 rb4 = make_float4(0.f, 0.f, 0.f, 0.f), dd4 = rb4;
          if (DUAL) { rb4 = stat[32 + c / 4]; dd4 = stat[48 + c / 4]; }
          const float lv[4] = {l4.x, l4.y, l4.z, l4.w}, dv[4] = {d4.x, d4.y, d4.z, d4.w};
          const float rv[4] = {rb4.x, rb4.y, rb4.z, rb4.w}, ddv[4] = {dd4.x, dd4.y, dd4.z, dd4.w};
          float pv[4], dsv[4], pdv[4], dsdv[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float pp = qbase + c + u >= key ? __expf(sv[e + u] - lv[u]) : 0.f;
            const float dpm = dp[e + u] - dv[u];
            pv[u] = pp;
            dsv[u] = pp * dpm;
            if (DUAL) {
              const float pd = pp * (sd[e + u] - rv[u]);
              pdv[u] = pd;
              dsdv[u] = pd * dpm + pp * (dpd[e + u] - ddv[u]);
            }
          }
          const int k = (16 * h + e) / 2;
          pk[k] = pack_bf16x2(pv[0], pv[1]);
          pk[k + 1] = pack_bf16x2(pv[2], pv[3]);
          dsk[k] = pack_bf16x2(dsv[0], dsv[1]);
          dsk[k + 1] = pack_bf16x2(dsv[2], dsv[3]);
          if (DUAL) {
            pdk[k] = pack_bf16x2(pdv[0], pdv[1]);
            pdk[k + 1] = pack_bf16x2(pdv[2], pdv[3]);
            dsdk[k] = pack_bf16x2(dsdv[0], dsdv[1]);
            dsdk[k + 1] = pack_bf16x2(dsdv[2], dsdv[3]);
          }
        }
      }
      // the previous tile's accumulating products have read the A operands
      if (i > 0 && !wwait(&o_done, (i - 1) & 1, p.status, abort)) { ok = false; break; }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t o = swz(r, cb / 8 + j);
        *reinterpret_cast<uint4*>(sOp + o) = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
        *reinterpret_cast<uint4*>(sOp + OPND_B + o) =
            make_uint4(dsk[4 * j], dsk[4 * j + 1], dsk[4 * j + 2], dsk[4 * j + 3]);
        if (DUAL) {
          *reinterpret_cast<uint4*>(sOp + 2 * OPND_B + o) =
              make_uint4(pdk[4 * j], pdk[4 * j + 1], pdk[4 * j + 2], pdk[4 * j + 3]);
          *reinterpret_cast<uint4*>(sOp + 3 * OPND_B + o) =
              make_uint4(dsdk[4 * j], dsdk[4 * j + 1], dsdk[4 * j + 2], dsdk[4 * j + 3]);
        }
      }
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_local(&p_full);
    }
    // ---- outputs: dV, dK (dV', dK') rows of this key, this thread's columns ---------------
    const bool have = ok && wwait(&o_done, (ntile - 1) & 1, p.status, abort);
    if (have) tc_fence_after();
    if (p.dqkv) {
      // merged rows: token b*S + key, k part (rotated) and v part of head h, staged in the
      // A-operand buffers (the last products have read them) and written row by row; every
      // elementwise thread meets the barrier, with or without a result (a timed-out call
      // reports its status and its outputs are void)
      if (have) {
        stage_merged_row(tb + lo + C::C_DK, cb, true, key, p.rope, 1.f, sOp, r);
        stage_merged_row(tb + lo + C::C_DV, cb, false, key, p.rope, 1.f, sOp + OPND_B, r);
        if (DUAL) {
          stage_merged_row(tb + lo + C::C_DKD, cb, true, key, p.rope, 1.f, sOp + 2 * OPND_B, r);
          stage_merged_row(tb + lo + C::C_DVD, cb, false, key, p.rope, 1.f, sOp + 3 * OPND_B, r);
        }
      }
      ew_bar();
      if (have) {
        const int hh = bh % p.H, bb = bh / p.H, dm = p.H * HD;
        const int et = threadIdx.x - 64;
        auto base = [&](__nv_bfloat16* out, int part) {
          return [=](int i) {
            return out + (static_cast<int64_t>(bb) * p.S + key0 + i) * p.ldq + part * dm + hh * HD;
          };
        };
        staged_rows_out(sOp, et, base(p.dqkv, 1));
        staged_rows_out(sOp + OPND_B, et, base(p.dqkv, 2));
        if (DUAL) {
          staged_rows_out(sOp + 2 * OPND_B, et, base(p.dqkvd, 1));
          staged_rows_out(sOp + 3 * OPND_B, et, base(p.dqkvd, 2));
        }
      }
    } else if (have) {
      const int64_t off = (static_cast<int64_t>(row0) + key) * HD;
      store_acc_row(tb + lo + C::C_DV, p.dV + off, cb);
      store_acc_row(tb + lo + C::C_DK, p.dK + off, cb);
      if (DUAL) {
        store_acc_row(tb + lo + C::C_DVD, p.dVd + off, cb);
        store_acc_row(tb + lo + C::C_DKD, p.dKd + off, cb);
      }
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
__global__ void __launch_bounds__(BW_THREADS, QCfg<DUAL>::CTAS)
    flash_tc_bwd_q_kernel(const __grid_constant__ CUtensorMap tmQ,
                          const __grid_constant__ CUtensorMap tmdO,
                          const __grid_constant__ CUtensorMap tmQd,
                          const __grid_constant__ CUtensorMap tmdOd,
                          const __grid_constant__ CUtensorMap tmK,
                          const __grid_constant__ CUtensorMap tmV,
                          const __grid_constant__ CUtensorMap tmKd,
                          const __grid_constant__ CUtensorMap tmVd, const FtbParams prm) {
  using C = QCfg<DUAL>;
  const FtbParams p = prm;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t res_full, s_full, s_free, p_full, o_done, drain;
  __shared__ __align__(8) uint64_t st_full[C::STAGES], st_empty[C::STAGES];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sRes = smem;                                  // Q, dO, Q', dO'
  uint8_t* sSt = smem + C::NRES * ROWS128_B;             // stage: K, V, K', V'
  uint8_t* sOp = sSt + C::STAGES * C::STAGE_B;           // dS, dS'
  // grid (heads, query tiles): heads fastest, the last query tile (most key tiles) first
  const int nq = p.S / 128;
  const int qt = nq - 1 - static_cast<int>(blockIdx.y);
  const int bh = static_cast<int>(blockIdx.x);
  const int row0 = bh * p.S;
  const int q0 = qt * 128;
  const int ntile = (q0 + 128) / BT_Q;                   // key tiles up to the diagonal
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&res_full, 1);
    mbar_init(&s_full, 1);
    mbar_init(&s_free, BW_EW);
    mbar_init(&p_full, BW_EW);
    mbar_init(&o_done, 1);
    mbar_init(&drain, 1);
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(&st_full[i], 1);
      mbar_init(&st_empty[i], 1);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmdO);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    if (DUAL) {
      prefetch_tmap(&tmQd);
      prefetch_tmap(&tmdOd);
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
      mbar_expect_tx(&res_full, C::NRES * ROWS128_B);
      tma_load_3d(sRes, &tmQ, &res_full, 0, row0 + q0, 0);
      tma_load_3d(sRes + ROWS128_B, &tmdO, &res_full, 0, row0 + q0, 0);
      if (DUAL) {
        tma_load_3d(sRes + 2 * ROWS128_B, &tmQd, &res_full, 0, row0 + q0, 0);
        tma_load_3d(sRes + 3 * ROWS128_B, &tmdOd, &res_full, 0, row0 + q0, 0);
      }
      int issued = 0;
      for (int i = 0; i < ntile; ++i, ++issued) {
        const int st = i % C::STAGES;
        const uint32_t ph = (i / C::STAGES) & 1;
        if (!fwait(&st_empty[st], ph ^ 1, p.status, abort)) break;
        mbar_expect_tx(&st_full[st], C::STAGE_B);
        uint8_t* b = sSt + st * C::STAGE_B;
        const int kr = row0 + i * BT_Q;
        tma_load_3d(b, &tmK, &st_full[st], 0, kr, 0);
        tma_load_3d(b + C::OFF_V, &tmV, &st_full[st], 0, kr, 0);
        if (DUAL) {
          tma_load_3d(b + ROWS64_B, &tmKd, &st_full[st], 0, kr, 0);
          tma_load_3d(b + 3 * ROWS64_B, &tmVd, &st_full[st], 0, kr, 0);
        }
      }
      mbar_wait(&res_full, 0, p.status, FTC_WAIT_NS);
      drain_loads(st_full, issued, C::STAGES, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer -------------------------------------------------------------------
      const uint32_t idS = idesc_bf16(128, BT_Q);
      const uint32_t idA = idesc_bf16(128, HD) | (1u << 16);   // B (K) read MN-major
      const uint32_t aQ = smem_u32(sRes), adO = aQ + ROWS128_B;
      const uint32_t aQd = aQ + 2 * ROWS128_B, adOd = aQ + 3 * ROWS128_B;
      const uint32_t adS = smem_u32(sOp), adSd = adS + OPND_B;
      // operand descriptors, built once: a byte offset moves a descriptor by offset >> 4
      const uint64_t dQ = sdesc_sw128(aQ), ddO = sdesc_sw128(adO);
      const uint64_t dQd = sdesc_sw128(aQd), ddOd = sdesc_sw128(adOd);
      const uint64_t ddS = sdesc_sw128(adS), ddSd = sdesc_sw128(adSd);
      const uint64_t dSt = sdesc_sw128(smem_u32(sSt)), mSt = sdesc_mn_sw128(smem_u32(sSt));
      constexpr uint64_t ST_STEP = C::STAGE_B >> 4, V_STEP = C::OFF_V >> 4;
      // dual: Q [K | K']^T -> [S | S'] and dO [V | V']^T -> [dP | dP'] as N = 128 MMAs,
      // then Q' K^T and dO' V^T accumulate into the tangents
      const uint32_t idS2 = idesc_bf16(128, 2 * BT_Q);
      auto scores = [&](int i) -> bool {
        const int st = i % C::STAGES;
        if (!fwait(&st_full[st], (i / C::STAGES) & 1, p.status, abort)) return false;
        tc_fence_after();
        const uint64_t dK = dSt + st * ST_STEP, dV = dK + V_STEP;
        if (DUAL) {
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dQ + 2 * kk, dK + 2 * kk, idS2, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DP, ddO + 2 * kk, dV + 2 * kk, idS2, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_SD, dQd + 2 * kk, dK + 2 * kk, idS, 1);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DPD, ddOd + 2 * kk, dV + 2 * kk, idS, 1);
        } else {
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_S, dQ + 2 * kk, dK + 2 * kk, idS, kk > 0);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16(tb + C::C_DP, ddO + 2 * kk, dV + 2 * kk, idS, kk > 0);
        }
        mma_commit(&s_full);
        return true;
      };
      bool ok = fwait(&res_full, 0, p.status, abort) && scores(0);
      for (int i = 0; ok && i < ntile; ++i) {
        if (!fwait(&s_free, i & 1, p.status, abort)) break;
        if (i + 1 < ntile && !scores(i + 1)) break;
        if (!fwait(&p_full, i & 1, p.status, abort)) break;
        tc_fence_after();
        const int st = i % C::STAGES;
        const uint64_t mK = mSt + st * ST_STEP;
        // dual: dS [K | K'] -> [dQ | dQ'] as one N = 128 MMA, then dS' K into dQ'
        const uint32_t idA2 = idesc_bf16(128, 2 * HD) | (1u << 16);
#pragma unroll
        for (int kk = 0; kk < BT_Q / 16; ++kk) {
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          const uint64_t bK = mK + 128 * kk;
          if (DUAL) {
            mma_bf16(tb + C::C_DQ, ddS + 2 * kk, bK, idA2, acc);
            mma_bf16(tb + C::C_DQD, ddSd + 2 * kk, bK, idA, 1);
          } else {
            mma_bf16(tb + C::C_DQ, ddS + 2 * kk, bK, idA, acc);
          }
        }
        mma_commit(&st_empty[st]);
        mma_commit(&o_done);
      }
      mma_commit(&drain);
      mbar_wait(&drain, 0, p.status, FTC_WAIT_NS);
    }
    __syncwarp();
  } else {
    // ---- elementwise: query row r (TMEM lane r), key columns cb .. cb + 31 -----------------
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const int cb = ((warp - 2) >> 2) * 32;
    const uint32_t lo = static_cast<uint32_t>(q4 * 32) << 16;
    const int q = q0 + r;
    const int64_t gi = static_cast<int64_t>(row0) + q;
    const float lse = p.lse[gi], Dv = p.D[gi];
    const float rb = DUAL ? p.rbar[gi] : 0.f, Ddv = DUAL ? p.Dd[gi] : 0.f;
    bool ok = true;
    for (int i = 0; i < ntile; ++i) {
      if (!wwait(&s_full, i & 1, p.status, abort)) { ok = false; break; }
      tc_fence_after();
      const int kbase = i * BT_Q;
      uint32_t dsk[16], dsdk[DUAL ? 16 : 1];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int c0 = cb + 16 * h;
        float sv[16], dp[16], sd[16], dpd[16];
        tmem_ld16_nowait(tb + lo + C::C_S + c0, sv);
        tmem_ld16_nowait(tb + lo + C::C_DP + c0, dp);
        if (DUAL) {
          tmem_ld16_nowait(tb + lo + C::C_SD + c0, sd);
          tmem_ld16_nowait(tb + lo + C::C_DPD + c0, dpd);
        }
        tmem_wait_ld();
        if (h == 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_local(&s_free);
        }
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          float dsv[2], dsdv[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int key = kbase + c0 + e + u;
            const float pp = key <= q ? __expf(sv[e + u] - lse) : 0.f;
            const float dpm = dp[e + u] - Dv;
            dsv[u] = pp * dpm;
            if (DUAL) {
              const float pd = pp * (sd[e + u] - rb);
              dsdv[u] = pd * dpm + pp * (dpd[e + u] - Ddv);
            }
          }
          dsk[(16 * h + e) / 2] = pack_bf16x2(dsv[0], dsv[1]);
          if (DUAL) dsdk[(16 * h + e) / 2] = pack_bf16x2(dsdv[0], dsdv[1]);
        }
      }
      if (i > 0 && !wwait(&o_done, (i - 1) & 1, p.status, abort)) { ok = false; break; }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t o = swz(r, cb / 8 + j);
        *reinterpret_cast<uint4*>(sOp + o) =
            make_uint4(dsk[4 * j], dsk[4 * j + 1], dsk[4 * j + 2], dsk[4 * j + 3]);
        if (DUAL)
          *reinterpret_cast<uint4*>(sOp + OPND_B + o) =
              make_uint4(dsdk[4 * j], dsdk[4 * j + 1], dsdk[4 * j + 2], dsdk[4 * j + 3]);
      }
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_local(&p_full);
    }
    const bool have = ok && wwait(&o_done, (ntile - 1) & 1, p.status, abort);
    if (have) tc_fence_after();
    if (p.dqkv) {
      // merged rows: token b*S + q, q part (rotated and scaled) of head h, staged in the
      // A-operand buffers and written row by row (every elementwise thread meets the barrier)
      if (have) {
        stage_merged_row(tb + lo + C::C_DQ, cb, true, q, p.rope, p.qscale, sOp, r);
        if (DUAL) stage_merged_row(tb + lo + C::C_DQD, cb, true, q, p.rope, p.qscale, sOp + OPND_B, r);
      }
      ew_bar();
      if (have) {
        const int hh = bh % p.H, bb = bh / p.H;
        const int et = threadIdx.x - 64;
        auto base = [&](__nv_bfloat16* out) {
          return [=](int i) {
            return out + (static_cast<int64_t>(bb) * p.S + q0 + i) * p.ldq + hh * HD;
          };
        };
        staged_rows_out(sOp, et, base(p.dqkv));
        if (DUAL) staged_rows_out(sOp + OPND_B, et, base(p.dqkvd));
      }
    } else if (have) {
      const int64_t off = gi * HD;
      store_acc_row(tb + lo + C::C_DQ, p.dQ + off, cb);
      if (DUAL) store_acc_row(tb + lo + C::C_DQD, p.dQd + off, cb);
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
cudaError_t launch_ftc_bwd(const FlashArgs& a, cudaStream_t s) {
  using KC = KvCfg<DUAL>;
  using QC = QCfg<DUAL>;
  const int rows = a.BH * a.S;
  CUtensorMap k128[4], q64[4], q128[4], k64[4];
  const void* kv[4] = {a.K, a.V, a.Kd, a.Vd};
  const void* qo[4] = {a.Q, a.dO, a.Qd, a.dOd};
  for (int i = 0; i < 4; ++i) {
    memset(&k128[i], 0, sizeof(CUtensorMap)); memset(&q64[i], 0, sizeof(CUtensorMap));
    memset(&q128[i], 0, sizeof(CUtensorMap)); memset(&k64[i], 0, sizeof(CUtensorMap));
    if (i >= 2 && !DUAL) continue;
    if (!make_map(&k128[i], kv[i], HD, rows, HD, 128) || !make_map(&k64[i], kv[i], HD, rows, HD, BT_Q) ||
        !make_map(&q128[i], qo[i], HD, rows, HD, 128) || !make_map(&q64[i], qo[i], HD, rows, HD, BT_Q))
      return cudaErrorInvalidValue;
  }
  static PerDeviceOnce attr_once;
  cudaError_t e = attr_once.run([](int&) {
    cudaError_t r = cudaFuncSetAttribute(flash_tc_bwd_kv_kernel<DUAL>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, KC::SMEM);
    if (r != cudaSuccess) return r;
    return cudaFuncSetAttribute(flash_tc_bwd_q_kernel<DUAL>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, QC::SMEM);
  });
  if (e != cudaSuccess) return e;
  FtbParams p;
  p.BH = a.BH;
  p.S = a.S;
  p.lse = a.lse;
  p.rbar = a.rbar;
  p.D = a.D;
  p.Dd = a.Dd;
  p.dQ = a.dQ; p.dQd = a.dQd;
  p.dK = a.dK; p.dKd = a.dKd;
  p.dV = a.dV; p.dVd = a.dVd;
  p.status = a.status;
  p.dqkv = a.dqkv;
  p.dqkvd = DUAL ? a.dqkvd : nullptr;
  p.H = a.H;
  p.ldq = a.ldq;
  p.rope = a.rope;
  p.qscale = a.qscale;
  const dim3 grid(a.BH, a.S / 128);
  e = launch_k(flash_tc_bwd_kv_kernel<DUAL>, grid, dim3(BW_THREADS), KC::SMEM, s, k128[0],
               k128[1], k128[2], k128[3], q64[0], q64[1], q64[2], q64[3], p);
  if (e != cudaSuccess) return e;
  return launch_k(flash_tc_bwd_q_kernel<DUAL>, grid, dim3(BW_THREADS), QC::SMEM, s, q128[0],
                  q128[1], q128[2], q128[3], k64[0], k64[1], k64[2], k64[3], p);
}

}  // namespace
}  // namespace mf

namespace mf {

bool flash_tc_supported(int S, int dh) { return dh == HD && S > 0 && S % TQ == 0; }

cudaError_t flash_tc_fwd(const FlashArgs& a, bool dual, cudaStream_t s) {
  if (!flash_tc_supported(a.S, HD) || a.BH < 1) return cudaErrorInvalidValue;
  return dual ? launch_ftc_fwd<true>(a, s) : launch_ftc_fwd<false>(a, s);
}

bool flash_tc_bwd_supported(const FlashArgs& a, bool dual) {
  if (!flash_tc_supported(a.S, HD) || a.BH < 1) return false;
  // merged outputs: 16-byte aligned rows, whole heads, a RoPE table
  if (a.dqkv && (a.H < 1 || a.BH % a.H || !a.rope || (a.ldq & 7) ||
                 (reinterpret_cast<uintptr_t>(a.dqkv) & 15) ||
                 (dual && (!a.dqkvd || (reinterpret_cast<uintptr_t>(a.dqkvd) & 15)))))
    return false;
  // the row statistics stream into shared memory by bulk copies of 64 floats
  const void* stats[4] = {a.lse, a.D, a.rbar, a.Dd};
  for (int i = 0; i < (dual ? 4 : 2); ++i)
    if (!stats[i] || (reinterpret_cast<uintptr_t>(stats[i]) & 15)) return false;
  return true;
}

cudaError_t flash_tc_bwd(const FlashArgs& a, bool dual, cudaStream_t s) {
  if (!flash_tc_bwd_supported(a, dual)) return cudaErrorInvalidValue;
  return dual ? launch_ftc_bwd<true>(a, s) : launch_ftc_bwd<false>(a, s);
}

}  // namespace mf
