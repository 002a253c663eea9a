// Persistent CTA-pair form of the tcgen05 dual GEMM (MF_OPT_GEMM_PERSISTENT, on by default).
//
// The one-tile kernels of tc_gemm_impl.cuh give every 256 x BN output tile its own CTA pair,
// so each tile pays the prologue (barrier init, TMEM allocation, tensor-map prefetch) and its
// epilogue (TMEM drain, activation, stores) never overlaps a main loop.  On short-K products
// (the weight tangent of Section 3's forward-over-reverse HVP has K = batch) the epilogue
// takes about as long as the main loop.  Here one cluster of two CTAs per SM pair stays
// resident for the whole GEMM and walks a static list of tiles: pair j of P takes tiles
// j, j + P, j + 2P, ...  TMEM holds two accumulator sets when they fit its 512 columns, so
// the epilogue warps drain tile i from one set while the MMA thread accumulates tile i + 1
// into the other, and the shared-memory stage ring runs on across tile boundaries, so the
// TMA producer fetches the next tile's first K blocks during the current tile's last MMAs.
//
// Roles per CTA (as in the one-tile pair kernel): warp 0 issues the TMA loads of this CTA's
// 128 rows of A and BN/2 rows of B; warp 1 owns TMEM, and in the even CTA one thread issues
// tcgen05.mma.cta_group::2 (M = 256) for the pair; epi_warps_p warps drain this CTA's 128
// accumulator rows, one TMEM lane quadrant and one column share per warp; full 16-column
// chunks are stored through a 2 KB row-block buffer per warp (8 rows x 64 bytes per warp
// store, see epilogue16_rows), ragged ones straight from registers.
//
// Barriers: full[s] / empty[s] per pipeline stage (full in the even CTA, completed by both
// CTAs' TMA bytes; empty in both, by the MMA commit multicast); per accumulator set,
// acc_full (MMA commit, multicast to both CTAs) and acc_empty (in the even CTA; every
// epilogue warp of both CTAs arrives once after its last TMEM read of the tile).  Every wait
// is bounded; the first role to time out records DEV_TIMEOUT and raises a CTA-local abort
// flag, after which the CTA's other roles stop waiting and leave their tile loops.
#include "tc_gemm_impl.cuh"

namespace mf {

int g_gemm_persist = 2;

namespace {

// Epilogue warps per CTA: twelve (three per TMEM lane quadrant) where the epilogue is the
// longer role, eight for the backward epilogues, whose prefetched pre-activations need the
// registers of a 320-thread CTA.
template <int MODE>
__host__ __device__ constexpr int epi_warps_p() { return MODE == EPI_ACT_BWD ? 8 : 12; }
template <int MODE>
__host__ __device__ constexpr int threads_p() { return 64 + 32 * epi_warps_p<MODE>(); }

// Accumulator blocks per logical accumulator (the rotation of mma_loop) when two sets of
// `nacc` accumulators must fit TMEM, else the one-set figure of the one-tile kernels.
__host__ __device__ constexpr int persist_nsub(int nacc, int bn) {
  return 2 * nacc * 4 * bn <= 512 ? 4
         : 2 * nacc * 2 * bn <= 512 ? 2
         : 2 * nacc * 1 * bn <= 512 ? 1
                                    : acc_blocks(nacc, bn);
}
__host__ __device__ constexpr int persist_sets(int nacc, int bn) {
  return 2 * nacc * persist_nsub(nacc, bn) * bn <= 512 ? 2 : 1;
}

// Tile list order (L2 reuse): per batch entry, groups of `group` 256-row blocks; inside a
// group the row blocks vary fastest, then the n tile; groups follow each other.  The pairs
// running at one time then share a few row blocks of A and a band of n tiles of B.
struct PersistParams {
  int tiles_n, pairs_m, ntiles, group;
  int nsets;                      // accumulator sets in TMEM (1 or 2)
  int set_cols;                   // TMEM columns of one set
};

__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Arrive on an mbarrier given by its shared::cluster address (this CTA's or the peer's).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}

// Bounded wait of the MMA issuer and the epilogue warps (limit_ns = TcParams::wait_ns) that
// gives up at once, unless the phase has already completed, when another of these roles in
// this CTA has timed out.  CLUSTER
// selects cluster-scope acquire (arrivals from the peer CTA).  The TMA producer never looks
// at the abort flag: it waits with DRAIN_NS only, so both CTAs' producers see the same MMA
// commits and stop at the same stage (see tc_gemm_impl.cuh).
template <bool CLUSTER>
__device__ __forceinline__ bool pwait(uint64_t* bar, uint32_t parity, int* status,
                                      volatile int* abort, long long limit_ns) {
  auto probe = [&]() {
    return CLUSTER ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity);
  };
  if (probe()) return true;
  if (*abort) return false;
  const long long t0 = global_ns();
  while (true) {
    if (probe()) return true;
    if (*abort) return false;
    if (global_ns() - t0 > limit_ns) {
      if (status) atomicMax(status, DEV_TIMEOUT);
      *abort = 1;
      return false;
    }
  }
}

// The same wait on a precomputed shared::cta address (this CTA's barrier, CTA-scope acquire).
__device__ __forceinline__ bool pwait_addr(uint32_t addr, uint32_t parity, int* status,
                                           volatile int* abort, long long limit_ns) {
  if (mbar_try_wait_addr(addr, parity)) return true;
  if (*abort) return false;
  const long long t0 = global_ns();
  while (true) {
    if (mbar_try_wait_addr(addr, parity)) return true;
    if (*abort) return false;
    if (global_ns() - t0 > limit_ns) {
      if (status) atomicMax(status, DEV_TIMEOUT);
      *abort = 1;
      return false;
    }
  }
}

// Commit of the MMA issuer's earlier tcgen05 work to a barrier of the even CTA only.
__device__ __forceinline__ void mma_commit_even(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(static_cast<uint16_t>(1))
      : "memory");
}

// The MMA issuer's ring state, carried across tiles: stage s and its phase, the barrier
// addresses of stage 0 and the stage-0 operand descriptors (see op_desc).
struct IssueRing {
  uint64_t a0s, a1s, b0s, b1s, stage_step, soff;
  uint32_t full0, empty0, ph;
  int s;
};

// The MMA issuer's loop over the K blocks of one tile, with the issue order and the
// accumulator-block rotation of mma_loop (KA = 1, pair form); the ring position continues
// from the pair's earlier tiles.  The tile's accumulators start at TMEM address tset.  Once
// `live` is false (a wait gave up) the stages are consumed without MMAs.  Returns false if
// even a drain wait gave up.
template <int BN, unsigned TERMS, int NSUB>
__device__ __forceinline__ bool mma_tile(const MmaLoop& L, IssueRing& R, uint32_t tset,
                                         unsigned terms_rt, int nsub_rt, volatile int* abort,
                                         bool& live) {
  const uint32_t idesc = idesc_bf16(2 * BM, BN) | (static_cast<uint32_t>(L.a_mn) << 15) |
                         (static_cast<uint32_t>(L.b_mn) << 16);
  const uint64_t stepA = L.a_mn ? 128u : 2u, stepB = L.b_mn ? 128u : 2u;
  const unsigned terms = TERMS ? TERMS : terms_rt;
  const uint32_t nsub = NSUB ? static_cast<uint32_t>(NSUB) : static_cast<uint32_t>(nsub_rt);
  const uint32_t p0 = __popc(terms & (T_C0_A0B0 | T_C0_A1B0 | T_C0_A0B1 | T_C0_A1B1));
  const uint32_t p1 = __popc(terms & (T_C1_A1B0 | T_C1_A0B1));
  for (int i = 0; i < L.nk; ++i) {
    const uint32_t fb = R.full0 + 8u * static_cast<uint32_t>(R.s);
    const uint32_t eb = R.empty0 + 8u * static_cast<uint32_t>(R.s);
    if (!live || !pwait_addr(fb, R.ph, L.status, abort, L.wait_ns)) {
      live = false;
      if (!mbar_wait_addr(fb, R.ph, L.status, DRAIN_NS)) return false;
      mma_commit_pair_addr(eb);
    } else {
      tc_fence_after();
      const uint64_t a0 = R.a0s + R.soff, a1 = R.a1s + R.soff;
      const uint64_t b0 = R.b0s + R.soff, b1 = R.b1s + R.soff;
#pragma unroll
      for (int kk = 0; kk < BK / 16; ++kk) {
        const uint64_t advA = static_cast<uint64_t>(kk) * stepA;
        const uint64_t advB = static_cast<uint64_t>(kk) * stepB;
        const bool first = i == 0;
        uint32_t q0 = static_cast<uint32_t>(kk) * p0, q1 = static_cast<uint32_t>(kk) * p1;
        auto mma = [&](uint32_t c, uint64_t ad, uint64_t bd) {
          uint32_t& q = c ? q1 : q0;
          const uint32_t blk = c * nsub + (q & (nsub - 1));
          const uint32_t f = (first && q < nsub) ? 0u : 1u;
          ++q;
          mma_bf16_pair(tset + blk * BN, ad, bd, idesc, f);
        };
        if (terms & T_C0_A0B0) mma(0, a0 + advA, b0 + advB);
        if (terms & T_C1_A1B0) mma(1, a1 + advA, b0 + advB);
        if (terms & T_C0_A1B0) mma(0, a1 + advA, b0 + advB);
        if (terms & T_C1_A0B1) mma(1, a0 + advA, b1 + advB);
        if (terms & T_C0_A0B1) mma(0, a0 + advA, b1 + advB);
        if (terms & T_C0_A1B1) mma(0, a1 + advA, b1 + advB);
      }
      mma_commit_pair_addr(eb);
    }
    if (++R.s == L.stages) {
      R.s = 0;
      R.ph ^= 1u;
      R.soff = 0;
    } else {
      R.soff += R.stage_step;
    }
  }
  return true;
}

// Product masks the library issues get straight-line MMA sequences (as mma_dispatch).
template <int BN, int MODE>
__device__ __forceinline__ bool mma_tile_dispatch(const MmaLoop& L, IssueRing& R, uint32_t tset,
                                                  unsigned terms, int nsub, volatile int* abort,
                                                  bool& live) {
  constexpr int N1 = persist_nsub(1, BN), N2 = persist_nsub(2, BN);
  switch (terms) {
    case T_C0_A0B0: return mma_tile<BN, T_C0_A0B0, N1>(L, R, tset, terms, nsub, abort, live);
    case T_C0_A0B0 | T_C1_A1B0 | T_C1_A0B1:
      return mma_tile<BN, T_C0_A0B0 | T_C1_A1B0 | T_C1_A0B1, N2>(L, R, tset, terms, nsub, abort, live);
    case T_C0_A0B0 | T_C1_A0B1:
      return mma_tile<BN, T_C0_A0B0 | T_C1_A0B1, N2>(L, R, tset, terms, nsub, abort, live);
    default: break;
  }
  if constexpr (MODE == EPI_STORE) {
    switch (terms) {
      case T_C0_A0B1: return mma_tile<BN, T_C0_A0B1, N1>(L, R, tset, terms, nsub, abort, live);
      case T_C0_A1B0 | T_C0_A0B1:
        return mma_tile<BN, T_C0_A1B0 | T_C0_A0B1, N1>(L, R, tset, terms, nsub, abort, live);
      case T_C0_A0B0 | T_C0_A1B1:
        return mma_tile<BN, T_C0_A0B0 | T_C0_A1B1, N1>(L, R, tset, terms, nsub, abort, live);
      default: break;
    }
  }
  return mma_tile<BN, 0, 0>(L, R, tset, terms, nsub, abort, live);
}

template <int BN, int MODE, int ACT>
__global__ void __launch_bounds__(threads_p<MODE>(), 1)
    tc2p_dual_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                          const __grid_constant__ CUtensorMap tmA1,
                          const __grid_constant__ CUtensorMap tmB0,
                          const __grid_constant__ CUtensorMap tmB1, const TcParams prm,
                          const PersistParams pp) {
  TcParams p = prm;
  float* const C0base = p.C0;
  float* const C1base = p.C1;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t empty_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t acc_full[2];
  __shared__ __align__(8) uint64_t acc_empty[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  constexpr int BH = BN / 2;                 // B rows staged by each CTA
  const uint32_t rank = cluster_rank();      // 0: issues the MMAs, 1: its peer
  const int pair = static_cast<int>(blockIdx.x >> 1);
  const int npairs = static_cast<int>(gridDim.x >> 1);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nk = (p.K + BK - 1) / BK;
  const unsigned terms = p.terms;
  const bool dual = (terms & (T_C1_A1B0 | T_C1_A0B1)) != 0;
  const uint32_t ncols = tmem_cols(pp.nsets * pp.set_cols);
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 2 * epi_warps_p<MODE>());
    }
    mbar_init(&drain_bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (p.a0_off >= 0) prefetch_tmap(&tmA0);
    if (p.a1_off >= 0) prefetch_tmap(&tmA1);
    if (p.b0_off >= 0) prefetch_tmap(&tmB0);
    if (p.b1_off >= 0) prefetch_tmap(&tmB1);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_slot)),
                 "r"(ncols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
  }
  tc_fence_before();
  cluster_sync_all();          // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  const uint32_t tbase = tmem_slot;
  volatile int* abort = &abort_flag;
  pdl_entry();

  // Tile t of the list (grouped order, see PersistParams).
  auto coords = [&](int t, int& bz, int& mp, int& tn) {
    const int per_batch = pp.tiles_n * pp.pairs_m;
    bz = t / per_batch;
    const int r = t % per_batch;
    const int gsz = pp.group * pp.tiles_n;
    const int g = r / gsz, w = r % gsz;
    const int rows = min(pp.group, pp.pairs_m - g * pp.group);
    mp = g * pp.group + w % rows;
    tn = w / rows;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer: this CTA's 128 rows of A and BN/2 rows of B per stage ------------
      const int stages = p.stages, stage_bytes = p.stage_bytes;
      const int a0_off = p.a0_off, a1_off = p.a1_off, b0_off = p.b0_off, b1_off = p.b1_off;
      int* const status = p.status;
      const uint32_t full0 = dsmem_addr(smem_u32(&full_bar[0]), 0);   // even CTA's barriers
      int g = 0;   // K blocks issued so far (ring position)
      bool live = true;
      for (int t = pair; t < pp.ntiles && live; t += npairs) {
        int bz, mp, tn;
        coords(t, bz, mp, tn);
        const int m0 = mp * (2 * BM) + static_cast<int>(rank) * BM;
        const int nb0 = tn * BN + static_cast<int>(rank) * BH;
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = g % stages;
          const uint32_t ph = (g / stages) & 1;
          if (!mbar_wait(&empty_bar[s], ph ^ 1, status, DRAIN_NS)) { live = false; break; }
          if (rank == 0) mbar_expect_tx(&full_bar[s], 2 * stage_bytes);
          const uint32_t bar = full0 + static_cast<uint32_t>(s) * 8u;
          uint8_t* st = smem + s * stage_bytes;
          const int k = i * BK;
          if (p.a_mn) {
            for (int j = 0; j < BM / 64; ++j) {
              if (a0_off >= 0) tma_load_3d_pair(st + a0_off + j * MN_BOX, &tmA0, bar, m0 + 64 * j, k, bz);
              if (a1_off >= 0) tma_load_3d_pair(st + a1_off + j * MN_BOX, &tmA1, bar, m0 + 64 * j, k, bz);
            }
          } else {
            if (a0_off >= 0) tma_load_3d_pair(st + a0_off, &tmA0, bar, k, m0, bz);
            if (a1_off >= 0) tma_load_3d_pair(st + a1_off, &tmA1, bar, k, m0, bz);
          }
          if (p.b_mn) {
            for (int j = 0; j < BH / 64; ++j) {
              if (b0_off >= 0) tma_load_3d_pair(st + b0_off + j * MN_BOX, &tmB0, bar, nb0 + 64 * j, k, bz);
              if (b1_off >= 0) tma_load_3d_pair(st + b1_off + j * MN_BOX, &tmB1, bar, nb0 + 64 * j, k, bz);
            }
          } else {
            if (b0_off >= 0) tma_load_3d_pair(st + b0_off, &tmB0, bar, k, nb0, bz);
            if (b1_off >= 0) tma_load_3d_pair(st + b1_off, &tmB1, bar, k, nb0, bz);
          }
        }
      }
      if (rank == 0) drain_loads(full_bar, g, stages, status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (rank == 0 && lane == 0) {
      // ---- MMA issuer (single thread of the even CTA) ------------------------------------
      MmaLoop L;
      L.nk = nk; L.stages = p.stages; L.stage_bytes = p.stage_bytes;
      L.a0_off = p.a0_off; L.a1_off = p.a1_off; L.b0_off = p.b0_off; L.b1_off = p.b1_off;
      L.sbase = smem_u32(smem); L.tbase = tbase;
      L.a_mn = p.a_mn; L.b_mn = p.b_mn;
      L.full_bar = full_bar; L.empty_bar = empty_bar; L.status = p.status;
      L.wait_ns = p.wait_ns;
      bool live = true;   // false once a wait gave up: the ring is consumed without MMAs
      IssueRing R;
      R.a0s = op_desc(L.sbase, L.a0_off, L.a_mn);
      R.a1s = op_desc(L.sbase, L.a1_off, L.a_mn);
      R.b0s = op_desc(L.sbase, L.b0_off, L.b_mn);
      R.b1s = op_desc(L.sbase, L.b1_off, L.b_mn);
      R.stage_step = static_cast<uint64_t>(L.stage_bytes >> 4);
      R.soff = 0;
      R.full0 = smem_u32(full_bar);
      R.empty0 = smem_u32(empty_bar);
      R.ph = 0;
      R.s = 0;
      int j = 0;
      for (int t = pair; t < pp.ntiles; t += npairs, ++j) {
        const int set = pp.nsets == 2 ? (j & 1) : 0;
        const int use = pp.nsets == 2 ? (j >> 1) : j;
        // the epilogue warps of both CTAs have read this set's previous tile
        if (live && !pwait<true>(&acc_empty[set], (use & 1) ^ 1, p.status, abort, p.wait_ns))
          live = false;
        tc_fence_after();
        const uint32_t tset = tbase + static_cast<uint32_t>(set * pp.set_cols);
        if (!mma_tile_dispatch<BN, MODE>(L, R, tset, terms, p.nsub, abort, live)) break;
        if (live) mma_commit_pair(&acc_full[set]);
      }
      mma_commit_even(&drain_bar);
      mbar_wait(&drain_bar, 0, p.status, DRAIN_NS);   // every MMA of the pair has completed
    }
    __syncwarp();
  } else {
    // ---- accumulator drain: TMEM lane quadrant = warp % 4, one column share per warp ----
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    // the quadrant's epi_warps_p / 4 warps take its 16-column chunks in turn
    constexpr int CSTEP = 16 * (epi_warps_p<MODE>() / 4);
    const int c_begin = ((warp - 2) >> 2) * 16, c_end = BN;
    const uint32_t empty0 = dsmem_addr(smem_u32(&acc_empty[0]), 0);   // even CTA's barriers
    // full chunks go through this warp's row-block buffer behind the pipeline stages
    uint8_t* const stg = smem + p.stages * p.stage_bytes + (warp - 2) * STG_ROWS_BYTES;
    const bool rows_ok = rows16_ok(p, MODE, dual) &&
                         (p.batch <= 1 || (!(p.bsC0 & 3) && !(p.bsC1 & 3)));
    int j = 0;
    for (int t = pair; t < pp.ntiles; t += npairs, ++j) {
      const int set = pp.nsets == 2 ? (j & 1) : 0;
      const int use = pp.nsets == 2 ? (j >> 1) : j;
      if (!pwait<false>(&acc_full[set], use & 1, p.status, abort, p.wait_ns)) break;
      tc_fence_after();
      int bz, mp, tn;
      coords(t, bz, mp, tn);
      const int m0 = mp * (2 * BM) + static_cast<int>(rank) * BM;
      const int n0 = tn * BN;
      p.C0 = C0base ? C0base + bz * p.bsC0 : nullptr;
      p.C1 = C1base ? C1base + bz * p.bsC1 : nullptr;
      const uint32_t taddr = tbase + lane_off + static_cast<uint32_t>(set * pp.set_cols);
      // backward epilogues: the next full chunk's stored pre-activations load while this
      // chunk is computed
      ZRows zq, zdq, zq_n, zdq_n;
      auto zissue = [&](int c, ZRows& a, ZRows& b) {
        if (rows_ok && n0 + c + 16 <= p.N) {
          zrows_issue(a, lane, m0 + q * 32, p.M, p.epi.Z, p.epi.ldz, n0 + c);
          if (dual) zrows_issue(b, lane, m0 + q * 32, p.M, p.epi.Zd, p.epi.ldz, n0 + c);
        }
      };
      if constexpr (MODE == EPI_ACT_BWD) zissue(c_begin, zq_n, zdq_n);
#pragma unroll 1
      for (int c = c_begin; c < c_end; c += CSTEP) {
        if constexpr (MODE == EPI_ACT_BWD) {
          zq = zq_n;
          zdq = zdq_n;
          if (c + CSTEP < c_end) zissue(c + CSTEP, zq_n, zdq_n);
        }
        float v0[16], v1[16];
        ld_acc16<BN>(taddr, 0, p.nsub, c, v0);
        if (dual) ld_acc16<BN>(taddr, 1, p.nsub, c, v1);
        else {
#pragma unroll
          for (int i = 0; i < 16; ++i) v1[i] = 0.f;
        }
        if (rows_ok && n0 + c + 16 <= p.N)
          epilogue16_rows<MODE, ACT>(p, stg, lane, m0 + q * 32, n0 + c, v0, v1, dual, zq, zdq);
        else if (n0 + c < p.N)
          epilogue16<MODE, ACT>(p, m0 + r, n0 + c, v0, v1, dual);
      }
      // every lane's TMEM reads of this tile are complete (tcgen05.wait::ld in ld_acc16)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(empty0 + static_cast<uint32_t>(set) * 8u);
    }
    tc_fence_before();
  }
  __syncthreads();
  cluster_sync_all();          // both CTAs are done with TMEM and with the peer's barriers
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tbase),
                 "r"(ncols));
  }
}

// Co-resident CTA pairs of one kernel instance (cluster occupancy), measured once per
// device and instance.
template <int BN, int MODE, int ACT>
int max_pairs_on_device(int smem) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int pairs = sms / 2;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(2 * (pairs > 0 ? pairs : 1), 1, 1);
  cfg.blockDim = dim3(threads_p<MODE>(), 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, tc2p_dual_gemm_kernel<BN, MODE, ACT>, &cfg) ==
          cudaSuccess &&
      clusters > 0)
    pairs = clusters;
  else
    cudaGetLastError();   // clear the query's error; keep the SM-count estimate
  if (pairs < 1) pairs = 1;
  return pairs;
}

template <int BN, int MODE, int ACT>
int max_pairs(int smem) {
  static PerDeviceOnce once;
  once.run([smem](int& v) {
    v = max_pairs_on_device<BN, MODE, ACT>(smem);
    return cudaSuccess;
  });
  const int v = once.get();
  return v > 0 ? v : 1;
}

template <int BN, int MODE, int ACT>
cudaError_t launch_cfg2p(const GemmArgs& a, cudaStream_t s, const char** why) {
  constexpr int BH = BN / 2;
  const unsigned t = a.terms;
  const bool useA0 = t & (T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1);
  const bool useA1 = t & (T_C0_A1B0 | T_C1_A1B0 | T_C0_A1B1);
  const bool useB0 = t & (T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0);
  const bool useB1 = t & (T_C0_A0B1 | T_C1_A0B1 | T_C0_A1B1);
  const bool dual = t & (T_C1_A1B0 | T_C1_A0B1);
  const int nacc = dual ? 2 : 1;
  TcParams p;
  memset(&p, 0, sizeof(p));
  p.M = a.M; p.N = a.N; p.K = a.K; p.terms = t;
  const int a_bytes = BM * BK * 2, b_bytes = BH * BK * 2;
  int off = 0;
  p.a0_off = useA0 ? (off += a_bytes, off - a_bytes) : -1;
  p.a1_off = useA1 ? (off += a_bytes, off - a_bytes) : -1;
  p.b0_off = useB0 ? (off += b_bytes, off - b_bytes) : -1;
  p.b1_off = useB1 ? (off += b_bytes, off - b_bytes) : -1;
  p.stage_bytes = off;
  p.tx_bytes = off;
  p.nsub = persist_nsub(nacc, BN);
  // pipeline stages, then one row-block buffer per epilogue warp
  int stages = (220 * 1024 - epi_warps_p<MODE>() * STG_ROWS_BYTES) / off;
  if (stages > MAX_STAGES) stages = MAX_STAGES;
  if (stages < 2) { *why = "tile does not fit shared memory"; return cudaErrorInvalidValue; }
  p.stages = stages;
  p.split = 1;
  p.C0 = a.C0; p.ldc0 = a.ldc0; p.bias0 = a.bias0;
  p.C1 = dual ? a.C1 : nullptr; p.ldc1 = a.ldc1; p.bias1 = a.bias1;
  p.epi = a.epi;
  p.status = a.status;
  p.wait_ns = g_wait_ns;
  p.tma_store = 0;
  const int nb = a.batch < 1 ? 1 : a.batch;

  CUtensorMap mA0, mA1, mB0, mB1;
  memset(&mA0, 0, sizeof(mA0)); memset(&mA1, 0, sizeof(mA1));
  memset(&mB0, 0, sizeof(mB0)); memset(&mB1, 0, sizeof(mB1));
  p.a_mn = a.a_mn ? 1 : 0;
  p.b_mn = a.b_mn ? 1 : 0;
  if (useA0 && !make_op_map(&mA0, a.A0, a.K, a.M, a.lda0, BM, nb, a.bsA0, a.a_mn)) { *why = "tensor map A0"; return cudaErrorInvalidValue; }
  if (useA1 && !make_op_map(&mA1, a.A1, a.K, a.M, a.lda1, BM, nb, a.bsA1, a.a_mn)) { *why = "tensor map A1"; return cudaErrorInvalidValue; }
  if (useB0 && !make_op_map(&mB0, a.B0, a.K, a.N, a.ldb0, BH, nb, a.bsB0, a.b_mn)) { *why = "tensor map B0"; return cudaErrorInvalidValue; }
  if (useB1 && !make_op_map(&mB1, a.B1, a.K, a.N, a.ldb1, BH, nb, a.bsB1, a.b_mn)) { *why = "tensor map B1"; return cudaErrorInvalidValue; }
  p.batch = nb;
  p.bsC0 = a.bsC0;
  p.bsC1 = a.bsC1;
  p.st_c0 = p.C0 != nullptr;
  p.st_c1 = p.C1 != nullptr;

  PersistParams pp;
  pp.tiles_n = (a.N + BN - 1) / BN;
  pp.pairs_m = (a.M + 2 * BM - 1) / (2 * BM);
  const int64_t ntiles = static_cast<int64_t>(pp.tiles_n) * pp.pairs_m * nb;
  if (ntiles > (1 << 30)) { *why = "too many tiles"; return cudaErrorInvalidValue; }
  pp.ntiles = static_cast<int>(ntiles);
  pp.group = pp.pairs_m < 8 ? pp.pairs_m : 8;
  pp.nsets = persist_sets(nacc, BN);
  pp.set_cols = nacc * p.nsub * BN;

  const int smem = stages * off + epi_warps_p<MODE>() * STG_ROWS_BYTES + 1024;
  static PerDeviceOnce attr_once;
  {
    cudaError_t e = attr_once.run([](int&) {
      return cudaFuncSetAttribute(tc2p_dual_gemm_kernel<BN, MODE, ACT>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, 225 * 1024);
    });
    if (e != cudaSuccess) return e;
  }
  if (smem > 225 * 1024) { *why = "shared memory budget exceeded"; return cudaErrorInvalidValue; }
  int npairs = max_pairs<BN, MODE, ACT>(225 * 1024);
  if (npairs > pp.ntiles) npairs = pp.ntiles;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(2 * npairs, 1, 1);
  cfg.blockDim = dim3(threads_p<MODE>(), 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = g_pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, tc2p_dual_gemm_kernel<BN, MODE, ACT>, mA0, mA1, mB0, mB1, p,
                            pp);
}

template <int MODE, int ACT>
cudaError_t launch_bn_p(const GemmArgs& a, cudaStream_t s, const char** why, int bn) {
  if (bn == 128) return launch_cfg2p<128, MODE, ACT>(a, s, why);
  if (bn == 256) return launch_cfg2p<256, MODE, ACT>(a, s, why);
  *why = "2-SM tiles are 128 or 256 columns wide";
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t tc_gemm_persist(const GemmArgs& a, cudaStream_t s, const char** why, int bn) {
  const int act = a.epi.act;
  // Dual products take 128-wide tiles, whose two accumulators fit TMEM twice, so that
  // epilogues overlap main loops; unless the caller fixed the width, mode 3 keeps them at
  // 256, and so does mode 2 for K > 2048, where the 256-wide tiles' halved operand bytes per
  // MMA outweigh the epilogue that a single accumulator set cannot overlap.
  const bool dual = a.terms & (T_C1_A1B0 | T_C1_A0B1);
  const bool wide = g_gemm_persist == 3 || (g_gemm_persist == 2 && a.K > 2048);
  if (bn == 256 && a.bn == 0 && dual && !wide) bn = 128;
  if (a.epi.mode == EPI_STORE) return launch_bn_p<EPI_STORE, ACT_IDENT>(a, s, why, bn);
  if (a.epi.mode == EPI_ACT_FWD) {
    switch (act) {
      case ACT_IDENT: return launch_bn_p<EPI_ACT_FWD, ACT_IDENT>(a, s, why, bn);
      case ACT_TANH: return launch_bn_p<EPI_ACT_FWD, ACT_TANH>(a, s, why, bn);
      case ACT_GELU: return launch_bn_p<EPI_ACT_FWD, ACT_GELU>(a, s, why, bn);
      case ACT_SILU: return launch_bn_p<EPI_ACT_FWD, ACT_SILU>(a, s, why, bn);
    }
  } else if (a.epi.mode == EPI_ACT_BWD) {
    switch (act) {
      case ACT_IDENT: return launch_bn_p<EPI_ACT_BWD, ACT_IDENT>(a, s, why, bn);
      case ACT_TANH: return launch_bn_p<EPI_ACT_BWD, ACT_TANH>(a, s, why, bn);
      case ACT_GELU: return launch_bn_p<EPI_ACT_BWD, ACT_GELU>(a, s, why, bn);
      case ACT_SILU: return launch_bn_p<EPI_ACT_BWD, ACT_SILU>(a, s, why, bn);
    }
  }
  *why = "unknown epilogue mode or activation";
  return cudaErrorInvalidValue;
}

}  // namespace mf
