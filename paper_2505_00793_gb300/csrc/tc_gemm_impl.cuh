// Dual-number bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// One launch evaluates a Linear layer of the forward-over-reverse pass (Section 2.2's
// forward-over-reverse HVP applied layer by layer): the primal product P = A B^T and its
// tangent P' = A' B^T + A B'^T share the A and B shared-memory tiles, so four TMA tiles
// feed three tensor-core products per K block.  Every product term is optional (bit mask),
// which gives the primal-only layer, the input layer (A' = 0) and the weight-tangent
// product [a'; a]^T [dz; dz'] from the same kernel.
//
// One-SM tiles: a CTA of 18 warps. Warp 0 issues the TMA loads, warp 1 owns TMEM and issues
// tcgen05.mma from one thread, and sixteen epilogue warps drain the accumulators
// (tcgen05.ld) and run the fused epilogue: bias, activation and its derivatives, and the
// bf16 operand stores that the next GEMM reads in place. Warps sharing a TMEM lane quadrant
// split its columns. Tile 128 x BN x (64 KA) (bf16, 128-byte swizzle, KA swizzle atoms per
// pipeline stage) with a multi-stage mbarrier pipeline. Operands are K-major or MN-major
// (64-row boxes), so no operand is ever stored transposed. Each product term (MMA) rotates over
// up to four TMEM accumulator blocks so that dependent MMAs do not serialise. CTA-pair tiles
// (cta_group::2, 256 rows) serve GEMMs whose pair grid fills the GPU. GEMMs with few output
// tiles split K across a thread-block cluster of S CTAs: the partial accumulators meet in
// distributed shared memory, and each CTA reduces 128/S rows in a fixed order, so results are
// deterministic. Every mbarrier wait is bounded; on expiry the CTA records DEV_TIMEOUT, stops
// issuing MMAs and drains the loads and MMAs it has issued before it releases its memory.
// Implementation of the tcgen05 dual GEMM, included by tc_gemm.cu (plain stores) and by
// tc_gemm_act.cu (activation epilogues).  The epilogue mode and the activation are template
// parameters so that each kernel instance carries only its own per-element code.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <string.h>

#include "device_math.cuh"
#include "internal.h"
#include "launch.cuh"

namespace mf {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;                 // bf16 elements per 128-byte swizzle row
constexpr int MAX_STAGES = 8;
// Epilogue warps: one-SM tiles (small grids, split K) drain with sixteen warps storing
// straight from registers; CTA-pair tiles with eight warps through TMA-store staging
// (STG_WARP bytes of shared memory per warp).  Warps sharing a TMEM lane quadrant split its
// columns.
constexpr int EPI_WARPS = 16;
constexpr int EPI_GROUPS = EPI_WARPS / 4;
constexpr bool EPI_TMA = false;
constexpr int EPI_THREADS = 32 * EPI_WARPS;
constexpr int THREADS = 64 + EPI_THREADS;        // producer warp, MMA warp, epilogue
constexpr int EPI_WARPS2 = 8;
constexpr int EPI_GROUPS2 = EPI_WARPS2 / 4;
constexpr bool EPI_TMA2 = true;
constexpr int THREADS2 = 64 + 32 * EPI_WARPS2;
// Bounded waits.  Every mbarrier wait gives up after a limit and records DEV_TIMEOUT.  The
// MMA issuer's and the epilogue's waits use the run-time limit g_wait_ns (TcParams::wait_ns,
// MF_OPT_WAIT_LIMIT_US; default 2 s).  The TMA producer's waits, and every wait that drains
// work already issued after a timeout, use the fixed DRAIN_NS, so that a CTA never releases
// shared memory or TMEM while a TMA load or an MMA it issued is still in flight:
//  - after a timeout the MMA issuer stops issuing MMAs but keeps consuming the pipeline
//    (waits for each stage's data, DRAIN_NS, and releases it), so the producer issues and
//    sees the end of every load of its schedule;
//  - the MMA issuer then commits and waits for its own last commit (all MMAs complete);
//  - the producer waits for the last phase it issued on every stage before the CTA's final
//    barrier (in a CTA pair, the even CTA, whose full barriers count both CTAs' bytes).
// Only a wait that a healthy GPU never exceeds can run past DRAIN_NS.
constexpr long long DRAIN_NS = 2000000000LL;

__device__ __forceinline__ long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return static_cast<long long>(t);
}

struct TcParams {
  int M, N, K;
  unsigned terms;
  int stages;
  int split;
  int tma_store;          // 1: row-major outputs through TMA stores
  int batch;              // independent GEMMs; blockIdx.z = batch index * split + split index
  int64_t bsC0, bsC1;     // batch strides of C0 / C1 (direct-store paths)
  int st_c0, st_c1, st_a, st_ad;   // which row-major outputs exist
  int a0_off, a1_off, b0_off, b1_off, stage_bytes, tx_bytes;
  int nsub;               // TMEM blocks per logical accumulator (1, 2 or 4)
  int a_mn, b_mn;         // operands stored MN-major ([K][rows]) instead of K-major
  float* C0; int ldc0; const float* bias0;
  float* C1; int ldc1; const float* bias1;
  EpiParams epi;
  int* status;
  long long wait_ns;      // limit of the MMA issuer's and the epilogue's waits
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and flags the status word) if the phase has not completed
// within limit_ns nanoseconds.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* status,
                                          long long limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = global_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > limit_ns) {
      if (status) atomicMax(status, DEV_TIMEOUT);
      return false;
    }
  }
}

// The producer's drain: wait for the last phase issued on every stage (issued = number of K
// blocks whose loads were issued, in ring order).
__device__ __forceinline__ void drain_loads(uint64_t* full_bar, int issued, int stages,
                                            int* status) {
  for (int j = issued - stages > 0 ? issued - stages : 0; j < issued; ++j)
    if (!mbar_wait(&full_bar[j % stages], (j / stages) & 1, status, DRAIN_NS)) return;
}

// Every operand map is 3-D {K, rows, batch}; non-batched GEMMs have batch extent 1.
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups of
// 1024 bytes (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1) << 16;              // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;      // stride byte offset
  d |= static_cast<uint64_t>(1) << 46;              // version
  d |= static_cast<uint64_t>(2) << 61;              // SWIZZLE_128B
  return d;
}

// MN-major operand ([K][rows] in memory, rows contiguous), 128-byte swizzle, staged as
// boxes of 64 rows x 64 K (8 KB, K rows of 128 bytes): 8-row K groups 1024 bytes apart
// (stride byte offset), 64-row blocks 8 KB apart (leading byte offset).
constexpr int MN_BOX = 64 * BK * 2;
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(MN_BOX >> 4) << 16;    // leading byte offset: next 64 rows
  d |= static_cast<uint64_t>(1024 >> 4) << 32;      // stride byte offset: next 8 K rows
  d |= static_cast<uint64_t>(1) << 46;              // version
  d |= static_cast<uint64_t>(2) << 61;              // SWIZZLE_128B
  return d;
}

// TMEM allocation size: a power of two >= 32 columns covering the accumulators.
__host__ __device__ constexpr uint32_t tmem_cols(int needed) {
  return needed <= 32 ? 32u : needed <= 64 ? 64u : needed <= 128 ? 128u : needed <= 256 ? 256u : 512u;
}

// Instruction descriptor, kind::f16: D f32, A/B bf16, both K-major, M = 128, N = BN.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t dtmem, uint64_t ad, uint64_t bd,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(dtmem),
      "l"(ad), "l"(bd), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Accumulators.  Logical accumulator c (0: C0, 1: C1) owns nsub blocks of BN TMEM columns
// at (c * nsub + j) * BN.  Successive products into one logical accumulator rotate over its
// blocks: an MMA into a block waits for the previous MMA into the same block (its
// read-modify-write of TMEM), so rotating keeps several MMAs in flight.  The epilogue sums
// the blocks in order j = 0..nsub-1 (deterministic).
template <int BN>
__device__ __forceinline__ void ld_acc16(uint32_t taddr, int c, int nsub, int col,
                                         float (&v)[16]) {
  tmem_ld16(taddr + static_cast<uint32_t>(c * nsub * BN + col), v);
  for (int j = 1; j < nsub; ++j) {
    float t[16];
    tmem_ld16(taddr + static_cast<uint32_t>((c * nsub + j) * BN + col), t);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] += t[i];
  }
}

// The most blocks (up to 4) that fit 512 TMEM columns.
__host__ __device__ constexpr int acc_blocks(int nlogical, int bn) {
  return nlogical * 4 * bn <= 512 ? 4 : nlogical * 2 * bn <= 512 ? 2 : 1;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t dsmem_addr(uint32_t local_addr, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local_addr), "r"(rank));
  return remote;
}

__device__ __forceinline__ void st_dsmem4(uint32_t remote_addr, float a, float b, float c, float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote_addr), "f"(a),
               "f"(b), "f"(c), "f"(d)
               : "memory");
}

__device__ __forceinline__ void epi_bar() {   // the epilogue warps only
  asm volatile("bar.sync 1, %0;" ::"n"(EPI_THREADS) : "memory");
}

// Row-per-thread epilogue for 16 consecutive columns (no split): float32 outputs and the
// row-major bf16 operand rows.
template <int MODE, int ACT>
__device__ __forceinline__ void epilogue16(const TcParams& p, int row, int col0,
                                           const float (&v0)[16], const float (&v1)[16],
                                           bool dual) {
  const EpiParams e = p.epi;
  const bool rowok = row < p.M;
  float o0[16], o1[16], c0[16], c1[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const int n = col0 + j;
    const bool ok = rowok && n < p.N;
    EpiOut o;
    if (ok) o = epi_eval_t<MODE, ACT>(e, row, n, v0[j], v1[j], p.bias0, p.bias1, dual);
    else o.c0 = o.c1 = o.o0 = o.o1 = 0.f;
    c0[j] = o.c0; c1[j] = o.c1; o0[j] = o.o0; o1[j] = o.o1;
  }
  const bool full = rowok && col0 + 16 <= p.N;
  if (rowok) {
    if (p.C0) {
      float* dst = p.C0 + static_cast<int64_t>(row) * p.ldc0 + col0;
      if (full && !(p.ldc0 & 3) && !(reinterpret_cast<uintptr_t>(p.C0) & 15)) {
#pragma unroll
        for (int j = 0; j < 16; j += 4)
          *reinterpret_cast<float4*>(dst + j) = make_float4(c0[j], c0[j + 1], c0[j + 2], c0[j + 3]);
      } else {
        for (int j = 0; j < 16; ++j) if (col0 + j < p.N) dst[j] = c0[j];
      }
    }
    if (p.C1 && dual) {
      float* dst = p.C1 + static_cast<int64_t>(row) * p.ldc1 + col0;
      if (full && !(p.ldc1 & 3) && !(reinterpret_cast<uintptr_t>(p.C1) & 15)) {
#pragma unroll
        for (int j = 0; j < 16; j += 4)
          *reinterpret_cast<float4*>(dst + j) = make_float4(c1[j], c1[j + 1], c1[j + 2], c1[j + 3]);
      } else {
        for (int j = 0; j < 16; ++j) if (col0 + j < p.N) dst[j] = c1[j];
      }
    }
  }
  if constexpr (MODE == EPI_STORE) return;
  // row-major operand copies (ld multiple of 8 elements, col0 multiple of 16)
  __nv_bfloat16* A = static_cast<__nv_bfloat16*>(e.A);
  __nv_bfloat16* Ad = static_cast<__nv_bfloat16*>(e.Ad);
  if (rowok) {
    for (int w = 0; w < 2; ++w) {
      __nv_bfloat16* X = w == 0 ? A : Ad;
      const float* o = w == 0 ? o0 : o1;
      if (!X || (w == 1 && !dual)) continue;
      __nv_bfloat16* dst = X + static_cast<int64_t>(row) * e.lda + col0;
      if (full) {
        uint4 q0 = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                              pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
        uint4 q1 = make_uint4(pack_bf16x2(o[8], o[9]), pack_bf16x2(o[10], o[11]),
                              pack_bf16x2(o[12], o[13]), pack_bf16x2(o[14], o[15]));
        reinterpret_cast<uint4*>(dst)[0] = q0;
        reinterpret_cast<uint4*>(dst)[1] = q1;
      } else {
        for (int j = 0; j < 16; ++j) if (col0 + j < p.N) dst[j] = __float2bfloat16_rn(o[j]);
      }
    }
  }
}

// ---- warp-cooperative row blocks through shared memory ---------------------------------
// The row-per-thread epilogues hold one accumulator row per lane (tcgen05.ld 32x32b), so a
// warp's direct 16-byte store touches 32 rows, 32 memory lines.  These helpers move a block
// of 32 rows x 64 bytes through a 2 KB per-warp buffer instead: lane l handles 16-byte quad
// l % 4 of rows l / 4 + 8 i (i = 0..3), so each warp access covers 8 rows x 64 bytes.  Row r's
// quad c sits at 128-byte line r >> 1, slot (r & 1) * 4 + (c ^ ((r >> 1) & 3)): both the
// row-wise and the quad-wise accesses of a warp are free of bank conflicts.
constexpr int STG_ROWS_BYTES = 32 * 64;

__device__ __forceinline__ int stg_quad(int r, int c) {
  return (r >> 1) * 128 + ((((r & 1) << 2) | (c ^ ((r >> 1) & 3))) << 4);
}

// A 32-row x 16-column float32 block read by quads (lane l: quad l % 4 of rows l / 4 + 8 i),
// in flight until zrows_finish turns it into rows.
struct ZRows {
  float4 q[4];
};

// Issue the loads of rows row0 .. row0 + 31 (those below M) of a float32 matrix, 16 columns
// from col0 (16-byte aligned rows).
__device__ __forceinline__ void zrows_issue(ZRows& z, int lane, int row0, int M, const float* src,
                                            int64_t ld, int col0) {
  const int rq = lane >> 2, cq = lane & 3;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = rq + 8 * i;
    z.q[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (row0 + r < M) z.q[i] = *reinterpret_cast<const float4*>(src + (row0 + r) * ld + col0 + 4 * cq);
  }
}

// ... and transpose them through the warp's buffer into this lane's row:
// out[j] = src[(row0 + lane) * ld + col0 + j].
__device__ __forceinline__ void zrows_finish(uint8_t* stg, int lane, const ZRows& z,
                                             float (&out)[16]) {
  const int rq = lane >> 2, cq = lane & 3;
#pragma unroll
  for (int i = 0; i < 4; ++i) *reinterpret_cast<float4*>(stg + stg_quad(rq + 8 * i, cq)) = z.q[i];
  __syncwarp();
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    const float4 v = *reinterpret_cast<const float4*>(stg + stg_quad(lane, c));
    out[4 * c] = v.x; out[4 * c + 1] = v.y; out[4 * c + 2] = v.z; out[4 * c + 3] = v.w;
  }
  __syncwarp();
}

__device__ __forceinline__ void warp_load_rows16(uint8_t* stg, int lane, int row0, int M,
                                                 const float* src, int64_t ld, int col0,
                                                 float (&out)[16]) {
  ZRows z;
  zrows_issue(z, lane, row0, M, src, ld, col0);
  zrows_finish(stg, lane, z, out);
}

// This lane's 64-byte row (quads q[0..3]) of a 32-row block, stored by quads: quad c of
// row r goes to dst(r, c) (nullptr: not stored) when row0 + r < M.
template <class Dst>
__device__ __forceinline__ void warp_store_rows(uint8_t* stg, int lane, int row0, int M,
                                                const uint4 (&q)[4], Dst dst) {
#pragma unroll
  for (int c = 0; c < 4; ++c) *reinterpret_cast<uint4*>(stg + stg_quad(lane, c)) = q[c];
  __syncwarp();
  const int rq = lane >> 2, cq = lane & 3;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = rq + 8 * i;
    const uint4 v = *reinterpret_cast<const uint4*>(stg + stg_quad(r, cq));
    void* d = dst(r, cq);
    if (d && row0 + r < M) *reinterpret_cast<uint4*>(d) = v;
  }
  __syncwarp();
}

__device__ __forceinline__ uint4 quad_f32(const float* v) {
  return make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                    __float_as_uint(v[3]));
}
__device__ __forceinline__ uint4 quad_bf16(const float* v) {
  return make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                    pack_bf16x2(v[6], v[7]));
}

// Whether the coalesced row-block epilogue may serve this GEMM: 16-byte aligned rows of
// every matrix it reads or writes.
__device__ __forceinline__ bool rows16_ok(const TcParams& p, int mode, bool dual) {
  auto al = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
  bool ok = true;
  if (p.C0) ok = ok && al(p.C0) && !(p.ldc0 & 3);
  if (p.C1 && dual) ok = ok && al(p.C1) && !(p.ldc1 & 3);
  if (mode != EPI_STORE) {
    if (p.epi.A) ok = ok && al(p.epi.A) && !(p.epi.lda & 7);
    if (p.epi.Ad && dual) ok = ok && al(p.epi.Ad) && !(p.epi.lda & 7);
  }
  if (mode == EPI_ACT_BWD) {
    ok = ok && al(p.epi.Z) && !(p.epi.ldz & 3);
    if (dual) ok = ok && al(p.epi.Zd);
  }
  return ok;
}

// epilogue16 for a full chunk (col0 + 16 <= N) of the warp's 32 rows row0 .. row0 + 31, with
// the outputs written through the per-warp buffer stg (STG_ROWS_BYTES).  Backward
// epilogues take the chunk's stored pre-activations as loads already issued (zq, zdq: see
// zrows_issue).  The arithmetic per element is epi_core_t's, as in epilogue16, computed in
// place (v0, v1 become the float32 outputs) with the activation outputs packed to bf16 pairs
// at once, so that few values stay live.  Rows at or past M are computed but not stored.
template <int MODE, int ACT, bool DUALE>
__device__ __forceinline__ void epilogue16_rows_t(const TcParams& p, uint8_t* stg, int lane,
                                                  int row0, int col0, float (&v0)[16],
                                                  float (&v1)[16], const ZRows& zq,
                                                  const ZRows& zdq) {
  constexpr bool dual = DUALE;
  const EpiParams e = p.epi;
  uint32_t pa[8], pad[8];       // bf16 pairs of A and Ad
  if constexpr (MODE == EPI_ACT_BWD) {
    float z[16];
    zrows_finish(stg, lane, zq, z);
    float zd[16];
    if constexpr (dual) zrows_finish(stg, lane, zdq, zd);
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      float o0[2], o1[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const EpiOut o = epi_core_t<MODE, ACT>(v0[j + h], v1[j + h], z[j + h],
                                               dual ? zd[j + h] : 0.f, 0.f, 0.f, dual);
        o0[h] = o.o0;
        o1[h] = o.o1;
      }
      pa[j / 2] = pack_bf16x2(o0[0], o0[1]);
      pad[j / 2] = pack_bf16x2(o1[0], o1[1]);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      float o0[2], o1[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int n = col0 + j + h;
        const float b0 = p.bias0 ? p.bias0[n] : 0.f;
        const float b1 = p.bias1 ? p.bias1[n] : 0.f;
        const EpiOut o = epi_core_t<MODE, ACT>(v0[j + h], v1[j + h], 0.f, 0.f, b0, b1, dual);
        v0[j + h] = o.c0;
        v1[j + h] = o.c1;
        o0[h] = o.o0;
        o1[h] = o.o1;
      }
      if constexpr (MODE != EPI_STORE) {
        pa[j / 2] = pack_bf16x2(o0[0], o0[1]);
        pad[j / 2] = pack_bf16x2(o1[0], o1[1]);
      }
    }
  }
  if (p.C0) {
    const uint4 q[4] = {quad_f32(v0), quad_f32(v0 + 4), quad_f32(v0 + 8), quad_f32(v0 + 12)};
    float* const C = p.C0;
    const int64_t ld = p.ldc0;
    warp_store_rows(stg, lane, row0, p.M, q, [&](int r, int c) -> void* {
      return C + (row0 + r) * ld + col0 + 4 * c;
    });
  }
  if (dual && p.C1) {
    const uint4 q[4] = {quad_f32(v1), quad_f32(v1 + 4), quad_f32(v1 + 8), quad_f32(v1 + 12)};
    float* const C = p.C1;
    const int64_t ld = p.ldc1;
    warp_store_rows(stg, lane, row0, p.M, q, [&](int r, int c) -> void* {
      return C + (row0 + r) * ld + col0 + 4 * c;
    });
  }
  if constexpr (MODE != EPI_STORE) {
    // A and Ad rows side by side: quads 0, 1 of A, quads 2, 3 of Ad
    __nv_bfloat16* const A = static_cast<__nv_bfloat16*>(e.A);
    __nv_bfloat16* const Ad = dual ? static_cast<__nv_bfloat16*>(e.Ad) : nullptr;
    if (A || Ad) {
      const uint4 q[4] = {make_uint4(pa[0], pa[1], pa[2], pa[3]),
                          make_uint4(pa[4], pa[5], pa[6], pa[7]),
                          make_uint4(pad[0], pad[1], pad[2], pad[3]),
                          make_uint4(pad[4], pad[5], pad[6], pad[7])};
      const int64_t ld = e.lda;
      warp_store_rows(stg, lane, row0, p.M, q, [&](int r, int c) -> void* {
        __nv_bfloat16* X = c < 2 ? A : Ad;
        return X ? X + (row0 + r) * ld + col0 + 8 * (c & 1) : nullptr;
      });
    }
  }
}

// The same with the dual flag as a compile-time constant, so that single-accumulator
// epilogues carry no tangent arithmetic.
template <int MODE, int ACT>
__device__ __forceinline__ void epilogue16_rows(const TcParams& p, uint8_t* stg, int lane,
                                                int row0, int col0, float (&v0)[16],
                                                float (&v1)[16], bool dual,
                                                const ZRows& zq, const ZRows& zdq) {
  if (dual) epilogue16_rows_t<MODE, ACT, true>(p, stg, lane, row0, col0, v0, v1, zq, zdq);
  else epilogue16_rows_t<MODE, ACT, false>(p, stg, lane, row0, col0, v0, v1, zq, zdq);
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int x, int y,
                                             int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(x), "r"(y), "r"(z), "r"(smem_u32(src))
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Per-warp staging of a 32-row slab of the tile for TMA stores (128-byte swizzle: the
// 16-byte chunk j of row r sits at chunk position j ^ (r % 8) of the row's 128 bytes).
// Layout per warp: C0 [2 boxes of 32x32 f32] | C1 [2 boxes] | A [32x64 bf16] | Ad [32x64],
constexpr int STG_F32_BOX = 32 * 32 * 4;          // 4 KB
constexpr int STG_BF16_BOX = 32 * 64 * 2;         // 4 KB
// ... followed by the row-block buffer (STG_ROWS_BYTES) through which the backward
// epilogues read the stored pre-activations.
constexpr int STG_ZROWS = 4 * STG_F32_BOX + 2 * STG_BF16_BOX;
constexpr int STG_WARP = STG_ZROWS + STG_ROWS_BYTES;              // 26 KB

// TMA-store epilogue of one warp (32 rows) over the tile's BN columns, 64 at a time.
template <int BN, int MODE, int ACT>
__device__ __forceinline__ void epilogue_tma(const TcParams& p, const CUtensorMap* mC0,
                                             const CUtensorMap* mC1, const CUtensorMap* mA,
                                             const CUtensorMap* mAd, uint8_t* stg, uint32_t taddr,
                                             int q, int lane, int m0, int n0, bool dual, int bz,
                                             int c_begin, int c_end) {
  const EpiParams e = p.epi;
  const int row = m0 + q * 32 + lane;
  const bool rowok = row < p.M;
  uint8_t* sC0 = stg;
  uint8_t* sC1 = stg + 2 * STG_F32_BOX;
  uint8_t* sA = stg + 4 * STG_F32_BOX;
  uint8_t* sAd = sA + STG_BF16_BOX;
  uint8_t* sZ = stg + STG_ZROWS;
  const int sw = lane & 7;
  // backward epilogues: the stored pre-activations of full chunks through sZ
  bool zrows_ok = false;
  if constexpr (MODE == EPI_ACT_BWD) {
    auto al = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
    zrows_ok = al(e.Z) && !(e.ldz & 3) && (!dual || al(e.Zd));
  }
  for (int c = c_begin; c < c_end; c += 64) {
    if (c > c_begin) {
      if (lane == 0) bulk_wait_read();
      __syncwarp();
    }
#pragma unroll 1
    for (int sub = 0; sub < 4; ++sub) {
      const int cc = c + sub * 16;          // tile column of this 16-column group
      if (cc >= BN) break;
      float v0[16], v1[16];
      ld_acc16<BN>(taddr, 0, p.nsub, cc, v0);
      if (dual) ld_acc16<BN>(taddr, 1, p.nsub, cc, v1);
      else {
#pragma unroll
        for (int j = 0; j < 16; ++j) v1[j] = 0.f;
      }
      float c0[16], c1[16], o0[16], o1[16];
      float z[16], zd[16];
      const bool zrows = zrows_ok && n0 + cc + 16 <= p.N;     // warp-uniform
      if constexpr (MODE == EPI_ACT_BWD) {
        if (zrows) {
          warp_load_rows16(sZ, lane, m0 + q * 32, p.M, e.Z, e.ldz, n0 + cc, z);
          if (dual) warp_load_rows16(sZ, lane, m0 + q * 32, p.M, e.Zd, e.ldz, n0 + cc, zd);
          else {
#pragma unroll
            for (int j = 0; j < 16; ++j) zd[j] = 0.f;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int n = n0 + cc + j;
        EpiOut o;
        if (rowok && n < p.N) {
          if (MODE == EPI_ACT_BWD && zrows) o = epi_core_t<MODE, ACT>(v0[j], v1[j], z[j], zd[j], 0.f, 0.f, dual);
          else o = epi_eval_t<MODE, ACT>(e, row, n, v0[j], v1[j], p.bias0, p.bias1, dual);
        } else {
          o.c0 = o.c1 = o.o0 = o.o1 = 0.f;
        }
        c0[j] = o.c0; c1[j] = o.c1; o0[j] = o.o0; o1[j] = o.o1;
      }
      // float32 slabs: box (sub / 2), chunks (sub % 2) * 4 .. + 3 of the 128-byte row
      const int fb = (sub >> 1) * STG_F32_BOX + lane * 128;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int pos = ((((sub & 1) * 4) + k) ^ sw) * 16;
        if (p.st_c0)
          *reinterpret_cast<float4*>(sC0 + fb + pos) =
              make_float4(c0[4 * k], c0[4 * k + 1], c0[4 * k + 2], c0[4 * k + 3]);
        if (p.st_c1)
          *reinterpret_cast<float4*>(sC1 + fb + pos) =
              make_float4(c1[4 * k], c1[4 * k + 1], c1[4 * k + 2], c1[4 * k + 3]);
      }
      // bf16 slabs: chunks sub * 2 .. + 1 of the 128-byte row
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int pos = (((sub * 2) + k) ^ sw) * 16;
        if (p.st_a)
          *reinterpret_cast<uint4*>(sA + lane * 128 + pos) =
              make_uint4(pack_bf16x2(o0[8 * k], o0[8 * k + 1]), pack_bf16x2(o0[8 * k + 2], o0[8 * k + 3]),
                         pack_bf16x2(o0[8 * k + 4], o0[8 * k + 5]), pack_bf16x2(o0[8 * k + 6], o0[8 * k + 7]));
        if (p.st_ad)
          *reinterpret_cast<uint4*>(sAd + lane * 128 + pos) =
              make_uint4(pack_bf16x2(o1[8 * k], o1[8 * k + 1]), pack_bf16x2(o1[8 * k + 2], o1[8 * k + 3]),
                         pack_bf16x2(o1[8 * k + 4], o1[8 * k + 5]), pack_bf16x2(o1[8 * k + 6], o1[8 * k + 7]));
      }
    }
    fence_proxy_async();
    __syncwarp();
    if (lane == 0) {
      const int y = m0 + q * 32;
      if (y < p.M) {
        for (int b = 0; b < 2; ++b) {
          const int x = n0 + c + 32 * b;
          if (x >= p.N) continue;
          if (p.st_c0) tma_store_3d(mC0, sC0 + b * STG_F32_BOX, x, y, bz);
          if (p.st_c1) tma_store_3d(mC1, sC1 + b * STG_F32_BOX, x, y, bz);
        }
        if (n0 + c < p.N) {
          if (p.st_a) tma_store_3d(mA, sA, n0 + c, y, bz);
          if (p.st_ad) tma_store_3d(mAd, sAd, n0 + c, y, bz);
        }
      }
      bulk_commit();
    }
  }
  if (lane == 0) bulk_wait_all();
  __syncwarp();
}

__device__ __forceinline__ void mma_bf16_pair(uint32_t dtmem, uint64_t ad, uint64_t bd,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(dtmem),
      "l"(ad), "l"(bd), "r"(idesc), "r"(accumulate));
}

// Arrive once on the barrier at this shared-memory offset in both CTAs of the pair when
// the pair's previously issued MMAs have completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// The MMA issuer's barrier operations on precomputed shared-memory addresses (the issue
// loop keeps its ring position and descriptors in registers: a single thread issues every
// MMA, and each instruction between two MMAs delays the tensor pipe).
__device__ __forceinline__ bool mbar_try_wait_addr(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_addr(uint32_t addr, uint32_t parity, int* status,
                                               long long limit_ns) {
  if (mbar_try_wait_addr(addr, parity)) return true;
  const long long t0 = global_ns();
  while (true) {
    if (mbar_try_wait_addr(addr, parity)) return true;
    if (global_ns() - t0 > limit_ns) {
      if (status) atomicMax(status, DEV_TIMEOUT);
      return false;
    }
  }
}

__device__ __forceinline__ void mma_commit_addr(uint32_t addr) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   addr)
               : "memory");
}

__device__ __forceinline__ void mma_commit_pair_addr(uint32_t addr) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(addr),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// Shared-memory descriptors of one operand for stage 0 of the ring.  The descriptor's
// address field holds (address & 0x3FFFF) >> 4 in its low 14 bits, and every stage, K atom
// and K slice lies inside the CTA's shared memory, so moving a descriptor by a byte offset
// is a 64-bit add of offset >> 4 that never carries out of the field.
__device__ __forceinline__ uint64_t op_desc(uint32_t sbase, int off, int mn) {
  if (off < 0) return 0;
  return mn ? sdesc_mn_sw128(sbase + off) : sdesc_sw128(sbase + off);
}

struct MmaLoop {
  int nk, stages, stage_bytes, a0_off, a1_off, b0_off, b1_off;
  int a_mn, b_mn;
  uint32_t sbase, tbase;
  uint64_t* full_bar;
  uint64_t* empty_bar;
  int* status;
  long long wait_ns;
};

// The MMA issuer's loop over K blocks.  TERMS != 0 fixes the product mask at compile time
// (TERMS = 0 reads `terms` at run time) so that the issue sequence is straight-line code:
// a single thread issues every tcgen05.mma, and instructions between MMAs delay the tensor
// pipe.  The ring position, the barrier addresses and the operand descriptors advance by
// additions (no division by the stage count, no descriptor rebuilt per K block).  Products
// of K slice kk go to accumulator block kk mod NSUB (see ld_acc16).  PAIR issues the M = 256
// form for a CTA pair and multicasts the commits to both CTAs.
template <int BN, int KA, unsigned TERMS, int NSUB, bool PAIR>
__device__ __forceinline__ void mma_loop(const MmaLoop& L, unsigned terms_rt, int nsub_rt) {
  constexpr int A_ATOM = BM * BK * 2, B_ATOM = (PAIR ? BN / 2 : BN) * BK * 2;
  // bits 15 / 16 of the instruction descriptor: A / B MN-major
  const uint32_t idesc = idesc_bf16(PAIR ? 2 * BM : BM, BN) | (static_cast<uint32_t>(L.a_mn) << 15) |
                         (static_cast<uint32_t>(L.b_mn) << 16);
  // descriptor advance per K=16 slice, in 16-byte units: 32 bytes K-major, 16 rows MN-major
  const uint64_t stepA = L.a_mn ? 128u : 2u, stepB = L.b_mn ? 128u : 2u;
  // per K atom (KA > 1, K-major operands only)
  const uint64_t atomA = L.a_mn ? 0u : static_cast<uint64_t>(A_ATOM >> 4);
  const uint64_t atomB = L.b_mn ? 0u : static_cast<uint64_t>(B_ATOM >> 4);
  const unsigned terms = TERMS ? TERMS : terms_rt;
  const uint32_t nsub = NSUB ? static_cast<uint32_t>(NSUB) : static_cast<uint32_t>(nsub_rt);
  // products into C0 / C1 per K slice
  const uint32_t p0 = __popc(terms & (T_C0_A0B0 | T_C0_A1B0 | T_C0_A0B1 | T_C0_A1B1));
  const uint32_t p1 = __popc(terms & (T_C1_A1B0 | T_C1_A0B1));
  const uint64_t a0s = op_desc(L.sbase, L.a0_off, L.a_mn), a1s = op_desc(L.sbase, L.a1_off, L.a_mn);
  const uint64_t b0s = op_desc(L.sbase, L.b0_off, L.b_mn), b1s = op_desc(L.sbase, L.b1_off, L.b_mn);
  const uint64_t stage_step = static_cast<uint64_t>(L.stage_bytes >> 4);
  const uint32_t full0 = smem_u32(L.full_bar), empty0 = smem_u32(L.empty_bar);
  int s = 0;
  uint32_t ph = 0;
  uint64_t soff = 0;   // descriptor offset of stage s
  bool live = true;   // false after a timed-out wait: consume the stages without MMAs
  for (int i = 0; i < L.nk; ++i) {
    const uint32_t fb = full0 + 8u * static_cast<uint32_t>(s);
    if (!live || !mbar_wait_addr(fb, ph, L.status, L.wait_ns)) {
      live = false;
      if (!mbar_wait_addr(fb, ph, L.status, DRAIN_NS)) break;
    }
    tc_fence_after();
    if (live) {
#pragma unroll
    for (int a = 0; a < KA; ++a) {
      const uint64_t a0 = a0s + soff + a * atomA, a1 = a1s + soff + a * atomA;
      const uint64_t b0 = b0s + soff + a * atomB, b1 = b1s + soff + a * atomB;
#pragma unroll
      for (int kk = 0; kk < BK / 16; ++kk) {
        // The j-th product of K slice kk into accumulator c goes to block
        // (kk * P_c + j) mod nsub (P_c products into c per slice); the first product into
        // a block overwrites it.
        const uint64_t advA = static_cast<uint64_t>(kk) * stepA;
        const uint64_t advB = static_cast<uint64_t>(kk) * stepB;
        const bool first = i == 0 && a == 0;
        uint32_t q0 = static_cast<uint32_t>(kk) * p0, q1 = static_cast<uint32_t>(kk) * p1;
        auto mma = [&](uint32_t c, uint64_t ad, uint64_t bd) {
          uint32_t& q = c ? q1 : q0;
          const uint32_t blk = c * nsub + (q & (nsub - 1));
          const uint32_t f = (first && q < nsub) ? 0u : 1u;
          ++q;
          if constexpr (PAIR) mma_bf16_pair(L.tbase + blk * BN, ad, bd, idesc, f);
          else mma_bf16(L.tbase + blk * BN, ad, bd, idesc, f);
        };
        if (terms & T_C0_A0B0) mma(0, a0 + advA, b0 + advB);
        if (terms & T_C1_A1B0) mma(1, a1 + advA, b0 + advB);
        if (terms & T_C0_A1B0) mma(0, a1 + advA, b0 + advB);
        if (terms & T_C1_A0B1) mma(1, a0 + advA, b1 + advB);
        if (terms & T_C0_A0B1) mma(0, a0 + advA, b1 + advB);
        if (terms & T_C0_A1B1) mma(0, a1 + advA, b1 + advB);
      }
    }
    }
    const uint32_t eb = empty0 + 8u * static_cast<uint32_t>(s);
    if constexpr (PAIR) mma_commit_pair_addr(eb);
    else mma_commit_addr(eb);
    if (++s == L.stages) {
      s = 0;
      ph ^= 1u;
      soff = 0;
    } else {
      soff += stage_step;
    }
  }
}

// Dispatch of the MMA loop over the product masks the library issues; anything else takes
// the run-time mask.  Plain-store GEMMs carry the weight products and the head layer,
// activation epilogues the forward and data products.
template <int BN, int KA, int MODE, bool PAIR>
__device__ __forceinline__ void mma_dispatch(const MmaLoop& L, unsigned terms, int nsub) {
  constexpr int N1 = acc_blocks(1, BN), N2 = acc_blocks(2, BN);
  switch (terms) {
    case T_C0_A0B0: mma_loop<BN, KA, T_C0_A0B0, N1, PAIR>(L, terms, nsub); return;
    case T_C0_A0B0 | T_C1_A1B0 | T_C1_A0B1:
      mma_loop<BN, KA, T_C0_A0B0 | T_C1_A1B0 | T_C1_A0B1, N2, PAIR>(L, terms, nsub); return;
    case T_C0_A0B0 | T_C1_A0B1:
      mma_loop<BN, KA, T_C0_A0B0 | T_C1_A0B1, N2, PAIR>(L, terms, nsub); return;
    default: break;
  }
  if constexpr (MODE == EPI_STORE) {
    switch (terms) {
      case T_C0_A0B1: mma_loop<BN, KA, T_C0_A0B1, N1, PAIR>(L, terms, nsub); return;
      case T_C0_A1B0 | T_C0_A0B1:
        mma_loop<BN, KA, T_C0_A1B0 | T_C0_A0B1, N1, PAIR>(L, terms, nsub); return;
      case T_C0_A0B0 | T_C0_A1B1:
        mma_loop<BN, KA, T_C0_A0B0 | T_C0_A1B1, N1, PAIR>(L, terms, nsub); return;
      default: break;
    }
  }
  mma_loop<BN, KA, 0, 0, PAIR>(L, terms, nsub);
}

template <int BN, int KA, int MODE, int ACT>
__global__ void __launch_bounds__(THREADS, 1)
    tc_dual_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                        const __grid_constant__ CUtensorMap tmA1,
                        const __grid_constant__ CUtensorMap tmB0,
                        const __grid_constant__ CUtensorMap tmB1,
                        const __grid_constant__ CUtensorMap tmC0,
                        const __grid_constant__ CUtensorMap tmC1,
                        const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmAd, const TcParams prm) {
  // Work on a register copy: a reference into the parameter block would be re-read after
  // every asm statement with a memory clobber (mbarrier waits, commits, stores).
  TcParams p = prm;
  const int bz = static_cast<int>(blockIdx.z) / p.split;     // batch index
  const int zs = static_cast<int>(blockIdx.z) % p.split;     // split index (cluster rank)
  if (p.C0) p.C0 += bz * p.bsC0;
  if (p.C1) p.C1 += bz * p.bsC1;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t empty_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_slot;

  constexpr int SK = BK * KA;            // K elements per pipeline stage
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * BM;
  const int n0 = blockIdx.x * BN;
  const int S = p.split;
  const int nkb = (p.K + SK - 1) / SK;
  const int kper = (nkb + S - 1) / S;
  const int kb0 = zs * kper;
  const int nk = max(0, min(nkb, kb0 + kper) - kb0);
  const unsigned terms = p.terms;
  const bool dual = (terms & (T_C1_A1B0 | T_C1_A0B1)) != 0;
  const uint32_t ncols = tmem_cols((dual ? 2 : 1) * p.nsub * BN);
  constexpr int A_ATOM = BM * BK * 2, B_ATOM = BN * BK * 2;

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&acc_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // the descriptors are kernel parameters, not data of the previous kernel
    if (p.a0_off >= 0) prefetch_tmap(&tmA0);
    if (p.a1_off >= 0) prefetch_tmap(&tmA1);
    if (p.b0_off >= 0) prefetch_tmap(&tmB0);
    if (p.b1_off >= 0) prefetch_tmap(&tmB1);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_slot)),
                 "r"(ncols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = tmem_slot;
  // Everything above overlaps the previous kernel under programmatic dependent launch;
  // from here on the kernel reads and writes global memory.
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer: KA swizzle atoms per operand per stage -------------------------
      const int stages = p.stages, stage_bytes = p.stage_bytes, tx_bytes = p.tx_bytes;
      const int a0_off = p.a0_off, a1_off = p.a1_off, b0_off = p.b0_off, b1_off = p.b1_off;
      int* const status = p.status;
      int issued = 0;
      for (int i = 0; i < nk; ++i, ++issued) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&empty_bar[s], ph ^ 1, status, DRAIN_NS)) break;
        uint8_t* st = smem + s * stage_bytes;
        mbar_expect_tx(&full_bar[s], tx_bytes);
        const int k = (kb0 + i) * SK;
#pragma unroll
        for (int a = 0; a < KA; ++a) {
          const int ka = k + a * BK;
          if (p.a_mn) {   // MN-major: boxes of 64 rows x 64 K at (row, k)
            for (int j = 0; j < BM / 64; ++j) {
              if (a0_off >= 0) tma_load_3d(st + a0_off + j * MN_BOX, &tmA0, &full_bar[s], m0 + 64 * j, ka, bz);
              if (a1_off >= 0) tma_load_3d(st + a1_off + j * MN_BOX, &tmA1, &full_bar[s], m0 + 64 * j, ka, bz);
            }
          } else {
            if (a0_off >= 0) tma_load_3d(st + a0_off + a * A_ATOM, &tmA0, &full_bar[s], ka, m0, bz);
            if (a1_off >= 0) tma_load_3d(st + a1_off + a * A_ATOM, &tmA1, &full_bar[s], ka, m0, bz);
          }
          if (p.b_mn) {
            for (int j = 0; j < BN / 64; ++j) {
              if (b0_off >= 0) tma_load_3d(st + b0_off + j * MN_BOX, &tmB0, &full_bar[s], n0 + 64 * j, ka, bz);
              if (b1_off >= 0) tma_load_3d(st + b1_off + j * MN_BOX, &tmB1, &full_bar[s], n0 + 64 * j, ka, bz);
            }
          } else {
            if (b0_off >= 0) tma_load_3d(st + b0_off + a * B_ATOM, &tmB0, &full_bar[s], ka, n0, bz);
            if (b1_off >= 0) tma_load_3d(st + b1_off + a * B_ATOM, &tmB1, &full_bar[s], ka, n0, bz);
          }
        }
      }
      drain_loads(full_bar, issued, stages, status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && nk > 0) {
      // ---- MMA issuer (single thread) -----------------------------------------------
      MmaLoop L;
      L.nk = nk; L.stages = p.stages; L.stage_bytes = p.stage_bytes;
      L.a0_off = p.a0_off; L.a1_off = p.a1_off; L.b0_off = p.b0_off; L.b1_off = p.b1_off;
      L.sbase = smem_u32(smem); L.tbase = tbase;
      L.a_mn = p.a_mn; L.b_mn = p.b_mn;
      L.full_bar = full_bar; L.empty_bar = empty_bar; L.status = p.status;
      L.wait_ns = p.wait_ns;
      mma_dispatch<BN, KA, MODE, false>(L, terms, p.nsub);
      mma_commit(&acc_bar);
      mbar_wait(&acc_bar, 0, p.status, DRAIN_NS);   // every MMA issued here has completed
    }
    __syncwarp();
  } else {
    // ---- accumulator drain: TMEM lane quadrant = warp % 4; the two warps of a quadrant
    // take one column half each (tiles of 128 or more columns) --------------------------
    const int q = warp & 3;
    const int r = q * 32 + lane;   // row within the tile
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    // columns of this warp: BN / EPI_GROUPS per group (16-column granularity; TMA-store
    // chunks of 64), narrow tiles on group 0 only
    const int grp = (warp - 2) >> 2;
    constexpr int GW = EPI_TMA ? 64 : 16;
    constexpr int CG = BN / EPI_GROUPS >= GW ? BN / EPI_GROUPS : BN;
    const int c_begin = CG < BN ? grp * CG : 0;
    const int c_end = CG < BN ? c_begin + CG : (grp == 0 ? BN : 0);
    const bool ok = nk > 0 && mbar_wait(&acc_bar, 0, p.status, p.wait_ns);
    tc_fence_after();
    if (S == 1) {
      if (ok) {
        if (p.tma_store) {
          epilogue_tma<BN, MODE, ACT>(p, &tmC0, &tmC1, &tmA, &tmAd, smem + (warp - 2) * STG_WARP,
                                      tbase + lane_off, q, lane, m0, n0, dual, bz, c_begin, c_end);
        } else {
#pragma unroll 1
          for (int c = c_begin; c < c_end; c += 16) {
            float v0[16], v1[16];
            ld_acc16<BN>(tbase + lane_off, 0, p.nsub, c, v0);
            if (dual) ld_acc16<BN>(tbase + lane_off, 1, p.nsub, c, v1);
            else {
#pragma unroll
              for (int j = 0; j < 16; ++j) v1[j] = 0.f;
            }
            if (n0 + c < p.N) epilogue16<MODE, ACT>(p, m0 + r, n0 + c, v0, v1, dual);
          }
        }
      }
    }
    tc_fence_before();
  }

  if (S > 1) {
    // Split K: CTA z of the cluster owns tile rows [z*128/S, (z+1)*128/S).  After a first
    // cluster barrier (every CTA is done with its pipeline buffers), each CTA pushes its
    // partial rows into the owner's receive buffer R[acc][src rank][row][BN + 4] with remote
    // shared-memory stores; after the second barrier each owner sums the S slabs in rank
    // order (deterministic) and runs the epilogue for its rows.
    constexpr int LDP = BN + 4;
    const int nacc = dual ? 2 : 1;
    const int rows_per = BM / S;
    const uint32_t z = static_cast<uint32_t>(zs);
    const uint32_t rbase = smem_u32(smem);
    __syncwarp();
    cluster_sync_all();
    if (warp >= 2) {
      tc_fence_after();
      const int q = warp & 3;
      const int r = q * 32 + lane;
      const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
      const int grp = (warp - 2) >> 2;
      constexpr int CG = BN / EPI_GROUPS >= 16 ? BN / EPI_GROUPS : BN;
      const int c_begin = CG < BN ? grp * CG : 0;
      const int c_end = CG < BN ? c_begin + CG : (grp == 0 ? BN : 0);
      const bool ok = nk > 0;
      const uint32_t owner = static_cast<uint32_t>(r / rows_per);
      const int rr = r % rows_per;
      for (int a = 0; a < nacc; ++a) {
        const uint32_t row_addr = dsmem_addr(
            rbase + static_cast<uint32_t>((((a * S + z) * rows_per + rr) * LDP) * 4), owner);
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += 16) {
          float v[16];
          if (ok) {
            ld_acc16<BN>(tbase + lane_off, a, p.nsub, c, v);
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.f;
          }
#pragma unroll
          for (int j = 0; j < 16; j += 4)
            st_dsmem4(row_addr + static_cast<uint32_t>((c + j) * 4), v[j], v[j + 1], v[j + 2], v[j + 3]);
        }
      }
      tc_fence_before();
    }
    __syncwarp();
    cluster_sync_all();   // every partial row has reached its owner
    if (warp >= 2) {
      const int e = threadIdx.x - 64;            // 0 .. EPI_THREADS-1
      const int r_begin = static_cast<int>(z) * rows_per;
      float* Rcv = reinterpret_cast<float*>(smem);          // [acc][S][rows_per][LDP]
      float* R = Rcv + nacc * BM * LDP;                     // reduced rows [acc][rows_per][LDP]
      // Phase A: sum the S received slabs in rank order (local shared memory).
      constexpr int VPR = BN / 4;                // float4 per row
      const int nvec = rows_per * VPR;
      for (int a = 0; a < nacc; ++a) {
        for (int it = e; it < nvec; it += EPI_THREADS) {
          const int rr = it / VPR, c4 = (it % VPR) * 4;
          float4 acc = *reinterpret_cast<const float4*>(Rcv + ((a * S) * rows_per + rr) * LDP + c4);
          for (int k = 1; k < S; ++k) {
            const float4 v = *reinterpret_cast<const float4*>(Rcv + ((a * S + k) * rows_per + rr) * LDP + c4);
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
          }
          *reinterpret_cast<float4*>(R + (a * rows_per + rr) * LDP + c4) = acc;
        }
      }
      epi_bar();
      // Phase B: fused epilogue, one column per thread, 8-row chunks (row-major stores are
      // coalesced across consecutive columns)
      constexpr int CW = BN < EPI_THREADS ? BN : EPI_THREADS;
      const int tpc = EPI_THREADS / CW;          // threads per column
      const EpiParams ep = p.epi;
      __nv_bfloat16* A = static_cast<__nv_bfloat16*>(ep.A);
      __nv_bfloat16* Ad = static_cast<__nv_bfloat16*>(ep.Ad);
      for (int col = e % BN; col < BN; col += EPI_THREADS) {
        const int n = n0 + col;
        for (int ch = e / CW; ch * 8 < rows_per; ch += tpc) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int rr = ch * 8 + j;
            const float v0 = R[rr * LDP + col];
            const float v1 = dual ? R[(rows_per + rr) * LDP + col] : 0.f;
            const int m = m0 + r_begin + rr;
            if (m < p.M && n < p.N) {
              const EpiOut o = epi_eval_t<MODE, ACT>(ep, m, n, v0, v1, p.bias0, p.bias1, dual);
              if (p.C0) p.C0[static_cast<int64_t>(m) * p.ldc0 + n] = o.c0;
              if (p.C1 && dual) p.C1[static_cast<int64_t>(m) * p.ldc1 + n] = o.c1;
              if (MODE != EPI_STORE) {
                if (A) A[static_cast<int64_t>(m) * ep.lda + n] = __float2bfloat16_rn(o.o0);
                if (Ad && dual) Ad[static_cast<int64_t>(m) * ep.lda + n] = __float2bfloat16_rn(o.o1);
              }
            }
          }
        }
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tbase),
                 "r"(ncols));
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// 2-D tensor map, 128-byte swizzle: inner extent `inner` elements, `rows` rows, row pitch
// `ld` elements, box box_inner x box_rows.
bool make_map2(CUtensorMap* m, CUtensorMapDataType dt, int esize, const void* ptr, int inner,
               int rows, int ld, int box_inner, int box_rows, int batch = 1,
               int64_t bstride = 0) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  if (batch < 1) batch = 1;
  if (batch == 1) bstride = static_cast<int64_t>(ld) * rows;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(batch)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(ld) * esize,
                           static_cast<cuuint64_t>(bstride) * esize};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, dt, 3, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// K-major bf16 operand [rows][K] (leading dimension ld), box 64 x box_rows.
bool make_map(CUtensorMap* m, const void* ptr, int K, int rows, int ld, int box_rows,
              int batch = 1, int64_t bstride = 0) {
  return make_map2(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ptr, K, rows, ld, BK, box_rows, batch,
                   bstride);
}

// Operand map: K-major [rows][K] (box 64 K x box_rows) or MN-major [K][rows] (boxes of 64
// rows x 64 K; the kernel issues box_rows / 64 of them per stage).
bool make_op_map(CUtensorMap* m, const void* ptr, int K, int rows, int ld, int box_rows, int batch,
                 int64_t bstride, bool mn) {
  if (!mn) return make_map(m, ptr, K, rows, ld, box_rows, batch, bstride);
  return make_map2(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ptr, rows, K, ld, 64, BK, batch, bstride);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// Split of K across a cluster: double S while the grid stays within ~1.2 waves of 152 SMs
// and every split keeps at least two K stages.
int choose_split(int tiles, int nkb) {
  int S = 1;
  while (S < 4 && tiles * S * 2 <= 184 && (nkb + 2 * S - 1) / (2 * S) >= 2) S *= 2;
  return S;
}

template <int BN, int KA, int MODE, int ACT>
cudaError_t launch_cfg(const GemmArgs& a, cudaStream_t s, const char** why) {
  const unsigned t = a.terms;
  const bool useA0 = t & (T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1);
  const bool useA1 = t & (T_C0_A1B0 | T_C1_A1B0 | T_C0_A1B1);
  const bool useB0 = t & (T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0);
  const bool useB1 = t & (T_C0_A0B1 | T_C1_A0B1 | T_C0_A1B1);
  const bool dual = t & (T_C1_A1B0 | T_C1_A0B1);
  TcParams p;
  memset(&p, 0, sizeof(p));
  p.M = a.M; p.N = a.N; p.K = a.K; p.terms = t;
  const int a_bytes = KA * BM * BK * 2, b_bytes = KA * BN * BK * 2;
  int off = 0;
  p.a0_off = useA0 ? (off += a_bytes, off - a_bytes) : -1;
  p.a1_off = useA1 ? (off += a_bytes, off - a_bytes) : -1;
  p.b0_off = useB0 ? (off += b_bytes, off - b_bytes) : -1;
  p.b1_off = useB1 ? (off += b_bytes, off - b_bytes) : -1;
  p.stage_bytes = off;
  p.tx_bytes = off;
  p.nsub = acc_blocks(dual ? 2 : 1, BN);
  const int budget = 220 * 1024;
  int stages = budget / off;
  if (stages > MAX_STAGES) stages = MAX_STAGES;
  if (stages < 2) { *why = "tile does not fit shared memory"; return cudaErrorInvalidValue; }
  p.stages = stages;
  p.C0 = a.C0; p.ldc0 = a.ldc0; p.bias0 = a.bias0;
  p.C1 = dual ? a.C1 : nullptr; p.ldc1 = a.ldc1; p.bias1 = a.bias1;
  p.epi = a.epi;
  p.status = a.status;
  p.wait_ns = g_wait_ns;

  const int tiles_n = (a.N + BN - 1) / BN, tiles_m = (a.M + BM - 1) / BM;
  const int nkb = (a.K + BK * KA - 1) / (BK * KA);
  int S = a.split_k > 0 ? a.split_k
                        : (BN > 128 ? 1 : choose_split(tiles_n * tiles_m * (a.batch < 1 ? 1 : a.batch), nkb));
  if (S != 1 && S != 2 && S != 4 && S != 8) { *why = "split_k must be 1, 2, 4 or 8"; return cudaErrorInvalidValue; }
  if (BN > 128) S = 1;
  if (S > nkb) S = 1;
  p.split = S;

  CUtensorMap mA0, mA1, mB0, mB1, mC0, mC1, mA, mAd;
  memset(&mA0, 0, sizeof(mA0)); memset(&mA1, 0, sizeof(mA1));
  memset(&mB0, 0, sizeof(mB0)); memset(&mB1, 0, sizeof(mB1));
  memset(&mC0, 0, sizeof(mC0)); memset(&mC1, 0, sizeof(mC1));
  memset(&mA, 0, sizeof(mA)); memset(&mAd, 0, sizeof(mAd));
  const int nb = a.batch < 1 ? 1 : a.batch;
  p.a_mn = a.a_mn ? 1 : 0;
  p.b_mn = a.b_mn ? 1 : 0;
  if (useA0 && !make_op_map(&mA0, a.A0, a.K, a.M, a.lda0, BM, nb, a.bsA0, a.a_mn)) { *why = "tensor map A0"; return cudaErrorInvalidValue; }
  if (useA1 && !make_op_map(&mA1, a.A1, a.K, a.M, a.lda1, BM, nb, a.bsA1, a.a_mn)) { *why = "tensor map A1"; return cudaErrorInvalidValue; }
  if (useB0 && !make_op_map(&mB0, a.B0, a.K, a.N, a.ldb0, BN, nb, a.bsB0, a.b_mn)) { *why = "tensor map B0"; return cudaErrorInvalidValue; }
  if (useB1 && !make_op_map(&mB1, a.B1, a.K, a.N, a.ldb1, BN, nb, a.bsB1, a.b_mn)) { *why = "tensor map B1"; return cudaErrorInvalidValue; }
  p.batch = nb;
  p.bsC0 = a.bsC0;
  p.bsC1 = a.bsC1;

  // Row-major outputs through TMA stores when every one of them is aligned for it.
  const bool act = a.epi.mode != EPI_STORE;
  p.st_c0 = p.C0 != nullptr;
  p.st_c1 = p.C1 != nullptr;
  p.st_a = act && a.epi.A != nullptr;
  p.st_ad = act && dual && a.epi.Ad != nullptr;
  bool tma_ok = EPI_TMA && S == 1 && BN >= 64;   // store boxes are 64 columns wide
  if (p.st_c0) tma_ok = tma_ok && aligned16(p.C0) && !(p.ldc0 & 3);
  if (p.st_c1) tma_ok = tma_ok && aligned16(p.C1) && !(p.ldc1 & 3);
  if (p.st_a) tma_ok = tma_ok && aligned16(a.epi.A) && !(a.epi.lda & 7);
  if (p.st_ad) tma_ok = tma_ok && aligned16(a.epi.Ad) && !(a.epi.lda & 7);
  if (nb > 1) tma_ok = tma_ok && !(a.bsC0 & 3) && !(a.bsC1 & 3);
  if (tma_ok && p.st_c0)
    tma_ok = make_map2(&mC0, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, p.C0, a.N, a.M, p.ldc0, 32, 32, nb,
                       a.bsC0);
  if (tma_ok && p.st_c1)
    tma_ok = make_map2(&mC1, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, p.C1, a.N, a.M, p.ldc1, 32, 32, nb,
                       a.bsC1);
  if (tma_ok && p.st_a)
    tma_ok = make_map2(&mA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a.epi.A, a.N, a.M, a.epi.lda, 64, 32);
  if (tma_ok && p.st_ad)
    tma_ok = make_map2(&mAd, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a.epi.Ad, a.N, a.M, a.epi.lda, 64, 32);
  p.tma_store = tma_ok ? 1 : 0;

  int need = stages * off;
  if (S > 1) {
    // split-K: partial tiles [acc][128][BN+4] plus this CTA's reduced rows [acc][128/S][BN+4]
    const int partial_bytes = (dual ? 2 : 1) * (BM + BM / S) * (BN + 4) * 4;
    if (partial_bytes > need) need = partial_bytes;
  }
  if (p.tma_store && EPI_WARPS * STG_WARP > need) need = EPI_WARPS * STG_WARP;
  const int smem = need + 1024;
  static PerDeviceOnce attr_once;
  {
    cudaError_t e = attr_once.run([](int&) {
      return cudaFuncSetAttribute(tc_dual_gemm_kernel<BN, KA, MODE, ACT>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, 225 * 1024);
    });
    if (e != cudaSuccess) return e;
  }
  if (smem > 225 * 1024) { *why = "shared memory budget exceeded"; return cudaErrorInvalidValue; }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(tiles_n, tiles_m, S * nb);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = S;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = g_pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, tc_dual_gemm_kernel<BN, KA, MODE, ACT>, mA0, mA1, mB0, mB1, mC0, mC1, mA,
                            mAd, p);
}

// ================================ 2-SM tiles (cta_group::2) ================================
// A cluster of two CTAs (a CTA pair on two SMs) computes a 256 x BN tile: each CTA stages
// its own 128 rows of A and one half (BN/2 rows) of B, the even CTA issues
// tcgen05.mma.cta_group::2 (M = 256) that reads both CTAs' shared memory and accumulates
// rows 0..127 in its TMEM and rows 128..255 in the odd CTA's TMEM.  Per SM this halves the
// B bytes per flop against the one-SM tile, so the same shared memory holds a deeper
// pipeline.  Both CTAs' TMA loads signal the even CTA's full barriers; the MMA completion
// is multicast to both CTAs' empty barriers and accumulator barrier.  No split of K.

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void tma_load_3d_pair(void* dst, const CUtensorMap* map,
                                                 uint32_t bar_cluster, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar_cluster)
      : "memory");
}

template <int BN, int MODE, int ACT>
__global__ void __launch_bounds__(THREADS2, 1)
    tc2_dual_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                         const __grid_constant__ CUtensorMap tmA1,
                         const __grid_constant__ CUtensorMap tmB0,
                         const __grid_constant__ CUtensorMap tmB1,
                         const __grid_constant__ CUtensorMap tmC0,
                         const __grid_constant__ CUtensorMap tmC1,
                         const __grid_constant__ CUtensorMap tmA,
                         const __grid_constant__ CUtensorMap tmAd, const TcParams prm) {
  TcParams p = prm;
  const int bz = static_cast<int>(blockIdx.z);
  if (p.C0) p.C0 += bz * p.bsC0;
  if (p.C1) p.C1 += bz * p.bsC1;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t empty_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_slot;

  constexpr int BH = BN / 2;                 // B rows staged by each CTA
  const uint32_t rank = cluster_rank();      // 0: issues the MMAs, 1: its peer
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m0 = static_cast<int>(blockIdx.x >> 1) * (2 * BM) + static_cast<int>(rank) * BM;
  const int n0 = blockIdx.y * BN;
  const int nk = (p.K + BK - 1) / BK;
  const unsigned terms = p.terms;
  const bool dual = (terms & (T_C1_A1B0 | T_C1_A0B1)) != 0;
  const uint32_t ncols = tmem_cols((dual ? 2 : 1) * p.nsub * BN);
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&acc_bar, 1);
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
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      const int stages = p.stages, stage_bytes = p.stage_bytes;
      const int a0_off = p.a0_off, a1_off = p.a1_off, b0_off = p.b0_off, b1_off = p.b1_off;
      int* const status = p.status;
      const uint32_t full0 = dsmem_addr(smem_u32(&full_bar[0]), 0);   // even CTA's barriers
      const int nb0 = n0 + static_cast<int>(rank) * BH;
      int issued = 0;
      for (int i = 0; i < nk; ++i, ++issued) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&empty_bar[s], ph ^ 1, status, DRAIN_NS)) break;
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
      // both CTAs' loads signal the even CTA's full barriers; the odd CTA's producer sees
      // the same commits and stops at the same stage, and waits at the final cluster barrier
      if (rank == 0) drain_loads(full_bar, issued, stages, status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (rank == 0 && lane == 0) {
      MmaLoop L;
      L.nk = nk; L.stages = p.stages; L.stage_bytes = p.stage_bytes;
      L.a0_off = p.a0_off; L.a1_off = p.a1_off; L.b0_off = p.b0_off; L.b1_off = p.b1_off;
      L.sbase = smem_u32(smem); L.tbase = tbase;
      L.a_mn = p.a_mn; L.b_mn = p.b_mn;
      L.full_bar = full_bar; L.empty_bar = empty_bar; L.status = p.status;
      L.wait_ns = p.wait_ns;
      mma_dispatch<BN, 1, MODE, true>(L, terms, p.nsub);
      mma_commit_pair(&acc_bar);
      mbar_wait(&acc_bar, 0, p.status, DRAIN_NS);   // every MMA of the pair has completed
    }
    __syncwarp();
  } else {
    // accumulator drain: this CTA's 128 rows of the pair tile, TMEM lane quadrant = warp % 4,
    // one column half per warp of a quadrant
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    constexpr int CG = BN / EPI_GROUPS2;
    const int c_begin = ((warp - 2) >> 2) * CG, c_end = c_begin + CG;
    const bool ok = mbar_wait(&acc_bar, 0, p.status, p.wait_ns);
    tc_fence_after();
    if (ok) {
      if (p.tma_store) {
        epilogue_tma<BN, MODE, ACT>(p, &tmC0, &tmC1, &tmA, &tmAd, smem + (warp - 2) * STG_WARP,
                                    tbase + lane_off, q, lane, m0, n0, dual, bz, c_begin, c_end);
      } else {
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += 16) {
          float v0[16], v1[16];
          ld_acc16<BN>(tbase + lane_off, 0, p.nsub, c, v0);
          if (dual) ld_acc16<BN>(tbase + lane_off, 1, p.nsub, c, v1);
          else {
#pragma unroll
            for (int j = 0; j < 16; ++j) v1[j] = 0.f;
          }
          if (n0 + c < p.N) epilogue16<MODE, ACT>(p, m0 + r, n0 + c, v0, v1, dual);
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  cluster_sync_all();          // both CTAs have drained their TMEM
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tbase),
                 "r"(ncols));
  }
}

template <int BN, int MODE, int ACT>
cudaError_t launch_cfg2(const GemmArgs& a, cudaStream_t s, const char** why) {
  constexpr int BH = BN / 2;
  const unsigned t = a.terms;
  const bool useA0 = t & (T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1);
  const bool useA1 = t & (T_C0_A1B0 | T_C1_A1B0 | T_C0_A1B1);
  const bool useB0 = t & (T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0);
  const bool useB1 = t & (T_C0_A0B1 | T_C1_A0B1 | T_C0_A1B1);
  const bool dual = t & (T_C1_A1B0 | T_C1_A0B1);
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
  p.nsub = acc_blocks(dual ? 2 : 1, BN);
  int stages = (220 * 1024) / off;
  if (stages > MAX_STAGES) stages = MAX_STAGES;
  if (stages < 2) { *why = "tile does not fit shared memory"; return cudaErrorInvalidValue; }
  p.stages = stages;
  p.split = 1;
  p.C0 = a.C0; p.ldc0 = a.ldc0; p.bias0 = a.bias0;
  p.C1 = dual ? a.C1 : nullptr; p.ldc1 = a.ldc1; p.bias1 = a.bias1;
  p.epi = a.epi;
  p.status = a.status;
  p.wait_ns = g_wait_ns;
  const int nb = a.batch < 1 ? 1 : a.batch;
  const int pairs_m = (a.M + 2 * BM - 1) / (2 * BM), tiles_n = (a.N + BN - 1) / BN;

  CUtensorMap mA0, mA1, mB0, mB1, mC0, mC1, mA, mAd;
  memset(&mA0, 0, sizeof(mA0)); memset(&mA1, 0, sizeof(mA1));
  memset(&mB0, 0, sizeof(mB0)); memset(&mB1, 0, sizeof(mB1));
  memset(&mC0, 0, sizeof(mC0)); memset(&mC1, 0, sizeof(mC1));
  memset(&mA, 0, sizeof(mA)); memset(&mAd, 0, sizeof(mAd));
  p.a_mn = a.a_mn ? 1 : 0;
  p.b_mn = a.b_mn ? 1 : 0;
  if (useA0 && !make_op_map(&mA0, a.A0, a.K, a.M, a.lda0, BM, nb, a.bsA0, a.a_mn)) { *why = "tensor map A0"; return cudaErrorInvalidValue; }
  if (useA1 && !make_op_map(&mA1, a.A1, a.K, a.M, a.lda1, BM, nb, a.bsA1, a.a_mn)) { *why = "tensor map A1"; return cudaErrorInvalidValue; }
  if (useB0 && !make_op_map(&mB0, a.B0, a.K, a.N, a.ldb0, BH, nb, a.bsB0, a.b_mn)) { *why = "tensor map B0"; return cudaErrorInvalidValue; }
  if (useB1 && !make_op_map(&mB1, a.B1, a.K, a.N, a.ldb1, BH, nb, a.bsB1, a.b_mn)) { *why = "tensor map B1"; return cudaErrorInvalidValue; }
  p.batch = nb;
  p.bsC0 = a.bsC0;
  p.bsC1 = a.bsC1;

  const bool act = a.epi.mode != EPI_STORE;
  p.st_c0 = p.C0 != nullptr;
  p.st_c1 = p.C1 != nullptr;
  p.st_a = act && a.epi.A != nullptr;
  p.st_ad = act && dual && a.epi.Ad != nullptr;
  bool tma_ok = EPI_TMA2;
  if (p.st_c0) tma_ok = tma_ok && aligned16(p.C0) && !(p.ldc0 & 3);
  if (p.st_c1) tma_ok = tma_ok && aligned16(p.C1) && !(p.ldc1 & 3);
  if (p.st_a) tma_ok = tma_ok && aligned16(a.epi.A) && !(a.epi.lda & 7);
  if (p.st_ad) tma_ok = tma_ok && aligned16(a.epi.Ad) && !(a.epi.lda & 7);
  if (nb > 1) tma_ok = tma_ok && !(a.bsC0 & 3) && !(a.bsC1 & 3);
  if (tma_ok && p.st_c0)
    tma_ok = make_map2(&mC0, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, p.C0, a.N, a.M, p.ldc0, 32, 32, nb,
                       a.bsC0);
  if (tma_ok && p.st_c1)
    tma_ok = make_map2(&mC1, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, p.C1, a.N, a.M, p.ldc1, 32, 32, nb,
                       a.bsC1);
  if (tma_ok && p.st_a)
    tma_ok = make_map2(&mA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a.epi.A, a.N, a.M, a.epi.lda, 64, 32);
  if (tma_ok && p.st_ad)
    tma_ok = make_map2(&mAd, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a.epi.Ad, a.N, a.M, a.epi.lda, 64, 32);
  p.tma_store = tma_ok ? 1 : 0;

  int need = stages * off;
  if (p.tma_store && EPI_WARPS2 * STG_WARP > need) need = EPI_WARPS2 * STG_WARP;
  const int smem = need + 1024;
  static PerDeviceOnce attr_once;
  {
    cudaError_t e = attr_once.run([](int&) {
      return cudaFuncSetAttribute(tc2_dual_gemm_kernel<BN, MODE, ACT>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, 225 * 1024);
    });
    if (e != cudaSuccess) return e;
  }
  if (smem > 225 * 1024) { *why = "shared memory budget exceeded"; return cudaErrorInvalidValue; }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(2 * pairs_m, tiles_n, nb);
  cfg.blockDim = dim3(THREADS2, 1, 1);
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
  return cudaLaunchKernelEx(&cfg, tc2_dual_gemm_kernel<BN, MODE, ACT>, mA0, mA1, mB0, mB1, mC0,
                            mC1, mA, mAd, p);
}

// Dispatch over the tile width for one epilogue (MODE, ACT).
// pair = 1 selects the 2-SM tile (bn 128 or 256).
template <int MODE, int ACT>
cudaError_t launch_bn(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair) {
  if (pair) {
    if (bn == 128) return launch_cfg2<128, MODE, ACT>(a, s, why);
    if (bn == 256) return launch_cfg2<256, MODE, ACT>(a, s, why);
    *why = "2-SM tiles are 128 or 256 columns wide";
    return cudaErrorInvalidValue;
  }
  switch (bn) {
    case 16: return launch_cfg<16, 1, MODE, ACT>(a, s, why);
    case 32: return launch_cfg<32, 1, MODE, ACT>(a, s, why);
    case 64: return launch_cfg<64, 1, MODE, ACT>(a, s, why);
    case 128: return launch_cfg<128, 1, MODE, ACT>(a, s, why);
    case 256: return launch_cfg<256, 1, MODE, ACT>(a, s, why);
  }
  *why = "unsupported tile width";
  return cudaErrorInvalidValue;
}

}  // namespace
}  // namespace mf
