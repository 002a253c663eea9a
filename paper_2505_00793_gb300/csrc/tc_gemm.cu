// Dual-number bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// One launch evaluates a Linear layer of the forward-over-reverse pass (Section 2.2's
// forward-over-reverse HVP applied layer by layer): the primal product P = A B^T and its
// tangent P' = A' B^T + A B'^T share the A and B shared-memory tiles, so four TMA tiles
// feed three tensor-core products per K block.  Every product term is optional (bit mask),
// which gives the primal-only layer, the input layer (A' = 0) and the weight-tangent
// product [a'; a]^T [dz; dz'] from the same kernel.
//
// CTA = 6 warps: warp 0 issues TMA loads, warp 1 owns TMEM and issues tcgen05.mma from
// one thread, warps 2..5 drain the accumulators (tcgen05.ld) and store float32 to global.
// Tile 128 x BN x 64 (bf16, 128-byte swizzle), multi-stage mbarrier pipeline.  Every
// mbarrier wait is bounded; on expiry the CTA records DEV_TIMEOUT and leaves.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <string.h>

#include "internal.h"

namespace mf {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;                 // bf16 elements per 128-byte swizzle row
constexpr int MAX_STAGES = 8;
constexpr int THREADS = 192;
constexpr long long WAIT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz

struct TcParams {
  int M, N, K;
  unsigned terms;
  int stages;
  int a0_off, a1_off, b0_off, b1_off, stage_bytes, tx_bytes;
  float* C0; int ldc0; const float* bias0;
  float* C1; int ldc1; const float* bias1;
  int* status;
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

// Bounded wait: returns false (and flags the status word) if the phase never completes.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (clock64() - t0 > WAIT_CYCLES) {
      if (status) atomicExch(status, DEV_TIMEOUT);
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
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

__device__ __forceinline__ void store_row16(float* C, int ldc, const float* bias, int row,
                                            int col0, int M, int N, const float (&v)[16]) {
  if (row >= M) return;
  float* dst = C + static_cast<int64_t>(row) * ldc + col0;
  const bool full = (col0 + 16 <= N) && ((ldc & 3) == 0) &&
                    ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
  if (full) {
#pragma unroll
    for (int j = 0; j < 16; j += 4) {
      float4 o;
      o.x = v[j] + (bias ? bias[col0 + j] : 0.f);
      o.y = v[j + 1] + (bias ? bias[col0 + j + 1] : 0.f);
      o.z = v[j + 2] + (bias ? bias[col0 + j + 2] : 0.f);
      o.w = v[j + 3] + (bias ? bias[col0 + j + 3] : 0.f);
      *reinterpret_cast<float4*>(dst + j) = o;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (col0 + j < N) dst[j] = v[j] + (bias ? bias[col0 + j] : 0.f);
  }
}

template <int BN>
__global__ void __launch_bounds__(THREADS, 1)
    tc_dual_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                        const __grid_constant__ CUtensorMap tmA1,
                        const __grid_constant__ CUtensorMap tmB0,
                        const __grid_constant__ CUtensorMap tmB1, const TcParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t empty_bar[MAX_STAGES];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_slot;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * BM;
  const int n0 = blockIdx.x * BN;
  const int nkb = (p.K + BK - 1) / BK;
  const unsigned terms = p.terms;
  const bool acc1 = (terms & (T_C1_A1B0 | T_C1_A0B1)) != 0;
  const uint32_t ncols = tmem_cols(acc1 ? 2 * BN : BN);

  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&acc_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
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

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer -------------------------------------------------------------
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % p.stages;
        const uint32_t ph = (kb / p.stages) & 1;
        if (!mbar_wait(&empty_bar[s], ph ^ 1, p.status)) break;
        uint8_t* st = smem + s * p.stage_bytes;
        mbar_expect_tx(&full_bar[s], p.tx_bytes);
        const int k = kb * BK;
        if (p.a0_off >= 0) tma_load_2d(st + p.a0_off, &tmA0, &full_bar[s], k, m0);
        if (p.a1_off >= 0) tma_load_2d(st + p.a1_off, &tmA1, &full_bar[s], k, m0);
        if (p.b0_off >= 0) tma_load_2d(st + p.b0_off, &tmB0, &full_bar[s], k, n0);
        if (p.b1_off >= 0) tma_load_2d(st + p.b1_off, &tmB1, &full_bar[s], k, n0);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer (single thread) -----------------------------------------------
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      const uint32_t d0 = tbase;
      const uint32_t d1 = tbase + BN;
      bool started0 = false, started1 = false;
      bool ok = true;
      for (int kb = 0; kb < nkb && ok; ++kb) {
        const int s = kb % p.stages;
        const uint32_t ph = (kb / p.stages) & 1;
        if (!mbar_wait(&full_bar[s], ph, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t st = smem_u32(smem + s * p.stage_bytes);
        const uint64_t a0 = p.a0_off >= 0 ? sdesc_sw128(st + p.a0_off) : 0;
        const uint64_t a1 = p.a1_off >= 0 ? sdesc_sw128(st + p.a1_off) : 0;
        const uint64_t b0 = p.b0_off >= 0 ? sdesc_sw128(st + p.b0_off) : 0;
        const uint64_t b1 = p.b1_off >= 0 ? sdesc_sw128(st + p.b1_off) : 0;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t adv = static_cast<uint64_t>(kk * 2);   // 32 bytes per K=16 step
          if (terms & T_C0_A0B0) { mma_bf16(d0, a0 + adv, b0 + adv, idesc, started0); started0 = true; }
          if (terms & T_C0_A1B0) { mma_bf16(d0, a1 + adv, b0 + adv, idesc, started0); started0 = true; }
          if (terms & T_C0_A0B1) { mma_bf16(d0, a0 + adv, b1 + adv, idesc, started0); started0 = true; }
          if (terms & T_C1_A1B0) { mma_bf16(d1, a1 + adv, b0 + adv, idesc, started1); started1 = true; }
          if (terms & T_C1_A0B1) { mma_bf16(d1, a0 + adv, b1 + adv, idesc, started1); started1 = true; }
        }
        mma_commit(&empty_bar[s]);
      }
      mma_commit(&acc_bar);
    }
    __syncwarp();
  } else {
    // ---- epilogue: warps 2..5, TMEM lane quadrant = warp % 4 ------------------------
    const int q = warp & 3;
    const bool ok = mbar_wait(&acc_bar, 0, p.status);
    tc_fence_after();
    if (ok) {
      const int row = m0 + q * 32 + lane;
      const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
#pragma unroll 1
      for (int c = 0; c < BN; c += 16) {
        float v[16];
        tmem_ld16(tbase + lane_off + c, v);
        if (p.C0 && n0 + c < p.N) store_row16(p.C0, p.ldc0, p.bias0, row, n0 + c, p.M, p.N, v);
      }
      if (acc1) {
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          float v[16];
          tmem_ld16(tbase + lane_off + BN + c, v);
          if (p.C1 && n0 + c < p.N) store_row16(p.C1, p.ldc1, p.bias1, row, n0 + c, p.M, p.N, v);
        }
      }
    }
    tc_fence_before();
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

// 2-D bf16 tensor map over a K-major operand [rows][K] with leading dimension ld.
bool make_map(CUtensorMap* m, const void* ptr, int K, int rows, int ld, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int BN>
cudaError_t launch_bn(const GemmArgs& a, cudaStream_t s, const char** why) {
  const unsigned t = a.terms;
  const bool useA0 = t & (T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1);
  const bool useA1 = t & (T_C0_A1B0 | T_C1_A1B0);
  const bool useB0 = t & (T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0);
  const bool useB1 = t & (T_C0_A0B1 | T_C1_A0B1);
  TcParams p;
  memset(&p, 0, sizeof(p));
  p.M = a.M; p.N = a.N; p.K = a.K; p.terms = t;
  const int a_bytes = BM * BK * 2, b_bytes = BN * BK * 2;
  int off = 0;
  p.a0_off = useA0 ? (off += a_bytes, off - a_bytes) : -1;
  p.a1_off = useA1 ? (off += a_bytes, off - a_bytes) : -1;
  p.b0_off = useB0 ? (off += b_bytes, off - b_bytes) : -1;
  p.b1_off = useB1 ? (off += b_bytes, off - b_bytes) : -1;
  p.stage_bytes = off;
  p.tx_bytes = off;
  const int budget = 220 * 1024;
  int stages = budget / off;
  if (stages > MAX_STAGES) stages = MAX_STAGES;
  if (stages < 2) { *why = "tile does not fit shared memory"; return cudaErrorInvalidValue; }
  p.stages = stages;
  p.C0 = a.C0; p.ldc0 = a.ldc0; p.bias0 = a.bias0;
  p.C1 = a.C1; p.ldc1 = a.ldc1; p.bias1 = a.bias1;
  p.status = a.status;

  CUtensorMap mA0, mA1, mB0, mB1;
  memset(&mA0, 0, sizeof(mA0)); memset(&mA1, 0, sizeof(mA1));
  memset(&mB0, 0, sizeof(mB0)); memset(&mB1, 0, sizeof(mB1));
  if (useA0 && !make_map(&mA0, a.A0, a.K, a.M, a.lda0, BM)) { *why = "tensor map A0"; return cudaErrorInvalidValue; }
  if (useA1 && !make_map(&mA1, a.A1, a.K, a.M, a.lda1, BM)) { *why = "tensor map A1"; return cudaErrorInvalidValue; }
  if (useB0 && !make_map(&mB0, a.B0, a.K, a.N, a.ldb0, BN)) { *why = "tensor map B0"; return cudaErrorInvalidValue; }
  if (useB1 && !make_map(&mB1, a.B1, a.K, a.N, a.ldb1, BN)) { *why = "tensor map B1"; return cudaErrorInvalidValue; }

  const int smem = stages * off + 1024;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(tc_dual_gemm_kernel<BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, 225 * 1024);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid((a.N + BN - 1) / BN, (a.M + BM - 1) / BM);
  tc_dual_gemm_kernel<BN><<<grid, THREADS, smem, s>>>(mA0, mA1, mB0, mB1, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t tc_gemm(const GemmArgs& a, cudaStream_t s, const char** why) {
  static const char* dummy;
  if (!why) why = &dummy;
  if (a.M <= 0 || a.N <= 0 || a.K <= 0 || (a.terms & 31u) == 0) {
    *why = "empty GEMM";
    return cudaErrorInvalidValue;
  }
  const void* ptrs[4] = {a.A0, a.A1, a.B0, a.B1};
  const int lds[4] = {a.lda0, a.lda1, a.ldb0, a.ldb1};
  const unsigned uses[4] = {T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1, T_C0_A1B0 | T_C1_A1B0,
                            T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0, T_C0_A0B1 | T_C1_A0B1};
  for (int i = 0; i < 4; ++i) {
    if (!(a.terms & uses[i])) continue;
    if (!ptrs[i] || (reinterpret_cast<uintptr_t>(ptrs[i]) & 15) || (lds[i] & 7) || lds[i] < a.K) {
      *why = "operand pointer must be 16-byte aligned with ld a multiple of 8 and >= K";
      return cudaErrorInvalidValue;
    }
  }
  if (a.N <= 16) return launch_bn<16>(a, s, why);
  if (a.N <= 32) return launch_bn<32>(a, s, why);
  if (a.N <= 64) return launch_bn<64>(a, s, why);
  return launch_bn<128>(a, s, why);
}

}  // namespace mf
