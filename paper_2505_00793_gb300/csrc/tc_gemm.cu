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
#include "tc_gemm_impl.cuh"

namespace mf {

int g_pair_mode = 1;
long long g_wait_ns = 2000000000LL;

cudaError_t tc_gemm(const GemmArgs& a, cudaStream_t s, const char** why) {
  static const char* dummy;
  if (!why) why = &dummy;
  if (a.M <= 0 || a.N <= 0 || a.K <= 0 || (a.terms & T_ALL) == 0 || (a.terms & ~T_ALL)) {
    *why = "empty GEMM";
    return cudaErrorInvalidValue;
  }
  const void* ptrs[4] = {a.A0, a.A1, a.B0, a.B1};
  const int lds[4] = {a.lda0, a.lda1, a.ldb0, a.ldb1};
  const unsigned uses[4] = {T_C0_A0B0 | T_C0_A0B1 | T_C1_A0B1, T_C0_A1B0 | T_C1_A1B0 | T_C0_A1B1,
                            T_C0_A0B0 | T_C0_A1B0 | T_C1_A1B0, T_C0_A0B1 | T_C1_A0B1 | T_C0_A1B1};
  for (int i = 0; i < 4; ++i) {
    if (!(a.terms & uses[i])) continue;
    const bool mn = i < 2 ? a.a_mn : a.b_mn;
    const int minld = mn ? (i < 2 ? a.M : a.N) : a.K;   // K-major rows hold K, MN-major rows M/N
    if (!ptrs[i] || (reinterpret_cast<uintptr_t>(ptrs[i]) & 15) || (lds[i] & 7) || lds[i] < minld) {
      *why = "operand pointer must be 16-byte aligned with ld a multiple of 8 and >= its row length";
      return cudaErrorInvalidValue;
    }
  }
  if (a.batch > 1 && a.epi.mode != EPI_STORE) {
    *why = "batched GEMMs support the plain-store epilogue only";
    return cudaErrorInvalidValue;
  }
  if (a.batch > 1) {
    const int64_t bs[4] = {a.bsA0, a.bsA1, a.bsB0, a.bsB1};
    for (int i = 0; i < 4; ++i)
      if ((a.terms & uses[i]) && (bs[i] & 7)) {
        *why = "operand batch strides must be multiples of 8 elements";
        return cudaErrorInvalidValue;
      }
  }
  if (a.epi.mode != EPI_STORE) {
    const void* outs[2] = {a.epi.A, a.epi.Ad};
    for (int i = 0; i < 2; ++i)
      if (outs[i] && (reinterpret_cast<uintptr_t>(outs[i]) & 15)) {
        *why = "epilogue outputs must be 16-byte aligned";
        return cudaErrorInvalidValue;
      }
    if (a.epi.lda & 7) {
      *why = "epilogue leading dimensions must be multiples of 8";
      return cudaErrorInvalidValue;
    }
  }
  int bn = a.bn, pair = 0;
  const int nbatch = a.batch < 1 ? 1 : a.batch;
  if (a.pair >= 0 && a.split_k <= 1 && a.M > 128 && (bn == 0 || bn == 128 || bn == 256)) {
    // 2-SM tiles (256 rows per CTA pair) when the pair grid fills the GPU
    const int pairs_m = ((a.M + 255) / 256) * nbatch;
    if (a.pair == 1 || g_pair_mode == 2) {
      pair = 1;
      if (bn == 0) bn = a.N > 128 ? 256 : 128;
    } else if (g_pair_mode == 1 && bn == 0 && a.M >= 256) {
      // 256-wide pairs when they fill a wave of 76 pairs, or when 128-wide pairs would spill
      // into a second wave while the 256-wide grid still holds 40 or more pairs
      const int p256 = pairs_m * ((a.N + 255) / 256), p128 = pairs_m * ((a.N + 127) / 128);
      if (p256 >= 76 || (p128 > 76 && p256 >= 40)) { pair = 1; bn = 256; }
      else if (p128 >= 60) { pair = 1; bn = 128; }
    }
  }
  if (bn == 0) {
    // Narrow outputs take the narrowest tile; otherwise 64-wide tiles while a 128-wide grid
    // would leave most SMs idle (small-batch layers), else 128 (dual) or 256 columns.
    const bool dual = a.terms & (T_C1_A1B0 | T_C1_A0B1);
    const int tiles_m = ((a.M + 127) / 128) * nbatch;
    const int nkb = (a.K + 63) / 64;
    if (a.N <= 16) bn = 16;
    else if (a.N <= 32) bn = 32;
    // Long K (weight products over thousands of tokens): 128-wide tiles stage twice the
    // MMA work per byte of 64-wide ones, and the cluster K split fills the GPU instead.
    else if (a.N > 64 && nkb >= 32) bn = 128;
    else if (a.N <= 64 || tiles_m * ((a.N + 127) / 128) < 76) bn = 64;
    else if (dual || tiles_m * ((a.N + 255) / 256) < 152) bn = 128;
    else bn = 256;
  }
  if (a.b_mn && bn < 64) bn = 64;   // MN-major B is staged in 64-row boxes
  if (pair && g_gemm_persist) return tc_gemm_persist(a, s, why, bn);
  if (a.epi.mode == EPI_STORE) return launch_bn<EPI_STORE, ACT_IDENT>(a, s, why, bn, pair);
  return tc_gemm_act(a, s, why, bn, pair);
}

}  // namespace mf
