// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <mutex>

namespace mf {

// Kernel attributes (cudaFuncSetAttribute) and occupancy figures belong to one device: a
// process that drives several GPUs sets and measures them once per device.  One instance per
// call site (a function-local static of the launching template), guarded by its own mutex.
constexpr int kMaxDevices = 64;
struct PerDeviceOnce {
  std::mutex mu;
  bool done[kMaxDevices] = {};
  int value[kMaxDevices] = {};
  // Runs f() -> cudaError_t on the current device unless it already succeeded there.
  template <typename F>
  cudaError_t run(F&& f) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (done[dev]) return cudaSuccess;
    e = f(value[dev]);
    if (e == cudaSuccess) done[dev] = true;
    return e;
  }
  // The value that f stored on the current device (0 before the first success).
  int get() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
    std::lock_guard<std::mutex> lock(mu);
    return value[dev];
  }
};

// Device status word values (also the mf_status codes they map to).
// Kernels raise the word with atomicMax, so the most severe condition of a call survives:
// a timed-out wait (whose skipped work leaves garbage behind) over a non-finite value over
// an out-of-range label (1).
enum : int { DEV_OK = 0, DEV_NONFINITE = 5, DEV_TIMEOUT = 6 };

// GEMM product terms (same bit meaning as mf_dual_gemm_bf16's `terms`).
enum : unsigned {
  T_C0_A0B0 = 1u, T_C0_A1B0 = 2u, T_C0_A0B1 = 4u, T_C1_A1B0 = 8u, T_C1_A0B1 = 16u,
  T_C0_A1B1 = 32u
};
constexpr unsigned T_ALL = 63u;

inline int term_count(unsigned t) { return __builtin_popcount(t & T_ALL); }

enum Act : int { ACT_IDENT = 0, ACT_TANH = 1, ACT_GELU = 2, ACT_SILU = 3 };
enum EpiMode : int { EPI_STORE = 0, EPI_ACT_FWD = 1, EPI_ACT_BWD = 2 };

// Fused epilogue of a dual GEMM (see device_math.cuh for the element rules).  The A family
// outputs have the operand element type of the GEMM backend (bf16 for tensor cores, float
// for the SIMT path): A/Ad row-major [M][lda], each nullable.  The next GEMM reads them in
// place (K- or MN-major), so no transposed copy is written.
struct EpiParams {
  int mode = EPI_STORE;
  int act = ACT_IDENT;
  void* A = nullptr; void* Ad = nullptr; int lda = 0;
  const float* Z = nullptr; const float* Zd = nullptr; int ldz = 0;   // EPI_ACT_BWD inputs
};

// C[m][n] (+)= sum over selected terms of X[m][k] * Y[n][k]   (both operands K-major).
struct GemmArgs {
  int M = 0, N = 0, K = 0;
  const void* A0 = nullptr; int lda0 = 0;
  const void* A1 = nullptr; int lda1 = 0;
  const void* B0 = nullptr; int ldb0 = 0;
  const void* B1 = nullptr; int ldb1 = 0;
  float* C0 = nullptr; int ldc0 = 0; const float* bias0 = nullptr;
  float* C1 = nullptr; int ldc1 = 0; const float* bias1 = nullptr;
  unsigned terms = 0;
  EpiParams epi;
  int batch = 1;           // independent GEMMs of the same shape (attention heads)
  int64_t bsA0 = 0, bsA1 = 0, bsB0 = 0, bsB1 = 0, bsC0 = 0, bsC1 = 0;   // batch strides (elements)
  int split_k = 0;         // 0 = choose automatically, else 1/2/4/8 (tensor-core path)
  int bn = 0, ka = 0;      // tile width / K atoms per stage; 0 = choose automatically
  int pair = 0;            // 2-SM tiles (tensor-core path): 0 automatic, 1 always, -1 never
  // Operand layouts: K-major (default, X[row][k] at row * ld + k) or MN-major
  // (X[row][k] at k * ld + row), for A0/A1 and for B0/B1.
  bool a_mn = false, b_mn = false;
  int* status = nullptr;   // device status word (timeouts), may be null
};

// tcgen05 bf16 GEMM (tc_gemm.cu).  Returns cudaSuccess or the launch error; sets *why on a
// host-side rejection (bad alignment/ld) and returns cudaErrorInvalidValue.
cudaError_t tc_gemm(const GemmArgs& a, cudaStream_t s, const char** why);
// Activation-epilogue instances (tc_gemm_act.cu dispatches to one translation unit per
// activation, tc_gemm_act_<activation>.cu), called by tc_gemm.
cudaError_t tc_gemm_act(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair);
cudaError_t tc_gemm_act_ident(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair);
cudaError_t tc_gemm_act_tanh(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair);
cudaError_t tc_gemm_act_gelu(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair);
cudaError_t tc_gemm_act_silu(const GemmArgs& a, cudaStream_t s, const char** why, int bn, int pair);
// Process-wide choice of 2-SM tiles for GEMMs that leave it automatic: 0 never, 1 when the
// grid fills the GPU (default), 2 whenever M > 128.
extern int g_pair_mode;
// Limit of the tensor-core GEMMs' MMA-issuer and epilogue waits, in nanoseconds
// (MF_OPT_WAIT_LIMIT_US; default 2 s).  Process-wide, read at launch.
extern long long g_wait_ns;
// Persistent CTA-pair form of the tcgen05 GEMM (tc_gemm_persist.cu), MF_OPT_GEMM_PERSISTENT:
// g_gemm_persist 0 = off; 1 = every 2-SM GEMM, dual products at 128-wide tiles with two
// TMEM accumulator sets; 2 (default) = as 1 except dual products with K > 2048, which take
// 256-wide tiles with one accumulator set; 3 = every 2-SM GEMM, dual products at their
// 256-wide tiles with one accumulator set.  bn is 128 or 256.
cudaError_t tc_gemm_persist(const GemmArgs& a, cudaStream_t s, const char** why, int bn);
extern int g_gemm_persist;
// SIMT float32 GEMM with the same semantics (simt_gemm.cu).
cudaError_t simt_gemm(const GemmArgs& a, cudaStream_t s);

// ---- elementwise / row kernels (kernels.cu); T is float or __nv_bfloat16 -------------

// Column fills: dst[n][r * ld[n] + col[n]] = value[n] for r < rows.
struct ColFill {
  int n = 0;
  void* dst[64];
  int col[64];
  int ld[64];
  float value[64];
};
template <typename T>
void fill_cols(const ColFill& f, int rows, cudaStream_t s);

struct LossArgs {
  int loss = 0;            // 0 squared, 1 softmax CE, 2 chain MSE (motivating example)
  int chain = 0;           // chain MSE: steps M of the recursion
  int rows = 0, cols = 0;
  const float* F = nullptr;  const float* Fd = nullptr;  // logits [rows][cols], tangent
  const float* Yf = nullptr; const int* Yi = nullptr;    // targets
  const float* eta_w = nullptr;   // example weight logits [rows] (weights = sigmoid), or
  const float* ex_w = nullptr;    // explicit weights [rows]; both null = 1
  float inv_norm = 1.f;    // 1/B
  float* l = nullptr;      // per-example loss [rows] (nullable)
  float* ld = nullptr;     // per-example tangent loss [rows] (nullable)
  float* d_eta = nullptr;  // += sigmoid'(eta_w) * ld * inv_norm  [rows] (nullable)
  void* dF = nullptr; void* dFd = nullptr; int ldo = 0; // seeds in T [rows][ldo]
  int* status = nullptr;
  // chain MSE by reverse-over-reverse: tape [2M][rows*cols] floats; ror = 1 records it in the
  // primal loss (writes dF), ror = 2 runs the adjoint of the chain's backward along Fd
  // (writes dFd, ld, d_eta) and overwrites the y-bar half with partial adjoints
  float* tape = nullptr;
  int ror = 0;
};
template <typename T>
void loss_seed(const LossArgs& a, cudaStream_t s);

// Fused narrow head (head_fused.cu): the output layer's forward product, the loss of
// loss_seed (squared or softmax CE) and the output layer's data product with the activation
// backward of the layer below, one block per example row.  Used for outputs of at most
// kHeadMaxOut units when g_fused_head is 1 (MF_OPT_FUSED_HEAD; default 0).
constexpr int kHeadMaxOut = 16;
struct HeadArgs {
  int rows = 0, D = 0, C = 0;      // example rows, head input width, head outputs
  bool dual = false;               // tangent pass along u
  int act = ACT_IDENT;             // activation of the layer below the head
  const void* A = nullptr; const void* Ad = nullptr; int lda = 0;   // head inputs [rows][lda] (T)
  const void* W = nullptr; const void* U = nullptr; int ldw = 0;    // [D][ldw] operand copies (T)
  const float* bias = nullptr; const float* ubias = nullptr;        // nullable
  LossArgs loss;                   // targets, weights, outputs and the head seeds (dF, dFd, ldo)
  const float* Z = nullptr; const float* Zd = nullptr; int ldz = 0;      // layer below: z, z'
  void* dz_prev = nullptr; void* dzd_prev = nullptr; int ld_prev = 0;    // its seeds (T); null:
                                                                         // no data product
};
template <typename T>
cudaError_t head_fused(const HeadArgs& a, cudaStream_t s);
extern int g_fused_head;

// out[0] = scale * sum_i x[i] (deterministic, one block)
void sum_scaled(const float* x, int n, float scale, float* out, cudaStream_t s);

struct LrArgs {
  float alpha = 0.f;
  const float* plr = nullptr;   // per-parameter log-lr [P]
  const float* slr = nullptr;   // scalar log-lr [1]
};

// Per-layer view of the flat parameter vector for the fused update/cast kernel.  Layer l
// occupies rows[l] x dout[l] floats at off[l] (W_l rows, then the bias row when present);
// its first din[l] rows are cast to the GEMM operand copy W (row-major [din][ldw]), or U for
// the tangent.
constexpr int kMaxLayers = 96;
// Fused update kernel geometry: UPD_THREADS threads of four parameters each per block;
// update_blocks is the block count of one layer (and the number of scalar-lr partials).
constexpr int UPD_THREADS = 256;
constexpr int UPD_ELEMS = UPD_THREADS * 4;
inline int update_blocks(int rows, int cols) {
  return static_cast<int>((static_cast<int64_t>(rows) * cols + UPD_ELEMS - 1) / UPD_ELEMS);
}

struct LayerTable {
  int n = 0;
  int rows[kMaxLayers], din[kMaxLayers], dout[kMaxLayers];
  int64_t off[kMaxLayers];
  int tile0[kMaxLayers + 1];
  int ldw[kMaxLayers];
  void* W[kMaxLayers]; void* U[kMaxLayers];
};

enum LuMode : int { LU_CAST = 0, LU_ROLLOUT = 1, LU_ADJOINT = 2 };
struct LayerUpdArgs {
  int mode = LU_CAST;
  const float* cast_src = nullptr;  // parameters to cast into W (nullable)
  bool cast_src_to_u = false;       // LU_CAST: write into U instead of W
  // LU_ROLLOUT (K4):  m' = mu m + g ; theta' = theta - lr m' ; cast theta' into W
  const float* theta = nullptr; const float* m = nullptr; const float* g = nullptr;
  float* theta_out = nullptr; float* m_out = nullptr;
  // LU_ADJOINT (K5):  theta_bar += Hu ; d eta_lr from m_adj ; u' = mu u - lr theta_bar ;
  //                   cast u' into U
  float* theta_bar = nullptr; const float* Hu = nullptr; const float* m_adj = nullptr;
  const float* u_in = nullptr; float* u_out = nullptr; float* d_plr = nullptr;
  float* partials = nullptr;       // scalar log-lr: one partial per block (tile)
  float mu = 0.f;
  LrArgs lr;
  int* status = nullptr;
  // Adam (adam = 1), for the step whose bias corrections are c1 = 1 - b1^(j+1), c2 = 1 - b2^(j+1):
  //  LU_ROLLOUT: m' = b1 m + (1-b1) g, v' = b2 v + (1-b2) g^2, theta' = theta - lr (m'/c1) /
  //              (sqrt(v'/c2) + eps); v (nullable = 0) in, v_out out.
  //  LU_ADJOINT with adam_pre: the reverse of step j from its outputs (m_adj = m_{j+1},
  //              v_adj = v_{j+1}) and input momentum m_prev = m_j (nullable = 0), with the
  //              cotangents theta_bar (after += Hu), mbar, vbar of theta_{j+1}, m_{j+1}, v_{j+1}
  //              (read only when bar_in): writes u_out = g-bar_j and mbar, vbar <- those of
  //              m_j, v_j; d eta_lr gets -lr theta_bar (m_{j+1}/c1) / (sqrt(v_{j+1}/c2) + eps).
  int adam = 0;
  bool adam_pre = false, bar_in = false;
  float b1 = 0.f, b2 = 0.f, eps = 0.f, c1 = 1.f, c2 = 1.f;
  const float* v = nullptr; float* v_out = nullptr;
  const float* v_adj = nullptr; const float* m_prev = nullptr;
  float* mbar = nullptr; float* vbar = nullptr;
  bool vec_ok = false;   // set by layer_update: every vector above is 16-byte aligned
};
template <typename T>
void layer_update(const LayerTable& tab, const LayerUpdArgs& a, cudaStream_t s);

void fill(float* p, int64_t n, float v, cudaStream_t s);

// Reverse-over-reverse element kernels (MLP): dabar = dzbar phi'(z), zpart = dzbar phi''(z) da;
// zbar = zpart + abar phi'(z).  T outputs row-major [rows][ld].
template <typename T>
void ror_fwd_elem(int act, const float* dzbar, const float* Z, const float* dA, int rows, int cols,
                  T* dab, int ld, float* zpart, cudaStream_t s);
template <typename T>
void ror_bwd_elem(int act, const float* zpart, const float* abar, const float* Z, int rows,
                  int cols, T* zb, int ld, cudaStream_t s);

// ---- fused dual attention (flash_attn.cu) -------------------------------------------------
// Heads [BH][S][64] bf16 (q pre-scaled by 1/sqrt(64)), causal.  Forward: O (and O') float32
// [BH][S][64], per-row lse and rbar [BH][S].  Backward: from dO (and dO') bf16 heads and
// D, D' [BH][S] (flash_prep), writes dQ, dK, dV (and tangents) float32 [BH][S][64].
struct FlashArgs {
  int BH = 0, S = 0;
  const __nv_bfloat16 *Q = nullptr, *K = nullptr, *V = nullptr;
  const __nv_bfloat16 *Qd = nullptr, *Kd = nullptr, *Vd = nullptr;
  const __nv_bfloat16 *dO = nullptr, *dOd = nullptr;
  float *O = nullptr, *Od = nullptr, *lse = nullptr, *rbar = nullptr;
  const float *D = nullptr, *Dd = nullptr;
  float *dQ = nullptr, *dQd = nullptr, *dK = nullptr, *dKd = nullptr, *dV = nullptr,
        *dVd = nullptr;
  // Forward outputs, head-merged: when Om is set the forward writes O (and O') as T, token
  // major [B*S][ldo] at column h*64 + e (H heads), instead of float32 O / Od per head.
  int H = 0, ldo = 0;
  __nv_bfloat16 *Om = nullptr, *Omd = nullptr;
  int tc = 1;              // tcgen05 forward where S is a multiple of 128: 0 never,
                           // 1 the dual kernel, 2 the dual and the primal kernels
  int tc_bwd = 0;          // 1: tcgen05 backward (primal and dual) where supported
  // tcgen05 backward only: when dqkv is set, the kernels write the gradient of the fused
  // q|k|v projection instead of float32 dQ, dK, dV: token-major bf16 rows [B*S][ldq], q at
  // column h*64 + e (scaled by qscale), k at H*64 + h*64 + e, v at 2*H*64 + h*64 + e, with
  // the inverse RoPE rotation of table rope ([S][32] (cos, sin) pairs) applied to q and k
  // (the output of dec_rope_merge); dqkvd likewise for the tangents.
  __nv_bfloat16 *dqkv = nullptr, *dqkvd = nullptr;
  int ldq = 0;
  const float* rope = nullptr;
  float qscale = 1.f;
  int* status = nullptr;   // device status word (bounded waits of the tcgen05 kernels)
};
bool flash_supported(int S, int dh);
// tcgen05 forward (flash_tc.cu): S a multiple of 128, 64-wide heads.
bool flash_tc_supported(int S, int dh);
cudaError_t flash_tc_fwd(const FlashArgs& a, bool dual, cudaStream_t s);
// tcgen05 backward (both kernels): S a multiple of 128, 64-wide heads, 16-byte aligned row
// statistics.
bool flash_tc_bwd_supported(const FlashArgs& a, bool dual);
// Whether flash_bwd runs the tcgen05 backward for these arguments (and so honours dqkv).
bool flash_bwd_merges(const FlashArgs& a, bool dual);
cudaError_t flash_tc_bwd(const FlashArgs& a, bool dual, cudaStream_t s);
void flash_fwd(const FlashArgs& a, bool dual, cudaStream_t s);
void flash_bwd(const FlashArgs& a, bool dual, cudaStream_t s);
// D = rowsum(dO (*) O), D' = rowsum(dO' (*) O + dO (*) O') per (token, head) from float32
// merged gradients [N][ld] and bf16 merged outputs; Dd / dOd / Od may be null (primal).
// The same pass writes dO (and dO') as bf16 per head, [B*H][S][64], for the backward kernels.
void flash_prep(int N, int S, int H, const float* dO, const float* dOd, const void* O,
                const void* Od, int ld, float* D, float* Dd, void* dOh, void* dOhd,
                cudaStream_t s);

// ---- decoder-only transformer kernels (decoder_kernels.cu) ------------------------------
void dec_embed_fwd(int N, int S, int d, int V, const int* ids, const float* E, const float* UE,
                   float* x, float* xd, int* status, cudaStream_t s);
template <typename T>
void dec_rmsnorm_fwd(int N, int d, float eps, const float* x_in, const float* y, const float* xd_in,
                     const float* yd, const float* g, const float* gd, float* x_out, float* xd_out,
                     float* r, float* rd, T* h, T* hd, int ldh, cudaStream_t s);
// dx (+=) the RMSNorm backward; when dxb / dxdb are given the updated dx / dx' are also
// written in T (the next GEMM seeds), row-major [N][d].  When dg (or dg' with dyd) is given,
// the gain gradient dg[j] = sum_r dy[r][j] x[r][j] r_r (and its tangent) is written too, in
// a fixed summation order.  part: scratch of 2 * dec_gain_chunks(N) * d floats.  Returns the
// number of kernels launched.
int dec_gain_chunks(int N);
template <typename T>
int dec_rmsnorm_bwd(int N, int d, const float* x, const float* xd, const float* r, const float* rd,
                    const float* g, const float* gd, const float* dy, const float* dyd, float* dx,
                    float* dxd, float* dg, float* dgd, float* part, cudaStream_t s,
                    T* dxb = nullptr, T* dxdb = nullptr);
// RoPE table [S][dh/2] of (cos, sin) pairs, float32, from double-precision angles.
void dec_rope_table(int S, int dh, float base, float* tab, cudaStream_t s);
template <typename T>
void dec_rope_split(int N, int S, int H, int dh, const float* rtab, float qscale, const float* qkv,
                    T* Q, T* K, T* V, cudaStream_t s);
template <typename T>
void dec_rope_merge(int N, int S, int H, int dh, const float* rtab, float qscale, const float* dQ,
                    const float* dK, const float* dV, T* out, int ldo, cudaStream_t s);
template <typename T>
void dec_head_merge(int N, int S, int H, int dh, const float* O, T* out, int ldo, cudaStream_t s);
template <typename T>
void dec_head_split(int N, int S, int H, int dh, const float* X, T* out, cudaStream_t s);
template <typename T>
void dec_softmax_fwd(int S, int rows, const float* Sc, const float* Scd, T* P, T* Pd,
                     cudaStream_t s);
template <typename T>
void dec_softmax_bwd(int S, int rows, const T* P, const T* Pd, const float* dP, const float* dPd,
                     T* dS, T* dSd, cudaStream_t s);
void dec_ce_stats(int N, int S, int V, const int* ids, const float* F, const float* Fd, float* lse,
                  float* l, float* pf, float* ld, int* status, cudaStream_t s);
template <typename T>
void dec_ce_seed(int N, int S, int V, const int* ids, const float* F, const float* Fd,
                 const float* lse, const float* pf, const float* eta_w, const float* ex_w,
                 float inv_norm, T* dF, T* dFd, int ldo, cudaStream_t s);
void dec_seq_reduce(int B, int S, const float* l, const float* ld, const float* eta_w, float invB,
                    float* l_seq, float* ld_seq, float* d_eta, cudaStream_t s);
// tmp: scratch of N ints
void dec_token_csr(int N, int S, int V, const int* ids, int* count, int* start, int* order,
                   int* tmp, cudaStream_t s);
void dec_embed_bwd(int V, int d, const int* start, const int* order, const float* dx,
                   const float* dxd, float* dE, float* dEd, cudaStream_t s);
template <typename T>
void cast_rows(const float* X, int rows, int cols, T* Y, int ldy, cudaStream_t s);

}  // namespace mf
