/*
 * mixflow.h - C ABI of the GB300 mixed-mode (forward-over-reverse) meta-gradient library.
 *
 * The library computes the meta-gradient dV/d eta of a Truncated-BPTT bilevel problem
 * (Eq. 1 of "Scalable Meta-Learning via Mixed-Mode Differentiation", unrolled as Eq. 2):
 *
 *     m_{t+1}     = mu * m_t + grad_theta L_t(theta_t),             m_0 = 0
 *     theta_{t+1} = theta_t - lr (*) m_{t+1},                        t = 0..T-1
 *     L_t(theta)  = (1/B) sum_b w_{t,b} l_b(theta; x_{t,b}),  w_{t,b} = sigmoid(eta_{t,b})
 *     V           = (1/B_outer) sum_b l_b(theta_T; outer batch)
 *
 * with lr = alpha, or exp(eta_lr) per parameter, or exp(eta_s) for one scalar log-lr.
 * The backward sweep walks t = T-1..0 using the reparameterisation of Eq. 3 and the
 * symmetry identities of Eqs. 6-7: every vector-Hessian and vector-mixed-derivative product
 * of the recurrence Eq. 5 is evaluated as a Hessian-vector product by forward-over-reverse
 * differentiation (Section 3, Proposition 3.1, Algorithm 2):
 *
 *     theta_bar_T = grad V(theta_T),  m_bar_T = 0
 *     u_t         = m_bar_{t+1} - lr (*) theta_bar_{t+1}
 *     theta_bar_t = theta_bar_{t+1} + H_t u_t              (H_t = Hessian of L_t at theta_t)
 *     m_bar_t     = mu * u_t
 *     d eta_{t,b} = sigmoid'(eta_{t,b}) / B * (grad l_b(theta_t) . u_t)
 *     d eta_lr   += -lr (*) m_{t+1} (*) theta_bar_{t+1}
 *
 * Inner models:
 *  - MF_ARCH_MLP: multilayer perceptrons.  Parameters are one flat float32 vector: for each
 *    layer l, W_l as [d_l][d_{l+1}] row-major, then b_l [d_{l+1}].
 *  - MF_ARCH_DECODER: decoder-only transformer (the language models of Section 5): token
 *    embedding, n_layers blocks of pre-RMSNorm causal multi-head attention with RoPE
 *    (rotate-half, angle s * rope_base^(-2j/dh)) and pre-RMSNorm GELU MLP with residual
 *    connections, final RMSNorm, untied head; per-sequence next-token cross-entropy (mean
 *    over the seq_len predicted positions).  No biases.  Flat parameter order: E [vocab][d];
 *    per block g1 [d], Wqkv [d][3d] (q | k | v columns, heads contiguous), Wo [d][d],
 *    g2 [d], W1 [d][d_ff], W2 [d_ff][d]; then gf [d], Wh [d][vocab].
 *
 * Conventions for every call:
 *  - Tensor arguments are device pointers owned by the caller (e.g. torch CUDA tensors),
 *    unless stated otherwise.  They must stay valid until the stream work completes.
 *  - Calls enqueue work on `stream` (a cudaStream_t; NULL = legacy default stream) and
 *    return without synchronising, except where stated.  Argument errors are returned
 *    immediately; errors found on the device (non-finite values, a kernel wait that ran out
 *    of time) are reported by mf_sync().
 *  - Library workspace (the theta_t checkpoint store, activations) is obtained through the
 *    allocator set with mf_set_allocator (default: cudaMalloc, freed with cudaFree),
 *    kept in the handle between calls with the same or smaller shape, and released by
 *    mf_release_workspace() or mf_destroy().
 *  - A handle is not thread-safe; use one handle per host thread.
 */
#ifndef MIXFLOW_H
#define MIXFLOW_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct mf_ctx* mf_handle;

typedef enum {
  MF_OK = 0,
  MF_ERR_INVALID_ARG = 1,   /* a NULL pointer, a bad size or an inconsistent descriptor */
  MF_ERR_UNSUPPORTED = 2,   /* valid request this build does not implement */
  MF_ERR_OOM = 3,           /* the allocator returned NULL */
  MF_ERR_CUDA = 4,          /* a CUDA runtime call failed; see mf_last_error() */
  MF_ERR_NONFINITE = 5,     /* a NaN/Inf reached the adjoint or the updated parameters */
  MF_ERR_TIMEOUT = 6        /* a bounded device-side wait ran out of time */
} mf_status;

enum { MF_ARCH_MLP = 0, MF_ARCH_DECODER = 1 };
enum { MF_ACT_IDENT = 0, MF_ACT_TANH = 1, MF_ACT_GELU = 2, MF_ACT_SILU = 3 };
enum { MF_LOSS_SQUARED = 0, MF_LOSS_SOFTMAX_CE = 1, MF_LOSS_NEXT_TOKEN_CE = 2,
       MF_LOSS_CHAIN_MSE = 3 };
enum { MF_PREC_FP32 = 0, MF_PREC_BF16 = 1 };
enum { MF_META_EXAMPLE_WEIGHTS = 1, MF_META_PARAM_LOGLR = 2, MF_META_SCALAR_LOGLR = 4 };
enum { MF_HVP_MIXED_FOR = 0, MF_HVP_REV_REV = 1 };
enum { MF_OPTIM_SGD = 0, MF_OPTIM_ADAM = 1 };

#define MF_MAX_LAYERS 32

/* Inner model (Eq. 1's L and V).
 *  arch       MF_ARCH_MLP.
 *  n_layers   number of Linear layers, 1..MF_MAX_LAYERS.
 *  dims       n_layers+1 widths: dims[0] = input size, dims[n_layers] = output size.
 *  act        activation after every layer but the last (MF_ACT_*).
 *  has_bias   1 = every layer has a bias vector.
 *  loss       MF_LOSS_SQUARED: l_b = 1/2 mean_o (f_bo - y_bo)^2, y float32 [rows][d_out];
 *             MF_LOSS_SOFTMAX_CE: l_b = logsumexp(f_b) - f_{b,y_b}, y int32 [rows];
 *             MF_LOSS_NEXT_TOKEN_CE (decoder only): x = y = int32 token ids [rows][seq_len+1],
 *             inputs ids[:, 0:S], targets ids[:, 1:S+1];
 *             MF_LOSS_CHAIN_MSE (MLP; the motivating example of Section 3, Eq. 8): the
 *             output f passes through y_0 = f, y_i = i (2 + sin y_{i-1})^cos y_{i-1},
 *             i = 1..chain_steps, and l_b = mean_o (y_M,bo - y_bo)^2 (no 1/2), y float32
 *             [rows][d_out].  In the mixed mode the recursion is evaluated inside the loss
 *             kernel with its first and second derivatives and nothing of it is stored;
 *             under MF_HVP_REV_REV the loss records the chain's tape (y_0..y_{M-1} and the
 *             adjoints ybar_1..ybar_M, 2 M floats per output element) and the adjoint of its
 *             backward reads it back, as reverse mode through the recursion does.
 *  precision  MF_PREC_FP32: float32 inputs, float32 GEMMs (SIMT);
 *             MF_PREC_BF16: bf16 inputs, bf16 tensor-core GEMMs with float32 accumulation;
 *             parameters, optimiser state, adjoints and meta-gradients stay float32.
 *  Decoder fields (MF_ARCH_DECODER; n_layers = blocks): d_model, n_heads (d_model/n_heads a
 *  multiple of 8), d_ff, vocab, seq_len (multiples of 8), rope_base (0 = 10000),
 *  rms_eps (0 = 1e-6).  dims/act/has_bias are ignored for decoders.
 *  chain_steps  M of MF_LOSS_CHAIN_MSE (0..4096; ignored for other losses). */
typedef struct {
  int arch;
  int n_layers;
  int dims[MF_MAX_LAYERS + 1];
  int act;
  int has_bias;
  int loss;
  int precision;
  int d_model, n_heads, d_ff, vocab, seq_len;
  float rope_base, rms_eps;
  int chain_steps;
} mf_model_desc;

/* Inner loop (Eq. 2) and meta-parameters.
 *  T          inner steps (>= 1);  B rows per inner batch;  B_outer rows of the outer batch.
 *  alpha      constant learning rate (used when no log-lr meta-parameter is set).
 *  momentum   heavy-ball coefficient mu in [0, 1) (0 = plain SGD); must be 0 with Adam.
 *  meta_kind  bit mask of MF_META_*; eta is laid out as [T*B example-weight logits]
 *             [P per-parameter log-lrs][1 scalar log-lr], in that order, for the bits set.
 *             PARAM_LOGLR and SCALAR_LOGLR are mutually exclusive.
 *  hvp_mode   MF_HVP_MIXED_FOR: each step's Hessian-vector product is forward-over-reverse
 *             (Algorithm 2, the mixed-mode sweep).  MF_HVP_REV_REV: reverse-over-reverse
 *             (Algorithm 1's schedule: the inner backward is kept whole and differentiated
 *             again in reverse), the standard-AD baseline; same result, more workspace.
 *             MLPs keep every layer's dz and da (and the chain loss its tape); the decoder
 *             keeps the residual-stream cotangent at every block output and recomputes the
 *             cotangents inside a block.
 *  ckpt_every k: segment length of the checkpoint store (Section 4).  0 or 1 keeps every
 *             theta_t (and m_t when needed): T+1 parameter slots.  k > 1 keeps theta_t only
 *             for t a multiple of k, plus k-1 slots for one segment; the sweep re-runs each
 *             earlier segment's rollout from its checkpoint before walking it back, with the
 *             same kernels, so results are bit-identical to k = 1 for one extra rollout's
 *             work.  theta slots: floor(T/k) + k (k = sqrt(T) minimises them).  m slots:
 *             floor(T/k) + k - 1 when the learning rate is a meta-parameter (the sweep reads
 *             every m_t); floor(T/k) + 1 for momentum alone with k > 1 (checkpoints plus one
 *             running slot, to restart segments); none otherwise.  k > T acts as T.
 *             Negative values are MF_ERR_INVALID_ARG.
 *  optimizer  MF_OPTIM_SGD (plain or heavy-ball, the default when the field is 0) or
 *             MF_OPTIM_ADAM, the inner optimiser of Section 5's language-model tasks
 *             (Kingma & Ba, with bias correction): m' = b1 m + (1-b1) g, v' = b2 v + (1-b2) g^2,
 *             theta' = theta - lr (m'/c1) / (sqrt(v'/c2) + eps), c1 = 1 - b1^(t+1),
 *             c2 = 1 - b2^(t+1), zero initial moments; lr as for SGD (alpha or exp of a
 *             log-lr meta-parameter).  The sweep reverses each step elementwise: the HVP's
 *             tangent is the gradient cotangent g-bar_t = (1-b1) M + 2 (1-b2) g_t V, with M, V
 *             the cotangents of m_{t+1}, v_{t+1}; g_t is recovered as (m_{t+1} - b1 m_t)/(1-b1).
 *             The store keeps m_t and v_t for every t (segmented like theta) plus two
 *             cotangent vectors: 2 (floor(T/k) + k - 1) + 2 extra |theta| slots.
 *  beta1, beta2, adam_eps  Adam's decays in [0, 1) and epsilon (> 0); ignored for SGD.
 *  ckpt_slots s (0 = off; 1..1024, exclusive with ckpt_every > 1; T <= 4096): binomial
 *             checkpointing (Section 4's "binomial checkpointing", Griewank's revolve).  The
 *             store keeps s + 3 states (theta_t, plus m_t whenever momentum, a learned
 *             learning rate or Adam needs it, plus v_t with Adam): S_0, s snapshots and two
 *             scratch states; the rollout leaves snapshots on its way, and the sweep
 *             recomputes every other state forward from a snapshot, following the schedule
 *             that re-runs the fewest inner steps for s snapshots (dynamic programming over
 *             the split points; mf_checkpoint_plan reports it).  The same kernels recompute
 *             the same values, so results are bit-identical to ckpt_every = 1.  Adam adds two
 *             |theta| buffers for a deferred reverse step.  s >= T - 1 stores every state. */
typedef struct {
  int T, B, B_outer;
  float alpha, momentum;
  int meta_kind;
  int hvp_mode;
  int ckpt_every;
  int optimizer;
  float beta1, beta2, adam_eps;
  int ckpt_slots;
} mf_loop_desc;

/* Create a handle for one inner-model architecture.  *out receives a library-owned handle.
 * Errors: MF_ERR_INVALID_ARG (bad descriptor), MF_ERR_CUDA (no usable device). */
mf_status mf_create(const mf_model_desc* desc, mf_handle* out);

/* Release the handle and its workspace (synchronises the device first). */
mf_status mf_destroy(mf_handle h);

/* Route workspace allocations through caller callbacks (e.g. PyTorch's caching allocator).
 * alloc(bytes, stream, ctx) returns a device pointer or NULL; free(ptr, bytes, stream, ctx).
 * Pass alloc = free = NULL to restore the default.  Releases the current workspace. */
mf_status mf_set_allocator(mf_handle h, void* (*alloc)(size_t, void*, void*),
                           void (*free_fn)(void*, size_t, void*, void*), void* ctx);

/* Number of parameters P = |theta| and of meta-parameters |eta| for loop descriptor `loop`
 * (loop may be NULL, then *n_eta is set to 0).  Host-only. */
mf_status mf_param_count(mf_handle h, const mf_loop_desc* loop, int64_t* n_params,
                         int64_t* n_eta);

/* Bytes of workspace mf_meta_grad needs for `loop` (checkpoint store + activations; with
 * MF_HVP_REV_REV also the stored inner backward graph). */
mf_status mf_workspace_bytes(mf_handle h, const mf_loop_desc* loop, size_t* bytes);

/* Checkpoint plan of a reverse sweep over T inner steps, host-only (no handle, no device):
 * *state_slots receives the number of stored states (theta_t, each with its optimiser state
 * where kept) and *recompute_steps the inner steps the sweep re-runs forward, for
 * ckpt_every = k (uniform segments; 0 or 1 = every state) or ckpt_slots = s > 0 (binomial;
 * then k must be 0 or 1).  State slots: T + 1 for k = 1; floor(T/k) + k for k > 1 (re-runs
 * about one rollout); s + 3 for the binomial schedule, with the fewest re-runs for s.
 * Errors: MF_ERR_INVALID_ARG (T < 1, negative or conflicting k and s, T > 4096 with s). */
mf_status mf_checkpoint_plan(int T, int ckpt_every, int ckpt_slots, int* state_slots,
                             int64_t* recompute_steps);

/* Free the cached workspace now (the next call allocates it again). */
mf_status mf_release_workspace(mf_handle h);

/* Inner rollout only (Eq. 2, Algorithm 2's loop): theta0 [P] float32, eta [n_eta] float32
 * (NULL allowed when n_eta = 0), inner_x [T][B][d_in] (bf16 for MF_PREC_BF16, float32 for
 * MF_PREC_FP32), inner_y [T][B] int32 labels (MF_LOSS_SOFTMAX_CE) or [T][B][d_out] float32
 * targets.  Decoders: inner_x = inner_y = int32 token ids [T][B][seq_len+1].  Writes
 * thetaT [P].  bf16 inputs must start on a 16-byte boundary with d_in a multiple of 8.
 * Errors: MF_ERR_INVALID_ARG (descriptor, NULL or misaligned tensor), MF_ERR_OOM (workspace),
 * MF_ERR_CUDA; device-side errors come from mf_sync(). */
mf_status mf_inner_rollout(mf_handle h, const mf_loop_desc* loop, const float* theta0,
                           const float* eta, const void* inner_x, const void* inner_y,
                           float* thetaT, void* stream);

/* One fwdrev_grad backward step (Section 3.1): at parameters theta [P], on the batch
 * x [B][d_in] / y [B] or [B][d_out] (decoders: x = y = token ids [B][seq_len+1]) with
 * per-example loss weights ex_w [B] (NULL = all 1), for L = (1/B) sum_b ex_w_b l_b:
 *   Hv [P]             = (d^2 L / d theta^2) v        (forward-over-reverse)
 *   tangent_losses [B] = grad l_b(theta) . v           (nullable; the mixed term per example)
 *   grad [P]           = grad L(theta)                 (nullable)
 * hvp_mode MF_HVP_MIXED_FOR (forward-over-reverse) or MF_HVP_REV_REV (reverse-over-reverse). */
mf_status mf_hvp(mf_handle h, int B, const float* theta, const void* x, const void* y,
                 const float* ex_w, const float* v, float* Hv, float* tangent_losses,
                 float* grad, int hvp_mode, void* stream);

/* The meta-gradient (Algorithm 2): rollout storing theta_t (and m_t when lr is a
 * meta-parameter; m_t and v_t with Adam), outer gradient (Eq. 4), then the reverse sweep
 * t = T-1..0 with the loop's hvp_mode.  Inputs as for mf_inner_rollout, plus
 * outer_x [B_outer][d_in], outer_y [B_outer] int32 or [B_outer][d_out] float32 (decoders:
 * outer_x = outer_y = token ids [B_outer][seq_len+1]).  Outputs (float32, device):
 *   d_eta [n_eta]      dV/d eta (same layout as eta; NULL allowed when n_eta = 0).
 *   d_theta0 [P]       dV/d theta_0 (nullable; required when n_eta = 0).
 *   outer_loss [1]     V (nullable).
 * Errors: as for mf_inner_rollout; device-side MF_ERR_NONFINITE (a NaN or Inf in theta_t or
 * an adjoint) and MF_ERR_TIMEOUT come from mf_sync(), after which the handle stays usable. */
mf_status mf_meta_grad(mf_handle h, const mf_loop_desc* loop, const float* theta0,
                       const float* eta, const void* inner_x, const void* inner_y,
                       const void* outer_x, const void* outer_y, float* d_eta,
                       float* d_theta0, float* outer_loss, void* stream);

/* Wait for the handle's last stream and report device-side errors (MF_ERR_NONFINITE,
 * MF_ERR_TIMEOUT, MF_ERR_CUDA).  Clears the device status word. */
mf_status mf_sync(mf_handle h);

/* Static description of a status code, and the handle's last error message. */
const char* mf_status_string(mf_status s);
const char* mf_last_error(mf_handle h);

/* Diagnostics.  mf_stats: kernel launches issued by the handle since creation and the
 * largest workspace it has held.  mf_set_kernel_timing(h, 1) records CUDA events around
 * every launch of the bf16 dual GEMM (inside the captured graph when graphs are in use);
 * mf_kernel_time synchronises and returns the summed milliseconds and launch count of that
 * kernel since the last reset - for graph replays, those of the most recent replay - plus
 * its algorithmic flops (2*M*N*K per accumulated product term), then resets.
 * mf_set_kernel_timing(h, 2) instead records the next call's GEMM launches for
 * mf_replay_gemms (below); 0 and 1 leave a pending record in place. */
mf_status mf_stats(mf_handle h, uint64_t* launches, size_t* peak_workspace_bytes);
mf_status mf_set_kernel_timing(mf_handle h, int enable);
mf_status mf_kernel_time(mf_handle h, double* ms, uint64_t* launches, double* flops);

/* Roofline timing of the bf16 dual GEMM without perturbing the call.  After
 * mf_set_kernel_timing(h, 2), the handle's next mf_meta_grad / mf_inner_rollout / mf_hvp runs
 * eagerly (no graph replay) and records the argument list of every bf16 dual GEMM it
 * launches.  mf_replay_gemms then launches that list back to back, in the recorded order, as
 * one captured CUDA graph on `stream`, `reps` times between two CUDA events, and returns the
 * milliseconds of one replay, the launches per replay and their algorithmic flops
 * (2*M*N*K per product term and batch entry).  The replay reads and overwrites the handle's
 * workspace and the buffers the recorded call was given: those must still be allocated, and
 * the outputs of the recorded call are not preserved.  The record is dropped with the
 * workspace (mf_release_workspace, a larger call, mf_set_allocator, mf_destroy) and replaced
 * by the next record.  Synchronises `stream`.  Errors: MF_ERR_INVALID_ARG (no record,
 * reps < 1), MF_ERR_CUDA. */
mf_status mf_replay_gemms(mf_handle h, int reps, void* stream, double* ms, uint64_t* launches,
                          double* flops);

/* Library options.  MF_OPT_CUDA_GRAPHS (default 1): a call of mf_meta_grad, mf_inner_rollout
 * or mf_hvp repeated with the same shapes and pointers is captured into a CUDA graph on its
 * second occurrence and replayed afterwards, on a library-owned stream that is ordered after
 * and before the caller's stream with events.  0 launches every kernel individually.
 * MF_OPT_PDL (default 1, process-wide): kernels are launched with programmatic dependent
 * launch, so each one's launch and prologue overlap the tail of the previous kernel on the
 * stream (memory effects keep stream order).  0 launches them with plain stream order.
 * Setting it drops the handle's captured graphs.
 * MF_OPT_CONCURRENT (default 1): in each backward layer the weight product and the data
 * product run on two streams (parallel branches of a captured graph); 0 runs them in
 * sequence on the call's stream.
 * MF_OPT_GEMM_2SM (process-wide): 1 (default) computes a bf16 GEMM with 256-row tiles on
 * CTA pairs (tcgen05 cta_group::2) when its grid of pairs fills the GPU, 0 never, 2 for
 * every GEMM with more than 128 rows (for tests).  Results are identical up to the
 * summation order within a tile, which both forms share.
 * MF_OPT_FLASH_ATTN (default 1): the decoder's dual attention runs fused, without the
 * S x S probabilities and their tangent in memory (bf16 decoders with d_model/n_heads = 64
 * and seq_len a multiple of 64; others always use the materialised form).  With 1, for
 * sequences of whole 128-token tiles, the dual (tangent-carrying) forward and both backward
 * kernels (primal and dual) run on tcgen05 tensor cores and the primal forward on
 * warp-level MMAs; 3 runs the primal forward on tcgen05 as well; 4 keeps the backward on
 * warp-level MMAs; 2 uses the warp-level kernels only.  0 materialises them (per
 * block, for the backward).  Setting it drops the handle's captured graphs and changes the
 * workspace size.
 * MF_OPT_GEMM_PERSISTENT (process-wide, default 2): GEMMs that take CTA-pair tiles run as a
 * persistent kernel: one pair per SM pair walks a static list of output tiles (grouped so
 * that the pairs running together share row blocks of A and a band of B), with two TMEM
 * accumulator sets when they fit so that a tile's epilogue overlaps the next tile's main
 * loop.  0 never; 1 every pair GEMM, dual products at 128-wide tiles (two sets of their two
 * accumulators fit); 2 as 1, except that dual products with K > 2048 take 256-wide tiles
 * with one accumulator set (half the operand bytes per MMA; their long main loops hide the
 * epilogue that one set cannot overlap); 3 every pair GEMM, dual products at 256-wide tiles
 * with one accumulator set.  Same products and summation
 * order within a tile as the one-tile form.  Setting it drops the handle's captured graphs.
 * MF_OPT_FUSED_HEAD (process-wide, default 0): 1 computes the output layer of an MLP with at
 * most 16 outputs and a squared or softmax cross-entropy loss in one kernel per pass: the
 * layer's forward product, the loss with its seeds and tangent losses, and its data product
 * into the layer below (one block per example row, float32 accumulation; the weight product
 * stays a GEMM).  The reverse-over-reverse sweep and the chain loss keep the separate
 * launches.  Setting it drops the handle's captured graphs.
 * MF_OPT_LAYER_UPDATES (default 0): 1 runs an MLP's inner-step and adjoint updates layer by
 * layer on a library stream of the handle, each as soon as its layer's products in the
 * backward pass are done, so that they overlap the layers below instead of following the
 * whole pass.  Element for element the same update.  Decoders and the reverse-over-reverse
 * sweep keep the single update.  Setting it drops the handle's captured graphs.
 * MF_OPT_WAIT_LIMIT_US (process-wide, default 2000000 = 2 s; 0..60000000): how long the
 * tensor-core GEMMs' MMA issuer and epilogue wait for a pipeline stage or an accumulator
 * before giving up (failure detection: a wait that gives up sets the device status word to
 * MF_ERR_TIMEOUT, reported by mf_sync).  After giving up, a CTA stops issuing MMAs, lets the
 * loads and MMAs it already issued complete, and ends; its outputs are then undefined.  A
 * short limit makes waits give up on a healthy GPU, which tests use.  Takes effect at the
 * next launch; drops every handle's graphs captured under another limit (graph keys include
 * it). */
enum { MF_OPT_CUDA_GRAPHS = 1, MF_OPT_PDL = 2, MF_OPT_CONCURRENT = 3, MF_OPT_GEMM_2SM = 4,
       MF_OPT_FLASH_ATTN = 5, MF_OPT_GEMM_PERSISTENT = 6, MF_OPT_FUSED_HEAD = 7,
       MF_OPT_LAYER_UPDATES = 8, MF_OPT_WAIT_LIMIT_US = 9 };
mf_status mf_set_option(mf_handle h, int option, int value);

/* Host-side fault injection for tests: kind 1 = the next workspace allocation fails;
 * kind 2 = the next mf_sync reports MF_ERR_TIMEOUT as if a device wait had expired;
 * kind 0 clears.  Nothing is done on the GPU. */
mf_status mf_inject_fault(mf_handle h, int kind);

/* mf_hvp without any device allocation.  The paper has no counterpart to this call; it
 * exists for callers that cannot allocate device memory: embedders whose device memory is
 * entirely reserved up front by their own allocator (a serving process that claims the GPU
 * at start-up and forbids later cudaMalloc, because a late allocation can fail or stall
 * the device), and hosts that only accept pre-registered buffers.  It computes exactly
 * what mf_hvp computes (MF_HVP_MIXED_FOR) for the MLP described by `desc`, without a
 * handle: inputs and outputs are caller-owned device pointers as in mf_hvp, and all
 * intermediate storage lives in one 32 MiB array in the library's device memory (a
 * file-scope __device__ array that every GPU loading the library holds until the process
 * exits).
 *  - MLP models only (every loss an MLP takes, the chain loss included); a decoder
 *    descriptor (MF_ARCH_DECODER or MF_LOSS_NEXT_TOKEN_CE) returns MF_ERR_UNSUPPORTED.
 *  - Returns MF_ERR_INVALID_ARG when the workspace for (desc, B) exceeds that array
 *    (about 32 MiB; e.g. a [128, 256, 256, 10] MLP at B = 64 needs well under 1 MiB).
 *  - The first call on a device looks up the array's device address (cudaGetSymbolAddress)
 *    with that device current; make that first call outside any stream capture.
 *  - Every call shares the array and leaves its contents behind; the call clears the
 *    status word it needs.  Calls whose GPU work overlaps (different streams, or several
 *    host threads) race on the array: serialise them.
 *  - Device-side conditions (non-finite values, a bounded wait that ran out) are not
 *    reported; the call is asynchronous on `stream` like mf_hvp. */
mf_status mf_hvp_noalloc(const mf_model_desc* desc, int B, const float* theta, const void* x,
                         const void* y, const float* ex_w, const float* v, float* Hv,
                         float* tangent_losses, float* grad, void* stream);

/* Building block exposed for tests and profiling: the bf16 dual GEMM of the sweep.
 * All operands K-major, row-major with leading dimension in elements (multiple of 8):
 *   A0, A1 [M][K] bf16;  B0, B1 [N][K] bf16;  C0, C1 [M][N] float32 (ldc).
 * `terms` selects the products summed into each accumulator:
 *   bit 0: C0 += A0 B0^T   bit 1: C0 += A1 B0^T   bit 2: C0 += A0 B1^T
 *   bit 3: C1 += A1 B0^T   bit 4: C1 += A0 B1^T   bit 5: C0 += A1 B1^T
 * The forward tangent of a dual Linear layer is terms = 1|8|16:  C0 = A0 B0^T (primal),
 * C1 = A1 B0^T + A0 B1^T (tangent).  bias0/bias1 [N] float32 are added when non-NULL.
 * Layout flags in the same word: bit 8 - A0, A1 are MN-major, stored [K][M] (element (m, k)
 * at k * lda + m, lda >= M); bit 9 - B0, B1 are MN-major, stored [K][N] (ldb >= N).
 * Runs on tcgen05 tensor cores with TMEM accumulators and TMA-fed shared memory. */
mf_status mf_dual_gemm_bf16(int M, int N, int K, const void* A0, int lda0, const void* A1,
                            int lda1, const void* B0, int ldb0, const void* B1, int ldb1,
                            float* C0, int ldc0, const float* bias0, float* C1, int ldc1,
                            const float* bias1, unsigned terms, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* MIXFLOW_H */
