// Host runtime of the library: handle, workspace, the MLP executor (dual forward, dual loss,
// dual backward as sequences of kernel launches), the rollout with its theta_t checkpoint
// store, the mixed-mode reverse sweep, and the C ABI of include/mixflow.h.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>
#include <type_traits>
#include <utility>
#include <vector>

#include "../../include/mixflow.h"
#include "decoder_layout.h"
#include "internal.h"
#include "launch.cuh"
#include "revolve.h"

using mf::GemmArgs;

namespace {

constexpr size_t ALIGN = 256;
inline size_t align_up(size_t x, size_t a = ALIGN) { return (x + a - 1) / a * a; }
inline int ld8(int x) { return (x + 7) / 8 * 8; }
inline uint32_t float_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof(u));
  return u;
}

}  // namespace

struct mf_ctx {
  mf_model_desc md;
  bool decoder = false;
  DecLayout Ly;
  int L = 0;
  std::vector<int> dims;
  std::vector<int64_t> woff, boff;
  int64_t P = 0;
  int maxd = 0;
  bool bf16 = false;

  void* (*ualloc)(size_t, void*, void*) = nullptr;
  void (*ufree)(void*, size_t, void*, void*) = nullptr;
  void* uctx = nullptr;

  void* ws = nullptr;
  size_t ws_bytes = 0;
  size_t peak = 0;
  int* d_status = nullptr;
  std::string err;
  uint64_t launches = 0;
  cudaStream_t last_stream = nullptr;
  int fault = 0;

  bool timing = false;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> evs;
  double timed_flops = 0.0;
  // GEMM launch record (mf_set_kernel_timing(h, 2)): the bf16 dual GEMMs of the next call in
  // launch order, with their algorithmic flops; mf_replay_gemms replays them back to back as
  // one captured graph.  Dropped with the workspace the recorded pointers refer to.
  bool record = false;
  std::vector<mf::GemmArgs> rec;
  double rec_flops = 0.0;
  cudaGraphExec_t rec_exec = nullptr;

  // CUDA graphs: a call repeated with the same shapes and pointers is captured once (on the
  // second occurrence) and replayed from then on, on the library's own stream.
  struct GraphCache {
    uint64_t key = 0, pending = 0;
    cudaGraphExec_t exec = nullptr;
    uint64_t launches = 0;
    // kernel timing: event pairs recorded inside the graph (re-recorded by each replay)
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> evs;
    double flops = 0.0;
  };
  GraphCache* timed_replay = nullptr;   // graph whose events hold the last replay's times
  bool use_graphs = true;
  GraphCache g_meta, g_roll, g_hvp;
  cudaStream_t gstream = nullptr;
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  // Side stream for independent GEMMs of one backward layer (the weight product runs next
  // to the data product); forked from and joined back into the working stream with events,
  // which a stream capture turns into parallel graph branches.
  cudaStream_t sstream = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // Decoder backward: the weight product of each linear layer runs on the side stream next
  // to the data product; ev_w[j] marks the end of the latest weight product that reads seed
  // buffer j, which the working stream waits for before it rewrites that buffer.
  cudaEvent_t ev_w[4] = {nullptr, nullptr, nullptr, nullptr};
  bool concurrent = true;
  int flash = 1;              // fused dual attention where supported (MF_OPT_FLASH_ATTN)
  // Per-layer parameter updates (MF_OPT_LAYER_UPDATES): an update stream that takes each
  // layer's update as soon as that layer's backward products are done, joined back into the
  // working stream at the end of the backward pass.
  bool layer_updates = false;
  cudaStream_t ustream = nullptr;
  cudaEvent_t ev_u_in = nullptr, ev_u_out = nullptr;
};

namespace {

mf_status fail(mf_ctx* h, mf_status s, const std::string& msg) {
  if (h) h->err = msg;
  return s;
}

#define MF_CUDA(h, call)                                                          \
  do {                                                                            \
    cudaError_t e_ = (call);                                                      \
    if (e_ != cudaSuccess)                                                        \
      return fail(h, MF_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

// ---- workspace layout -------------------------------------------------------------------
struct Plan {
  int rows = 0;          // max rows of any batch
  int T = 0;
  int n_theta_slots = 0, n_m_slots = 0;
  int nb = 0;            // blocks (tiles) of the per-layer update kernel
  size_t bytes = 0;
  size_t o_theta = 0, o_m = 0, o_g = 0, o_tbar = 0, o_u = 0, o_part = 0, o_l = 0, o_ld = 0;
  std::vector<size_t> o_Wb, o_Ub, o_A, o_Ad, o_Z, o_Zd;
  std::vector<int> lda;  // leading dim of layer l's input activations (room for the bias column)
  size_t o_dZ[2] = {0, 0}, o_dZd[2] = {0, 0};
  // fused narrow head (MF_OPT_FUSED_HEAD): the output layer's seeds in buffers of their own,
  // so that its weight product does not hold up the layers below
  bool head_bufs = false;
  size_t o_dZh = 0, o_dZdh = 0;
  // reverse-over-reverse: the stored reverse graph (per-layer dz, da) and the adjoints
  bool ror = false;
  std::vector<size_t> o_SZ, o_SA, o_DAB, o_ZP;
  size_t o_DZB = 0, o_ZB = 0, o_AB = 0;
  // ... and, for the chain loss, its tape: y_0..y_{M-1} and y-bar_1..y-bar_M per element
  size_t o_CH = 0;
};

int n_update_tiles(const mf_ctx* h) {
  int tiles = 0;
  for (int l = 0; l < h->L; ++l) {
    const int rows = h->dims[l] + (h->md.has_bias ? 1 : 0);
    tiles += mf::update_blocks(rows, h->dims[l + 1]);
  }
  return tiles;
}

// Activations a [rows][din] carry one extra column (ones for a, zeros for a') so that the
// weight product [a 1]^T dz, read MN-major straight from the row-major activations, yields
// the weight and the bias gradient (stored contiguously in theta).  No operand is stored
// transposed: the forward product reads W [din][dout] MN-major as well.
Plan make_plan(const mf_ctx* h, int rows, int T, int n_theta_slots, int n_m_slots,
               bool with_partials, bool ror = false) {
  Plan p;
  p.ror = ror;
  p.rows = rows;
  p.T = T;
  p.n_theta_slots = n_theta_slots;
  p.n_m_slots = n_m_slots;
  const size_t es = h->bf16 ? 2 : 4;
  const int hb = h->md.has_bias ? 1 : 0;
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t r = o; o += align_up(bytes); return r; };
  const size_t P4 = static_cast<size_t>(h->P) * 4;
  p.o_theta = take(P4 * n_theta_slots);
  p.o_m = take(P4 * n_m_slots);
  p.o_g = take(P4);
  p.o_tbar = take(P4);
  p.o_u = take(P4);
  p.nb = n_update_tiles(h);
  p.o_part = take(with_partials ? static_cast<size_t>(p.nb) * (T > 0 ? T : 1) * 4 : 4);
  p.o_l = take(static_cast<size_t>(rows) * 4);
  p.o_ld = take(static_cast<size_t>(rows) * 4);
  const int L = h->L;
  p.o_Wb.resize(L); p.o_Ub.resize(L); p.o_A.resize(L); p.o_Ad.resize(L);
  p.o_Z.resize(L); p.o_Zd.resize(L); p.lda.resize(L);
  for (int l = 0; l < L; ++l) {
    const int din = h->dims[l], dout = h->dims[l + 1];
    p.lda[l] = ld8(din + hb);
    p.o_Wb[l] = take(static_cast<size_t>(din) * ld8(dout) * es);
    p.o_Ub[l] = take(static_cast<size_t>(din) * ld8(dout) * es);
    p.o_A[l] = take(static_cast<size_t>(rows) * p.lda[l] * es);
    p.o_Ad[l] = take(static_cast<size_t>(rows) * p.lda[l] * es);
    p.o_Z[l] = take(static_cast<size_t>(rows) * dout * 4);
    p.o_Zd[l] = take(static_cast<size_t>(rows) * dout * 4);
  }
  const int md = h->maxd;
  for (int b = 0; b < 2; ++b) {
    p.o_dZ[b] = take(static_cast<size_t>(rows) * ld8(md) * es);
    p.o_dZd[b] = take(static_cast<size_t>(rows) * ld8(md) * es);
  }
  if (mf::g_fused_head && !h->decoder && h->dims[L] <= mf::kHeadMaxOut &&
      h->md.loss != MF_LOSS_CHAIN_MSE) {
    p.head_bufs = true;
    p.o_dZh = take(static_cast<size_t>(rows) * ld8(h->dims[L]) * es);
    p.o_dZdh = take(static_cast<size_t>(rows) * ld8(h->dims[L]) * es);
  }
  if (ror) {
    p.o_SZ.resize(L); p.o_SA.resize(L); p.o_DAB.resize(L); p.o_ZP.resize(L);
    for (int l = 0; l < L; ++l) {
      const int din = h->dims[l], dout = h->dims[l + 1];
      p.o_SZ[l] = take(static_cast<size_t>(rows) * ld8(dout) * es);
      p.o_SA[l] = take(static_cast<size_t>(rows) * din * 4);
      p.o_DAB[l] = take(static_cast<size_t>(rows) * ld8(dout + hb) * es);
      p.o_ZP[l] = take(static_cast<size_t>(rows) * dout * 4);
    }
    p.o_DZB = take(static_cast<size_t>(rows) * md * 4);
    p.o_ZB = take(static_cast<size_t>(rows) * ld8(md) * es);
    p.o_AB = take(static_cast<size_t>(rows) * md * 4);
    if (h->md.loss == MF_LOSS_CHAIN_MSE && h->md.chain_steps > 0)
      p.o_CH = take(2 * static_cast<size_t>(h->md.chain_steps) * rows * h->dims[L] * 4);
  }
  p.bytes = o;
  return p;
}

void drop_graphs(mf_ctx* h);

void drop_record(mf_ctx* h) {
  if (h->rec_exec) cudaGraphExecDestroy(h->rec_exec);
  h->rec_exec = nullptr;
  h->rec.clear();
  h->rec_flops = 0.0;
}

// Algorithmic flops of one GEMM launch: 2 M N K per accumulated product term and batch entry.
double gemm_flops(const GemmArgs& g) {
  return 2.0 * g.M * g.N * static_cast<double>(g.K) * mf::term_count(g.terms) *
         (g.batch > 1 ? g.batch : 1);
}

// Called by the executors for every tensor-core GEMM they launch.
void note_gemm(mf_ctx* h, const GemmArgs& g) {
  if (!h->record) return;
  h->rec.push_back(g);
  h->rec_flops += gemm_flops(g);
}

void release_ws(mf_ctx* h) {
  drop_graphs(h);
  drop_record(h);
  if (!h->ws) return;
  cudaDeviceSynchronize();
  if (h->ufree) h->ufree(h->ws, h->ws_bytes, nullptr, h->uctx);
  else cudaFree(h->ws);
  h->ws = nullptr;
  h->ws_bytes = 0;
}

mf_status ensure_ws(mf_ctx* h, size_t bytes, cudaStream_t s) {
  if (h->fault == 1) {
    h->fault = 0;
    return fail(h, MF_ERR_OOM, "injected allocation failure");
  }
  if (h->ws && h->ws_bytes >= bytes) return MF_OK;
  release_ws(h);
  void* p = nullptr;
  if (h->ualloc) {
    p = h->ualloc(bytes, static_cast<void*>(s), h->uctx);
  } else if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    p = nullptr;
  }
  if (!p) return fail(h, MF_ERR_OOM, "workspace allocation of " + std::to_string(bytes) + " bytes failed");
  h->ws = p;
  h->ws_bytes = bytes;
  h->peak = std::max(h->peak, bytes);
  return MF_OK;
}

// ---- CUDA graph replay ---------------------------------------------------------------------
uint64_t mix_key(uint64_t h, uint64_t v) {
  h ^= v + 0x9e3779b97f4a7c15ULL + (h << 6) + (h >> 2);
  return h;
}

void drop_graph(mf_ctx::GraphCache& g) {
  if (g.exec) cudaGraphExecDestroy(g.exec);
  g.exec = nullptr;
  g.key = g.pending = 0;
  for (auto& e : g.evs) { cudaEventDestroy(e.first); cudaEventDestroy(e.second); }
  g.evs.clear();
  g.flops = 0.0;
}

void drop_graphs(mf_ctx* h) {
  h->timed_replay = nullptr;
  drop_graph(h->g_meta);
  drop_graph(h->g_roll);
  drop_graph(h->g_hvp);
}

mf_status graph_launch(mf_ctx* h, mf_ctx::GraphCache& g, cudaStream_t user) {
  MF_CUDA(h, cudaEventRecord(h->ev_in, user));
  MF_CUDA(h, cudaStreamWaitEvent(h->gstream, h->ev_in, 0));
  MF_CUDA(h, cudaGraphLaunch(g.exec, h->gstream));
  MF_CUDA(h, cudaEventRecord(h->ev_out, h->gstream));
  MF_CUDA(h, cudaStreamWaitEvent(user, h->ev_out, 0));
  h->launches += g.launches;
  h->timed_replay = g.evs.empty() ? nullptr : &g;
  return MF_OK;
}

// Runs body(stream) eagerly, or replays / captures it as a CUDA graph.  The first call with
// a given key runs eagerly (it may allocate the workspace and set kernel attributes); the
// second captures on the library stream; later ones replay.
template <typename F>
mf_status run_graphed(mf_ctx* h, mf_ctx::GraphCache& g, uint64_t key, cudaStream_t user, F&& body) {
  key = mix_key(key, reinterpret_cast<uintptr_t>(h->ws));
  key = mix_key(key, h->ws_bytes);
  key = mix_key(key, h->timing ? 1 : 0);
  // Process-wide options change which kernels a call launches; another handle may have set
  // them since this handle captured its graphs, so they are part of every graph's key.
  key = mix_key(key, static_cast<uint64_t>(mf::g_pdl));
  key = mix_key(key, static_cast<uint64_t>(mf::g_pair_mode));
  key = mix_key(key, static_cast<uint64_t>(mf::g_gemm_persist));
  key = mix_key(key, static_cast<uint64_t>(mf::g_fused_head));
  key = mix_key(key, static_cast<uint64_t>(mf::g_wait_ns));
  if (h->record) {
    // one eager execution whose GEMM launches are recorded for mf_replay_gemms
    drop_record(h);
    h->record = true;
    const mf_status st = body(user);
    h->record = false;
    return st;
  }
  if (!h->use_graphs || !h->gstream) return body(user);
  if (g.exec && g.key == key) return graph_launch(h, g, user);
  if (g.pending != key) {
    if (g.exec) drop_graph(g);
    g.pending = key;
    return body(user);
  }
  // second identical call: capture
  if (h->ws == nullptr) return body(user);
  const uint64_t l0 = h->launches;
  // events recorded while capturing belong to the graph
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> outer_evs;
  outer_evs.swap(h->evs);
  const double outer_flops = h->timed_flops;
  h->timed_flops = 0.0;
  MF_CUDA(h, cudaStreamBeginCapture(h->gstream, cudaStreamCaptureModeThreadLocal));
  const mf_status st = body(h->gstream);
  cudaGraph_t graph = nullptr;
  const cudaError_t ce = cudaStreamEndCapture(h->gstream, &graph);
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> graph_evs;
  graph_evs.swap(h->evs);
  h->evs.swap(outer_evs);
  const double graph_flops = h->timed_flops;
  h->timed_flops = outer_flops;
  if (st != MF_OK || ce != cudaSuccess || !graph) {
    if (graph) cudaGraphDestroy(graph);
    for (auto& e : graph_evs) { cudaEventDestroy(e.first); cudaEventDestroy(e.second); }
    cudaGetLastError();
    h->launches = l0;
    g.pending = 0;
    if (st != MF_OK) return st;
    return fail(h, MF_ERR_CUDA, std::string("graph capture failed: ") + cudaGetErrorString(ce));
  }
  cudaGraphExec_t exec = nullptr;
  const cudaError_t ie = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (ie != cudaSuccess) {
    for (auto& e : graph_evs) { cudaEventDestroy(e.first); cudaEventDestroy(e.second); }
    cudaGetLastError();
    h->launches = l0;
    g.pending = 0;
    return fail(h, MF_ERR_CUDA, std::string("graph instantiate failed: ") + cudaGetErrorString(ie));
  }
  g.exec = exec;
  g.key = key;
  g.evs.swap(graph_evs);
  g.flops = graph_flops;
  g.launches = h->launches - l0;
  h->launches = l0;
  return graph_launch(h, g, user);
}

size_t y_stride_bytes(const mf_ctx* h, int rows);

// ---- the MLP executor --------------------------------------------------------------------
template <typename T>
struct Exec {
  mf_ctx* h;
  const Plan& p;
  cudaStream_t s;
  char* base;
  mf_status st = MF_OK;
  mf::LayerTable tab;
  bool ror_store = false;   // primal backward keeps every layer's dz (and da) for RoR

  // backward seed buffers of layer l (ping-pong, or the stored reverse graph)
  T* dz_buf(int l) const { return ror_store ? at<T>(p.o_SZ[l]) : at<T>(p.o_dZ[l & 1]); }
  // loss kernel selector: 0 squared, 1 softmax CE, 2 chain MSE
  int loss_kind() const {
    return h->md.loss == MF_LOSS_SOFTMAX_CE ? 1 : h->md.loss == MF_LOSS_CHAIN_MSE ? 2 : 0;
  }
  // The output layer's forward product, loss and data product as one kernel
  // (MF_OPT_FUSED_HEAD); never inside the reverse-over-reverse HVP, whose adjoint passes
  // read the logits and the stored reverse graph.
  bool no_fuse = false;
  const float* fwd_theta = nullptr;   // parameters and tangent of the last forward pass
  const float* fwd_u = nullptr;
  bool fused_head() const {
    return mf::g_fused_head && p.head_bufs && !no_fuse && !ror_store && loss_kind() != 2 &&
           h->dims[h->L] <= mf::kHeadMaxOut;
  }

  Exec(mf_ctx* h_, const Plan& p_, cudaStream_t s_)
      : h(h_), p(p_), s(s_), base(static_cast<char*>(h_->ws)) {
    tab.n = h->L;
    int tiles = 0;
    for (int l = 0; l < h->L; ++l) {
      const int din = h->dims[l], dout = h->dims[l + 1];
      tab.rows[l] = din + (h->md.has_bias ? 1 : 0);
      tab.din[l] = din;
      tab.dout[l] = dout;
      tab.off[l] = h->woff[l];
      tab.tile0[l] = tiles;
      tiles += mf::update_blocks(tab.rows[l], dout);
      tab.ldw[l] = ld8(dout);
      tab.W[l] = at<T>(p.o_Wb[l]);
      tab.U[l] = at<T>(p.o_Ub[l]);
    }
    tab.tile0[h->L] = tiles;
  }

  template <typename U> U* at(size_t off) const { return reinterpret_cast<U*>(base + off); }
  float* theta_slot(int t) const { return at<float>(p.o_theta) + static_cast<int64_t>(t) * h->P; }
  float* m_slot(int j) const { return at<float>(p.o_m) + static_cast<int64_t>(j) * h->P; }
  float* g_buf() const { return at<float>(p.o_g); }
  float* tbar_buf() const { return at<float>(p.o_tbar); }
  float* u_buf() const { return at<float>(p.o_u); }
  float* part_buf() const { return at<float>(p.o_part); }
  float* l_buf() const { return at<float>(p.o_l); }
  float* ld_buf() const { return at<float>(p.o_ld); }
  int nb() const { return p.nb; }
  size_t x_step_bytes(int rows) const {
    return static_cast<size_t>(rows) * h->dims[0] * (h->bf16 ? 2 : 4);
  }
  size_t y_step_bytes(int rows) const { return y_stride_bytes(h, rows); }

  void launched(int n = 1) { h->launches += n; }

  // Fork the side stream off the working stream / join it back (see mf_ctx::sstream).
  bool can_fork() const { return h->concurrent && h->sstream && h->ev_fork && h->ev_join; }
  void fork() {
    if (cudaEventRecord(h->ev_fork, s) != cudaSuccess ||
        cudaStreamWaitEvent(h->sstream, h->ev_fork, 0) != cudaSuccess) {
      st = MF_ERR_CUDA; h->err = "stream fork failed";
    }
  }
  void join() {
    if (cudaEventRecord(h->ev_join, h->sstream) != cudaSuccess ||
        cudaStreamWaitEvent(s, h->ev_join, 0) != cudaSuccess) {
      st = MF_ERR_CUDA; h->err = "stream join failed";
    }
  }

  void gemm(GemmArgs g, cudaStream_t on = nullptr) {
    if (st != MF_OK) return;
    const cudaStream_t s = on ? on : this->s;
    g.status = h->d_status;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    unsigned ev_flags = cudaEventRecordDefault;
    const bool tc = h->bf16;
    if (tc && h->timing) {
      cudaEventCreate(&e0);
      cudaEventCreate(&e1);
      // inside a stream capture an external record becomes an event-record graph node
      cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
      cudaStreamIsCapturing(s, &cs);
      ev_flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
      cudaEventRecordWithFlags(e0, s, ev_flags);
    }
    cudaError_t e;
    const char* why = "";
    if (tc) e = mf::tc_gemm(g, s, &why);
    else e = mf::simt_gemm(g, s);
    if (e != cudaSuccess) {
      st = MF_ERR_CUDA;
      h->err = std::string("dual GEMM launch failed: ") + cudaGetErrorString(e) + " " + why;
      return;
    }
    launched();
    if (tc) note_gemm(h, g);
    if (tc && h->timing) {
      cudaEventRecordWithFlags(e1, s, ev_flags);
      h->evs.emplace_back(e0, e1);
      h->timed_flops += gemm_flops(g);
    }
  }

  // Bias columns of the augmented activations (ones for a, zeros for a' and for the
  // reverse-over-reverse adjoint activations).
  void prepare() {
    if (!h->md.has_bias) return;
    mf::ColFill f;
    for (int l = 0; l < h->L; ++l) {
      f.dst[f.n] = at<T>(p.o_A[l]); f.col[f.n] = h->dims[l]; f.ld[f.n] = p.lda[l]; f.value[f.n] = 1.f; ++f.n;
      f.dst[f.n] = at<T>(p.o_Ad[l]); f.col[f.n] = h->dims[l]; f.ld[f.n] = p.lda[l]; f.value[f.n] = 0.f; ++f.n;
    }
    if (p.ror) {
      for (int l = 0; l + 1 < h->L; ++l) {
        f.dst[f.n] = at<T>(p.o_DAB[l]); f.col[f.n] = h->dims[l + 1]; f.ld[f.n] = p.lda[l + 1];
        f.value[f.n] = 0.f; ++f.n;
      }
    }
    mf::fill_cols<T>(f, p.rows, s);
    launched();
  }

  void update(const mf::LayerUpdArgs& a) {
    mf::layer_update<T>(tab, a, s);
    launched();
  }

  // Per-layer updates (MF_OPT_LAYER_UPDATES).  With upd_after set, backward() runs that
  // update for layer l on the update stream as soon as layer l's weight and data products are
  // done (the update overwrites the layer's operand copies, which the data product reads),
  // and joins the update stream back before it returns; the caller then skips its update of
  // the whole vector.  Every update element reads and writes only its own parameter, so the
  // layers' updates are independent of each other and of the layers still in the pass.
  const mf::LayerUpdArgs* upd_after = nullptr;
  bool layer_updates_ok() const {
    return h->layer_updates && h->ustream && h->ev_u_in && h->ev_u_out;
  }
  void update_layer(const mf::LayerUpdArgs& a, int l) {
    mf::LayerTable t1;
    t1.n = 1;
    t1.rows[0] = tab.rows[l]; t1.din[0] = tab.din[l]; t1.dout[0] = tab.dout[l];
    t1.off[0] = tab.off[l];
    t1.tile0[0] = 0;
    t1.tile0[1] = tab.tile0[l + 1] - tab.tile0[l];
    t1.ldw[0] = tab.ldw[l];
    t1.W[0] = tab.W[l]; t1.U[0] = tab.U[l];
    mf::LayerUpdArgs b = a;
    if (b.partials) b.partials += tab.tile0[l];   // this layer's blocks' scalar-lr partials
    mf::layer_update<T>(t1, b, h->ustream);
    launched();
  }
  // Layer l's products are enqueued on `on`: the update stream waits for them, then updates l.
  void upd_layer_after(int l, cudaStream_t on) {
    if (!upd_after || st != MF_OK) return;
    if (cudaEventRecord(h->ev_u_in, on) != cudaSuccess ||
        cudaStreamWaitEvent(h->ustream, h->ev_u_in, 0) != cudaSuccess) {
      st = MF_ERR_CUDA; h->err = "update stream fork failed";
      return;
    }
    update_layer(*upd_after, l);
  }
  void upd_join() {
    if (!upd_after) return;
    if (cudaEventRecord(h->ev_u_out, h->ustream) != cudaSuccess ||
        cudaStreamWaitEvent(s, h->ev_u_out, 0) != cudaSuccess) {
      st = MF_ERR_CUDA; h->err = "update stream join failed";
    }
  }

  // Cast parameters (or the tangent) into the GEMM operand copies.
  void cast_params(const float* theta, bool tangent) {
    mf::LayerUpdArgs a;
    a.mode = mf::LU_CAST;
    a.cast_src = theta;
    a.cast_src_to_u = tangent;
    update(a);
  }

  // Forward pass of `rows` examples: primal (z) or dual (z, z_dot along u).  Hidden layers
  // fuse bias, activation and its tangent into the GEMM epilogue.
  void forward(int rows, const void* xv, const float* theta, const float* u, bool dual) {
    fwd_theta = theta;
    fwd_u = u;
    const int din0 = h->dims[0];
    const size_t es = sizeof(T);
    // inputs into the augmented layer-0 activations (the bias column is already set)
    if (cudaMemcpy2DAsync(at<T>(p.o_A[0]), p.lda[0] * es, xv, din0 * es, din0 * es, rows,
                          cudaMemcpyDeviceToDevice, s) != cudaSuccess && st == MF_OK) {
      st = MF_ERR_CUDA;
      h->err = "input copy failed";
    }
    for (int l = 0; l < h->L; ++l) {
      if (l == h->L - 1 && fused_head()) break;   // the output layer runs in loss()
      const int din = h->dims[l], dout = h->dims[l + 1];
      GemmArgs g;
      g.M = rows; g.N = dout; g.K = din;
      g.A0 = at<T>(p.o_A[l]); g.lda0 = p.lda[l];
      g.A1 = l == 0 ? nullptr : at<T>(p.o_Ad[l]);
      g.lda1 = p.lda[l];
      g.B0 = at<T>(p.o_Wb[l]); g.ldb0 = ld8(dout);   // W [din][dout]: MN-major
      g.B1 = at<T>(p.o_Ub[l]); g.ldb1 = ld8(dout);
      g.b_mn = true;
      g.C0 = at<float>(p.o_Z[l]); g.ldc0 = dout;
      g.bias0 = h->md.has_bias ? theta + h->boff[l] : nullptr;
      g.terms = mf::T_C0_A0B0;
      if (dual) {
        g.terms |= mf::T_C1_A0B1 | (l > 0 ? mf::T_C1_A1B0 : 0u);
        g.C1 = at<float>(p.o_Zd[l]); g.ldc1 = dout;
        g.bias1 = h->md.has_bias ? u + h->boff[l] : nullptr;
      }
      if (l + 1 < h->L) {
        g.epi.mode = mf::EPI_ACT_FWD;
        g.epi.act = h->md.act;
        g.epi.A = at<T>(p.o_A[l + 1]);
        g.epi.Ad = dual ? at<T>(p.o_Ad[l + 1]) : nullptr;
        g.epi.lda = p.lda[l + 1];
      }
      gemm(g);
    }
  }

  // Loss seeds at the head: d f (and its tangent) into backward buffer set (L-1) & 1.
  void loss(int rows, bool dual, const void* y, const float* eta_w, const float* ex_w,
            float* l_out, float* ld_out, float* d_eta) {
    const int L = h->L, C = h->dims[L];
    mf::LossArgs a;
    a.loss = loss_kind();
    a.chain = h->md.chain_steps;
    a.rows = rows; a.cols = C;
    a.F = at<float>(p.o_Z[L - 1]);
    a.Fd = dual ? at<float>(p.o_Zd[L - 1]) : nullptr;
    if (a.loss != 1) a.Yf = static_cast<const float*>(y);
    else a.Yi = static_cast<const int*>(y);
    a.eta_w = eta_w; a.ex_w = ex_w;
    a.inv_norm = 1.f / static_cast<float>(rows);
    a.l = l_out; a.ld = ld_out; a.d_eta = d_eta;
    const int b = (L - 1) & 1;
    a.dF = dz_buf(L - 1); a.dFd = dual ? at<T>(p.o_dZd[b]) : nullptr;
    a.ldo = ld8(C);
    a.status = h->d_status;
    if (ror_store && a.loss == 2 && a.chain > 0) {   // reverse mode records the chain's tape
      a.tape = at<float>(p.o_CH);
      a.ror = 1;
    }
    if (fused_head()) {
      a.dF = at<T>(p.o_dZh);
      a.dFd = dual ? at<T>(p.o_dZdh) : nullptr;
      head(rows, dual, a, fwd_theta, fwd_u);
      return;
    }
    mf::loss_seed<T>(a, s);
    launched();
  }

  // Fused output layer (see fused_head): forward product of layer L-1 from the activations
  // the forward pass left, the loss `a`, and the data product into layer L-2's seeds.
  void head(int rows, bool dual, const mf::LossArgs& a, const float* theta, const float* u) {
    if (st != MF_OK) return;
    const int L = h->L, l = L - 1, din = h->dims[l], dout = h->dims[L];
    mf::HeadArgs ha;
    ha.rows = rows; ha.D = din; ha.C = dout; ha.dual = dual;
    ha.act = h->md.act;
    ha.A = at<T>(p.o_A[l]);
    ha.Ad = dual && l > 0 ? at<T>(p.o_Ad[l]) : nullptr;
    ha.lda = p.lda[l];
    ha.W = at<T>(p.o_Wb[l]); ha.U = at<T>(p.o_Ub[l]); ha.ldw = ld8(dout);
    ha.bias = h->md.has_bias ? theta + h->boff[l] : nullptr;
    ha.ubias = dual && h->md.has_bias ? u + h->boff[l] : nullptr;
    ha.loss = a;
    if (l > 0) {
      ha.Z = at<float>(p.o_Z[l - 1]);
      ha.Zd = dual ? at<float>(p.o_Zd[l - 1]) : nullptr;
      ha.ldz = din;
      ha.dz_prev = dz_buf(l - 1);
      ha.dzd_prev = dual ? at<T>(p.o_dZd[(l - 1) & 1]) : nullptr;
      ha.ld_prev = ld8(din);
    }
    const cudaError_t e = mf::head_fused<T>(ha, s);
    if (e != cudaSuccess) {
      st = MF_ERR_CUDA;
      h->err = std::string("fused head launch failed: ") + cudaGetErrorString(e);
      return;
    }
    launched();
  }

  // Backward pass.  Primal: out_g = grad L.  Dual: out_h = H u (and out_g = grad L if given).
  // Weight products write the weight and bias rows of theta's layout in one GEMM; the data
  // products fuse the activation backward (and its tangent) into the epilogue.
  void backward(int rows, bool dual, float* out_h, float* out_g) {
    const int hb = h->md.has_bias ? 1 : 0;
    const bool fused = fused_head();
    bool side_pending = false;   // a weight product on the side stream not joined yet
    for (int l = h->L - 1; l >= 0; --l) {
      const int din = h->dims[l], dout = h->dims[l + 1], b = l & 1;
      const bool head_seeds = fused && l == h->L - 1;
      // [a 1]^T dz and [a' 0]^T dz + [a 1]^T dz': activations [rows][din+1] and seeds
      // [rows][dout] are read MN-major (K = rows)
      GemmArgs g;
      g.M = din + hb; g.N = dout; g.K = rows;
      g.A0 = at<T>(p.o_A[l]); g.lda0 = p.lda[l];
      g.A1 = at<T>(p.o_Ad[l]); g.lda1 = p.lda[l];
      g.B0 = head_seeds ? at<T>(p.o_dZh) : dz_buf(l); g.ldb0 = ld8(dout);
      g.B1 = head_seeds ? at<T>(p.o_dZdh) : at<T>(p.o_dZd[b]); g.ldb1 = ld8(dout);
      g.a_mn = g.b_mn = true;
      if (!dual) {
        g.terms = mf::T_C0_A0B0;
        g.C0 = out_g + h->woff[l]; g.ldc0 = dout;
      } else if (out_g) {
        g.terms = mf::T_C0_A0B0 | mf::T_C1_A0B1 | (l > 0 ? mf::T_C1_A1B0 : 0u);
        g.C0 = out_g + h->woff[l]; g.ldc0 = dout;
        g.C1 = out_h + h->woff[l]; g.ldc1 = dout;
      } else {
        g.terms = mf::T_C0_A0B1 | (l > 0 ? mf::T_C0_A1B0 : 0u);
        g.C0 = out_h + h->woff[l]; g.ldc0 = dout;
      }
      const bool wgemm = dual || out_g;
      if (l == 0) {
        if (wgemm) gemm(g);
        upd_layer_after(0, s);
        break;
      }
      if (head_seeds) {
        // the fused head kernel has written layer l-1's seeds already, and this weight
        // product reads the head's own seed buffers, which nothing below overwrites: it runs
        // on the side stream next to the layers below, joined with their weight products
        if (wgemm && can_fork()) {
          fork();
          gemm(g, h->sstream);
          side_pending = true;
          upd_layer_after(l, h->sstream);
        } else {
          if (wgemm) gemm(g);
          upd_layer_after(l, s);
        }
        continue;
      }
      // data product: da = dz W^T ; da' = dz' W^T + dz U^T ; epilogue -> dz, dz' of layer l-1
      GemmArgs d;
      d.M = rows; d.N = din; d.K = dout;
      d.A0 = dz_buf(l); d.lda0 = ld8(dout);
      d.A1 = at<T>(p.o_dZd[b]); d.lda1 = ld8(dout);
      d.B0 = at<T>(p.o_Wb[l]); d.ldb0 = ld8(dout);
      d.B1 = at<T>(p.o_Ub[l]); d.ldb1 = ld8(dout);
      d.terms = dual ? (mf::T_C0_A0B0 | mf::T_C1_A1B0 | mf::T_C1_A0B1) : mf::T_C0_A0B0;
      d.epi.mode = mf::EPI_ACT_BWD;
      d.epi.act = h->md.act;
      d.epi.Z = at<float>(p.o_Z[l - 1]);
      d.epi.Zd = dual ? at<float>(p.o_Zd[l - 1]) : nullptr;
      d.epi.ldz = din;
      if (ror_store) { d.C0 = at<float>(p.o_SA[l]); d.ldc0 = din; }
      d.epi.A = dz_buf(l - 1);
      d.epi.Ad = dual ? at<T>(p.o_dZd[b ^ 1]) : nullptr;
      d.epi.lda = ld8(din);
      // The weight product reads layer l's seeds and writes its slice of the output; the
      // data product reads the same seeds and writes layer l-1's (the other ping-pong set):
      // they are independent and run side by side, joined before layer l-1 overwrites.
      if (wgemm && can_fork()) {
        fork();
        gemm(g, h->sstream);
        gemm(d);
        join();
        side_pending = false;
      } else {
        if (wgemm) gemm(g);
        gemm(d);
      }
      upd_layer_after(l, s);
    }
    if (side_pending) join();
    upd_join();
  }

  // Hessian-vector product by reverse-over-reverse (Algorithm 1's schedule): primal forward,
  // primal backward keeping every layer's dz and da (the reverse graph), then the adjoint of
  // the backward in forward layer order and the adjoint of the forward in reverse order.
  // Writes Hv, and per example l'_b (ld_out) and d eta (from the loss Hessian step).
  void ror_hvp(int rows, const void* x, const float* theta, const float* u, const void* y,
               const float* eta_w, const float* ex_w, float* Hv, float* grad, float* ld_out,
               float* d_eta) {
    const int L = h->L, hb = h->md.has_bias ? 1 : 0;
    no_fuse = true;
    forward(rows, x, theta, nullptr, false);
    ror_store = true;
    loss(rows, false, y, eta_w, ex_w, nullptr, nullptr, nullptr);
    backward(rows, false, nullptr, grad);
    ror_store = false;
    // adjoint of the backward pass, layers 0..L-1: dzbar_l = a_{l-1} V_l + c_l + dabar_{l-1} W_l
    for (int l = 0; l < L; ++l) {
      const int din = h->dims[l], dout = h->dims[l + 1];
      GemmArgs g;
      g.M = rows; g.N = dout; g.K = din;
      g.A0 = at<T>(p.o_A[l]); g.lda0 = p.lda[l];
      g.A1 = l == 0 ? nullptr : at<T>(p.o_DAB[l - 1]);
      g.lda1 = p.lda[l];
      g.B0 = at<T>(p.o_Wb[l]); g.ldb0 = ld8(dout);
      g.B1 = at<T>(p.o_Ub[l]); g.ldb1 = ld8(dout);
      g.b_mn = true;
      g.terms = mf::T_C0_A0B1 | (l > 0 ? mf::T_C0_A1B0 : 0u);
      g.C0 = at<float>(p.o_DZB); g.ldc0 = dout;
      g.bias0 = h->md.has_bias ? u + h->boff[l] : nullptr;
      gemm(g);
      if (l + 1 < L) {
        mf::ror_fwd_elem<T>(h->md.act, at<float>(p.o_DZB), at<float>(p.o_Z[l]),
                            at<float>(p.o_SA[l + 1]), rows, dout, at<T>(p.o_DAB[l]), p.lda[l + 1],
                            at<float>(p.o_ZP[l]), s);
        launched();
      } else {
        // loss Hessian along dzbar (this is the forward tangent of the logits): zbar_{L-1},
        // the per-example directional losses and the weight meta-gradient
        mf::LossArgs a;
        a.loss = loss_kind();
        a.chain = h->md.chain_steps;
        a.rows = rows; a.cols = dout;
        a.F = at<float>(p.o_Z[l]);
        a.Fd = at<float>(p.o_DZB);
        if (a.loss != 1) a.Yf = static_cast<const float*>(y);
        else a.Yi = static_cast<const int*>(y);
        a.eta_w = eta_w; a.ex_w = ex_w;
        a.inv_norm = 1.f / static_cast<float>(rows);
        a.ld = ld_out; a.d_eta = d_eta;
        a.dF = nullptr; a.dFd = at<T>(p.o_ZB);
        a.ldo = ld8(dout);
        a.status = h->d_status;
        if (a.loss == 2 && a.chain > 0) {   // adjoint of the chain's backward, from its tape
          a.tape = at<float>(p.o_CH);
          a.ror = 2;
        }
        mf::loss_seed<T>(a, s);
        launched();
      }
    }
    // adjoint of the forward pass, layers L-1..0
    for (int l = L - 1; l >= 0; --l) {
      const int din = h->dims[l], dout = h->dims[l + 1];
      if (l + 1 < L) {
        mf::ror_bwd_elem<T>(h->md.act, at<float>(p.o_ZP[l]), at<float>(p.o_AB), at<float>(p.o_Z[l]),
                            rows, dout, at<T>(p.o_ZB), ld8(dout), s);
        launched();
      }
      // (H v)_{W_l, b_l} = [a_{l-1}^T; 1] zbar_l + [dabar_{l-1}^T; 0] dz_l
      GemmArgs g;
      g.M = din + hb; g.N = dout; g.K = rows;
      g.A0 = at<T>(p.o_A[l]); g.lda0 = p.lda[l];
      g.A1 = l > 0 ? at<T>(p.o_DAB[l - 1]) : nullptr; g.lda1 = p.lda[l];
      g.B0 = at<T>(p.o_ZB); g.ldb0 = ld8(dout);
      g.B1 = at<T>(p.o_SZ[l]); g.ldb1 = ld8(dout);
      g.a_mn = g.b_mn = true;
      g.terms = mf::T_C0_A0B0 | (l > 0 ? mf::T_C0_A1B1 : 0u);
      g.C0 = Hv + h->woff[l]; g.ldc0 = dout;
      gemm(g);
      if (l == 0) break;
      // abar_{l-1} = zbar_l W_l^T + dz_l V_l^T
      GemmArgs d;
      d.M = rows; d.N = din; d.K = dout;
      d.A0 = at<T>(p.o_ZB); d.lda0 = ld8(dout);
      d.A1 = at<T>(p.o_SZ[l]); d.lda1 = ld8(dout);
      d.B0 = at<T>(p.o_Wb[l]); d.ldb0 = ld8(dout);
      d.B1 = at<T>(p.o_Ub[l]); d.ldb1 = ld8(dout);
      d.terms = mf::T_C0_A0B0 | mf::T_C0_A1B1;
      d.C0 = at<float>(p.o_AB); d.ldc0 = din;
      gemm(d);
    }
    no_fuse = false;
  }
};

#include "decoder_exec.cuh"

// Per-layer updates run inside the MLP executor's backward pass (Exec::upd_after); the
// decoder executor updates the whole vector after the pass.
template <typename X>
bool per_layer_updates(X&) { return false; }
template <typename X>
void set_upd_after(X&, const mf::LayerUpdArgs*) {}
template <typename T>
bool per_layer_updates(Exec<T>& ex) { return ex.layer_updates_ok(); }
template <typename T>
void set_upd_after(Exec<T>& ex, const mf::LayerUpdArgs* a) { ex.upd_after = a; }

mf_status validate_loop(mf_ctx* h, const mf_loop_desc* lp) {
  if (!lp) return fail(h, MF_ERR_INVALID_ARG, "loop descriptor is NULL");
  if (lp->T < 1 || lp->B < 1 || lp->B_outer < 1)
    return fail(h, MF_ERR_INVALID_ARG, "T, B and B_outer must be >= 1");
  if (lp->meta_kind & ~7) return fail(h, MF_ERR_INVALID_ARG, "unknown meta_kind bits");
  if ((lp->meta_kind & MF_META_PARAM_LOGLR) && (lp->meta_kind & MF_META_SCALAR_LOGLR))
    return fail(h, MF_ERR_INVALID_ARG, "PARAM_LOGLR and SCALAR_LOGLR are mutually exclusive");
  if (!(lp->momentum >= 0.f && lp->momentum < 1.f))
    return fail(h, MF_ERR_INVALID_ARG, "momentum must be in [0, 1)");
  if (lp->hvp_mode != MF_HVP_MIXED_FOR && lp->hvp_mode != MF_HVP_REV_REV)
    return fail(h, MF_ERR_INVALID_ARG, "unknown hvp_mode");

  if (lp->ckpt_every < 0) return fail(h, MF_ERR_INVALID_ARG, "ckpt_every must be >= 0");
  if (lp->ckpt_slots < 0 || lp->ckpt_slots > 1024)
    return fail(h, MF_ERR_INVALID_ARG, "ckpt_slots must be in 0..1024");
  if (lp->ckpt_slots > 0 && lp->ckpt_every > 1)
    return fail(h, MF_ERR_INVALID_ARG, "ckpt_slots and ckpt_every > 1 are exclusive");
  if (lp->ckpt_slots > 0 && lp->T > 4096)
    return fail(h, MF_ERR_INVALID_ARG, "binomial checkpointing takes T <= 4096");
  if (lp->optimizer != MF_OPTIM_SGD && lp->optimizer != MF_OPTIM_ADAM)
    return fail(h, MF_ERR_INVALID_ARG, "unknown optimizer");
  if (lp->optimizer == MF_OPTIM_ADAM &&
      (lp->momentum != 0.f || !(lp->beta1 >= 0.f && lp->beta1 < 1.f) ||
       !(lp->beta2 >= 0.f && lp->beta2 < 1.f) || !(lp->adam_eps > 0.f) ||
       !std::isfinite(lp->adam_eps)))
    return fail(h, MF_ERR_INVALID_ARG,
                "Adam needs momentum 0, beta1 and beta2 in [0, 1) and a finite adam_eps > 0");
  return MF_OK;
}

int64_t n_eta_of(const mf_ctx* h, const mf_loop_desc* lp) {
  int64_t n = 0;
  if (lp->meta_kind & MF_META_EXAMPLE_WEIGHTS) n += static_cast<int64_t>(lp->T) * lp->B;
  if (lp->meta_kind & MF_META_PARAM_LOGLR) n += h->P;
  if (lp->meta_kind & MF_META_SCALAR_LOGLR) n += 1;
  return n;
}

mf_status check_x(mf_ctx* h, const void* x, int rows) {
  if (!h->bf16 || h->decoder) return MF_OK;
  const int din = h->dims[0];
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (din % 8) != 0 ||
      ((static_cast<int64_t>(rows) * din * 2) % 16) != 0)
    return fail(h, MF_ERR_INVALID_ARG,
                "bf16 inputs must be 16-byte aligned with d_in a multiple of 8");
  return MF_OK;
}

size_t y_stride_bytes(const mf_ctx* h, int rows) {
  return h->md.loss == MF_LOSS_SOFTMAX_CE ? static_cast<size_t>(rows) * 4
                                          : static_cast<size_t>(rows) * h->dims[h->L] * 4;
}

// Checkpoint store of the sweep (Section 4; segment rematerialisation when k > 1).  theta_t
// lives in checkpoint slot t/k when t is a multiple of k, else in segment slot (t mod k) - 1;
// the segment slots hold one segment at a time and the sweep refills them from the segment's
// checkpoint.  m_t (t >= 1) is kept the same way, without a slot for m_0 = 0, when the sweep
// reads it (a log-learning-rate meta-parameter).  When only a recompute needs it (momentum
// with k > 1), the checkpoints keep it and one running slot carries it inside a segment.
struct Store {
  int k = 1, T = 0, n_ck = 1;
  bool m_kept = false, m_run_only = false;
  bool adam = false;   // Adam: v_t kept like m_t after the m slots, then m-bar and v-bar
  // Binomial schedule (ckpt_slots = s > 0): s + 3 state slots (S_0, s snapshots, two
  // scratch), each theta plus, when kept, m (and v with Adam); see revolve.h.
  int bin = 0;
  int theta_idx(int t) const { return t % k == 0 ? t / k : n_ck + t % k - 1; }
  int m_idx(int t) const {
    return t % k == 0 ? t / k - 1 : (m_run_only ? n_ck - 1 : n_ck - 1 + t % k - 1);
  }
  int theta_slots() const { return bin ? bin + 3 : n_ck + k - 1; }
  int m_slots() const {
    if (bin) return !m_kept ? 0 : adam ? 2 * (bin + 3) + 4 : bin + 3;
    const int nm = !m_kept ? 0 : m_run_only ? n_ck : n_ck - 1 + k - 1;
    return adam ? 2 * nm + 2 : nm;
  }
  int v_idx(int t) const { return n_ck - 1 + k - 1 + m_idx(t); }
  int mbar_idx() const { return 2 * (n_ck - 1 + k - 1); }
  // binomial slot j: m at m slot j, v at m slot n + j; then m-bar, v-bar and the two
  // buffers that keep m_{t+1}, v_{t+1} of a deferred Adam reverse step
  int bin_v(int j) const { return bin + 3 + j; }
  int bin_mbar() const { return 2 * (bin + 3); }
  int bin_pend() const { return 2 * (bin + 3) + 2; }
};

Store make_store(const mf_loop_desc* lp) {
  Store st;
  st.T = lp->T;
  if (lp->ckpt_slots > 0) {
    st.bin = std::min(lp->ckpt_slots, std::max(lp->T - 1, 1));
    st.adam = lp->optimizer == MF_OPTIM_ADAM;
    const bool lr_meta = lp->meta_kind & (MF_META_PARAM_LOGLR | MF_META_SCALAR_LOGLR);
    // recomputation restarts from snapshots, so every kept state carries its momentum
    st.m_kept = lr_meta || st.adam || lp->momentum != 0.f;
    return st;
  }
  st.k = lp->ckpt_every <= 1 ? 1 : std::min(lp->ckpt_every, lp->T);
  st.n_ck = lp->T / st.k + 1;
  const bool lr_meta = lp->meta_kind & (MF_META_PARAM_LOGLR | MF_META_SCALAR_LOGLR);
  st.adam = lp->optimizer == MF_OPTIM_ADAM;
  st.m_kept = lr_meta || st.adam || (lp->momentum != 0.f && st.k > 1);
  st.m_run_only = st.m_kept && !lr_meta && !st.adam;
  return st;
}

// Adam's hyper-parameters and the bias corrections of inner step j on an update.
void set_adam(mf::LayerUpdArgs& a, const mf_loop_desc* lp, int j) {
  a.adam = 1;
  a.b1 = lp->beta1;
  a.b2 = lp->beta2;
  a.eps = lp->adam_eps;
  a.c1 = static_cast<float>(1.0 - std::pow(static_cast<double>(lp->beta1), j + 1));
  a.c2 = static_cast<float>(1.0 - std::pow(static_cast<double>(lp->beta2), j + 1));
}

struct LrSel {
  mf::LrArgs lr;
  bool lr_meta = false;
  int64_t off_plr = -1, off_slr = -1;
};

LrSel lr_select(const mf_ctx* h, const mf_loop_desc* lp, const float* eta) {
  LrSel r;
  int64_t o = 0;
  if (lp->meta_kind & MF_META_EXAMPLE_WEIGHTS) o += static_cast<int64_t>(lp->T) * lp->B;
  r.lr.alpha = lp->alpha;
  if (lp->meta_kind & MF_META_PARAM_LOGLR) {
    r.off_plr = o;
    r.lr.plr = eta + o;
    r.lr_meta = true;
    o += h->P;
  }
  if (lp->meta_kind & MF_META_SCALAR_LOGLR) {
    r.off_slr = o;
    r.lr.slr = eta + o;
    r.lr_meta = true;
  }
  return r;
}

// One inner step (Eq. 2): forward, loss and backward at theta, then K4 writes theta' (and m'
// when m_out is set) and casts theta' into the GEMM operand copies.  m = null reads m_t = 0.
template <typename X>
void inner_step(X& ex, const mf_loop_desc* lp, const float* eta, const void* inner_x,
                const void* inner_y, const LrSel& lr, int t, const float* theta, const float* m,
                float* theta_out, float* m_out, const float* v = nullptr,
                float* v_out = nullptr) {
  mf_ctx* h = ex.h;
  const int B = lp->B;
  const void* x = static_cast<const char*>(inner_x) + ex.x_step_bytes(B) * t;
  const void* y = static_cast<const char*>(inner_y) + ex.y_step_bytes(B) * t;
  ex.forward(B, x, theta, nullptr, false);
  const float* ew = (lp->meta_kind & MF_META_EXAMPLE_WEIGHTS) ? eta + static_cast<int64_t>(t) * B : nullptr;
  ex.loss(B, false, y, ew, nullptr, nullptr, nullptr, nullptr);
  float* g = ex.g_buf();
  mf::LayerUpdArgs a;
  a.mode = mf::LU_ROLLOUT;
  a.theta = theta;
  a.m = m;
  a.g = g;
  a.theta_out = theta_out;
  a.m_out = m_out;
  a.mu = lp->momentum;
  a.lr = lr.lr;
  a.status = h->d_status;
  if (lp->optimizer == MF_OPTIM_ADAM) {
    set_adam(a, lp, t);
    a.v = v;
    a.v_out = v_out;
  }
  const bool per_layer = per_layer_updates(ex);
  if (per_layer) set_upd_after(ex, &a);
  ex.backward(B, false, nullptr, g);
  if (per_layer) set_upd_after(ex, nullptr);
  else ex.update(a);
}

// Inner rollout over steps [t0, t1) into the checkpoint store: theta_{t+1} (and m_{t+1} when
// kept) go to their slots.  Without kept momentum slots a running m lives in the u buffer
// (only on the first pass, before the sweep uses u).  Expects theta_{t0} cast already.
template <typename X>
void rollout_store(X& ex, const mf_loop_desc* lp, const Store& st, const float* eta,
                   const void* inner_x, const void* inner_y, const LrSel& lr, int t0, int t1) {
  float* m_run = (lp->momentum != 0.f && !st.m_kept) ? ex.u_buf() : nullptr;
  for (int t = t0; t < t1; ++t) {
    const float* m_in = m_run ? (t > t0 ? m_run : nullptr)
                              : (st.m_kept && t > 0 ? ex.m_slot(st.m_idx(t)) : nullptr);
    float* m_out = m_run ? m_run : (st.m_kept ? ex.m_slot(st.m_idx(t + 1)) : nullptr);
    const float* v_in = st.adam && t > 0 ? ex.m_slot(st.v_idx(t)) : nullptr;
    float* v_out = st.adam ? ex.m_slot(st.v_idx(t + 1)) : nullptr;
    inner_step(ex, lp, eta, inner_x, inner_y, lr, t, ex.theta_slot(st.theta_idx(t)), m_in,
               ex.theta_slot(st.theta_idx(t + 1)), m_out, v_in, v_out);
    if (ex.st != MF_OK) return;
  }
}

// Inner rollout without a store (mf_inner_rollout): two theta slots ping-pong; m runs in the
// u buffer, or in m slot 0 when the learning rate is a meta-parameter.
template <typename X>
void rollout_plain(X& ex, const mf_loop_desc* lp, const float* eta, const void* inner_x,
                   const void* inner_y, const LrSel& lr, float** theta_T) {
  const bool adam = lp->optimizer == MF_OPTIM_ADAM;
  float* m_run = adam || lr.lr_meta ? ex.m_slot(0) : lp->momentum != 0.f ? ex.u_buf() : nullptr;
  float* v_run = adam ? ex.m_slot(1) : nullptr;
  ex.cast_params(ex.theta_slot(0), false);
  for (int t = 0; t < lp->T; ++t) {
    inner_step(ex, lp, eta, inner_x, inner_y, lr, t, ex.theta_slot(t & 1),
               t > 0 ? m_run : nullptr, ex.theta_slot((t + 1) & 1), m_run,
               t > 0 ? v_run : nullptr, v_run);
    if (ex.st != MF_OK) return;
  }
  *theta_T = ex.theta_slot(lp->T & 1);
}

// Algorithm 2 once the workspace is in place: rollout, outer gradient (Eq. 4), then the
// reverse sweep t = T-1..0 with forward-over-reverse Hessian-vector products.
template <typename X>
mf_status meta_grad_run(X& ex, const mf_loop_desc* lp, const float* theta0, const float* eta,
                        const void* inner_x, const void* inner_y, const void* outer_x,
                        const void* outer_y, float* d_eta, float* d_theta0, float* outer_loss) {
  mf_ctx* h = ex.h;
  cudaStream_t s = ex.s;
  const int T = lp->T, B = lp->B, Bo = lp->B_outer;
  const LrSel lr = lr_select(h, lp, eta);
  const Store st = make_store(lp);
  const int k = st.k;
  auto theta_at = [&](int t) { return ex.theta_slot(st.theta_idx(t)); };
  auto m_at = [&](int t) { return ex.m_slot(st.m_idx(t)); };   // m_t, t >= 1
  const bool scalar_lr = lp->meta_kind & MF_META_SCALAR_LOGLR;
  MF_CUDA(h, cudaMemcpyAsync(theta_at(0), theta0, h->P * 4, cudaMemcpyDeviceToDevice, s));
  const int64_t ne = n_eta_of(h, lp);
  if (ne > 0) MF_CUDA(h, cudaMemsetAsync(d_eta, 0, ne * 4, s));
  ex.prepare();

  // 1. rollout into the checkpoint store; the last segment stays in the segment slots
  ex.cast_params(theta_at(0), false);
  rollout_store(ex, lp, st, eta, inner_x, inner_y, lr, 0, T);
  if (ex.st != MF_OK) return ex.st;
  float* thT = theta_at(T);

  // 2. outer gradient theta_bar_T = grad V(theta_T)  (Eq. 4); theta_T is already cast
  float* tbar = ex.tbar_buf();
  float* u = ex.u_buf();
  float* Hu = ex.g_buf();
  float* part = ex.part_buf();
  const int nb = ex.nb();
  ex.forward(Bo, outer_x, thT, nullptr, false);
  ex.loss(Bo, false, outer_y, nullptr, nullptr, ex.l_buf(), nullptr, nullptr);
  ex.backward(Bo, false, nullptr, tbar);
  if (outer_loss) {
    mf::sum_scaled(ex.l_buf(), Bo, 1.f / Bo, outer_loss, s);
    ex.launched();
  }
  float* d_plr = lr.off_plr >= 0 ? d_eta + lr.off_plr : nullptr;
  // Adam: reverse of inner step j from its stored outputs; u = g-bar_j, and the cotangents of
  // m_j, v_j replace those of m_{j+1}, v_{j+1} in place
  auto adam_pre = [&](mf::LayerUpdArgs& a, int j, bool bar_in) {
    set_adam(a, lp, j);
    a.adam_pre = true;
    a.bar_in = bar_in;
    a.m_adj = m_at(j + 1);
    a.v_adj = ex.m_slot(st.v_idx(j + 1));
    a.m_prev = j > 0 ? m_at(j) : nullptr;
    a.mbar = ex.m_slot(st.mbar_idx());
    a.vbar = ex.m_slot(st.mbar_idx() + 1);
    a.u_out = u;
  };
  // u_{T-1} = -lr theta_bar_T ;  d eta_lr += -lr m_T theta_bar_T ; cast theta_{T-1}, u_{T-1}
  // (Adam: u_{T-1} = g-bar_{T-1} from theta_bar_T and zero moment cotangents)
  {
    mf::LayerUpdArgs a;
    a.mode = mf::LU_ADJOINT;
    a.theta_bar = tbar;
    a.m_adj = lr.lr_meta ? m_at(T) : nullptr;
    a.u_out = u;
    if (st.adam) adam_pre(a, T - 1, false);
    a.d_plr = d_plr;
    a.partials = scalar_lr ? part + static_cast<int64_t>(T - 1) * nb : nullptr;
    a.cast_src = theta_at(T - 1);
    a.mu = lp->momentum;
    a.lr = lr.lr;
    a.status = h->d_status;
    ex.update(a);
  }

  // 3. reverse sweep
  const size_t xs = ex.x_step_bytes(B);
  const size_t ys = ex.y_step_bytes(B);
  const bool exw = lp->meta_kind & MF_META_EXAMPLE_WEIGHTS;
  bool adam_pending = false;   // Adam's reverse of step t waits for its segment's recompute
  for (int t = T - 1; t >= 0; --t) {
    // entering an earlier segment [t+1-k, t+1): rebuild theta and m of its steps from the
    // segment's checkpoint (the rollout's own kernels, so bit-identical); this leaves
    // theta_t cast for the forward below
    if (t + 1 < T && (t + 1) % k == 0 && k > 1) {
      const int a0 = t + 1 - k;
      ex.cast_params(theta_at(a0), false);
      rollout_store(ex, lp, st, eta, inner_x, inner_y, lr, a0, t);
      if (ex.st != MF_OK) return ex.st;
    }
    if (adam_pending) {
      mf::LayerUpdArgs a;
      a.mode = mf::LU_ADJOINT;
      a.theta_bar = tbar;
      adam_pre(a, t, true);
      a.d_plr = d_plr;
      a.partials = scalar_lr ? part + static_cast<int64_t>(t) * nb : nullptr;
      a.lr = lr.lr;
      a.status = h->d_status;
      ex.update(a);
      adam_pending = false;
    }
    const float* th = theta_at(t);
    const void* x = static_cast<const char*>(inner_x) + xs * t;
    const void* y = static_cast<const char*>(inner_y) + ys * t;
    const float* ew = exw ? eta + static_cast<int64_t>(t) * B : nullptr;
    float* de = exw ? d_eta + static_cast<int64_t>(t) * B : nullptr;
    // theta_bar_t = theta_bar_{t+1} + H u ; d eta_lr += -lr m_t theta_bar_t ;
    // u_{t-1} = mu u_t - lr theta_bar_t ; cast theta_{t-1}, u_{t-1}
    mf::LayerUpdArgs a;
    a.mode = mf::LU_ADJOINT;
    a.theta_bar = tbar;
    a.Hu = Hu;
    const bool in_store = t % k != 0 || k == 1;   // theta_{t-1}, m_{t-1} in the store now
    if (t > 0 && st.adam && !in_store) {
      a.adam = 1;            // theta_bar only; the reverse of step t-1 follows the recompute
      adam_pending = true;
    } else if (t > 0) {
      a.m_adj = lr.lr_meta ? m_at(t) : nullptr;
      a.u_in = u;
      a.u_out = u;
      if (st.adam) adam_pre(a, t - 1, true);
      a.d_plr = d_plr;
      a.partials = scalar_lr ? part + static_cast<int64_t>(t - 1) * nb : nullptr;
      // theta_{t-1} is in the store only within this segment or at a checkpoint; otherwise
      // the recompute of its segment casts it
      if (in_store) a.cast_src = theta_at(t - 1);
    }
    a.mu = lp->momentum;
    a.lr = lr.lr;
    a.status = h->d_status;
    // H u at theta_t; with per-layer updates the backward pass runs the update above layer by
    // layer, else it runs once over the whole vector afterwards
    const bool per_layer = lp->hvp_mode != MF_HVP_REV_REV && per_layer_updates(ex);
    if (lp->hvp_mode == MF_HVP_REV_REV) {
      ex.ror_hvp(B, x, th, u, y, ew, nullptr, Hu, nullptr, ex.ld_buf(), de);
    } else {
      ex.forward(B, x, th, u, true);
      ex.loss(B, true, y, ew, nullptr, nullptr, ex.ld_buf(), de);
      if (per_layer) set_upd_after(ex, &a);
      ex.backward(B, true, Hu, nullptr);
      if (per_layer) set_upd_after(ex, nullptr);
    }
    if (!per_layer) ex.update(a);
    if (ex.st != MF_OK) return ex.st;
  }
  if (scalar_lr) {
    mf::sum_scaled(part, T * nb, 1.f, d_eta + lr.off_slr, s);
    ex.launched();
  }
  if (d_theta0) MF_CUDA(h, cudaMemcpyAsync(d_theta0, tbar, h->P * 4, cudaMemcpyDeviceToDevice, s));
  MF_CUDA(h, cudaGetLastError());
  return ex.st;
}

// ---- binomial checkpointing (ckpt_slots > 0; the schedule of revolve.h) ------------------
// State slot j: theta in theta slot j; m (when kept) in m slot j, v (Adam) in m slot n + j.
struct BinSlots {
  const Store* st;
  template <typename X> float* theta(X& ex, int j) const { return ex.theta_slot(j); }
  template <typename X> float* m(X& ex, int j) const { return st->m_kept ? ex.m_slot(j) : nullptr; }
  template <typename X> float* v(X& ex, int j) const { return st->adam ? ex.m_slot(st->bin_v(j)) : nullptr; }
};

// S_t0 in slot src -> S_t1 in slot dst by inner steps t0..t1-1.  The intermediate states
// alternate between dst and the scratch slot that is not dst, so that the last lands in dst;
// src is never written.  Each step casts the parameters it produces, so theta_t1 is cast at
// the end.
template <typename X>
void bin_advance(X& ex, const mf_loop_desc* lp, const mf::RevolveSchedule& rs, const BinSlots& sl,
                 const float* eta, const void* inner_x, const void* inner_y, const LrSel& lr,
                 int t0, int t1, int src, int dst) {
  const int other = dst == rs.scratch(0) ? rs.scratch(1) : rs.scratch(0);
  ex.cast_params(sl.theta(ex, src), false);
  int cur = src;
  const int n = t1 - t0;
  for (int k = 0; k < n && ex.st == MF_OK; ++k) {
    const int t = t0 + k;
    const int out = (n - 1 - k) % 2 == 0 ? dst : other;
    inner_step(ex, lp, eta, inner_x, inner_y, lr, t, sl.theta(ex, cur),
               t > 0 ? sl.m(ex, cur) : nullptr, sl.theta(ex, out), sl.m(ex, out),
               t > 0 ? sl.v(ex, cur) : nullptr, sl.v(ex, out));
    cur = out;
  }
}

// Algorithm 2 with the binomial store: the rollout leaves the schedule's snapshots on its
// way and S_T in a scratch slot; the sweep runs the schedule's actions, recomputing states
// before it reverses them.  The reverse step itself is meta_grad_run's.  The cast of
// theta_{t-1} (and, with Adam, the reverse of step t-1's moments) fuses into step t's update
// only when S_{t-1} sits in a slot and the next action reverses it; otherwise the recompute
// casts theta_{t-1}, and Adam's reverse of step t-1 waits for it, with m_t and v_t copied
// aside because the recompute may overwrite their slot.
template <typename X>
mf_status meta_grad_run_binomial(X& ex, const mf_loop_desc* lp, const float* theta0,
                                 const float* eta, const void* inner_x, const void* inner_y,
                                 const void* outer_x, const void* outer_y, float* d_eta,
                                 float* d_theta0, float* outer_loss) {
  mf_ctx* h = ex.h;
  cudaStream_t s = ex.s;
  const int T = lp->T, B = lp->B, Bo = lp->B_outer;
  const LrSel lr = lr_select(h, lp, eta);
  const Store st = make_store(lp);
  const BinSlots sl{&st};
  const mf::RevolveSchedule rs = mf::revolve_schedule(T, st.bin);
  const bool scalar_lr = lp->meta_kind & MF_META_SCALAR_LOGLR;
  MF_CUDA(h, cudaMemcpyAsync(sl.theta(ex, 0), theta0, h->P * 4, cudaMemcpyDeviceToDevice, s));
  const int64_t ne = n_eta_of(h, lp);
  if (ne > 0) MF_CUDA(h, cudaMemsetAsync(d_eta, 0, ne * 4, s));
  ex.prepare();

  // 1. rollout S_0 -> S_T, leaving S_t in slot keep[t] for the schedule's snapshots
  {
    int cur = 0, tc = 0;
    for (int t = 1; t < T && ex.st == MF_OK; ++t) {
      if (rs.keep[t] < 0) continue;
      bin_advance(ex, lp, rs, sl, eta, inner_x, inner_y, lr, tc, t, cur, rs.keep[t]);
      cur = rs.keep[t];
      tc = t;
    }
    if (ex.st == MF_OK)
      bin_advance(ex, lp, rs, sl, eta, inner_x, inner_y, lr, tc, T, cur, rs.slot_T);
  }
  if (ex.st != MF_OK) return ex.st;
  const int sT = rs.slot_T;

  // 2. outer gradient at theta_T (cast by the rollout's last step)
  float* tbar = ex.tbar_buf();
  float* u = ex.u_buf();
  float* Hu = ex.g_buf();
  float* part = ex.part_buf();
  const int nb = ex.nb();
  ex.forward(Bo, outer_x, sl.theta(ex, sT), nullptr, false);
  ex.loss(Bo, false, outer_y, nullptr, nullptr, ex.l_buf(), nullptr, nullptr);
  ex.backward(Bo, false, nullptr, tbar);
  if (outer_loss) {
    mf::sum_scaled(ex.l_buf(), Bo, 1.f / Bo, outer_loss, s);
    ex.launched();
  }
  float* d_plr = lr.off_plr >= 0 ? d_eta + lr.off_plr : nullptr;
  float* pend_m = st.adam ? ex.m_slot(st.bin_pend()) : nullptr;
  float* pend_v = st.adam ? ex.m_slot(st.bin_pend() + 1) : nullptr;
  // Adam's reverse of inner step j: m_{j+1}, v_{j+1} from (mj1, vj1), m_j from slot prev
  auto adam_pre = [&](mf::LayerUpdArgs& a, int j, bool bar_in, float* mj1, float* vj1,
                      int prev) {
    set_adam(a, lp, j);
    a.adam_pre = true;
    a.bar_in = bar_in;
    a.m_adj = mj1;
    a.v_adj = vj1;
    a.m_prev = j > 0 ? sl.m(ex, prev) : nullptr;
    a.mbar = ex.m_slot(st.bin_mbar());
    a.vbar = ex.m_slot(st.bin_mbar() + 1);
    a.u_out = u;
  };
  size_t ai = 0;    // next action of the schedule
  // slot of S_{t-1} if the next action reverses step t-1 at once, else -1
  auto next_rev = [&](int t) {
    return ai < rs.acts.size() && rs.acts[ai].kind == mf::RevolveAct::REV &&
                   rs.acts[ai].t0 == t - 1
               ? rs.acts[ai].src
               : -1;
  };
  bool adam_pending = false, pend_bar_in = false;
  auto defer_adam = [&](int slot, bool bar_in) {
    MF_CUDA(h, cudaMemcpyAsync(pend_m, sl.m(ex, slot), h->P * 4, cudaMemcpyDeviceToDevice, s));
    MF_CUDA(h, cudaMemcpyAsync(pend_v, sl.v(ex, slot), h->P * 4, cudaMemcpyDeviceToDevice, s));
    adam_pending = true;
    pend_bar_in = bar_in;
    return MF_OK;
  };
  // u_{T-1} = -lr theta_bar_T ; d eta_lr += -lr m_T theta_bar_T ; cast theta_{T-1}, u_{T-1}
  {
    const int prev = next_rev(T);
    if (st.adam && prev < 0) {
      const mf_status e = defer_adam(sT, false);
      if (e != MF_OK) return e;
    } else {
      mf::LayerUpdArgs a;
      a.mode = mf::LU_ADJOINT;
      a.theta_bar = tbar;
      a.m_adj = lr.lr_meta ? sl.m(ex, sT) : nullptr;
      a.u_out = u;
      if (st.adam) adam_pre(a, T - 1, false, sl.m(ex, sT), sl.v(ex, sT), prev);
      a.d_plr = d_plr;
      a.partials = scalar_lr ? part + static_cast<int64_t>(T - 1) * nb : nullptr;
      a.cast_src = prev >= 0 ? sl.theta(ex, prev) : nullptr;
      a.mu = lp->momentum;
      a.lr = lr.lr;
      a.status = h->d_status;
      ex.update(a);
    }
  }

  // 3. reverse sweep along the schedule
  const size_t xs = ex.x_step_bytes(B);
  const size_t ys = ex.y_step_bytes(B);
  const bool exw = lp->meta_kind & MF_META_EXAMPLE_WEIGHTS;
  for (int t = T - 1; t >= 0; --t) {
    while (ai < rs.acts.size() && rs.acts[ai].kind == mf::RevolveAct::ADV) {
      const mf::RevolveAct& c = rs.acts[ai++];
      bin_advance(ex, lp, rs, sl, eta, inner_x, inner_y, lr, c.t0, c.t1, c.src, c.dst);
      if (ex.st != MF_OK) return ex.st;
    }
    if (ai >= rs.acts.size() || rs.acts[ai].kind != mf::RevolveAct::REV || rs.acts[ai].t0 != t)
      return fail(h, MF_ERR_CUDA, "binomial schedule out of order");
    const int cs = rs.acts[ai++].src;      // slot of S_t
    if (adam_pending) {   // the reverse of step t's moments, now that m_t is in slot cs
      mf::LayerUpdArgs a;
      a.mode = mf::LU_ADJOINT;
      a.theta_bar = tbar;
      adam_pre(a, t, pend_bar_in, pend_m, pend_v, cs);
      a.d_plr = d_plr;
      a.partials = scalar_lr ? part + static_cast<int64_t>(t) * nb : nullptr;
      a.lr = lr.lr;
      a.status = h->d_status;
      ex.update(a);
      adam_pending = false;
    }
    const float* th = sl.theta(ex, cs);
    const void* x = static_cast<const char*>(inner_x) + xs * t;
    const void* y = static_cast<const char*>(inner_y) + ys * t;
    const float* ew = exw ? eta + static_cast<int64_t>(t) * B : nullptr;
    float* de = exw ? d_eta + static_cast<int64_t>(t) * B : nullptr;
    // theta_bar_t = theta_bar_{t+1} + H u ; d eta_lr += -lr m_t theta_bar_t ;
    // u_{t-1} = mu u_t - lr theta_bar_t ; cast theta_{t-1} (when in a slot), u_{t-1}
    mf::LayerUpdArgs a;
    a.mode = mf::LU_ADJOINT;
    a.theta_bar = tbar;
    a.Hu = Hu;
    const int prev = t > 0 ? next_rev(t) : -1;
    bool defer = false;
    if (t > 0 && st.adam && prev < 0) {
      a.adam = 1;            // theta_bar only; the reverse of step t-1 follows the recompute
      defer = true;
    } else if (t > 0) {
      a.m_adj = lr.lr_meta ? sl.m(ex, cs) : nullptr;
      a.u_in = u;
      a.u_out = u;
      if (st.adam) adam_pre(a, t - 1, true, sl.m(ex, cs), sl.v(ex, cs), prev);
      a.d_plr = d_plr;
      a.partials = scalar_lr ? part + static_cast<int64_t>(t - 1) * nb : nullptr;
      if (prev >= 0) a.cast_src = sl.theta(ex, prev);
    }
    a.mu = lp->momentum;
    a.lr = lr.lr;
    a.status = h->d_status;
    const bool per_layer = lp->hvp_mode != MF_HVP_REV_REV && per_layer_updates(ex);
    if (lp->hvp_mode == MF_HVP_REV_REV) {
      ex.ror_hvp(B, x, th, u, y, ew, nullptr, Hu, nullptr, ex.ld_buf(), de);
    } else {
      ex.forward(B, x, th, u, true);
      ex.loss(B, true, y, ew, nullptr, nullptr, ex.ld_buf(), de);
      if (per_layer) set_upd_after(ex, &a);
      ex.backward(B, true, Hu, nullptr);
      if (per_layer) set_upd_after(ex, nullptr);
    }
    if (!per_layer) ex.update(a);
    if (ex.st != MF_OK) return ex.st;
    if (defer) {
      const mf_status e = defer_adam(cs, true);
      if (e != MF_OK) return e;
    }
  }
  if (scalar_lr) {
    mf::sum_scaled(part, T * nb, 1.f, d_eta + lr.off_slr, s);
    ex.launched();
  }
  if (d_theta0) MF_CUDA(h, cudaMemcpyAsync(d_theta0, tbar, h->P * 4, cudaMemcpyDeviceToDevice, s));
  MF_CUDA(h, cudaGetLastError());
  return ex.st;
}

template <typename X>
mf_status rollout_run(X& ex, const mf_loop_desc* lp, const float* theta0, const float* eta,
                      const void* inner_x, const void* inner_y, float* thetaT) {
  mf_ctx* h = ex.h;
  const LrSel lr = lr_select(h, lp, eta);
  MF_CUDA(h, cudaMemcpyAsync(ex.theta_slot(0), theta0, h->P * 4, cudaMemcpyDeviceToDevice, ex.s));
  ex.prepare();
  float* thT = nullptr;
  rollout_plain(ex, lp, eta, inner_x, inner_y, lr, &thT);
  if (ex.st != MF_OK) return ex.st;
  MF_CUDA(h, cudaMemcpyAsync(thetaT, thT, h->P * 4, cudaMemcpyDeviceToDevice, ex.s));
  return MF_OK;
}

template <typename X>
mf_status hvp_run(X& ex, int B, const float* theta, const void* x, const void* y,
                  const float* ex_w, const float* v, float* Hv, float* tl, float* grad,
                  bool ror) {
  mf_ctx* h = ex.h;
  ex.prepare();
  ex.cast_params(theta, false);
  ex.cast_params(v, true);
  if (ror) {
    ex.ror_hvp(B, x, theta, v, y, nullptr, ex_w, Hv, grad, tl, nullptr);
  } else {
    ex.forward(B, x, theta, v, true);
    ex.loss(B, true, y, nullptr, ex_w, nullptr, tl, nullptr);
    ex.backward(B, true, Hv, grad);
  }
  MF_CUDA(h, cudaGetLastError());
  return ex.st;
}

// Plan the workspace for the handle's model, allocate it, and run f(executor).
template <typename E, typename F>
mf_status with_exec(mf_ctx* h, int rows, int T, int theta_slots, int m_slots, bool partials,
                    bool ror, cudaStream_t s, F&& f) {
  if (h->decoder) {
    DecPlan plan = make_dec_plan(h, h->Ly, rows, T, theta_slots, m_slots, partials, ror);
    mf_status st = ensure_ws(h, plan.bytes, s);
    if (st != MF_OK) return st;
    DecExec<E> ex(h, plan, h->Ly, s);
    return f(ex);
  }
  Plan plan = make_plan(h, rows, T, theta_slots, m_slots, partials, ror);
  mf_status st = ensure_ws(h, plan.bytes, s);
  if (st != MF_OK) return st;
  Exec<E> ex(h, plan, s);
  return f(ex);
}

template <typename E>
mf_status meta_grad_impl(mf_ctx* h, const mf_loop_desc* lp, const float* theta0,
                         const float* eta, const void* inner_x, const void* inner_y,
                         const void* outer_x, const void* outer_y, float* d_eta,
                         float* d_theta0, float* outer_loss, cudaStream_t s) {
  const Store store = make_store(lp);
  return with_exec<E>(h, std::max(lp->B, lp->B_outer), lp->T, store.theta_slots(),
                      store.m_slots(), lp->meta_kind & MF_META_SCALAR_LOGLR,
                      lp->hvp_mode == MF_HVP_REV_REV, s,
                      [&](auto& ex) {
                        if (store.bin)
                          return meta_grad_run_binomial(ex, lp, theta0, eta, inner_x, inner_y,
                                                        outer_x, outer_y, d_eta, d_theta0,
                                                        outer_loss);
                        return meta_grad_run(ex, lp, theta0, eta, inner_x, inner_y, outer_x,
                                             outer_y, d_eta, d_theta0, outer_loss);
                      });
}

template <typename E>
mf_status rollout_impl(mf_ctx* h, const mf_loop_desc* lp, const float* theta0, const float* eta,
                       const void* inner_x, const void* inner_y, float* thetaT, cudaStream_t s) {
  const bool lr_meta = lp->meta_kind & (MF_META_PARAM_LOGLR | MF_META_SCALAR_LOGLR);
  const int m_slots = lp->optimizer == MF_OPTIM_ADAM ? 2 : lr_meta ? 1 : 0;
  return with_exec<E>(h, lp->B, lp->T, 2, m_slots, false, false, s, [&](auto& ex) {
    return rollout_run(ex, lp, theta0, eta, inner_x, inner_y, thetaT);
  });
}

template <typename E>
mf_status hvp_impl(mf_ctx* h, int B, const float* theta, const void* x, const void* y,
                   const float* ex_w, const float* v, float* Hv, float* tl, float* grad,
                   bool ror, cudaStream_t s) {
  return with_exec<E>(h, B, 1, 0, 0, false, ror, s, [&](auto& ex) {
    return hvp_run(ex, B, theta, x, y, ex_w, v, Hv, tl, grad, ror);
  });
}

void destroy_handle_objects(mf_ctx* h) {
  if (h->d_status) cudaFree(h->d_status);
  if (h->gstream) cudaStreamDestroy(h->gstream);
  if (h->sstream) cudaStreamDestroy(h->sstream);
  if (h->ustream) cudaStreamDestroy(h->ustream);
  for (cudaEvent_t e : {h->ev_in, h->ev_out, h->ev_fork, h->ev_join, h->ev_u_in, h->ev_u_out,
                        h->ev_w[0], h->ev_w[1], h->ev_w[2], h->ev_w[3]})
    if (e) cudaEventDestroy(e);
  for (cudaEvent_t& e : h->ev_w) e = nullptr;
  h->d_status = nullptr;
  h->gstream = h->sstream = h->ustream = nullptr;
  h->ev_in = h->ev_out = h->ev_fork = h->ev_join = h->ev_u_in = h->ev_u_out = nullptr;
}

}  // namespace

// ======================================= C ABI ============================================
extern "C" {

const char* mf_status_string(mf_status s) {
  switch (s) {
    case MF_OK: return "ok";
    case MF_ERR_INVALID_ARG: return "invalid argument";
    case MF_ERR_UNSUPPORTED: return "unsupported";
    case MF_ERR_OOM: return "out of memory";
    case MF_ERR_CUDA: return "CUDA error";
    case MF_ERR_NONFINITE: return "non-finite value";
    case MF_ERR_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

const char* mf_last_error(mf_handle h) { return h ? h->err.c_str() : "NULL handle"; }

mf_status mf_create(const mf_model_desc* d, mf_handle* out) {
  if (!d || !out) return MF_ERR_INVALID_ARG;
  *out = nullptr;
  if (d->precision != MF_PREC_FP32 && d->precision != MF_PREC_BF16) return MF_ERR_INVALID_ARG;
  const bool decoder = d->arch == MF_ARCH_DECODER;
  if (decoder) {
    if (d->loss != MF_LOSS_NEXT_TOKEN_CE || d->n_layers < 1 || d->n_layers > 30 ||
        d->d_model < 8 || d->n_heads < 1 || d->d_model % d->n_heads != 0 ||
        (d->d_model / d->n_heads) % 8 != 0 || d->d_ff < 8 || d->d_ff % 8 != 0 ||
        d->d_model % 8 != 0 || d->vocab < 2 || d->vocab % 8 != 0 || d->seq_len < 8 ||
        d->seq_len % 8 != 0)
      return MF_ERR_INVALID_ARG;
  } else {
    if (d->arch != MF_ARCH_MLP) return MF_ERR_INVALID_ARG;
    if (d->n_layers < 1 || d->n_layers > MF_MAX_LAYERS) return MF_ERR_INVALID_ARG;
    for (int i = 0; i <= d->n_layers; ++i)
      if (d->dims[i] < 1 || d->dims[i] > (1 << 20)) return MF_ERR_INVALID_ARG;
    if (d->act < MF_ACT_IDENT || d->act > MF_ACT_SILU) return MF_ERR_INVALID_ARG;
    if (d->loss != MF_LOSS_SQUARED && d->loss != MF_LOSS_SOFTMAX_CE && d->loss != MF_LOSS_CHAIN_MSE)
      return MF_ERR_INVALID_ARG;
    if (d->loss == MF_LOSS_CHAIN_MSE && (d->chain_steps < 0 || d->chain_steps > 4096))
      return MF_ERR_INVALID_ARG;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return MF_ERR_CUDA; }
  mf_ctx* h = new mf_ctx();
  h->md = *d;
  h->decoder = decoder;
  if (decoder) {
    h->Ly = dec_layout(*d);
    h->P = dec_param_count(h->Ly);
    h->bf16 = d->precision == MF_PREC_BF16;
    h->dims.assign(1, d->d_model);
    h->maxd = d->d_model;
  }
  h->L = decoder ? 0 : d->n_layers;
  if (!decoder) h->dims.assign(d->dims, d->dims + d->n_layers + 1);
  int64_t o = 0;
  for (int l = 0; l < h->L; ++l) {
    h->woff.push_back(o);
    o += static_cast<int64_t>(h->dims[l]) * h->dims[l + 1];
    h->boff.push_back(d->has_bias ? o : -1);
    if (d->has_bias) o += h->dims[l + 1];
  }
  if (!decoder) {
    h->P = o;
    h->maxd = *std::max_element(h->dims.begin(), h->dims.end());
    h->bf16 = d->precision == MF_PREC_BF16;
  }
  if (cudaMalloc(&h->d_status, sizeof(int)) != cudaSuccess ||
      cudaMemset(h->d_status, 0, sizeof(int)) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->gstream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_in, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_out, cudaEventDisableTiming) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->sstream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->ustream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_u_in, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_u_out, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_w[0], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_w[1], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_w[2], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_w[3], cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    destroy_handle_objects(h);
    delete h;
    return MF_ERR_CUDA;
  }
  *out = h;
  return MF_OK;
}

mf_status mf_destroy(mf_handle h) {
  if (!h) return MF_ERR_INVALID_ARG;
  cudaDeviceSynchronize();
  release_ws(h);
  for (auto& e : h->evs) { cudaEventDestroy(e.first); cudaEventDestroy(e.second); }
  drop_graphs(h);
  destroy_handle_objects(h);
  delete h;
  return MF_OK;
}

mf_status mf_set_allocator(mf_handle h, void* (*alloc)(size_t, void*, void*),
                           void (*free_fn)(void*, size_t, void*, void*), void* ctx) {
  if (!h) return MF_ERR_INVALID_ARG;
  if ((alloc == nullptr) != (free_fn == nullptr))
    return fail(h, MF_ERR_INVALID_ARG, "alloc and free must both be set or both NULL");
  release_ws(h);
  h->ualloc = alloc;
  h->ufree = free_fn;
  h->uctx = ctx;
  return MF_OK;
}

mf_status mf_param_count(mf_handle h, const mf_loop_desc* lp, int64_t* n_params, int64_t* n_eta) {
  if (!h) return MF_ERR_INVALID_ARG;
  if (n_params) *n_params = h->P;
  if (n_eta) *n_eta = lp ? n_eta_of(h, lp) : 0;
  return MF_OK;
}

mf_status mf_workspace_bytes(mf_handle h, const mf_loop_desc* lp, size_t* bytes) {
  if (!h || !bytes) return MF_ERR_INVALID_ARG;
  mf_status st = validate_loop(h, lp);
  if (st != MF_OK) return st;
  const Store store = make_store(lp);
  if (h->decoder) {
    *bytes = make_dec_plan(h, h->Ly, std::max(lp->B, lp->B_outer), lp->T, store.theta_slots(),
                           store.m_slots(), lp->meta_kind & MF_META_SCALAR_LOGLR,
                           lp->hvp_mode == MF_HVP_REV_REV).bytes;
    return MF_OK;
  }
  *bytes = make_plan(h, std::max(lp->B, lp->B_outer), lp->T, store.theta_slots(),
                     store.m_slots(), lp->meta_kind & MF_META_SCALAR_LOGLR,
                     lp->hvp_mode == MF_HVP_REV_REV).bytes;
  return MF_OK;
}

mf_status mf_checkpoint_plan(int T, int ckpt_every, int ckpt_slots, int* state_slots,
                             int64_t* recompute_steps) {
  if (T < 1 || ckpt_every < 0 || ckpt_slots < 0 || ckpt_slots > 1024 ||
      (ckpt_slots > 0 && (ckpt_every > 1 || T > 4096)))
    return MF_ERR_INVALID_ARG;
  mf_loop_desc lp;
  memset(&lp, 0, sizeof(lp));
  lp.T = T;
  lp.ckpt_every = ckpt_every;
  lp.ckpt_slots = ckpt_slots;
  const Store st = make_store(&lp);
  int64_t re = 0;
  if (st.bin) {
    re = mf::revolve_recompute_steps(mf::revolve_schedule(T, st.bin));
  } else if (st.k > 1) {
    // every segment but the last is re-run from its checkpoint: k - 1 steps each
    re = static_cast<int64_t>((T - 1) / st.k) * (st.k - 1);
  }
  if (state_slots) *state_slots = st.theta_slots();
  if (recompute_steps) *recompute_steps = re;
  return MF_OK;
}

mf_status mf_release_workspace(mf_handle h) {
  if (!h) return MF_ERR_INVALID_ARG;
  release_ws(h);
  return MF_OK;
}

mf_status mf_inner_rollout(mf_handle h, const mf_loop_desc* lp, const float* theta0,
                           const float* eta, const void* inner_x, const void* inner_y,
                           float* thetaT, void* stream) {
  if (!h) return MF_ERR_INVALID_ARG;
  mf_status st = validate_loop(h, lp);
  if (st != MF_OK) return st;
  if (!theta0 || !inner_x || !inner_y || !thetaT || (n_eta_of(h, lp) > 0 && !eta))
    return fail(h, MF_ERR_INVALID_ARG, "NULL tensor argument");
  if ((st = check_x(h, inner_x, lp->B)) != MF_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  h->last_stream = s;
  uint64_t key = 0x726f6c6cULL;
  for (uint64_t v : {static_cast<uint64_t>(lp->T), static_cast<uint64_t>(lp->B),
                     static_cast<uint64_t>(lp->meta_kind),
                     static_cast<uint64_t>(float_bits(lp->alpha)),
                     static_cast<uint64_t>(float_bits(lp->momentum)),
                     static_cast<uint64_t>(lp->optimizer),
                     static_cast<uint64_t>(float_bits(lp->beta1)),
                     static_cast<uint64_t>(float_bits(lp->beta2)),
                     static_cast<uint64_t>(float_bits(lp->adam_eps)),
                     reinterpret_cast<uint64_t>(theta0), reinterpret_cast<uint64_t>(eta),
                     reinterpret_cast<uint64_t>(inner_x), reinterpret_cast<uint64_t>(inner_y),
                     reinterpret_cast<uint64_t>(thetaT)})
    key = mix_key(key, v);
  return run_graphed(h, h->g_roll, key, s, [&](cudaStream_t st) {
    return h->bf16 ? rollout_impl<__nv_bfloat16>(h, lp, theta0, eta, inner_x, inner_y, thetaT, st)
                   : rollout_impl<float>(h, lp, theta0, eta, inner_x, inner_y, thetaT, st);
  });
}

mf_status mf_hvp(mf_handle h, int B, const float* theta, const void* x, const void* y,
                 const float* ex_w, const float* v, float* Hv, float* tangent_losses, float* grad,
                 int hvp_mode, void* stream) {
  if (!h) return MF_ERR_INVALID_ARG;
  if (B < 1) return fail(h, MF_ERR_INVALID_ARG, "B must be >= 1");
  if (hvp_mode != MF_HVP_MIXED_FOR && hvp_mode != MF_HVP_REV_REV)
    return fail(h, MF_ERR_INVALID_ARG, "unknown hvp_mode");

  const bool ror = hvp_mode == MF_HVP_REV_REV;
  if (!theta || !x || !y || !v || !Hv) return fail(h, MF_ERR_INVALID_ARG, "NULL tensor argument");
  mf_status st = check_x(h, x, B);
  if (st != MF_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  h->last_stream = s;
  uint64_t key = 0x687670ULL;
  for (uint64_t v2 : {static_cast<uint64_t>(B), static_cast<uint64_t>(hvp_mode),
                      reinterpret_cast<uint64_t>(theta),
                      reinterpret_cast<uint64_t>(x), reinterpret_cast<uint64_t>(y),
                      reinterpret_cast<uint64_t>(ex_w), reinterpret_cast<uint64_t>(v),
                      reinterpret_cast<uint64_t>(Hv), reinterpret_cast<uint64_t>(tangent_losses),
                      reinterpret_cast<uint64_t>(grad)})
    key = mix_key(key, v2);
  return run_graphed(h, h->g_hvp, key, s, [&](cudaStream_t st) {
    return h->bf16 ? hvp_impl<__nv_bfloat16>(h, B, theta, x, y, ex_w, v, Hv, tangent_losses, grad, ror, st)
                   : hvp_impl<float>(h, B, theta, x, y, ex_w, v, Hv, tangent_losses, grad, ror, st);
  });
}

mf_status mf_meta_grad(mf_handle h, const mf_loop_desc* lp, const float* theta0, const float* eta,
                       const void* inner_x, const void* inner_y, const void* outer_x,
                       const void* outer_y, float* d_eta, float* d_theta0, float* outer_loss,
                       void* stream) {
  if (!h) return MF_ERR_INVALID_ARG;
  mf_status st = validate_loop(h, lp);
  if (st != MF_OK) return st;
  if (!theta0 || !inner_x || !inner_y || !outer_x || !outer_y)
    return fail(h, MF_ERR_INVALID_ARG, "NULL tensor argument");
  if (n_eta_of(h, lp) > 0 && (!eta || !d_eta))
    return fail(h, MF_ERR_INVALID_ARG, "eta and d_eta are required when meta_kind != 0");
  if (n_eta_of(h, lp) == 0 && !d_theta0)
    return fail(h, MF_ERR_INVALID_ARG, "nothing to compute: meta_kind = 0 and d_theta0 = NULL");
  if ((st = check_x(h, inner_x, lp->B)) != MF_OK) return st;
  if ((st = check_x(h, outer_x, lp->B_outer)) != MF_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  h->last_stream = s;
  uint64_t key = 0x6d657461ULL;
  for (uint64_t v : {static_cast<uint64_t>(lp->T), static_cast<uint64_t>(lp->B),
                     static_cast<uint64_t>(lp->B_outer), static_cast<uint64_t>(lp->meta_kind),
                     static_cast<uint64_t>(lp->hvp_mode),
                     static_cast<uint64_t>(make_store(lp).k),
                     static_cast<uint64_t>(make_store(lp).bin),
                     static_cast<uint64_t>(lp->optimizer),
                     static_cast<uint64_t>(float_bits(lp->beta1)),
                     static_cast<uint64_t>(float_bits(lp->beta2)),
                     static_cast<uint64_t>(float_bits(lp->adam_eps)),
                     static_cast<uint64_t>(float_bits(lp->alpha)),
                     static_cast<uint64_t>(float_bits(lp->momentum)),
                     reinterpret_cast<uint64_t>(theta0), reinterpret_cast<uint64_t>(eta),
                     reinterpret_cast<uint64_t>(inner_x), reinterpret_cast<uint64_t>(inner_y),
                     reinterpret_cast<uint64_t>(outer_x), reinterpret_cast<uint64_t>(outer_y),
                     reinterpret_cast<uint64_t>(d_eta), reinterpret_cast<uint64_t>(d_theta0),
                     reinterpret_cast<uint64_t>(outer_loss)})
    key = mix_key(key, v);
  return run_graphed(h, h->g_meta, key, s, [&](cudaStream_t st) {
    return h->bf16 ? meta_grad_impl<__nv_bfloat16>(h, lp, theta0, eta, inner_x, inner_y, outer_x,
                                                   outer_y, d_eta, d_theta0, outer_loss, st)
                   : meta_grad_impl<float>(h, lp, theta0, eta, inner_x, inner_y, outer_x, outer_y,
                                           d_eta, d_theta0, outer_loss, st);
  });
}

mf_status mf_sync(mf_handle h) {
  if (!h) return MF_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(h->last_stream);
  if (e == cudaSuccess && h->gstream) e = cudaStreamSynchronize(h->gstream);
  if (e != cudaSuccess) return fail(h, MF_ERR_CUDA, std::string("stream: ") + cudaGetErrorString(e));
  int v = 0;
  e = cudaMemcpy(&v, h->d_status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(h, MF_ERR_CUDA, std::string("status read: ") + cudaGetErrorString(e));
  if (h->fault == 2) { h->fault = 0; v = mf::DEV_TIMEOUT; }
  if (v != 0) {
    cudaMemset(h->d_status, 0, sizeof(int));
    if (v == mf::DEV_TIMEOUT) return fail(h, MF_ERR_TIMEOUT, "a device-side wait ran out of time");
    if (v == mf::DEV_NONFINITE) return fail(h, MF_ERR_NONFINITE, "non-finite value in the adjoint or the parameters");
    if (v == 1) return fail(h, MF_ERR_INVALID_ARG, "a class label is out of range");
    return fail(h, MF_ERR_CUDA, "device status " + std::to_string(v));
  }
  return MF_OK;
}

mf_status mf_stats(mf_handle h, uint64_t* launches, size_t* peak) {
  if (!h) return MF_ERR_INVALID_ARG;
  if (launches) *launches = h->launches;
  if (peak) *peak = h->peak;
  return MF_OK;
}

mf_status mf_set_kernel_timing(mf_handle h, int enable) {
  if (!h || enable < 0 || enable > 2) return MF_ERR_INVALID_ARG;
  if (enable == 2) {
    h->record = true;
    return MF_OK;
  }
  h->timing = enable != 0;
  return MF_OK;
}

mf_status mf_replay_gemms(mf_handle h, int reps, void* stream, double* ms, uint64_t* launches,
                          double* flops) {
  if (!h || reps < 1) return MF_ERR_INVALID_ARG;
  if (h->rec.empty()) return fail(h, MF_ERR_INVALID_ARG, "no recorded GEMM launches");
  if (!h->gstream) return fail(h, MF_ERR_UNSUPPORTED, "no library stream for the capture");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!h->rec_exec) {
    MF_CUDA(h, cudaStreamBeginCapture(h->gstream, cudaStreamCaptureModeThreadLocal));
    cudaError_t le = cudaSuccess;
    const char* why = "";
    for (const GemmArgs& g : h->rec) {
      le = mf::tc_gemm(g, h->gstream, &why);
      if (le != cudaSuccess) break;
    }
    cudaGraph_t graph = nullptr;
    const cudaError_t ce = cudaStreamEndCapture(h->gstream, &graph);
    if (le != cudaSuccess || ce != cudaSuccess || !graph) {
      if (graph) cudaGraphDestroy(graph);
      cudaGetLastError();
      return fail(h, MF_ERR_CUDA, std::string("GEMM replay capture failed: ") +
                                      cudaGetErrorString(le != cudaSuccess ? le : ce) + " " + why);
    }
    const cudaError_t ie = cudaGraphInstantiate(&h->rec_exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ie != cudaSuccess) {
      h->rec_exec = nullptr;
      cudaGetLastError();
      return fail(h, MF_ERR_CUDA, std::string("GEMM replay instantiate failed: ") + cudaGetErrorString(ie));
    }
  }
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  MF_CUDA(h, cudaEventCreate(&e0));
  if (cudaEventCreate(&e1) != cudaSuccess) {
    cudaEventDestroy(e0);
    return fail(h, MF_ERR_CUDA, "event creation failed");
  }
  cudaError_t e = cudaEventRecord(e0, s);
  for (int r = 0; r < reps && e == cudaSuccess; ++r) e = cudaGraphLaunch(h->rec_exec, s);
  if (e == cudaSuccess) e = cudaEventRecord(e1, s);
  if (e == cudaSuccess) e = cudaEventSynchronize(e1);
  float t = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&t, e0, e1);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (e != cudaSuccess) return fail(h, MF_ERR_CUDA, std::string("GEMM replay: ") + cudaGetErrorString(e));
  h->launches += static_cast<uint64_t>(reps) * h->rec.size();
  if (ms) *ms = static_cast<double>(t) / reps;
  if (launches) *launches = h->rec.size();
  if (flops) *flops = h->rec_flops;
  return MF_OK;
}

mf_status mf_kernel_time(mf_handle h, double* ms, uint64_t* launches, double* flops) {
  if (!h) return MF_ERR_INVALID_ARG;
  double tot = 0.0;
  uint64_t n = 0;
  double fl = h->timed_flops;
  if (h->timed_replay) {
    // one replay's worth of in-graph event pairs (each replay re-records them)
    auto& g = *h->timed_replay;
    cudaError_t e = cudaEventSynchronize(g.evs.back().second);
    if (e != cudaSuccess) return fail(h, MF_ERR_CUDA, cudaGetErrorString(e));
    for (auto& pr : g.evs) {
      float t = 0.f;
      if (cudaEventElapsedTime(&t, pr.first, pr.second) == cudaSuccess) { tot += t; ++n; }
    }
    fl += g.flops;
    h->timed_replay = nullptr;
  }
  if (!h->evs.empty()) {
    cudaError_t e = cudaEventSynchronize(h->evs.back().second);
    if (e != cudaSuccess) return fail(h, MF_ERR_CUDA, cudaGetErrorString(e));
  }
  for (auto& pr : h->evs) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, pr.first, pr.second) == cudaSuccess) { tot += t; ++n; }
    cudaEventDestroy(pr.first);
    cudaEventDestroy(pr.second);
  }
  h->evs.clear();
  if (ms) *ms = tot;
  if (launches) *launches = n;
  if (flops) *flops = fl;
  h->timed_flops = 0.0;
  return MF_OK;
}

mf_status mf_set_option(mf_handle h, int option, int value) {
  if (!h) return MF_ERR_INVALID_ARG;
  if (option == MF_OPT_CUDA_GRAPHS) {
    h->use_graphs = value != 0;
    if (!h->use_graphs) drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_PDL) {
    mf::g_pdl = value != 0;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_GEMM_2SM) {
    if (value < 0 || value > 2) return fail(h, MF_ERR_INVALID_ARG, "MF_OPT_GEMM_2SM takes 0, 1 or 2");
    mf::g_pair_mode = value;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_GEMM_PERSISTENT) {
    if (value < 0 || value > 3) return fail(h, MF_ERR_INVALID_ARG, "MF_OPT_GEMM_PERSISTENT takes 0..3");
    mf::g_gemm_persist = value;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_FUSED_HEAD) {
    if (value < 0 || value > 1) return fail(h, MF_ERR_INVALID_ARG, "MF_OPT_FUSED_HEAD takes 0 or 1");
    mf::g_fused_head = value;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_WAIT_LIMIT_US) {
    if (value < 0 || value > 60000000)
      return fail(h, MF_ERR_INVALID_ARG, "MF_OPT_WAIT_LIMIT_US takes 0..60000000");
    mf::g_wait_ns = static_cast<long long>(value) * 1000LL;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_LAYER_UPDATES) {
    h->layer_updates = value != 0;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_CONCURRENT) {
    h->concurrent = value != 0;
    drop_graphs(h);
    return MF_OK;
  }
  if (option == MF_OPT_FLASH_ATTN) {
    if (value < 0 || value > 4) return fail(h, MF_ERR_INVALID_ARG, "MF_OPT_FLASH_ATTN takes 0..4");
    h->flash = value;
    drop_graphs(h);
    return MF_OK;
  }
  return fail(h, MF_ERR_INVALID_ARG, "unknown option");
}

mf_status mf_inject_fault(mf_handle h, int kind) {
  if (!h || kind < 0 || kind > 2) return MF_ERR_INVALID_ARG;
  h->fault = kind;
  return MF_OK;
}

mf_status mf_dual_gemm_bf16(int M, int N, int K, const void* A0, int lda0, const void* A1,
                            int lda1, const void* B0, int ldb0, const void* B1, int ldb1,
                            float* C0, int ldc0, const float* bias0, float* C1, int ldc1,
                            const float* bias1, unsigned terms, void* stream) {
  constexpr unsigned kAmn = 1u << 8, kBmn = 1u << 9;
  const bool a_mn = terms & kAmn, b_mn = terms & kBmn;
  terms &= ~(kAmn | kBmn);
  if (M < 1 || N < 1 || K < 1 || (terms & ~mf::T_ALL) || !(terms & mf::T_ALL)) return MF_ERR_INVALID_ARG;
  const bool acc0 = terms & (mf::T_C0_A0B0 | mf::T_C0_A1B0 | mf::T_C0_A0B1 | mf::T_C0_A1B1);
  const bool acc1 = terms & (mf::T_C1_A1B0 | mf::T_C1_A0B1);
  if ((acc0 && (!C0 || ldc0 < N)) || (acc1 && (!C1 || ldc1 < N))) return MF_ERR_INVALID_ARG;
  GemmArgs g;
  g.M = M; g.N = N; g.K = K;
  g.A0 = A0; g.lda0 = lda0; g.A1 = A1; g.lda1 = lda1;
  g.B0 = B0; g.ldb0 = ldb0; g.B1 = B1; g.ldb1 = ldb1;
  g.C0 = acc0 ? C0 : nullptr; g.ldc0 = ldc0; g.bias0 = bias0;
  g.C1 = acc1 ? C1 : nullptr; g.ldc1 = ldc1; g.bias1 = bias1;
  g.terms = terms;
  g.a_mn = a_mn;
  g.b_mn = b_mn;
  const char* why = "";
  cudaError_t e = mf::tc_gemm(g, static_cast<cudaStream_t>(stream), &why);
  if (e == cudaErrorInvalidValue) { cudaGetLastError(); return MF_ERR_INVALID_ARG; }
  return e == cudaSuccess ? MF_OK : MF_ERR_CUDA;
}

}  // extern "C"

// ================================ no-allocation HVP =======================================
// Callers that cannot allocate device memory - embedders whose memory is fully reserved up
// front by their own allocator, or hosts that only hand out pre-registered buffers - use
// mf_hvp_noalloc.  Its workspace is one file-scope device array; nothing is allocated per
// call or per handle.
namespace {

constexpr size_t kNoAllocScratchBytes = static_cast<size_t>(32) << 20;   // 32 MiB
constexpr size_t kNoAllocStatusBytes = 256;   // status word, then the workspace
constexpr int kMaxDevices = 64;

// Held by every GPU that loads the library until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up once per device.
// The symbol name is only a host-side stand-in; kernels must be given this address.
cudaError_t noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" mf_status mf_hvp_noalloc(const mf_model_desc* d, int B, const float* theta,
                                    const void* x, const void* y, const float* ex_w,
                                    const float* v, float* Hv, float* tangent_losses,
                                    float* grad, void* stream) {
  if (!d || B < 1 || !theta || !x || !y || !v || !Hv) return MF_ERR_INVALID_ARG;
  if (d->arch == MF_ARCH_DECODER) return MF_ERR_UNSUPPORTED;   // MLP models only
  if (d->arch != MF_ARCH_MLP || d->n_layers < 1 || d->n_layers > MF_MAX_LAYERS)
    return MF_ERR_INVALID_ARG;
  for (int i = 0; i <= d->n_layers; ++i)
    if (d->dims[i] < 1 || d->dims[i] > (1 << 20)) return MF_ERR_INVALID_ARG;
  if (d->act < MF_ACT_IDENT || d->act > MF_ACT_SILU) return MF_ERR_INVALID_ARG;
  if (d->loss != MF_LOSS_SQUARED && d->loss != MF_LOSS_SOFTMAX_CE && d->loss != MF_LOSS_CHAIN_MSE)
    return d->loss == MF_LOSS_NEXT_TOKEN_CE ? MF_ERR_UNSUPPORTED : MF_ERR_INVALID_ARG;
  if (d->loss == MF_LOSS_CHAIN_MSE && (d->chain_steps < 0 || d->chain_steps > 4096))
    return MF_ERR_INVALID_ARG;
  if (d->precision != MF_PREC_FP32 && d->precision != MF_PREC_BF16) return MF_ERR_INVALID_ARG;

  // A handle-free context on the host stack; its workspace is the static device array.
  mf_ctx h;
  h.md = *d;
  h.L = d->n_layers;
  h.dims.assign(d->dims, d->dims + d->n_layers + 1);
  int64_t o = 0;
  for (int l = 0; l < h.L; ++l) {
    h.woff.push_back(o);
    o += static_cast<int64_t>(h.dims[l]) * h.dims[l + 1];
    h.boff.push_back(d->has_bias ? o : -1);
    if (d->has_bias) o += h.dims[l + 1];
  }
  h.P = o;
  h.maxd = *std::max_element(h.dims.begin(), h.dims.end());
  h.bf16 = d->precision == MF_PREC_BF16;
  const Plan plan = make_plan(&h, B, 1, 0, 0, false);
  if (plan.bytes > kNoAllocScratchBytes - kNoAllocStatusBytes) return MF_ERR_INVALID_ARG;
  if (check_x(&h, x, B) != MF_OK) return MF_ERR_INVALID_ARG;

  void* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) {
    cudaGetLastError();
    return MF_ERR_CUDA;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  h.d_status = static_cast<int*>(scratch);
  if (cudaMemsetAsync(h.d_status, 0, sizeof(int), s) != cudaSuccess) {
    cudaGetLastError();
    return MF_ERR_CUDA;
  }
  h.ws = static_cast<char*>(scratch) + kNoAllocStatusBytes;
  h.ws_bytes = kNoAllocScratchBytes - kNoAllocStatusBytes;
  const mf_status st =
      h.bf16 ? hvp_impl<__nv_bfloat16>(&h, B, theta, x, y, ex_w, v, Hv, tangent_losses, grad, false, s)
             : hvp_impl<float>(&h, B, theta, x, y, ex_w, v, Hv, tangent_losses, grad, false, s);
  h.ws = nullptr;   // not owned: never released
  return st;
}
