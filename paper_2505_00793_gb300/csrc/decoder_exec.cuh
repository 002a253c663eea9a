// Decoder-only transformer executor (included by capi.cu inside its anonymous namespace).
//
// Forward-over-reverse for the transformer of the language-modelling tasks: every block is
// pre-RMSNorm causal multi-head attention with RoPE followed by a pre-RMSNorm GELU MLP, with
// residual connections; an untied head produces next-token logits.  The dual forward carries
// the tangent along u of every activation; the dual backward carries the tangent of every
// gradient, so the weight products yield H u directly (no stored reverse graph).
//
// Linear layers run on the tcgen05 dual GEMM (the W1 GEMM fuses GELU and its derivatives,
// the W2 data product fuses the GELU backward).  Attention runs in the fused dual attention
// kernels (flash_tc.cu on tcgen05 for bf16 sequences of whole 128-token tiles, flash_attn.cu
// otherwise); where those do not apply (float32 decoders, heads other than 64 wide,
// sequences that are not whole 64-token tiles), the scores, P V and the four backward
// products run as batched dual GEMMs over batch x heads with the softmax row kernels between
// them.  RMSNorm, RoPE, the embedding gradient and the loss are row kernels
// (decoder_kernels.cu).

// A parameter tensor as seen by the fused update/cast kernel: rows x cols at off; the first
// `cast` rows (0 or all) get bf16 operand copies.
struct DecTensor {
  int64_t off;
  int rows, cols, cast;
};

std::vector<DecTensor> dec_tensors(const DecLayout& Ly) {
  std::vector<DecTensor> t;
  t.push_back({Ly.E, Ly.V, Ly.d, 0});
  for (int l = 0; l < Ly.L; ++l) {
    t.push_back({Ly.g1[l], 1, Ly.d, 0});
    t.push_back({Ly.Wqkv[l], Ly.d, 3 * Ly.d, Ly.d});
    t.push_back({Ly.Wo[l], Ly.d, Ly.d, Ly.d});
    t.push_back({Ly.g2[l], 1, Ly.d, 0});
    t.push_back({Ly.W1[l], Ly.d, Ly.F, Ly.d});
    t.push_back({Ly.W2[l], Ly.F, Ly.d, Ly.F});
  }
  t.push_back({Ly.gf, 1, Ly.d, 0});
  t.push_back({Ly.Wh, Ly.d, Ly.V, Ly.d});
  return t;
}

struct DecPlan {
  int rows = 0, N = 0, ldN = 0, T = 0;
  int nb = 0;
  size_t bytes = 0;
  size_t o_theta = 0, o_m = 0, o_g = 0, o_tbar = 0, o_u = 0, o_part = 0, o_l = 0, o_ld = 0;
  size_t o_count = 0, o_start = 0, o_order = 0, o_order_tmp = 0, gpart = 0;
  // per tensor operand copies (index = tensor index; 0 when not cast)
  std::vector<size_t> o_W, o_U;
  // per block activations
  std::vector<size_t> x1, x1d, r1, r1d, x2, x2d, r2, r2d, h1, h1d, h2, h2d;
  std::vector<size_t> Q, Qd, K, Kd, Vv, Vd, P, Pd, Om, Omd;
  std::vector<size_t> z1, z1d, a1, a1d;
  size_t x0 = 0, x0d = 0, xf = 0, xfd = 0, rf = 0, rfd = 0, hf = 0, hfd = 0;
  size_t Fl = 0, Fld = 0, lse = 0, ltok = 0, pf = 0, ldtok = 0, dF = 0, dFd = 0;
  // scratch reused by every block
  size_t qkv = 0, qkvd = 0, Sc = 0, Scd = 0, O = 0, Od = 0, y = 0, yd = 0, yprev = 0;
  size_t dx = 0, dxd = 0, dh = 0, dhd = 0, dy = 0, dyd = 0;
  size_t dOh = 0, dOhd = 0, dP = 0, dPd = 0, dS = 0, dSd = 0;
  size_t dQ = 0, dQd = 0, dK = 0, dKd = 0, dV = 0, dVd = 0;
  size_t dqkv = 0, dqkvd = 0, dz1 = 0, dz1d = 0;
  // reverse-over-reverse: the inner backward's residual-stream cotangent at the output of
  // every block (the stored reverse graph, at block granularity)
  bool ror = false;
  std::vector<size_t> dxs;
  // fused dual attention: per block the row statistics (lse, then rbar) instead of P and P';
  // D and D' of the block being differentiated
  bool flash = false;
  std::vector<size_t> fst;
  size_t fD = 0;
  size_t rope = 0;   // RoPE (cos, sin) table [S][dh/2]
};

DecPlan make_dec_plan(const mf_ctx* h, const DecLayout& Ly, int rows, int T, int n_theta_slots,
                      int n_m_slots, bool with_partials, bool ror = false) {
  DecPlan p;
  p.ror = ror;
  p.rows = rows;
  p.N = rows * Ly.S;
  p.ldN = ld8(p.N);
  p.T = T;
  const size_t es = h->bf16 ? 2 : 4;
  const int64_t N = p.N, d = Ly.d, F = Ly.F, V = Ly.V, S = Ly.S, BH = rows * Ly.H;
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t r = o; o += align_up(bytes); return r; };
  const size_t P4 = static_cast<size_t>(h->P) * 4;
  p.o_theta = take(P4 * n_theta_slots);
  p.o_m = take(P4 * n_m_slots);
  p.o_g = take(P4);
  p.o_tbar = take(P4);
  p.o_u = take(P4);
  const auto tens = dec_tensors(Ly);
  int tiles = 0;
  for (const auto& t : tens) tiles += mf::update_blocks(t.rows, t.cols);
  p.nb = tiles;
  p.o_part = take(with_partials ? static_cast<size_t>(p.nb) * (T > 0 ? T : 1) * 4 : 4);
  p.o_l = take(static_cast<size_t>(rows) * 4);
  p.o_ld = take(static_cast<size_t>(rows) * 4);
  p.o_count = take(static_cast<size_t>(V) * 4);
  p.o_start = take(static_cast<size_t>(V + 1) * 4);
  p.o_order = take(static_cast<size_t>(N) * 4);
  p.o_order_tmp = take(static_cast<size_t>(N) * 4);
  p.gpart = take(static_cast<size_t>(2) * mf::dec_gain_chunks(static_cast<int>(N)) * d * 4);
  for (const auto& t : tens) {
    if (t.cast) {
      p.o_W.push_back(take(static_cast<size_t>(t.rows) * ld8(t.cols) * es));
      p.o_U.push_back(take(static_cast<size_t>(t.rows) * ld8(t.cols) * es));
    } else {
      p.o_W.push_back(0); p.o_U.push_back(0);
    }
  }
  const size_t Nd4 = N * d * 4, NdT = N * d * es;
  const size_t head = static_cast<size_t>(BH) * S * Ly.dh * es;
  p.flash = h->flash && h->bf16 && mf::flash_supported(static_cast<int>(S), Ly.dh);
  const size_t SS = p.flash ? 0 : static_cast<size_t>(BH) * S * S;
  const size_t stat = static_cast<size_t>(BH) * S * 4;
  for (int l = 0; l < Ly.L; ++l) {
    p.x1.push_back(take(Nd4)); p.x1d.push_back(take(Nd4));
    p.r1.push_back(take(N * 4)); p.r1d.push_back(take(N * 4));
    p.x2.push_back(take(Nd4)); p.x2d.push_back(take(Nd4));
    p.r2.push_back(take(N * 4)); p.r2d.push_back(take(N * 4));
    p.h1.push_back(take(NdT)); p.h1d.push_back(take(NdT));
    p.h2.push_back(take(NdT)); p.h2d.push_back(take(NdT));
    p.Q.push_back(take(head)); p.Qd.push_back(take(head));
    p.K.push_back(take(head)); p.Kd.push_back(take(head));
    p.Vv.push_back(take(head)); p.Vd.push_back(take(head));
    p.P.push_back(take(SS * es)); p.Pd.push_back(take(SS * es));
    if (p.flash) p.fst.push_back(take(2 * stat));
    p.Om.push_back(take(NdT)); p.Omd.push_back(take(NdT));
    p.z1.push_back(take(N * F * 4)); p.z1d.push_back(take(N * F * 4));
    p.a1.push_back(take(N * F * es)); p.a1d.push_back(take(N * F * es));
  }
  p.x0 = take(Nd4); p.x0d = take(Nd4);
  p.xf = take(Nd4); p.xfd = take(Nd4); p.rf = take(N * 4); p.rfd = take(N * 4);
  p.hf = take(NdT); p.hfd = take(NdT);
  p.Fl = take(N * V * 4); p.Fld = take(N * V * 4);
  p.lse = take(N * 4); p.ltok = take(N * 4); p.pf = take(N * 4); p.ldtok = take(N * 4);
  p.dF = take(N * V * es); p.dFd = take(N * V * es);
  p.qkv = take(N * 3 * d * 4); p.qkvd = take(N * 3 * d * 4);
  p.Sc = take(SS * 4); p.Scd = take(SS * 4);
  // per-head float32 attention outputs (the fused attention writes them head-merged instead)
  const size_t osz = p.flash ? 0 : static_cast<size_t>(BH) * S * Ly.dh * 4;
  p.O = take(osz); p.Od = take(osz);
  p.y = take(Nd4); p.yd = take(Nd4);
  p.dx = take(Nd4); p.dxd = take(Nd4); p.dh = take(Nd4); p.dhd = take(Nd4);
  p.dy = take(NdT); p.dyd = take(NdT);
  p.dOh = take(head); p.dOhd = take(head);
  p.dP = take(SS * 4); p.dPd = take(SS * 4);
  p.dS = take(SS * es); p.dSd = take(SS * es);
  if (p.flash) p.fD = take(2 * stat);
  p.rope = take(static_cast<size_t>(S) * (Ly.dh / 2) * 2 * 4);
  const size_t head4 = static_cast<size_t>(BH) * S * Ly.dh * 4;
  p.dQ = take(head4); p.dQd = take(head4); p.dK = take(head4); p.dKd = take(head4);
  p.dV = take(head4); p.dVd = take(head4);
  if (ror)
    for (int l = 0; l < Ly.L; ++l) p.dxs.push_back(take(Nd4));
  p.dqkv = take(N * 3 * d * es); p.dqkvd = take(N * 3 * d * es);
  p.dz1 = take(N * F * es); p.dz1d = take(N * F * es);
  p.bytes = o;
  return p;
}

template <typename T>
struct DecExec {
  mf_ctx* h;
  const DecPlan& p;
  const DecLayout& Ly;
  cudaStream_t s;
  char* base;
  mf_status st = MF_OK;
  mf::LayerTable tab;
  std::vector<DecTensor> tens;
  int rows_cur = 0;
  const int* ids_cur = nullptr;
  bool dual_cur = false;
  const float* theta_cur = nullptr;
  const float* u_cur = nullptr;
  // reverse-over-reverse: 1 = the primal backward stores each block's output cotangent,
  // 2 = the second-order backward restarts every block from the stored cotangent
  int ror_mode = 0;

  DecExec(mf_ctx* h_, const DecPlan& p_, const DecLayout& L_, cudaStream_t s_)
      : h(h_), p(p_), Ly(L_), s(s_), base(static_cast<char*>(h_->ws)) {
    tens = dec_tensors(Ly);
    tab.n = static_cast<int>(tens.size());
    int tiles = 0;
    for (int i = 0; i < tab.n; ++i) {
      const auto& t = tens[i];
      tab.rows[i] = t.rows;
      tab.din[i] = t.cast;
      tab.dout[i] = t.cols;
      tab.off[i] = t.off;
      tab.tile0[i] = tiles;
      tiles += mf::update_blocks(t.rows, t.cols);
      tab.ldw[i] = ld8(t.cols);
      tab.W[i] = t.cast ? at<T>(p.o_W[i]) : nullptr;   // read K- or MN-major, never transposed
      tab.U[i] = t.cast ? at<T>(p.o_U[i]) : nullptr;
    }
    tab.tile0[tab.n] = tiles;
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
  size_t x_step_bytes(int rows) const { return static_cast<size_t>(rows) * (Ly.S + 1) * 4; }
  size_t y_step_bytes(int rows) const { return x_step_bytes(rows); }

  void launched(int n = 1) { h->launches += n; }
  void chk(const char* what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess && st == MF_OK) {
      st = MF_ERR_CUDA;
      h->err = std::string(what) + ": " + cudaGetErrorString(e);
    }
  }

  // index of a cast tensor in `tens`
  int tidx(int64_t off) const {
    for (int i = 0; i < static_cast<int>(tens.size()); ++i)
      if (tens[i].off == off) return i;
    return -1;
  }
  T* W(int64_t off) const { return at<T>(p.o_W[tidx(off)]); }

  T* Uw(int64_t off) const { return at<T>(p.o_U[tidx(off)]); }


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
      cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
      cudaStreamIsCapturing(s, &cs);
      ev_flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
      cudaEventRecordWithFlags(e0, s, ev_flags);
    }
    const char* why = "";
    cudaError_t e = tc ? mf::tc_gemm(g, s, &why) : mf::simt_gemm(g, s);
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

  // C = X Y^T style linear product; dual adds X' Y^T + X Y'^T (or the weight-tangent sum).
  // Operands of the fused attention of block l: its heads and row statistics.
  mf::FlashArgs flash_args(int l, int BH) const {
    auto hb = [&](size_t o) { return reinterpret_cast<const __nv_bfloat16*>(at<T>(o)); };
    mf::FlashArgs fa;
    fa.BH = BH;
    fa.S = Ly.S;
    fa.tc = h->flash == 1 || h->flash == 4 ? 1 : h->flash == 3 ? 2 : 0;
    fa.tc_bwd = h->flash == 1 || h->flash == 3 ? 1 : 0;
    fa.status = h->d_status;
    fa.Q = hb(p.Q[l]); fa.K = hb(p.K[l]); fa.V = hb(p.Vv[l]);
    fa.Qd = hb(p.Qd[l]); fa.Kd = hb(p.Kd[l]); fa.Vd = hb(p.Vd[l]);
    fa.lse = at<float>(p.fst[l]);
    fa.rbar = fa.lse + static_cast<int64_t>(BH) * Ly.S;
    return fa;
  }

  GemmArgs lin(int M, int N, int K, const void* A0, const void* A1, int lda, const void* B0,
               const void* B1, int ldb, bool dual) const {
    GemmArgs g;
    g.M = M; g.N = N; g.K = K;
    g.A0 = A0; g.A1 = A1; g.lda0 = g.lda1 = lda;
    g.B0 = B0; g.B1 = B1; g.ldb0 = g.ldb1 = ldb;
    g.terms = dual ? (mf::T_C0_A0B0 | mf::T_C1_A1B0 | mf::T_C1_A0B1) : mf::T_C0_A0B0;
    return g;
  }

  void batched(GemmArgs& g, int batch, int64_t bsA, int64_t bsB, int64_t bsC) const {
    g.batch = batch;
    g.bsA0 = g.bsA1 = bsA;
    g.bsB0 = g.bsB1 = bsB;
    g.bsC0 = g.bsC1 = bsC;
  }

  void prepare() {
    mf::dec_rope_table(Ly.S, Ly.dh, Ly.base, at<float>(p.rope), s);
    launched();
  }

  void update(const mf::LayerUpdArgs& a) {
    mf::layer_update<T>(tab, a, s);
    launched();
  }

  void cast_params(const float* theta, bool tangent) {
    mf::LayerUpdArgs a;
    a.mode = mf::LU_CAST;
    a.cast_src = theta;
    a.cast_src_to_u = tangent;
    update(a);
  }

  void forward(int rows, const void* x, const float* theta, const float* u, bool dual) {
    const int S = Ly.S, d = Ly.d, H = Ly.H, dh = Ly.dh, F = Ly.F, V = Ly.V;
    const int N = rows * S, BH = rows * H;
    const int* ids = static_cast<const int*>(x);
    rows_cur = rows;
    ids_cur = ids;
    dual_cur = dual;
    theta_cur = theta;
    u_cur = u;
    const int64_t hs = static_cast<int64_t>(S) * dh, ss = static_cast<int64_t>(S) * S;
    mf::dec_embed_fwd(N, S, d, V, ids, theta + Ly.E, dual ? u + Ly.E : nullptr, at<float>(p.x0),
                      dual ? at<float>(p.x0d) : nullptr, h->d_status, s);
    launched();
    const float* xin = at<float>(p.x0);
    const float* xind = at<float>(p.x0d);
    const float* yin = nullptr;
    const float* yind = nullptr;
    for (int l = 0; l < Ly.L; ++l) {
      // residual + attention RMSNorm
      mf::dec_rmsnorm_fwd<T>(N, d, Ly.eps, xin, yin, dual ? xind : nullptr, yind, theta + Ly.g1[l],
                             dual ? u + Ly.g1[l] : nullptr, at<float>(p.x1[l]), at<float>(p.x1d[l]),
                             at<float>(p.r1[l]), at<float>(p.r1d[l]), at<T>(p.h1[l]), at<T>(p.h1d[l]),
                             d, s);
      launched();
      // q k v = h Wqkv   (weights [d][3d] read MN-major)
      {
        GemmArgs g = lin(N, 3 * d, d, at<T>(p.h1[l]), at<T>(p.h1d[l]), d, W(Ly.Wqkv[l]),
                         Uw(Ly.Wqkv[l]), ld8(3 * d), dual);
        g.b_mn = true;
        g.C0 = at<float>(p.qkv); g.ldc0 = 3 * d;
        g.C1 = at<float>(p.qkvd); g.ldc1 = 3 * d;
        if (!dual) g.terms = mf::T_C0_A0B0;
        gemm(g);
      }
      const float qscale = 1.f / sqrtf(static_cast<float>(dh));
      mf::dec_rope_split<T>(N, S, H, dh, at<float>(p.rope), qscale, at<float>(p.qkv), at<T>(p.Q[l]),
                            at<T>(p.K[l]), at<T>(p.Vv[l]), s);
      launched();
      if (dual) {
        mf::dec_rope_split<T>(N, S, H, dh, at<float>(p.rope), qscale, at<float>(p.qkvd), at<T>(p.Qd[l]),
                              at<T>(p.Kd[l]), at<T>(p.Vd[l]), s);
        launched();
      }

      if (p.flash) {
        // fused causal attention and its tangent: O, O' and the row statistics
        // fused causal attention and its tangent, written head-merged as the Wo operands
        mf::FlashArgs fa = flash_args(l, BH);
        fa.H = H;
        fa.ldo = d;
        fa.Om = reinterpret_cast<__nv_bfloat16*>(at<T>(p.Om[l]));
        fa.Omd = dual ? reinterpret_cast<__nv_bfloat16*>(at<T>(p.Omd[l])) : nullptr;
        mf::flash_fwd(fa, dual, s);
        launched();
      } else {
      // scores S = Q K^T (dual: Q' K^T + Q K'^T), batch over B*H
      {
        GemmArgs g = lin(S, S, dh, at<T>(p.Q[l]), at<T>(p.Qd[l]), dh, at<T>(p.K[l]), at<T>(p.Kd[l]),
                         dh, dual);
        batched(g, BH, hs, hs, ss);
        g.C0 = at<float>(p.Sc); g.ldc0 = S;
        g.C1 = at<float>(p.Scd); g.ldc1 = S;
        gemm(g);
      }
      mf::dec_softmax_fwd<T>(S, BH * S, at<float>(p.Sc), dual ? at<float>(p.Scd) : nullptr,
                             at<T>(p.P[l]), dual ? at<T>(p.Pd[l]) : nullptr, s);
      launched();
      // O = P V (dual: P' V + P V'); V [S][dh] read MN-major
      {
        GemmArgs g = lin(S, dh, S, at<T>(p.P[l]), at<T>(p.Pd[l]), S, at<T>(p.Vv[l]),
                         at<T>(p.Vd[l]), dh, dual);
        g.b_mn = true;
        batched(g, BH, ss, hs, hs);
        g.C0 = at<float>(p.O); g.ldc0 = dh;
        g.C1 = at<float>(p.Od); g.ldc1 = dh;
        gemm(g);
      }
      mf::dec_head_merge<T>(N, S, H, dh, at<float>(p.O), at<T>(p.Om[l]), d, s);
      launched();
      if (dual) {
        mf::dec_head_merge<T>(N, S, H, dh, at<float>(p.Od), at<T>(p.Omd[l]), d, s);
        launched();
      }
      }
      // y = O Wo
      {
        GemmArgs g = lin(N, d, d, at<T>(p.Om[l]), at<T>(p.Omd[l]), d, W(Ly.Wo[l]), Uw(Ly.Wo[l]),
                         ld8(d), dual);
        g.b_mn = true;
        g.C0 = at<float>(p.y); g.ldc0 = d;
        g.C1 = at<float>(p.yd); g.ldc1 = d;
        gemm(g);
      }
      // residual + MLP RMSNorm
      mf::dec_rmsnorm_fwd<T>(N, d, Ly.eps, at<float>(p.x1[l]), at<float>(p.y),
                             dual ? at<float>(p.x1d[l]) : nullptr, dual ? at<float>(p.yd) : nullptr,
                             theta + Ly.g2[l], dual ? u + Ly.g2[l] : nullptr, at<float>(p.x2[l]),
                             at<float>(p.x2d[l]), at<float>(p.r2[l]), at<float>(p.r2d[l]),
                             at<T>(p.h2[l]), at<T>(p.h2d[l]), d, s);
      launched();
      // a = GELU(h2 W1) fused; z kept for the backward
      {
        GemmArgs g = lin(N, F, d, at<T>(p.h2[l]), at<T>(p.h2d[l]), d, W(Ly.W1[l]), Uw(Ly.W1[l]),
                         ld8(F), dual);
        g.b_mn = true;
        g.C0 = at<float>(p.z1[l]); g.ldc0 = F;
        g.C1 = at<float>(p.z1d[l]); g.ldc1 = F;
        g.epi.mode = mf::EPI_ACT_FWD;
        g.epi.act = mf::ACT_GELU;
        g.epi.A = at<T>(p.a1[l]);
        g.epi.Ad = dual ? at<T>(p.a1d[l]) : nullptr;
        g.epi.lda = F;
        gemm(g);
      }
      // y = a W2  (added to x2 by the next RMSNorm)
      {
        GemmArgs g = lin(N, d, F, at<T>(p.a1[l]), at<T>(p.a1d[l]), F, W(Ly.W2[l]), Uw(Ly.W2[l]),
                         ld8(d), dual);
        g.b_mn = true;
        g.C0 = at<float>(p.y); g.ldc0 = d;
        g.C1 = at<float>(p.yd); g.ldc1 = d;
        gemm(g);
      }
      xin = at<float>(p.x2[l]);
      xind = at<float>(p.x2d[l]);
      yin = at<float>(p.y);
      yind = dual ? at<float>(p.yd) : nullptr;
    }
    mf::dec_rmsnorm_fwd<T>(N, d, Ly.eps, xin, yin, dual ? xind : nullptr, yind, theta + Ly.gf,
                           dual ? u + Ly.gf : nullptr, at<float>(p.xf), at<float>(p.xfd),
                           at<float>(p.rf), at<float>(p.rfd), at<T>(p.hf), at<T>(p.hfd), d, s);
    launched();
    {
      GemmArgs g = lin(N, V, d, at<T>(p.hf), at<T>(p.hfd), d, W(Ly.Wh), Uw(Ly.Wh), ld8(V), dual);
      g.b_mn = true;
      g.C0 = at<float>(p.Fl); g.ldc0 = V;
      g.C1 = at<float>(p.Fld); g.ldc1 = V;
      gemm(g);
    }
    chk("decoder forward");
  }

  // Next-token cross-entropy; l_out / ld_out are per sequence; d_eta per sequence.
  void loss(int rows, bool dual, const void* y, const float* eta_w, const float* ex_w,
            float* l_out, float* ld_out, float* d_eta) {
    (void)y;
    const int S = Ly.S, V = Ly.V, N = rows * S;
    mf::dec_ce_stats(N, S, V, ids_cur, at<float>(p.Fl), dual ? at<float>(p.Fld) : nullptr,
                     at<float>(p.lse), at<float>(p.ltok), at<float>(p.pf), at<float>(p.ldtok),
                     h->d_status, s);
    launched();
    mf::dec_ce_seed<T>(N, S, V, ids_cur, at<float>(p.Fl), dual ? at<float>(p.Fld) : nullptr,
                       at<float>(p.lse), at<float>(p.pf), eta_w, ex_w,
                       1.f / (static_cast<float>(rows) * S), at<T>(p.dF),
                       dual ? at<T>(p.dFd) : nullptr, V, s);
    launched();
    mf::dec_seq_reduce(rows, S, at<float>(p.ltok), dual ? at<float>(p.ldtok) : nullptr, eta_w,
                       1.f / rows, l_out, ld_out, d_eta, s);
    launched();
    chk("decoder loss");
  }

  // Weight products on the side stream (MF_OPT_CONCURRENT): each runs next to the data
  // product of its layer, after the seeds it reads are written on the working stream.
  // Seed buffers: 0 = dy (read by the W2 and Wo products), 1 = dz1 (W1), 2 = dqkv (Wqkv).
  enum { WS_W2 = 0, WS_WO = 1, WS_W1 = 2, WS_QKV = 3, WS_NONE = -1 };
  bool w_rec[4] = {false, false, false, false};
  bool side_used = false;
  bool conc() const {
    return h->concurrent && h->sstream && h->ev_fork && h->ev_join && h->ev_w[0] &&
           h->ev_w[1] && h->ev_w[2] && h->ev_w[3];
  }
  void chk_cuda(cudaError_t e, const char* what) {
    if (e != cudaSuccess && st == MF_OK) {
      st = MF_ERR_CUDA;
      h->err = std::string(what) + ": " + cudaGetErrorString(e);
    }
  }
  // the working stream waits until every weight product reading seed buffer `buf` is done
  void wait_seed_readers(int buf) {
    const int slots[2][2] = {{WS_W2, WS_WO}, {WS_W1, WS_NONE}};
    const int* sl = buf == 0 ? slots[0] : buf == 1 ? slots[1] : nullptr;
    auto wait1 = [&](int j) {
      if (j >= 0 && w_rec[j]) chk_cuda(cudaStreamWaitEvent(s, h->ev_w[j], 0), "seed wait");
    };
    if (sl) { wait1(sl[0]); wait1(sl[1]); }
    else wait1(WS_QKV);
  }
  void side_join() {
    if (!side_used) return;
    chk_cuda(cudaEventRecord(h->ev_join, h->sstream), "side join");
    chk_cuda(cudaStreamWaitEvent(s, h->ev_join, 0), "side join");
    side_used = false;
    for (bool& r : w_rec) r = false;
  }

  // weight product into out (grad) / outh (tangent): A^T seed with K = tokens; the
  // activations A [tokens][M] and the seeds [tokens][Nn] are read MN-major
  void wprod(int M, int Nn, const T* A_, const T* Ad_, const T* S_, const T* Sd_, bool dual,
             float* outg, float* outh, int slot = WS_NONE) {
    if (!dual && !outg) return;   // primal backward kept only for its cotangents
    GemmArgs g;
    g.M = M; g.N = Nn; g.K = rows_cur * Ly.S;
    g.A0 = A_; g.A1 = Ad_; g.lda0 = g.lda1 = M;
    g.B0 = S_; g.B1 = Sd_; g.ldb0 = g.ldb1 = Nn;
    g.a_mn = g.b_mn = true;
    if (!dual) {
      g.terms = mf::T_C0_A0B0;
      g.C0 = outg; g.ldc0 = Nn;
    } else if (outg) {
      g.terms = mf::T_C0_A0B0 | mf::T_C1_A1B0 | mf::T_C1_A0B1;
      g.C0 = outg; g.ldc0 = Nn;
      g.C1 = outh; g.ldc1 = Nn;
    } else {
      g.terms = mf::T_C0_A1B0 | mf::T_C0_A0B1;
      g.C0 = outh; g.ldc0 = Nn;
    }
    if (!conc()) {
      gemm(g);
      return;
    }
    chk_cuda(cudaEventRecord(h->ev_fork, s), "side fork");
    chk_cuda(cudaStreamWaitEvent(h->sstream, h->ev_fork, 0), "side fork");
    gemm(g, h->sstream);
    side_used = true;
    if (slot >= 0) {
      chk_cuda(cudaEventRecord(h->ev_w[slot], h->sstream), "side event");
      w_rec[slot] = true;
    }
  }

  // residual gradient (float32) -> operand-type seed
  // bf16 seeds dy (dy') of the next products from the residual-stream gradient dx (dx');
  // skipped when the RMSNorm backward that produced dx already wrote them (fresh)
  void seed_from(const float* X, const float* Xd, bool dual, bool fresh = false) {
    if (fresh) return;
    wait_seed_readers(0);
    const int N = rows_cur * Ly.S, d = Ly.d;
    mf::cast_rows<T>(X, N, d, at<T>(p.dy), d, s);
    launched();
    if (dual) {
      mf::cast_rows<T>(Xd, N, d, at<T>(p.dyd), d, s);
      launched();
    }
  }

  void backward(int rows, bool dual, float* out_h, float* out_g) {
    const int S = Ly.S, d = Ly.d, H = Ly.H, dh = Ly.dh, F = Ly.F, V = Ly.V;
    const int N = rows * S, BH = rows * H;
    const int64_t hs = static_cast<int64_t>(S) * dh, ss = static_cast<int64_t>(S) * S;
    const float* u = u_cur;
    auto G = [&](int64_t off) { return out_g ? out_g + off : nullptr; };
    auto Hh = [&](int64_t off) { return dual ? out_h + off : nullptr; };
    mf::dec_token_csr(N, S, V, ids_cur, at<int>(p.o_count), at<int>(p.o_start), at<int>(p.o_order),
                      at<int>(p.o_order_tmp), s);
    launched(4);
    // head: dWh = hf^T dF ; dhf = dF Wh^T
    wprod(d, V, at<T>(p.hf), at<T>(p.hfd), at<T>(p.dF), at<T>(p.dFd), dual, G(Ly.Wh), Hh(Ly.Wh));
    {
      GemmArgs g = lin(N, d, V, at<T>(p.dF), at<T>(p.dFd), V, W(Ly.Wh), Uw(Ly.Wh), ld8(V), dual);
      g.C0 = at<float>(p.dh); g.ldc0 = d;
      g.C1 = at<float>(p.dhd); g.ldc1 = d;
      gemm(g);
    }
    cudaMemsetAsync(at<float>(p.dx), 0, static_cast<size_t>(N) * d * 4, s);
    if (dual) cudaMemsetAsync(at<float>(p.dxd), 0, static_cast<size_t>(N) * d * 4, s);
    wait_seed_readers(0);
    launched(mf::dec_rmsnorm_bwd<T>(N, d, at<float>(p.xf), at<float>(p.xfd), at<float>(p.rf),
                                    at<float>(p.rfd), theta_cur + Ly.gf, dual ? u + Ly.gf : nullptr,
                                    at<float>(p.dh), dual ? at<float>(p.dhd) : nullptr,
                                    at<float>(p.dx), at<float>(p.dxd), G(Ly.gf), Hh(Ly.gf),
                                    at<float>(p.gpart), s, at<T>(p.dy),
                                    dual ? at<T>(p.dyd) : nullptr));
    for (int l = Ly.L - 1; l >= 0; --l) {
      if (ror_mode == 1) {
        cudaMemcpyAsync(at<float>(p.dxs[l]), at<float>(p.dx), static_cast<size_t>(N) * d * 4,
                        cudaMemcpyDeviceToDevice, s);
      } else if (ror_mode == 2) {
        cudaMemcpyAsync(at<float>(p.dx), at<float>(p.dxs[l]), static_cast<size_t>(N) * d * 4,
                        cudaMemcpyDeviceToDevice, s);
      }
      // ---- MLP branch: seed = dx (already in bf16 unless dx was just restored) ---------
      seed_from(at<float>(p.dx), at<float>(p.dxd), dual, ror_mode != 2);
      wprod(F, d, at<T>(p.a1[l]), at<T>(p.a1d[l]), at<T>(p.dy), at<T>(p.dyd), dual, G(Ly.W2[l]),
            Hh(Ly.W2[l]), WS_W2);
      wait_seed_readers(1);   // the data product's epilogue rewrites dz1
      {
        GemmArgs g = lin(N, F, d, at<T>(p.dy), at<T>(p.dyd), d, W(Ly.W2[l]), Uw(Ly.W2[l]), ld8(d), dual);
        g.epi.mode = mf::EPI_ACT_BWD;
        g.epi.act = mf::ACT_GELU;
        g.epi.Z = at<float>(p.z1[l]);
        g.epi.Zd = dual ? at<float>(p.z1d[l]) : nullptr;
        g.epi.ldz = F;
        g.epi.A = at<T>(p.dz1);
        g.epi.Ad = dual ? at<T>(p.dz1d) : nullptr;
        g.epi.lda = F;
        gemm(g);
      }
      wprod(d, F, at<T>(p.h2[l]), at<T>(p.h2d[l]), at<T>(p.dz1), at<T>(p.dz1d), dual, G(Ly.W1[l]),
            Hh(Ly.W1[l]), WS_W1);
      {
        GemmArgs g = lin(N, d, F, at<T>(p.dz1), at<T>(p.dz1d), F, W(Ly.W1[l]), Uw(Ly.W1[l]), ld8(F), dual);
        g.C0 = at<float>(p.dh); g.ldc0 = d;
        g.C1 = at<float>(p.dhd); g.ldc1 = d;
        gemm(g);
      }
      wait_seed_readers(0);
      launched(mf::dec_rmsnorm_bwd<T>(N, d, at<float>(p.x2[l]), at<float>(p.x2d[l]),
                                      at<float>(p.r2[l]), at<float>(p.r2d[l]), theta_cur + Ly.g2[l],
                                      dual ? u + Ly.g2[l] : nullptr, at<float>(p.dh),
                                      dual ? at<float>(p.dhd) : nullptr, at<float>(p.dx),
                                      at<float>(p.dxd), G(Ly.g2[l]), Hh(Ly.g2[l]),
                                      at<float>(p.gpart), s, at<T>(p.dy),
                                      dual ? at<T>(p.dyd) : nullptr));
      // ---- attention branch: seed = dx (written in bf16 by the norm backward above) -----
      seed_from(at<float>(p.dx), at<float>(p.dxd), dual, true);
      wprod(d, d, at<T>(p.Om[l]), at<T>(p.Omd[l]), at<T>(p.dy), at<T>(p.dyd), dual, G(Ly.Wo[l]),
            Hh(Ly.Wo[l]), WS_WO);
      {
        GemmArgs g = lin(N, d, d, at<T>(p.dy), at<T>(p.dyd), d, W(Ly.Wo[l]), Uw(Ly.Wo[l]), ld8(d), dual);
        g.C0 = at<float>(p.dh); g.ldc0 = d;
        g.C1 = at<float>(p.dhd); g.ldc1 = d;
        gemm(g);
      }
      if (!p.flash) {
        mf::dec_head_split<T>(N, S, H, dh, at<float>(p.dh), at<T>(p.dOh), s);
        launched();
        if (dual) {
          mf::dec_head_split<T>(N, S, H, dh, at<float>(p.dhd), at<T>(p.dOhd), s);
          launched();
        }
      }
      bool merged = false;   // the attention backward writes dqkv itself (no RoPE merge)
      if (p.flash) {
        // fused backward of the attention and its tangent, from D = rowsum(dO O) (and D')
        float* D = at<float>(p.fD);
        float* Dd = D + static_cast<int64_t>(BH) * S;
        // D, D' and the per-head bf16 copies of dO, dO' in one pass over dO
        mf::flash_prep(N, S, H, at<float>(p.dh), dual ? at<float>(p.dhd) : nullptr,
                       at<T>(p.Om[l]), dual ? at<T>(p.Omd[l]) : nullptr, d, D,
                       dual ? Dd : nullptr, at<T>(p.dOh), dual ? at<T>(p.dOhd) : nullptr, s);
        mf::FlashArgs fa = flash_args(l, BH);
        fa.dO = reinterpret_cast<const __nv_bfloat16*>(at<T>(p.dOh));
        fa.dOd = dual ? reinterpret_cast<const __nv_bfloat16*>(at<T>(p.dOhd)) : nullptr;
        fa.D = D;
        fa.Dd = dual ? Dd : nullptr;
        fa.dQ = at<float>(p.dQ); fa.dK = at<float>(p.dK); fa.dV = at<float>(p.dV);
        if (dual) { fa.dQd = at<float>(p.dQd); fa.dKd = at<float>(p.dKd); fa.dVd = at<float>(p.dVd); }
        // the tcgen05 backward writes the merged, RoPE-inverted bf16 rows of dqkv directly
        fa.H = H;
        fa.ldq = 3 * d;
        fa.rope = at<float>(p.rope);
        fa.qscale = 1.f / sqrtf(static_cast<float>(dh));
        fa.dqkv = reinterpret_cast<__nv_bfloat16*>(at<T>(p.dqkv));
        fa.dqkvd = dual ? reinterpret_cast<__nv_bfloat16*>(at<T>(p.dqkvd)) : nullptr;
        merged = std::is_same<T, __nv_bfloat16>::value && mf::flash_bwd_merges(fa, dual);
        if (merged) {
          wait_seed_readers(2);    // dqkv's previous readers (the side stream) are done
        } else {
          fa.dqkv = fa.dqkvd = nullptr;
        }
        mf::flash_bwd(fa, dual, s);
        launched(3);
      } else {
      // dP = dO V^T (dual: dO' V^T + dO V'^T)
      {
        GemmArgs g = lin(S, S, dh, at<T>(p.dOh), at<T>(p.dOhd), dh, at<T>(p.Vv[l]), at<T>(p.Vd[l]), dh, dual);
        batched(g, BH, hs, hs, ss);
        g.C0 = at<float>(p.dP); g.ldc0 = S;
        g.C1 = at<float>(p.dPd); g.ldc1 = S;
        gemm(g);
      }
      mf::dec_softmax_bwd<T>(S, BH * S, at<T>(p.P[l]), dual ? at<T>(p.Pd[l]) : nullptr,
                             at<float>(p.dP), dual ? at<float>(p.dPd) : nullptr, at<T>(p.dS),
                             dual ? at<T>(p.dSd) : nullptr, s);
      launched();
      // dV = P^T dO ; dQ = dS K ; dK = dS^T Q   (each with its tangent); P, dS, dO, K, Q
      // are read in place (MN-major where the product contracts over their row index)
      {
        GemmArgs g = lin(S, dh, S, at<T>(p.P[l]), at<T>(p.Pd[l]), S, at<T>(p.dOh), at<T>(p.dOhd), dh, dual);
        g.a_mn = g.b_mn = true;
        batched(g, BH, ss, hs, hs);
        g.C0 = at<float>(p.dV); g.ldc0 = dh;
        g.C1 = at<float>(p.dVd); g.ldc1 = dh;
        gemm(g);
      }
      {
        GemmArgs g = lin(S, dh, S, at<T>(p.dS), at<T>(p.dSd), S, at<T>(p.K[l]), at<T>(p.Kd[l]), dh, dual);
        g.b_mn = true;
        batched(g, BH, ss, hs, hs);
        g.C0 = at<float>(p.dQ); g.ldc0 = dh;
        g.C1 = at<float>(p.dQd); g.ldc1 = dh;
        gemm(g);
      }
      {
        GemmArgs g = lin(S, dh, S, at<T>(p.dS), at<T>(p.dSd), S, at<T>(p.Q[l]), at<T>(p.Qd[l]), dh, dual);
        g.a_mn = g.b_mn = true;
        batched(g, BH, ss, hs, hs);
        g.C0 = at<float>(p.dK); g.ldc0 = dh;
        g.C1 = at<float>(p.dKd); g.ldc1 = dh;
        gemm(g);
      }
      }
      if (!merged) {
        const float qscale = 1.f / sqrtf(static_cast<float>(dh));
        wait_seed_readers(2);
        mf::dec_rope_merge<T>(N, S, H, dh, at<float>(p.rope), qscale, at<float>(p.dQ), at<float>(p.dK),
                              at<float>(p.dV), at<T>(p.dqkv), 3 * d, s);
        launched();
        if (dual) {
          mf::dec_rope_merge<T>(N, S, H, dh, at<float>(p.rope), qscale, at<float>(p.dQd), at<float>(p.dKd),
                                at<float>(p.dVd), at<T>(p.dqkvd), 3 * d, s);
          launched();
        }
      }
      wprod(d, 3 * d, at<T>(p.h1[l]), at<T>(p.h1d[l]), at<T>(p.dqkv), at<T>(p.dqkvd), dual,
            G(Ly.Wqkv[l]), Hh(Ly.Wqkv[l]), WS_QKV);
      {
        GemmArgs g = lin(N, d, 3 * d, at<T>(p.dqkv), at<T>(p.dqkvd), 3 * d, W(Ly.Wqkv[l]),
                         Uw(Ly.Wqkv[l]), ld8(3 * d), dual);
        g.C0 = at<float>(p.dh); g.ldc0 = d;
        g.C1 = at<float>(p.dhd); g.ldc1 = d;
        gemm(g);
      }
      if (l > 0) wait_seed_readers(0);
      launched(mf::dec_rmsnorm_bwd<T>(N, d, at<float>(p.x1[l]), at<float>(p.x1d[l]),
                                      at<float>(p.r1[l]), at<float>(p.r1d[l]), theta_cur + Ly.g1[l],
                                      dual ? u + Ly.g1[l] : nullptr, at<float>(p.dh),
                                      dual ? at<float>(p.dhd) : nullptr, at<float>(p.dx),
                                      at<float>(p.dxd), G(Ly.g1[l]), Hh(Ly.g1[l]),
                                      at<float>(p.gpart), s, l > 0 ? at<T>(p.dy) : nullptr,
                                      l > 0 && dual ? at<T>(p.dyd) : nullptr));
    }
    mf::dec_embed_bwd(V, d, at<int>(p.o_start), at<int>(p.o_order), at<float>(p.dx),
                      dual ? at<float>(p.dxd) : nullptr, G(Ly.E), Hh(Ly.E), s);
    launched();
    side_join();
    chk("decoder backward");
  }

  // Hessian-vector product by reverse-over-reverse (Algorithm 1's schedule) at block
  // granularity: primal forward and primal backward, which stores the residual-stream
  // cotangent at the output of every block (the reverse graph); then the tangent pass in
  // forward order (the adjoint of the backward, by the symmetry of Eqs. 6-7) and the
  // second-order backward in reverse order, which restarts each block from its stored
  // cotangent and recomputes the cotangents inside the block (block rematerialisation of
  // the inner backward, the granularity at which the forward keeps its activations).
  void ror_hvp(int rows, const void* x, const float* theta, const float* u, const void* y,
               const float* eta_w, const float* ex_w, float* Hv, float* grad, float* ld_out,
               float* d_eta) {
    forward(rows, x, theta, nullptr, false);
    loss(rows, false, y, eta_w, ex_w, nullptr, nullptr, nullptr);
    ror_mode = 1;
    backward(rows, false, nullptr, grad);
    ror_mode = 0;
    forward(rows, x, theta, u, true);
    loss(rows, true, y, eta_w, ex_w, nullptr, ld_out, d_eta);
    ror_mode = 2;
    backward(rows, true, Hv, nullptr);
    ror_mode = 0;
  }
};
