// Flat-parameter layout of the decoder-only transformer (shared by the runtime and its
// executor).  Order: embedding E [V][d]; per block g1 [d], Wqkv [d][3d], Wo [d][d], g2 [d],
// W1 [d][dff], W2 [dff][d]; final gain gf [d]; head Wh [d][V].
#pragma once
#include <stdint.h>

#include <vector>

#include "../../include/mixflow.h"

struct DecLayout {
  int d = 0, H = 0, dh = 0, F = 0, V = 0, S = 0, L = 0;
  float base = 10000.f, eps = 1e-6f;
  int64_t E = 0, gf = 0, Wh = 0;
  std::vector<int64_t> g1, Wqkv, Wo, g2, W1, W2;
};

inline DecLayout dec_layout(const mf_model_desc& md) {
  DecLayout Ly;
  Ly.d = md.d_model; Ly.H = md.n_heads; Ly.dh = md.d_model / md.n_heads; Ly.F = md.d_ff;
  Ly.V = md.vocab; Ly.S = md.seq_len; Ly.L = md.n_layers;
  Ly.base = md.rope_base > 0.f ? md.rope_base : 10000.f;
  Ly.eps = md.rms_eps > 0.f ? md.rms_eps : 1e-6f;
  int64_t o = 0;
  const int64_t d = Ly.d;
  Ly.E = o; o += static_cast<int64_t>(Ly.V) * d;
  for (int l = 0; l < Ly.L; ++l) {
    Ly.g1.push_back(o); o += d;
    Ly.Wqkv.push_back(o); o += d * 3 * d;
    Ly.Wo.push_back(o); o += d * d;
    Ly.g2.push_back(o); o += d;
    Ly.W1.push_back(o); o += d * Ly.F;
    Ly.W2.push_back(o); o += static_cast<int64_t>(Ly.F) * d;
  }
  Ly.gf = o; o += d;
  Ly.Wh = o; o += d * Ly.V;
  return Ly;
}

inline int64_t dec_param_count(const DecLayout& Ly) {
  return Ly.Wh + static_cast<int64_t>(Ly.d) * Ly.V;
}

