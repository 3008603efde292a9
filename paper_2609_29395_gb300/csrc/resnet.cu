// Rounds of the CIFAR ResNet-18 split (architecture 2), grouped over the C
// replicas on the same kernels as the SplitCNN path plus the normalisation
// kernels.
//
// Model (Section V-A's ResNet-18 workload split after stage 1):
//   client: stem conv 3x3 3->64 (no bias) + GroupNorm(32) + ReLU, stage 1
//           (two basic blocks of 64 channels, GroupNorm);
//   server: stages 2-4 (128 / 256 / 512 channels, two basic blocks each, the
//           first with stride 2 and a 1x1 stride-2 convolution + norm on the
//           shortcut), train-mode BatchNorm, global average pool, linear
//           512 -> 10.
//   basic block: out = relu(N2(conv2(relu(N1(conv1(x))))) + s), s = x or
//           Ns(conv_s(x)).
//
// bf16 storage (fp32 accumulation and statistics): the stem input (its
// im2col), every convolution output y, every norm(+residual)+ReLU output,
// the pooled features, the gradient entering the last block, every
// norm-backward output and every block-input gradient.
//
// Backward of a block, given d = dL/d(out):
//   dz  = d [out > 0]                    (norm-2 backward sums; dz kept)
//   dy2 = N2'(dz), dys = Ns'(dz)         (norm backward)
//   dW2 = wgrad(dy2, a1); da1 = dgrad(conv2, dy2) [a1 > 0] (fused mask)
//   dy1 = N1'(da1); dW1 = wgrad(dy1, x); dWs = wgrad(dys, x)
//   dx  = dgrad(conv1, dy1) + dz (identity; fused add), or for stride 2 the
//         four input-pixel parities of dgrad(conv1, dy1), parity (0, 0) also
//         taking the shortcut's dgrad(conv_s, dys) in the same accumulator.
#include <algorithm>
#include <cmath>
#include <functional>

#include "ctx.h"

namespace gcpsl {

struct RnConv {
  int cin, cout, k, stride, hin, win, hout, wout;
  int64_t off_w;                    // kernel layout [co][k*k][ci]
  int bw, hb, bb, tiles_w, tiles_h; // M tile over the output grid
  int bn_f, bkc_f, bn_d, bkc_d, bn_w;
  int whb, wbb, kb_total, kb_per_split, splits;
  CUtensorMap fA, fB, dA, dB, wA, wB;
  // halo-tiled forward / data gradient (3x3 stride 1 on 8 x 16 M tiles,
  // resident weights, N tiles of 64): activation boxes of 10 x 18 pixels
  bool halo_f, halo_d;
  CUtensorMap hfA, hfB, hdA;
  bool wg_halo;                     // weight gradient from halo tiles of x
  CUtensorMap wH;
  float* part;                      // weight-gradient split partials (null: direct)
  const bf16* x;                    // input activation
  bf16* y;                          // output (pre-norm)
  bf16* g;                          // its gradient dL/dy (scratch shared with other layers)
  int stage;                        // 0 stem, 1..4
};

struct RnNorm {
  int ch, gn, hw;
  int64_t off_g, off_b, s_off;      // affine offsets in the blob; BatchNorm state offset
  float* mean;                      // [C][sets]
  float* rstd;
  float2* ss;                       // [C][B or 1][ch] forward affine form
};

struct RnBlock {
  RnConv c1, c2, cs;
  RnNorm n1, n2, ns;
  bool sc;
  bf16 *y1, *a1, *y2, *ys, *out;
};

struct RnState {
  RnConv stem;
  RnNorm stem_n;
  bf16 *ystem, *astem;
  RnBlock blk[8];
  bf16* h;                          // pooled features [C][B][512]
  bf16 *gin[2], *cutg;              // block gradients (ping-pong) and the cut gradient
  bf16 *dz, *dy, *dys, *dt;
  float* sums;
  float4* kk;                       // backward affine form of the norm being differentiated
  float* bn;                        // [C][S_pad] running mean / var per BatchNorm
  int64_t S, S_pad;
  int64_t fcw, fcb, p_client, p_total;
  int J;                            // classes
};

namespace {

constexpr int kStages[4][2] = {{64, 1}, {128, 2}, {256, 2}, {512, 2}};

// parameter and state offsets in the order of PyTorch's named_parameters()
void rn_layout(RnState& r, int J) {
  int64_t p = 0, s = 0;
  r.J = J;
  auto conv = [&](RnConv& c, int cin, int cout, int k, int stride, int hin, int stage) {
    c = RnConv{};
    c.cin = cin; c.cout = cout; c.k = k; c.stride = stride;
    c.hin = c.win = hin; c.hout = c.wout = hin / stride;
    c.off_w = p; p += (int64_t)cout * cin * k * k;
    c.stage = stage;
  };
  auto norm = [&](RnNorm& n, int ch, int gn, int hw) {
    n = RnNorm{};
    n.ch = ch; n.gn = gn; n.hw = hw;
    n.off_g = p; n.off_b = p + ch; p += 2 * ch;
    n.s_off = -1;
    if (!gn) { n.s_off = s; s += 2 * ch; }
  };
  conv(r.stem, 3, 64, 3, 1, 32, 0);
  norm(r.stem_n, 64, 1, 1024);
  int cin = 64, hw = 32;
  for (int st = 0; st < 4; ++st)
    for (int j = 0; j < 2; ++j) {
      RnBlock& b = r.blk[st * 2 + j];
      const int cout = kStages[st][0], stride = j == 0 ? kStages[st][1] : 1, gn = st == 0;
      const int ho = hw / stride;
      conv(b.c1, cin, cout, 3, stride, hw, st + 1);
      norm(b.n1, cout, gn, ho * ho);
      conv(b.c2, cout, cout, 3, 1, ho, st + 1);
      norm(b.n2, cout, gn, ho * ho);
      b.sc = stride != 1 || cin != cout;
      if (b.sc) {
        conv(b.cs, cin, cout, 1, stride, hw, st + 1);
        norm(b.ns, cout, gn, ho * ho);
      }
      if (st == 0 && j == 1) r.p_client = p;
      cin = cout; hw = ho;
    }
  r.fcw = p; p += (int64_t)J * 512;
  r.fcb = p; p += J;
  r.p_total = p;
  r.S = s;
  r.S_pad = (s + 63) / 64 * 64;
}

void for_each_conv(RnState& r, const std::function<void(RnConv&)>& f) {
  f(r.stem);
  for (auto& b : r.blk) {
    f(b.c1); f(b.c2);
    if (b.sc) f(b.cs);
  }
}

// names of the launches in the kernel timer, per stage
const char* const kFwdName[5] = {"rn_conv_fwd.stem", "rn_conv_fwd.s1", "rn_conv_fwd.s2",
                                 "rn_conv_fwd.s3", "rn_conv_fwd.s4"};
const char* const kDgradName[5] = {"rn_conv_dgrad.stem", "rn_conv_dgrad.s1", "rn_conv_dgrad.s2",
                                   "rn_conv_dgrad.s3", "rn_conv_dgrad.s4"};
const char* const kWgradName[5] = {"rn_conv_wgrad.stem", "rn_conv_wgrad.s1", "rn_conv_wgrad.s2",
                                   "rn_conv_wgrad.s3", "rn_conv_wgrad.s4"};

// GroupNorm statistics keep a stride of 32 sets per example (the most groups)
int64_t sets_of(const RnNorm& n, int B) { return n.gn ? (int64_t)B * 32 : n.ch; }

}  // namespace

int64_t rn_num_params(int J, int segment) {
  RnState r;
  rn_layout(r, J);
  if (segment == GCPSL_CLIENT) return r.p_client;
  if (segment == GCPSL_SERVER) return r.p_total - r.p_client;
  if (segment == GCPSL_BN_STATE) return r.S;
  return -1;
}

// canonical (OIHW) <-> kernel ([co][ky][kx][ci]) conv weights; the rest is
// copied unchanged
void rn_to_kernel_layout(int J, const float* can, float* ker) {
  RnState r;
  rn_layout(r, J);
  std::memcpy(ker, can, sizeof(float) * (size_t)r.p_total);
  for_each_conv(r, [&](RnConv& c) {
    const int kk = c.k * c.k;
    for (int co = 0; co < c.cout; ++co)
      for (int ci = 0; ci < c.cin; ++ci)
        for (int t = 0; t < kk; ++t)
          ker[c.off_w + ((int64_t)co * kk + t) * c.cin + ci] =
              can[c.off_w + ((int64_t)co * c.cin + ci) * kk + t];
  });
}

void rn_to_canonical_layout(int J, const float* ker, float* can) {
  RnState r;
  rn_layout(r, J);
  std::memcpy(can, ker, sizeof(float) * (size_t)r.p_total);
  for_each_conv(r, [&](RnConv& c) {
    const int kk = c.k * c.k;
    for (int co = 0; co < c.cout; ++co)
      for (int ci = 0; ci < c.cin; ++ci)
        for (int t = 0; t < kk; ++t)
          can[c.off_w + ((int64_t)co * c.cin + ci) * kk + t] =
              ker[c.off_w + ((int64_t)co * kk + t) * c.cin + ci];
  });
}

// PyTorch-style initial parameters: conv / linear weights U(+-1/sqrt(fan_in)),
// linear bias likewise, norm weight 1 and bias 0 (deterministic LCG stream)
void rn_seeded_init(int J, uint64_t seed, float* can) {
  RnState r;
  rn_layout(r, J);
  uint64_t st = seed * 6364136223846793005ull + 1442695040888963407ull;
  auto uni = [&](float bound) {
    st = st * 6364136223846793005ull + 1442695040888963407ull;
    const double u = (double)(st >> 11) * (1.0 / 9007199254740992.0);
    return (float)((2.0 * u - 1.0) * bound);
  };
  for (int64_t i = 0; i < r.p_total; ++i) can[i] = 0.f;
  for_each_conv(r, [&](RnConv& c) {
    const float b = 1.f / std::sqrt((float)(c.cin * c.k * c.k));
    for (int64_t i = 0; i < (int64_t)c.cout * c.cin * c.k * c.k; ++i) can[c.off_w + i] = uni(b);
  });
  auto ones = [&](const RnNorm& n) { for (int i = 0; i < n.ch; ++i) can[n.off_g + i] = 1.f; };
  ones(r.stem_n);
  for (auto& b : r.blk) {
    ones(b.n1); ones(b.n2);
    if (b.sc) ones(b.ns);
  }
  const float bf = 1.f / std::sqrt(512.f);
  for (int i = 0; i < J * 512; ++i) can[r.fcw + i] = uni(bf);
  for (int i = 0; i < J; ++i) can[r.fcb + i] = uni(bf);
}

void rn_free(gcpsl_ctx* c) {
  delete c->rn;
  c->rn = nullptr;
}

// buffers, tile shapes and tensor maps of every layer
gcpsl_status rn_setup(gcpsl_ctx* c) {
  c->rn = new (std::nothrow) RnState();
  if (!c->rn) return fail(c, GCPSL_E_NOMEM, "host allocation failed");
  RnState& r = *c->rn;
  rn_layout(r, c->J);
  // the GroupNorm layers take the context's group count
  r.stem_n.gn = c->gn_groups;
  for (auto& b : r.blk)
    for (RnNorm* n : {&b.n1, &b.n2, &b.ns})
      if (n->gn) n->gn = c->gn_groups;
  const int C = c->C, B = c->B;
  const int64_t P = c->P_pad;
  auto act = [&](bf16*& p, int64_t elems) -> gcpsl_status {
    DALLOC(p, sizeof(bf16) * (size_t)(C * B * elems));
    return GCPSL_OK;
  };
  // activations of one round
  gcpsl_status st;
#define RN_ACT(p, e) do { st = act(p, e); if (st != GCPSL_OK) return st; } while (0)
  RN_ACT(r.ystem, 64 * 1024);
  RN_ACT(r.astem, 64 * 1024);
  const int64_t big = 64 * 1024;                    // largest activation per example
  for (auto& b : r.blk) {
    const int64_t e = (int64_t)b.c1.cout * b.c1.hout * b.c1.wout;
    RN_ACT(b.y1, e); RN_ACT(b.a1, e); RN_ACT(b.y2, e); RN_ACT(b.out, e);
    if (b.sc) RN_ACT(b.ys, e);
  }
  RN_ACT(r.h, 512);
  RN_ACT(r.gin[0], big); RN_ACT(r.gin[1], big); RN_ACT(r.cutg, big);
  RN_ACT(r.dz, big); RN_ACT(r.dy, big); RN_ACT(r.dys, big); RN_ACT(r.dt, big);
#undef RN_ACT
  auto stats = [&](RnNorm& n) -> gcpsl_status {
    const int64_t sets = sets_of(n, B);
    DALLOC(n.mean, sizeof(float) * (size_t)(C * sets));
    DALLOC(n.rstd, sizeof(float) * (size_t)(C * sets));
    DALLOC(n.ss, sizeof(float2) * (size_t)C * (n.gn ? B : 1) * n.ch);
    return GCPSL_OK;
  };
  if ((st = stats(r.stem_n)) != GCPSL_OK) return st;
  for (auto& b : r.blk) {
    if ((st = stats(b.n1)) != GCPSL_OK) return st;
    if ((st = stats(b.n2)) != GCPSL_OK) return st;
    if (b.sc && (st = stats(b.ns)) != GCPSL_OK) return st;
  }
  DALLOC(r.kk, sizeof(float4) * (size_t)C * B * 512);
  DALLOC(r.sums, sizeof(float) * (size_t)C * B * 512 * 2);
  // BatchNorm running statistics: mean 0, variance 1
  DALLOC(r.bn, sizeof(float) * (size_t)(C * r.S_pad));
  {
    std::vector<float> h((size_t)(C * r.S_pad), 0.f);
    auto init = [&](const RnNorm& n) {
      if (n.gn) return;
      for (int k = 0; k < C; ++k)
        for (int i = 0; i < n.ch; ++i) h[(size_t)(k * r.S_pad + n.s_off + n.ch + i)] = 1.f;
    };
    for (auto& b : r.blk) { init(b.n1); init(b.n2); if (b.sc) init(b.ns); }
    CK(cudaMemcpy(r.bn, h.data(), sizeof(float) * h.size(), cudaMemcpyHostToDevice));
  }

  // wiring: inputs, outputs and gradient buffers of every convolution
  r.stem.x = (const bf16*)c->d_act[0];
  r.stem.y = r.ystem;
  r.stem.g = r.dy;
  const bf16* x = r.astem;
  for (auto& b : r.blk) {
    b.c1.x = x; b.c1.y = b.y1; b.c1.g = r.dy;
    b.c2.x = b.a1; b.c2.y = b.y2; b.c2.g = r.dy;
    if (b.sc) { b.cs.x = x; b.cs.y = b.ys; b.cs.g = r.dys; }
    x = b.out;
  }

  // tensor maps
  auto setup = [&](RnConv& v, bool im2col) -> gcpsl_status {
    if (!m_tile(v.wout, v.hout, v.bw, v.hb, v.bb))
      return fail(c, GCPSL_E_UNSUPPORTED, "no M tile for a %dx%d output", v.wout, v.hout);
    v.tiles_w = v.wout / v.bw;
    v.tiles_h = v.hout / v.hb;
    const int cin_op = im2col ? 32 : v.cin;          // channels of the A operand
    v.bn_f = std::min(v.cout, 256);
    v.bkc_f = std::min(cin_op, 64);
    v.bn_d = std::min(v.cin, 256);
    v.bkc_d = std::min(v.cout, 64);
    v.bn_w = std::min(v.cin, 128);
    const uint64_t rs = (uint64_t)P * 2;
    const uint32_t s = (uint32_t)v.stride;
    const uint32_t es[5] = {1, s, s, 1, 1};
    const uint64_t xd[5] = {(uint64_t)cin_op, (uint64_t)v.win, (uint64_t)v.hin, (uint64_t)B,
                            (uint64_t)C};
    const uint64_t gd[5] = {(uint64_t)v.cout, (uint64_t)v.wout, (uint64_t)v.hout, (uint64_t)B,
                            (uint64_t)C};
    const uint64_t wd[4] = {(uint64_t)v.cin, (uint64_t)(v.k * v.k), (uint64_t)v.cout, (uint64_t)C};
    const uint32_t fa[5] = {(uint32_t)v.bkc_f, s * v.bw, s * v.hb, (uint32_t)v.bb, 1};
    bool ok;
    if (im2col) {
      const uint64_t w0d[4] = {32, 1, (uint64_t)v.cout, (uint64_t)C};
      const uint32_t w0b[4] = {32, 1, (uint32_t)v.cout, 1};
      ok = tensor_map_bf16(&v.fA, v.x, 5, xd, fa, 64, es) &&
           tensor_map_bf16(&v.fB, c->d_w0p, 4, w0d, w0b, 64);
    } else {
      const uint32_t fb[4] = {(uint32_t)v.bkc_f, 1, (uint32_t)v.bn_f, 1};
      const int nbw = std::min(v.bn_d, 64);
      const uint32_t da[5] = {(uint32_t)v.bkc_d, (uint32_t)v.bw, (uint32_t)v.hb, (uint32_t)v.bb, 1};
      const uint32_t db[4] = {(uint32_t)nbw, 1, (uint32_t)v.bkc_d, 1};
      ok = tensor_map_bf16(&v.fA, v.x, 5, xd, fa, v.bkc_f * 2, es) &&
           tensor_map_bf16_strided(&v.fB, c->d_shadow + v.off_w, 4, wd, rs, fb, v.bkc_f * 2) &&
           tensor_map_bf16(&v.dA, v.g, 5, gd, da, v.bkc_d * 2) &&
           tensor_map_bf16_strided(&v.dB, c->d_shadow + v.off_w, 4, wd, rs, db, nbw * 2);
    }
    // weight gradient: 64-pixel K blocks of the output grid
    v.whb = std::min(v.hout, 64 / v.wout);
    v.wbb = v.whb > 0 ? 64 / (v.wout * v.whb) : 0;
    if (v.wout * v.whb * v.wbb != 64 || v.hout % v.whb)
      return fail(c, GCPSL_E_UNSUPPORTED, "no weight-gradient K block for %dx%d", v.wout, v.hout);
    v.kb_total = ((B + v.wbb - 1) / v.wbb) * (v.hout / v.whb);
    int tiles;
    v.wg_halo = !im2col && v.whb * v.wout == 64 &&
                wgrad_halo_supported(v.hout, v.wout, v.cin, v.cout, v.k * v.k, v.stride);
    if (im2col) {
      tiles = 1;
    } else if (v.wg_halo) {
      tiles = wgrad_halo_tiles(v.cin, v.cout);
    } else {
      tiles = wgrad_tc_tiles(v.cin, v.cout, v.k * v.k, v.bn_w);
    }
    // per-replica shape only: C grouped replicas equal C one-replica runs
    const int64_t per = im2col ? (int64_t)v.cout * 27 + v.cout
                               : (int64_t)v.cout * v.k * v.k * v.cin;
    int splits = wgrad_splits(tiles, v.kb_total, per);
    if (im2col) splits = std::max(1, std::min(64, (v.kb_total + 15) / 16));
    v.kb_per_split = (v.kb_total + splits - 1) / splits;
    v.splits = (v.kb_total + v.kb_per_split - 1) / v.kb_per_split;
    // several splits write partials that the update sums; the stem's
    // partial also holds its ones-column sums (no parameter), so it always
    // goes through one
    v.part = nullptr;
    if (im2col || v.splits > 1 || v.off_w % 4) {
      v.part = partial_range(c, v.off_w, im2col ? (int64_t)v.cout * 27 : per, per, v.splits);
      if (!v.part) return fail(c, GCPSL_E_NOMEM, "device allocation failed");
    }
    const uint32_t wa[5] = {64, (uint32_t)v.wout, (uint32_t)v.whb, (uint32_t)v.wbb, 1};
    if (im2col) {
      const uint32_t wa0[5] = {(uint32_t)v.cout, (uint32_t)v.wout, (uint32_t)v.whb, 1, 1};
      const uint32_t xb0[5] = {32, (uint32_t)v.wout, (uint32_t)v.whb, 1, 1};
      ok = ok && tensor_map_bf16(&v.wA, v.g, 5, gd, wa0, v.cout * 2) &&
           tensor_map_bf16(&v.wB, v.x, 5, xd, xb0, 64);
    } else {
      if (v.wg_halo) {
        const int cb = v.cin == 32 ? 32 : 64;
        const int hrows = wgrad_halo_rows(v.cin) == 3 ? v.whb + 2 : v.whb;
        const uint32_t hx[5] = {(uint32_t)cb, (uint32_t)v.wout + 2, (uint32_t)hrows, 1, 1};
        ok = ok && tensor_map_bf16(&v.wH, v.x, 5, xd, hx, cb * 2);
      }
      const int wx = std::min(v.cin, 64);
      const uint32_t wb[5] = {(uint32_t)wx, s * v.wout, s * v.whb, (uint32_t)v.wbb, 1};
      ok = ok && tensor_map_bf16(&v.wA, v.g, 5, gd, wa, 128) &&
           tensor_map_bf16(&v.wB, v.x, 5, xd, wb, wx * 2, es);
    }
    v.halo_f = v.halo_d = false;
    if (!im2col && v.k == 3 && v.stride == 1) {
      v.halo_f = halo_supported(v.hout, v.wout, v.cin, 64, 64, EPI_STORE);
      v.halo_d = halo_supported(v.hout, v.wout, v.cout, 64, 64, EPI_DRELU) &&
                 halo_supported(v.hout, v.wout, v.cout, 64, 64, EPI_ADD);
      const uint32_t hb[5] = {64, 10, 18, 1, 1};
      const uint32_t hw[4] = {64, 1, 64, 1};
      if (v.halo_f)
        ok = ok && tensor_map_bf16(&v.hfA, v.x, 5, xd, hb, 128) &&
             tensor_map_bf16_strided(&v.hfB, c->d_shadow + v.off_w, 4, wd, rs, hw, 128);
      if (v.halo_d) ok = ok && tensor_map_bf16(&v.hdA, v.g, 5, gd, hb, 128);
    }
    if (!ok) return fail(c, GCPSL_E_CUDA, "cuTensorMapEncodeTiled failed (stage %d conv)", v.stage);
    return GCPSL_OK;
  };
  if ((st = setup(r.stem, true)) != GCPSL_OK) return st;
  for (auto& b : r.blk) {
    if ((st = setup(b.c1, false)) != GCPSL_OK) return st;
    if ((st = setup(b.c2, false)) != GCPSL_OK) return st;
    if (b.sc && (st = setup(b.cs, false)) != GCPSL_OK) return st;
  }
  return GCPSL_OK;
}

namespace {

// M tiles of the halo-tiled kernel: 8 columns x 16 rows of one image
void halo_tiles(ConvTcArgs& p, const RnConv& v) {
  p.bw = 8;
  p.hb = 16;
  p.bb = 1;
  p.tiles_w = v.wout / 8;
  p.tiles_h = v.hout / 16;
}

// forward convolution: raw bf16 output (the norm follows)
gcpsl_status conv_fwd(gcpsl_ctx* c, const RnConv& v, bool im2col) {
  ConvTcArgs p{v.hout, v.wout, c->B, im2col ? 32 : v.cin, v.bw, v.hb, v.bb, v.tiles_w,
               v.tiles_h, v.cout, nullptr, 0, v.y, nullptr, c->d_err};
  if (v.k == 3 && !im2col) conv_taps_fwd3(p);
  else conv_taps_one(p);                         // 1x1, or the stem's im2col (K = 32)
  p.stride = v.stride;
  if (v.halo_f) {
    halo_tiles(p, v);
    LAUNCH(kFwdName[v.stage], launch_conv_halo(c->stream, v.hfA, v.hfB, p, 64, 64, EPI_STORE,
                                               c->C));
    return GCPSL_OK;
  }
  LAUNCH(kFwdName[v.stage], launch_conv_tc(c->stream, v.fA, v.fB, p, v.bn_f, v.bkc_f, EPI_STORE,
                                           c->C));
  return GCPSL_OK;
}

gcpsl_status conv_wgrad(gcpsl_ctx* c, const RnConv& v) {
  WgradTcArgs w{v.hout, v.wout, c->B, v.cout, v.cin, v.whb, v.wbb, v.kb_total, v.kb_per_split,
                v.splits, v.part, c->d_err};
  w.taps = v.k * v.k;
  w.bias = 0;
  w.stride = v.stride;
  w.pad = v.k / 2;
  // a single split writes the gradient directly; several write the layer's
  // partials, which the update sums
  if (!v.part) {
    w.out = c->d_grad + v.off_w;
    w.out_rs = c->P_pad;
  }
  if (v.wg_halo)
    LAUNCH(kWgradName[v.stage], launch_wgrad_halo(c->stream, v.wA, v.wH, w, c->C));
  else
    LAUNCH(kWgradName[v.stage], launch_wgrad_tc(c->stream, v.wA, v.wB, w, v.bn_w, c->C));
  return GCPSL_OK;
}

gcpsl_status norm_stats(gcpsl_ctx* c, const RnNorm& n, const bf16* y) {
  RnState& r = *c->rn;
  const float* th = c->d_theta;
  LAUNCH("rn_norm_sums", launch_norm_sums(c->stream, false, y, nullptr, nullptr, nullptr,
                                          nullptr, nullptr, r.sums, c->C, c->B, n.hw, n.ch,
                                          n.gn));
  LAUNCH("rn_norm_finalize",
         launch_norm_finalize_fwd(c->stream, r.sums, th + n.off_g, th + n.off_b, c->P_pad, n.mean,
                                  n.rstd, n.ss, n.gn ? nullptr : r.bn + n.s_off, r.S_pad, c->C,
                                  c->B, n.hw, n.ch, n.gn, c->norm_eps, c->bn_momentum,
                                  c->d_upd));
  return GCPSL_OK;
}

// GroupNorm forward in one launch per layer: out = relu(norm(y) + res)
gcpsl_status gn_fwd(gcpsl_ctx* c, const RnNorm& n, const bf16* y, const bf16* res, bf16* out) {
  const float* th = c->d_theta;
  LAUNCH("rn_norm_gn", launch_gn_fused_fwd(c->stream, y, res, th + n.off_g, th + n.off_b,
                                           c->P_pad, n.mean, n.rstd, out, c->C, c->B, n.hw, n.ch,
                                           1, n.gn, c->norm_eps, c->d_err));
  return GCPSL_OK;
}

// dy = N'(dz) for dz = d [mask > 0] (mask nullable); dz_out (nullable)
// keeps dz; affine gradients go to the gradient store
gcpsl_status norm_bwd(gcpsl_ctx* c, const RnNorm& n, const bf16* y, const bf16* d,
                      const bf16* mask, bf16* dz_out, bf16* dy) {
  RnState& r = *c->rn;
  const float* th = c->d_theta;
  if (n.gn) {
    // one example per block: sums, the per-set affine form and dy together;
    // then dgamma / dbeta over the batch
    LAUNCH("rn_norm_gn_bwd",
           launch_gn_fused_bwd(c->stream, y, d, mask, dz_out, th + n.off_g, c->P_pad, n.mean,
                               n.rstd, r.sums, dy, c->C, c->B, n.hw, n.ch, n.gn, c->d_err));
    LAUNCH("rn_norm_bwd_finalize",
           launch_norm_finalize_bwd_channels(c->stream, r.sums, c->d_grad + n.off_g,
                                             c->d_grad + n.off_b, c->P_pad, c->C, c->B, n.ch));
    return GCPSL_OK;
  }
  LAUNCH("rn_norm_bwd_sums", launch_norm_sums(c->stream, true, y, d, mask, n.mean, n.rstd,
                                              dz_out, r.sums, c->C, c->B, n.hw, n.ch, n.gn));
  LAUNCH("rn_norm_bwd_finalize",
         launch_norm_finalize_bwd(c->stream, r.sums, th + n.off_g, c->P_pad, n.mean, n.rstd, r.kk,
                                  c->d_grad + n.off_g, c->d_grad + n.off_b, c->P_pad, c->C, c->B,
                                  n.hw, n.ch, n.gn));
  LAUNCH("rn_norm_bwd_apply",
         launch_norm_apply_bwd(c->stream, y, r.kk, n.gn, dz_out ? dz_out : d,
                               dz_out ? nullptr : mask, dy, c->C, c->B, n.hw, n.ch));
  return GCPSL_OK;
}

}  // namespace

// One local round of every cluster (after sampling and the gather).
gcpsl_status rn_enqueue_round(gcpsl_ctx* c) {
  RnState& r = *c->rn;
  cudaStream_t s = c->stream;
  const int C = c->C, B = c->B;
  const int64_t P = c->P_pad;
  const float* th = c->d_theta;
  gcpsl_status st;
#define RN(call) do { st = (call); if (st != GCPSL_OK) return st; } while (0)

  // ---- forward ----
  RN(conv_fwd(c, r.stem, true));
  RN(gn_fwd(c, r.stem_n, r.ystem, nullptr, r.astem));
  for (auto& b : r.blk) {
    RN(conv_fwd(c, b.c1, false));
    if (b.n1.gn) {
      RN(gn_fwd(c, b.n1, b.y1, nullptr, b.a1));
    } else {
      RN(norm_stats(c, b.n1, b.y1));
      LAUNCH("rn_norm_apply", launch_norm_apply_fwd(s, b.y1, b.n1.ss, 0, nullptr, nullptr,
                                                    nullptr, 0, b.a1, C, B, b.n1.hw, b.n1.ch, 1));
    }
    RN(conv_fwd(c, b.c2, false));
    if (b.n2.gn && !b.sc) {
      RN(gn_fwd(c, b.n2, b.y2, b.c1.x, b.out));       // + the identity shortcut
      continue;
    }
    RN(norm_stats(c, b.n2, b.y2));
    if (b.sc) {
      RN(conv_fwd(c, b.cs, false));
      RN(norm_stats(c, b.ns, b.ys));
    }
    LAUNCH("rn_norm_apply",
           launch_norm_apply_fwd(s, b.y2, b.n2.ss, b.n2.gn, b.sc ? nullptr : b.c1.x,
                                 b.sc ? b.ys : nullptr, b.sc ? b.ns.ss : nullptr, b.ns.gn, b.out, C,
                                 B, b.n2.hw, b.n2.ch, 1));
  }
  LAUNCH("rn_avgpool", launch_avgpool(s, r.blk[7].out, r.h, C * B, 16, 512));
  LAUNCH("fc_fwd_ce", launch_fc_fwd_ce<bf16>(s, r.h, c->d_shadow + r.fcw, P, th + r.fcb, P,
                                              c->d_y, c->d_loss_ex, c->d_dlogits, C, B, 512, r.J,
                                              c->desc.label_smoothing));
  // ---- backward ----
  bf16* d = r.gin[1];
  LAUNCH("fc_bwd", launch_fc_bwd<bf16>(s, c->d_dlogits, c->d_loss_ex, r.h, c->d_shadow + r.fcw, P,
                                        c->d_grad + r.fcw, c->d_grad + r.fcb, P, d, c->d_loss, C,
                                        B, 512, r.J, FC_DH_AVG, nullptr, nullptr, 4, 4, 512));
  if (fc_bwd_split_dh(r.J))
    LAUNCH("fc_bwd_dh", launch_fc_bwd_dh<bf16>(s, c->d_dlogits, c->d_shadow + r.fcw, P, d, C, B,
                                                512, r.J, FC_DH_AVG, nullptr, nullptr, 4, 4, 512));
  for (int i = 7; i >= 0; --i) {
    RnBlock& b = r.blk[i];
    bf16* dx = i == 2 ? r.cutg : (d == r.gin[1] ? r.gin[0] : r.gin[1]);
    // through the output ReLU and norm 2 (dz kept for the shortcut)
    RN(norm_bwd(c, b.n2, b.y2, d, b.out, r.dz, r.dy));
    if (b.sc) {
      RN(norm_bwd(c, b.ns, b.ys, r.dz, nullptr, nullptr, r.dys));
      RN(conv_wgrad(c, b.cs));
    }
    RN(conv_wgrad(c, b.c2));
    {
      ConvTcArgs p{b.c2.hout, b.c2.wout, B, b.c2.cout, b.c2.bw, b.c2.hb, b.c2.bb, b.c2.tiles_w,
                   b.c2.tiles_h, b.c2.cin, nullptr, 0, nullptr, nullptr, c->d_err, b.a1, r.dt};
      conv_taps_dgrad3(p);
      if (b.c2.halo_d) {
        halo_tiles(p, b.c2);
        LAUNCH(kDgradName[b.c2.stage], launch_conv_halo(s, b.c2.hdA, b.c2.dB, p, 64, 64,
                                                        EPI_DRELU, C));
      } else {
        LAUNCH(kDgradName[b.c2.stage], launch_conv_tc(s, b.c2.dA, b.c2.dB, p, b.c2.bn_d,
                                                      b.c2.bkc_d, EPI_DRELU, C));
      }
    }
    RN(norm_bwd(c, b.n1, b.y1, r.dt, nullptr, nullptr, r.dy));
    RN(conv_wgrad(c, b.c1));
    const RnConv& v = b.c1;
    if (!b.sc) {
      ConvTcArgs p{v.hout, v.wout, B, v.cout, v.bw, v.hb, v.bb, v.tiles_w, v.tiles_h, v.cin,
                   nullptr, 0, dx, nullptr, c->d_err};
      conv_taps_dgrad3(p);
      p.res = r.dz;
      if (v.halo_d) {
        halo_tiles(p, v);
        LAUNCH(kDgradName[v.stage], launch_conv_halo(s, v.hdA, v.dB, p, 64, 64, EPI_ADD, C));
      } else {
        LAUNCH(kDgradName[v.stage], launch_conv_tc(s, v.dA, v.dB, p, v.bn_d, v.bkc_d, EPI_ADD,
                                                   C));
      }
    } else {
      for (int py = 0; py < 2; ++py)
        for (int px = 0; px < 2; ++px) {
          ConvTcArgs p{v.hout, v.wout, B, v.cout, v.bw, v.hb, v.bb, v.tiles_w, v.tiles_h, v.cin,
                       nullptr, 0, dx, nullptr, c->d_err};
          conv_taps_dgrad3_s2(p, py, px, true);
          p.out_H = v.hin;
          p.out_W = v.win;
          LAUNCH(kDgradName[v.stage], launch_conv_tc(s, v.dA, v.dB, p, v.bn_d, v.bkc_d,
                                                     EPI_DSTORE, C, &b.cs.dA, &b.cs.dB));
        }
    }
    d = dx;
    if (i == 2 && c->desc.client_average)
      // the per-client average: the cut gradient, per example by B / (|A| b_k)
      LAUNCH("client_avg", launch_client_avg_scale<bf16>(s, r.cutg, (int64_t)64 * 32 * 32,
                                                         (bf16*)nullptr, 0, c->d_cut_scale,
                                                         C * B));
  }
  // stem: its ReLU and GroupNorm, then the weight gradient over the im2col
  RN(norm_bwd(c, r.stem_n, r.ystem, d, r.astem, nullptr, r.dy));
  {
    const RnConv& v = r.stem;
    WgradTcArgs w{v.hout, v.wout, B, v.cout, 3, v.whb, v.wbb, v.kb_total, v.kb_per_split, v.splits,
                  v.part, c->d_err};
    // weights only: the update skips the ones column's sums (a bias
    // gradient, not a parameter here)
    LAUNCH(kWgradName[0], launch_wgrad0_tc(s, v.wA, v.wB, w, C));
  }
#undef RN
  return GCPSL_OK;
}

// ReLU decisions of the last round, [C][B][E] bytes, per example the stem's
// then every block's a1 and output, each in NCHW order: 1 where the stored
// value (the ReLU output) is positive
gcpsl_status rn_relu_masks(gcpsl_ctx* c, uint8_t* dst, size_t len, size_t* needed) {
  RnState& r = *c->rn;
  const int64_t CB = (int64_t)c->C * c->B;
  struct Src { const bf16* p; int ch, hw; };
  std::vector<Src> srcs;
  srcs.push_back({r.astem, 64, 1024});
  for (auto& b : r.blk) {
    const int hw = b.c1.hout * b.c1.wout;
    srcs.push_back({b.a1, b.c1.cout, hw});
    srcs.push_back({b.out, b.c1.cout, hw});
  }
  int64_t E = 0;
  for (auto& q : srcs) E += (int64_t)q.ch * q.hw;
  if (needed) *needed = (size_t)(CB * E);
  if (!dst) return GCPSL_OK;
  if (len < (size_t)(CB * E)) return fail(c, GCPSL_E_INVAL, "dst too small");
  SYNC_CHECK(c);
  int64_t off = 0;
  for (auto& q : srcs) {
    const int64_t per = (int64_t)q.ch * q.hw;
    std::vector<uint16_t> h((size_t)(CB * per));
    CK(cudaMemcpy(h.data(), q.p, sizeof(uint16_t) * h.size(), cudaMemcpyDeviceToHost));
    for (int64_t cb = 0; cb < CB; ++cb)
      for (int p = 0; p < q.hw; ++p)
        for (int k = 0; k < q.ch; ++k) {
          const uint16_t v = h[(size_t)((cb * q.hw + p) * q.ch + k)];
          dst[cb * E + off + (int64_t)k * q.hw + p] = (uint8_t)(v != 0 && !(v & 0x8000u));
        }
    off += per;
  }
  return GCPSL_OK;
}

// cut tensors (NHWC bf16 [C][B][32][32][64]) for the getters
const bf16* rn_cut(const gcpsl_ctx* c, int which) {
  return which == GCPSL_CUT_ACT ? c->rn->blk[1].out : c->rn->cutg;
}

float* rn_bn_state(const gcpsl_ctx* c, int64_t* S, int64_t* S_pad) {
  *S = c->rn->S;
  *S_pad = c->rn->S_pad;
  return c->rn->bn;
}

}  // namespace gcpsl
