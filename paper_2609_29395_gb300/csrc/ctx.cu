// Host side of libgcpsl.so: the C ABI declared in include/gcpsl.h.
//
// A context holds C cluster workloads (the paper's N execution slots,
// Section III-A) resident on one GPU: every replica's fp32 parameters,
// momentum and gradients as one [C][P] store, the bf16 operand shadow, the
// activations of the current round as [C][B][H][W][ch] tensors, the sampler
// state, and the dataset.  gcpsl_step enqueues one local round of every
// cluster (Algorithm 2's inner loop body) as grouped kernels on one stream.
#include <algorithm>
#include <cmath>

#include "ctx.h"

using namespace gcpsl;

// ---------------------------------------------------------------------------
// Architectures
// ---------------------------------------------------------------------------
bool gcpsl::make_arch(int id, ArchSpec* a) {
  std::memset(a, 0, sizeof(*a));
  if (id == GCPSL_TINY_CNN) {
    a->ncl = 1; a->nsv = 1;
    a->conv[0] = {3, 16, 32, 32, 1};
    a->conv[1] = {16, 32, 16, 16, 1};
  } else if (id == GCPSL_SPLIT_CNN) {
    a->ncl = 2; a->nsv = 2;
    a->conv[0] = {3, 32, 32, 32, 0};
    a->conv[1] = {32, 64, 32, 32, 1};
    a->conv[2] = {64, 128, 16, 16, 1};
    a->conv[3] = {128, 128, 8, 8, 1};
  } else {
    return false;
  }
  a->fc_in = 2048; a->fc_out = 10;
  int64_t p = 0;
  for (int i = 0; i < a->L(); ++i) {
    if (i == a->ncl) a->p_client = p;
    a->off_w[i] = p; p += (int64_t)a->conv[i].cout * 9 * a->conv[i].cin;
    a->off_b[i] = p; p += a->conv[i].cout;
  }
  a->off_fcw = p; p += (int64_t)a->fc_out * a->fc_in;
  a->off_fcb = p; p += a->fc_out;
  a->p_total = p;
  return true;
}

namespace {

// classes of a ResNet-18 split architecture, 0 for any other id
int resnet_classes(int arch) {
  return arch == GCPSL_RESNET18 ? 10 : arch == GCPSL_RESNET18_C100 ? 100 : 0;
}

// classes of any built architecture, 0 for an unknown id
int arch_classes(int arch) {
  if (resnet_classes(arch)) return resnet_classes(arch);
  ArchSpec a;
  return make_arch(arch, &a) ? a.fc_out : 0;
}

thread_local std::string g_init_error;

}  // namespace

void gcpsl::set_global_error(const char* msg) { g_init_error = msg; }

gcpsl_status gcpsl::fail(gcpsl_ctx* c, gcpsl_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (c) {
    c->err = buf;
    if (st == GCPSL_E_CUDA || st == GCPSL_E_TIMEOUT) c->sticky = st;
  } else {
    g_init_error = buf;
  }
  return st;
}


namespace {

// canonical (PyTorch) <-> kernel layout of one replica's parameters.
// conv weight: OIHW <-> [co][kh][kw][ci]; linear weight: input index
// ch*HoWo + h*Wo + w <-> (h*Wo + w)*ch + ch_idx.
void to_kernel_layout(const ArchSpec& a, const float* can, float* ker) {
  std::memcpy(ker, can, sizeof(float) * (size_t)a.p_total);
  for (int i = 0; i < a.L(); ++i) {
    const ConvSpec& s = a.conv[i];
    const float* src = can + a.off_w[i];
    float* dst = ker + a.off_w[i];
    for (int co = 0; co < s.cout; ++co)
      for (int ci = 0; ci < s.cin; ++ci)
        for (int t = 0; t < 9; ++t)
          dst[((int64_t)co * 9 + t) * s.cin + ci] = src[((int64_t)co * s.cin + ci) * 9 + t];
  }
  const int l = a.L() - 1, ch = a.conv[l].cout, hw = a.out_h(l) * a.out_w(l);
  for (int j = 0; j < a.fc_out; ++j)
    for (int cc = 0; cc < ch; ++cc)
      for (int p = 0; p < hw; ++p)
        ker[a.off_fcw + (int64_t)j * a.fc_in + (int64_t)p * ch + cc] =
            can[a.off_fcw + (int64_t)j * a.fc_in + (int64_t)cc * hw + p];
}

void to_canonical_layout(const ArchSpec& a, const float* ker, float* can) {
  std::memcpy(can, ker, sizeof(float) * (size_t)a.p_total);
  for (int i = 0; i < a.L(); ++i) {
    const ConvSpec& s = a.conv[i];
    const float* src = ker + a.off_w[i];
    float* dst = can + a.off_w[i];
    for (int co = 0; co < s.cout; ++co)
      for (int ci = 0; ci < s.cin; ++ci)
        for (int t = 0; t < 9; ++t)
          dst[((int64_t)co * s.cin + ci) * 9 + t] = src[((int64_t)co * 9 + t) * s.cin + ci];
  }
  const int l = a.L() - 1, ch = a.conv[l].cout, hw = a.out_h(l) * a.out_w(l);
  for (int j = 0; j < a.fc_out; ++j)
    for (int cc = 0; cc < ch; ++cc)
      for (int p = 0; p < hw; ++p)
        can[a.off_fcw + (int64_t)j * a.fc_in + (int64_t)cc * hw + p] =
            ker[a.off_fcw + (int64_t)j * a.fc_in + (int64_t)p * ch + cc];
}

// U(-1/sqrt(fan_in), 1/sqrt(fan_in)) from Philox(counter = (p, 0, 0, 0x5eed))
void seeded_init(const ArchSpec& a, uint64_t seed, float* can) {
  auto fill = [&](int64_t off, int64_t cnt, int64_t fan_in) {
    const float bound = 1.0f / std::sqrt((float)fan_in);
    for (int64_t p = off; p < off + cnt; ++p) {
      uint32_t ctr[4] = {(uint32_t)p, (uint32_t)(p >> 32), 0u, 0x5eedu};
      philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32));
      const float u = (float)(ctr[0] >> 8) * (1.0f / 16777216.0f);
      can[p] = (2.0f * u - 1.0f) * bound;
    }
  };
  for (int i = 0; i < a.L(); ++i) {
    const int64_t fan = (int64_t)a.conv[i].cin * 9;
    fill(a.off_w[i], (int64_t)a.conv[i].cout * fan, fan);
    fill(a.off_b[i], a.conv[i].cout, fan);
  }
  fill(a.off_fcw, (int64_t)a.fc_out * a.fc_in, a.fc_in);
  fill(a.off_fcb, a.fc_out, a.fc_in);
}

}  // namespace

gcpsl_status gcpsl::check_usable(gcpsl_ctx* c) {
  if (!c) return GCPSL_E_INVAL;
  if (c->sticky != GCPSL_OK) return GCPSL_E_STATE;
  return GCPSL_OK;
}

namespace {

int64_t act_elems(const gcpsl_ctx* c, int i) {   // elements of d_act[i]
  if (i == 0) return (int64_t)c->C * c->B * 1024 * c->x0c;
  const int l = i - 1;
  return (int64_t)c->C * c->B * c->a.out_h(l) * c->a.out_w(l) * c->a.conv[l].cout;
}

// ---------------------------------------------------------------------------
// One local round of every cluster
// ---------------------------------------------------------------------------
// the packed input-layer weights, from the shadow (after every update)
gcpsl_status refresh_derived(gcpsl_ctx* c) {
  if (c->tc0.on || c->rn)
    LAUNCH("pack_w0", launch_pack_w0(c->stream, c->d_shadow + c->w0_off, c->d_w0p, c->P_pad,
                                     c->w0_cout, c->C));
  return GCPSL_OK;
}

// canonical <-> kernel parameter layout of the context's architecture
void to_kernel(const gcpsl_ctx* c, const float* can, float* ker) {
  if (c->rn) rn_to_kernel_layout(c->J, can, ker);
  else to_kernel_layout(c->a, can, ker);
}
void to_canonical(const gcpsl_ctx* c, const float* ker, float* can) {
  if (c->rn) rn_to_canonical_layout(c->J, ker, can);
  else to_canonical_layout(c->a, ker, can);
}

}  // namespace

// a device-side wait that gave up leaves a nonzero error word; the context
// then refuses further work
gcpsl_status gcpsl::check_device_error(gcpsl_ctx* c) {
  int e = 0;
  CK(cudaMemcpy(&e, c->d_err, sizeof(int), cudaMemcpyDeviceToHost));
  if (e) return fail(c, GCPSL_E_TIMEOUT, "device-side wait gave up (error word 0x%x)", e);
  return GCPSL_OK;
}

float* gcpsl::partial_range(gcpsl_ctx* c, int64_t off, int64_t count, int64_t per, int splits) {
  float* buf = nullptr;
  if (dalloc(c, &buf, sizeof(float) * (size_t)c->C * splits * per) != GCPSL_OK) return nullptr;
  c->pranges.push_back({off, count, per, splits, buf});
  return buf;
}

gcpsl_status gcpsl::build_sgd_segments(gcpsl_ctx* c) {
  if (c->pranges.empty()) return GCPSL_OK;
  std::vector<gcpsl_ctx::PartialRange> r = c->pranges;
  std::sort(r.begin(), r.end(), [](const auto& a, const auto& b) { return a.off < b.off; });
  std::vector<SgdSeg> segs;
  std::vector<int4> blocks;
  int64_t at = 0;
  bool aligned = true;
  auto add = [&](const float* src, int64_t off, int64_t count, int64_t per, int splits) {
    aligned = aligned && off % 4 == 0 && count % 4 == 0 && per % 4 == 0 &&
              (uintptr_t)src % 16 == 0;
    const int64_t quads = (int64_t)c->C * count / 4;
    const int chunk = sgd_chunk(splits);
    for (int64_t e = 0; e < quads; e += chunk)
      blocks.push_back(make_int4((int)segs.size(), (int)e, (int)std::min<int64_t>(chunk, quads - e),
                                 0));
    // the input layer's weights also go packed to w0p (bf16 mode)
    const bool w0 = c->d_w0p && off == c->w0_off;
    segs.push_back({src, off, count, per, (int64_t)c->C * count, splits, w0 ? c->d_w0p : nullptr,
                    w0 ? c->w0_cout : 0});
    if (w0) c->sgd_packs_w0 = true;
  };
  for (const auto& q : r) {
    if (q.off < at || q.off + q.count > c->P_pad)
      return fail(c, GCPSL_E_INVAL, "overlapping weight-gradient partial ranges");
    if (q.off > at) add(c->d_grad + at, at, q.off - at, c->P_pad, 1);
    add(q.buf, q.off, q.count, q.per, q.splits);
    at = q.off + q.count;
  }
  if (at < c->P_pad) add(c->d_grad + at, at, c->P_pad - at, c->P_pad, 1);
  if ((int64_t)c->C * c->P_pad >= ((int64_t)1 << 31) || !aligned)
    return fail(c, GCPSL_E_UNSUPPORTED, "parameter segments not supported by the update");
  DALLOC(c->d_sgd_segs, sizeof(SgdSeg) * segs.size());
  DALLOC(c->d_sgd_blocks, sizeof(int4) * blocks.size());
  CK(cudaMemcpy(c->d_sgd_segs, segs.data(), sizeof(SgdSeg) * segs.size(), cudaMemcpyHostToDevice));
  CK(cudaMemcpy(c->d_sgd_blocks, blocks.data(), sizeof(int4) * blocks.size(),
                cudaMemcpyHostToDevice));
  c->n_sgd_blocks = (int)blocks.size();
  return GCPSL_OK;
}

namespace {

// per-layer names of the tensor-core launches in the kernel timer
const char* const kFwdTc[4] = {"conv_fwd_tc.L0", "conv_fwd_tc.L1", "conv_fwd_tc.L2",
                               "conv_fwd_tc.L3"};
const char* const kDgradTc[4] = {"conv_dgrad_tc.L0", "conv_dgrad_tc.L1", "conv_dgrad_tc.L2",
                                 "conv_dgrad_tc.L3"};
const char* const kWgradTc[4] = {"conv_wgrad_tc.L0", "conv_wgrad_tc.L1", "conv_wgrad_tc.L2",
                                 "conv_wgrad_tc.L3"};

// true when some cluster starts an epoch in round c->t (0-based)
bool epoch_boundary(const gcpsl_ctx* c) {
  for (int n = 0; n < c->C; ++n)
    if (c->t % c->h_period[n] == 0) return true;
  return false;
}

// GPSL sampling (Eq. 1) and the gather of the sampled images.  The epoch
// permutation is rebuilt only when some cluster starts an epoch; the host
// round count equals the device one, so other rounds skip those launches
// (the kernels also check the device counter themselves).
template <typename T>
gcpsl_status enqueue_sample(gcpsl_ctx* c, bool boundary) {
  cudaStream_t s = c->stream;
  const int C = c->C, B = c->B;
  if (boundary) {
    LAUNCH("epoch_keys", launch_epoch_keys(s, c->d_ids, c->d_off, c->d_period, c->d_t,
                                           c->desc.cluster_id_base, c->seed, c->d_keys, C,
                                           c->max_nc));
    LAUNCH("epoch_rank", launch_epoch_rank(s, c->d_ids, c->d_off, c->d_period, c->d_t,
                                           c->d_keys, c->d_perm, C, c->max_nc));
  }
  LAUNCH("sample", launch_sample(s, c->d_perm, c->d_off, c->d_rounds, c->d_period, c->d_t,
                                 c->d_owner, c->d_labels, c->K, B, C, c->d_idx, c->d_counts,
                                 c->d_active, c->d_y, c->d_upd, c->d_cut_scale));
  const AugArgs aug{c->desc.augment, (uint32_t)c->seed, (uint32_t)(c->seed >> 32), c->d_t,
                    c->desc.cluster_id_base, B};
  LAUNCH("gather", launch_gather<T>(s, c->d_images, c->d_idx, C * B, (T*)c->d_act[0], aug));
  return GCPSL_OK;
}

gcpsl_status enqueue_sgd(gcpsl_ctx* c) {
  if (c->n_sgd_blocks)
    LAUNCH("sgd", launch_sgd_seg(c->stream, c->d_theta, c->d_mom, c->d_shadow, c->d_sgd_segs,
                                 c->d_sgd_blocks, c->n_sgd_blocks, c->P_pad, c->desc.lr,
                                 c->desc.momentum, c->desc.weight_decay, c->desc.nesterov,
                                 c->d_upd, c->d_t));
  else
    LAUNCH("sgd", launch_sgd(c->stream, c->d_theta, c->d_mom, c->d_grad, c->d_shadow,
                             (int64_t)c->C * c->P_pad, c->P_pad, c->desc.lr, c->desc.momentum,
                             c->desc.weight_decay, c->desc.nesterov, c->d_upd, c->d_t));
  // the segment update also rewrites the packed input-layer weights
  return c->sgd_packs_w0 ? GCPSL_OK : refresh_derived(c);
}


template <typename T>
gcpsl_status enqueue_round(gcpsl_ctx* c, bool boundary) {
  gcpsl_status st0 = enqueue_sample<T>(c, boundary);
  if (st0 != GCPSL_OK) return st0;
  if (c->rn) {
    st0 = rn_enqueue_round(c);
    if (st0 != GCPSL_OK) return st0;
    return enqueue_sgd(c);
  }
  cudaStream_t s = c->stream;
  const ArchSpec& a = c->a;
  const int C = c->C, B = c->B;
  const int64_t P = c->P_pad;
  const T* wts = c->bf ? (const T*)(const void*)c->d_shadow : (const T*)(const void*)c->d_theta;
  T* act[5];
  T* dact[5];
  for (int i = 0; i <= a.L(); ++i) { act[i] = (T*)c->d_act[i]; dact[i] = (T*)c->d_dact[i]; }

  // client segment to the cut, then the server segment
  for (int i = 0; i < a.L(); ++i) {
    const auto& L = c->tc[i];
    if (i == 0 && c->tc0.on) {
      // one tap over the im2col: K = 32 columns
      const auto& L0 = c->tc0;
      ConvTcArgs p{a.conv[0].h, a.conv[0].w, B, 32, L0.bw, L0.hb, L0.bb, L0.tiles_w, L0.tiles_h,
                   a.conv[0].cout, c->d_theta + a.off_b[0], P, (bf16*)(void*)act[1],
                   c->d_code[0], c->d_err};
      conv_taps_one(p);
      LAUNCH(kFwdTc[0], launch_conv_tc(s, L0.A, L0.B, p, a.conv[0].cout, 32,
                                       a.conv[0].pool ? EPI_POOL : EPI_RELU, C));
    } else if (L.on) {
      ConvTcArgs p{a.conv[i].h, a.conv[i].w, B, a.conv[i].cin, L.bw, L.hb, L.bb, L.tiles_w,
                   L.tiles_h, a.conv[i].cout, c->d_theta + a.off_b[i], P,
                   (bf16*)(void*)act[i + 1], c->d_code[i], c->d_err};
      conv_taps_fwd3(p);
      const int epi = a.conv[i].pool ? EPI_POOL : EPI_RELU;
      if (L.halo_f) {
        p.bw = 8; p.hb = 16; p.bb = 1;
        p.tiles_w = a.conv[i].w / 8;
        p.tiles_h = a.conv[i].h / 16;
        LAUNCH(kFwdTc[i], launch_conv_halo(s, L.hfA, L.fwdB, p, L.bn_f, L.bkc_f, epi, C));
      } else {
        LAUNCH(kFwdTc[i], launch_conv_tc(s, L.fwdA, L.fwdB, p, L.bn_f, L.bkc_f, epi, C));
      }
    } else {
      LAUNCH("conv_fwd", launch_conv_fwd_simt<T>(s, act[i], wts + a.off_w[i], P,
                                                 c->d_theta + a.off_b[i], P, act[i + 1],
                                                 c->d_code[i], C, B, a.conv[i]));
    }
  }
  LAUNCH("fc_fwd_ce", launch_fc_fwd_ce<T>(s, act[a.L()], wts + a.off_fcw, P,
                                          c->d_theta + a.off_fcb, P, c->d_y, c->d_loss_ex,
                                          c->d_dlogits, C, B, a.fc_in, a.fc_out,
                                          c->desc.label_smoothing));
  // The head hands dh straight through the last conv layer's max-pool /
  // ReLU backward into its g; so does every tensor-core data gradient for
  // the layer below it.  g_ready[i]: g_i has been written.
  bool g_ready[4] = {};
  {
    const int l = a.L() - 1;
    const ConvSpec& cs = a.conv[l];
    LAUNCH("fc_bwd", launch_fc_bwd<T>(s, c->d_dlogits, c->d_loss_ex, act[a.L()], wts + a.off_fcw,
                                      P, c->d_grad + a.off_fcw, c->d_grad + a.off_fcb, P,
                                      (T*)c->gbuf(l), c->d_loss, C, B, a.fc_in, a.fc_out,
                                      cs.pool ? FC_DH_POOL : FC_DH_RELU, c->d_code[l], act[a.L()],
                                      a.out_h(l), a.out_w(l), cs.cout));
    g_ready[l] = true;
  }
  // backward to the cut gradient (dact[ncl]) and through the client segment
  for (int i = a.L() - 1; i >= 0; --i) {
    const auto& L = c->tc[i];
    const ConvSpec& cs = a.conv[i];
    T* g = (T*)c->gbuf(i);
    if (!g_ready[i])
      LAUNCH("relu_pool_bwd", launch_relu_pool_bwd<T>(s, dact[i + 1], c->d_code[i], act[i + 1],
                                                      g, C, B, cs));
    if (i == a.ncl - 1 && c->desc.client_average)
      // the per-client average: g of the client's last layer and the stored
      // cut gradient, per example by B / (|A| b_k)
      LAUNCH("client_avg", launch_client_avg_scale<T>(
                               s, g, (int64_t)cs.h * cs.w * cs.cout, dact[a.ncl],
                               act_elems(c, a.ncl) / ((int64_t)C * B), c->d_cut_scale, C * B));
    const auto& R = c->red[i];
    if (L.on) {
      // weights and bias together (the bias follows the weight in the store);
      // a single split writes the gradient directly, several write the
      // layer's partials, which the update sums
      WgradTcArgs w{cs.h, cs.w, B, cs.cout, cs.cin, L.whb, L.wbb, L.kb_total, L.kb_per_split,
                    L.splits, L.part, c->d_err};
      if (!L.part) {
        w.out = c->d_grad + a.off_w[i];
        w.out_rs = P;
      }
      if (L.wg_halo)
        LAUNCH(kWgradTc[i], launch_wgrad_halo(s, L.wgA, L.wgH, w, C));
      else
        LAUNCH(kWgradTc[i], launch_wgrad_tc(s, L.wgA, L.wgB, w, L.bn_w, C));
    } else if (i == 0 && c->tc0.wg_on) {
      const auto& L0 = c->tc0;
      WgradTcArgs w{cs.h, cs.w, B, cs.cout, cs.cin, L0.whb, L0.wbb, L0.kb_total, L0.kb_per_split,
                    L0.splits, L0.part, c->d_err};
      LAUNCH(kWgradTc[0], launch_wgrad0_tc(s, L0.wgA, L0.wgB, w, C));
    } else {
      // weights and bias together (the bias follows the weight in the store)
      LAUNCH("conv_wgrad", launch_wgrad_simt<T>(s, act[i], i == 0 ? c->x0c : cs.cin, g,
                                                c->d_bpartial, C, B, cs, R.tr, R.splits,
                                                R.tiles_per_split));
      LAUNCH("wgrad_reduce", launch_wgrad_reduce(s, c->d_bpartial, c->d_grad + a.off_w[i], P,
                                                 R.splits,
                                                 (int64_t)cs.cout * 9 * cs.cin + cs.cout, C));
    }
    if (i == 0) continue;
    if (L.on) {
      // dx of layer i, routed into g_{i-1}; the cut gradient itself is kept
      const ConvSpec& pv = a.conv[i - 1];
      ConvTcArgs p{cs.h, cs.w, B, cs.cout, L.bw, L.hb, L.bb, L.tiles_w, L.tiles_h, cs.cin,
                   nullptr, 0, i == a.ncl ? (bf16*)(void*)dact[i] : nullptr,
                   pv.pool ? c->d_code[i - 1] : nullptr, c->d_err,
                   pv.pool ? nullptr : (const bf16*)(const void*)act[i],
                   (bf16*)c->gbuf(i - 1)};
      conv_taps_dgrad3(p);
      const int epi = pv.pool ? EPI_DPOOL : EPI_DRELU;
      if (L.halo_d) {
        p.bw = 8; p.hb = 16; p.bb = 1;
        p.tiles_w = cs.w / 8;
        p.tiles_h = cs.h / 16;
        LAUNCH(kDgradTc[i], launch_conv_halo(s, L.hdA, L.dgrB, p, std::min(L.bn_d, 64),
                                             L.bkc_d, epi, C));
      } else {
        LAUNCH(kDgradTc[i], launch_conv_tc(s, L.dgrA, L.dgrB, p, L.bn_d, L.bkc_d, epi, C));
      }
      g_ready[i - 1] = true;
    } else {
      LAUNCH("conv_dgrad", launch_conv_dgrad_simt<T>(s, g, wts + a.off_w[i], P, dact[i], C, B,
                                                     cs));
    }
  }
  return enqueue_sgd(c);
}

// One round through a CUDA graph: captured on first use of its variant
// (epoch boundary or not; untimed or timed), then replayed.  Every launch
// parameter is fixed for the context's lifetime (buffers, tensor maps,
// hyper-parameters) and the round counter lives in device memory, so a
// replay is the same round the eager path would enqueue.
gcpsl_status run_round_graph(gcpsl_ctx* c) {
  const bool boundary = epoch_boundary(c);
  const int k = c->timing ? 1 + (c->timed_phase ^= 1) : 0;
  auto& g = c->graph[boundary][k];
  if (g.unread) {                 // event pairs of this copy's previous launch
    c->timer.account(g.marks);
    g.unread = false;
  }
  if (!g.exec) {
    const int64_t before = c->enqueued;
    CK(cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal));
    if (c->timing) c->timer.capture = &g.marks;
    c->capturing = true;
    gcpsl_status st = c->bf ? enqueue_round<bf16>(c, boundary) : enqueue_round<float>(c, boundary);
    c->capturing = false;
    c->timer.capture = nullptr;
    cudaGraph_t graph = nullptr;
    cudaError_t e = cudaStreamEndCapture(c->stream, &graph);
    if (st != GCPSL_OK || e != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      for (auto& m : g.marks) { c->timer.pool.push_back(m.a); c->timer.pool.push_back(m.b); }
      g.marks.clear();
      if (st != GCPSL_OK) return st;
      return fail(c, GCPSL_E_CUDA, "graph capture of a round failed: %s", cudaGetErrorString(e));
    }
    e = cudaGraphInstantiate(&g.exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
      g.exec = nullptr;
      return fail(c, GCPSL_E_CUDA, "graph instantiation failed: %s", cudaGetErrorString(e));
    }
    g.kernels = c->enqueued - before;
  }
  CK(cudaGraphLaunch(g.exec, c->stream));
  c->launched += g.kernels;
  g.unread = c->timing;
  return GCPSL_OK;
}

// add the event pairs of every timed graph launch not yet read
void account_graph_marks(gcpsl_ctx* c) {
  for (auto& v : c->graph)
    for (auto& g : v)
      if (g.unread) { c->timer.account(g.marks); g.unread = false; }
}

void destroy_graphs(gcpsl_ctx* c) {
  for (auto& v : c->graph)
    for (auto& g : v) {
      if (g.exec) cudaGraphExecDestroy(g.exec);
      g.exec = nullptr;
      for (auto& m : g.marks) { cudaEventDestroy(m.a); cudaEventDestroy(m.b); }
      g.marks.clear();
      g.unread = false;
    }
}

gcpsl_status enqueue_fuse(gcpsl_ctx* c) {
  if (c->C == 1) return GCPSL_OK;                 // q_1 = 1: the identity
  LAUNCH("fuse", launch_fuse(c->stream, c->d_theta, c->d_shadow, c->d_q, c->C, c->P_pad));
  if (c->rn) {                                    // BatchNorm running statistics, same q
    int64_t S, S_pad;
    float* bn = rn_bn_state(c, &S, &S_pad);
    LAUNCH("fuse", launch_fuse(c->stream, bn, nullptr, c->d_q, c->C, S_pad));
  }
  return refresh_derived(c);
}

}  // namespace

// 128-pixel M tile of a W x H image: bw <= 16 columns (so a warp holds whole
// 2x2 pooling windows), hb rows, bb images
bool gcpsl::m_tile(int W, int H, int& bw, int& hb, int& bb) {
  bw = std::min(W, 16);
  if (bw < 2 || W % bw || 128 % bw) return false;
  hb = std::min(H, 128 / bw);
  bb = 128 / (bw * hb);
  return bw * hb * bb == 128 && H % hb == 0 && hb % 2 == 0;
}

namespace {

// Tile shapes, split-K factors and TMA descriptors of every layer that runs on
// the tensor cores: 3x3 layers with 32k input and 64k output channels and
// rows of at most 64 pixels.  Layers outside that shape (the 3-channel input
// layer) stay on the CUDA-core kernels.
gcpsl_status setup_tensor_core_layers(gcpsl_ctx* c) {
  const ArchSpec& a = c->a;
  const int C = c->C, B = c->B;
  for (int i = 0; i < a.L(); ++i) {
    const ConvSpec& s = a.conv[i];
    auto& L = c->tc[i];
    L.on = false;
    // (16-byte aligned weight rows and bias vectors)
    if (s.cin < 32 || s.cin % 32 || s.cout % 64 || s.w > 64 || 64 % s.w || a.off_w[i] % 8 ||
        a.off_b[i] % 4)
      continue;
    if (!m_tile(s.w, s.h, L.bw, L.hb, L.bb)) continue;
    L.whb = std::min(s.h, 64 / s.w);
    L.wbb = 64 / (s.w * L.whb);
    if (s.w * L.whb * L.wbb != 64 || s.h % L.whb) continue;
    L.tiles_w = s.w / L.bw;
    L.tiles_h = s.h / L.hb;
    L.bn_f = std::min(s.cout, 256);
    L.bkc_f = std::min(s.cin, 64);
    L.bn_d = std::min(s.cin, 256);
    L.bkc_d = std::min(s.cout, 64);
    L.bn_w = std::min(s.cin, 128);
    if (s.cout % L.bn_f || s.cin % L.bn_d || s.cin % L.bkc_f || s.cin % L.bn_w) continue;
    L.wg_halo = wgrad_halo_supported(s.h, s.w, s.cin, s.cout, 9, 1) && L.whb * s.w == 64;
    const int tiles = L.wg_halo ? wgrad_halo_tiles(s.cin, s.cout)
                                : wgrad_tc_tiles(s.cin, s.cout, 9, L.bn_w);
    L.kb_total = ((B + L.wbb - 1) / L.wbb) * (s.h / L.whb);
    const int64_t per = (int64_t)s.cout * 9 * s.cin + s.cout;
    const int splits = wgrad_splits(tiles, L.kb_total, per);
    L.kb_per_split = (L.kb_total + splits - 1) / splits;
    L.splits = (L.kb_total + L.kb_per_split - 1) / L.kb_per_split;
    L.part = nullptr;
    if (L.splits > 1 || a.off_w[i] % 4) {
      L.part = partial_range(c, a.off_w[i], per, per, L.splits);
      if (!L.part) return fail(c, GCPSL_E_NOMEM, "device allocation failed");
    }

    const uint64_t act_in[5] = {(uint64_t)s.cin, (uint64_t)s.w, (uint64_t)s.h, (uint64_t)B,
                                (uint64_t)C};
    const uint64_t g_dims[5] = {(uint64_t)s.cout, (uint64_t)s.w, (uint64_t)s.h, (uint64_t)B,
                                (uint64_t)C};
    const uint64_t wf[4] = {(uint64_t)s.cin, 9, (uint64_t)s.cout, (uint64_t)C};
    const uint64_t rs = (uint64_t)c->P_pad * 2;
    const uint32_t bA[5] = {(uint32_t)L.bkc_f, (uint32_t)L.bw, (uint32_t)L.hb, (uint32_t)L.bb, 1};
    const uint32_t bB[4] = {(uint32_t)L.bkc_f, 1, (uint32_t)L.bn_f, 1};
    const uint32_t dA[5] = {(uint32_t)L.bkc_d, (uint32_t)L.bw, (uint32_t)L.hb, (uint32_t)L.bb, 1};
    // data gradient: W[co][tap][ci] read MN-major, N blocks of <= 64 ci
    const int nbw = std::min(L.bn_d, 64);
    const uint32_t dB[4] = {(uint32_t)nbw, 1, (uint32_t)L.bkc_d, 1};
    const uint32_t wA[5] = {64, (uint32_t)s.w, (uint32_t)L.whb, (uint32_t)L.wbb, 1};
    const int wx = std::min(s.cin, 64);
    const uint32_t wB[5] = {(uint32_t)wx, (uint32_t)s.w, (uint32_t)L.whb, (uint32_t)L.wbb, 1};
    bool ok = tensor_map_bf16(&L.fwdA, c->d_act[i], 5, act_in, bA, L.bkc_f * 2) &&
              tensor_map_bf16_strided(&L.fwdB, c->d_shadow + a.off_w[i], 4, wf, rs, bB,
                                      L.bkc_f * 2) &&
              tensor_map_bf16(&L.dgrA, c->gbuf(i), 5, g_dims, dA, L.bkc_d * 2) &&
              tensor_map_bf16_strided(&L.dgrB, c->d_shadow + a.off_w[i], 4, wf, rs, dB,
                                      nbw * 2) &&
              tensor_map_bf16(&L.wgA, c->gbuf(i), 5, g_dims, wA, 128) &&
              tensor_map_bf16(&L.wgB, c->d_act[i], 5, act_in, wB, wx * 2);
    // halo-tiled forward / data gradient where the shape allows: one box of
    // 10 x 18 pixels per K block
    L.halo_f = halo_supported(s.h, s.w, s.cin, L.bn_f, L.bkc_f, s.pool ? EPI_POOL : EPI_RELU);
    L.halo_d = i > 0 && halo_supported(s.h, s.w, s.cout, std::min(L.bn_d, 64), L.bkc_d,
                                       a.conv[i - 1].pool ? EPI_DPOOL : EPI_DRELU);
    const uint32_t hbf[5] = {(uint32_t)L.bkc_f, 10, 18, 1, 1};
    const uint32_t hbd[5] = {(uint32_t)L.bkc_d, 10, 18, 1, 1};
    if (L.halo_f) ok = ok && tensor_map_bf16(&L.hfA, c->d_act[i], 5, act_in, hbf, L.bkc_f * 2);
    if (L.halo_d) ok = ok && tensor_map_bf16(&L.hdA, c->gbuf(i), 5, g_dims, hbd, L.bkc_d * 2);
    if (L.wg_halo) {
      const int cb = s.cin == 32 ? 32 : 64;
      const int hrows = wgrad_halo_rows(s.cin) == 3 ? L.whb + 2 : L.whb;
      const uint32_t hx[5] = {(uint32_t)cb, (uint32_t)s.w + 2, (uint32_t)hrows, 1, 1};
      ok = ok && tensor_map_bf16(&L.wgH, c->d_act[i], 5, act_in, hx, cb * 2);
    }
    if (!ok) return fail(c, GCPSL_E_CUDA, "cuTensorMapEncodeTiled failed for layer %d", i);
    L.on = true;
  }

  // the input layer (3 channels): with bf16 operands the gather writes its
  // im2col (32 columns per pixel), so its forward is a one-tap K = 32
  // convolution and its weight gradient a GEMM over the pixels
  const ConvSpec& s0 = a.conv[0];
  auto& L0 = c->tc0;
  L0.on = false;
  if (s0.cin != 3 || (s0.cout != 32 && s0.cout != 64) || s0.w != 32 || s0.h != 32 ||
      a.off_b[0] % 4 || !m_tile(s0.w, s0.h, L0.bw, L0.hb, L0.bb))
    return fail(c, GCPSL_E_UNSUPPORTED, "input layer shape not supported with bf16 operands");
  L0.tiles_w = s0.w / L0.bw;
  L0.tiles_h = s0.h / L0.hb;
  DALLOC(c->d_w0p, sizeof(bf16) * (size_t)C * s0.cout * 32);
  const uint64_t xdims[5] = {32, (uint64_t)s0.w, (uint64_t)s0.h, (uint64_t)B, (uint64_t)C};
  const uint32_t xbox[5] = {32, (uint32_t)L0.bw, (uint32_t)L0.hb, (uint32_t)L0.bb, 1};
  const uint64_t wdims[4] = {32, 1, (uint64_t)s0.cout, (uint64_t)C};
  const uint32_t wbox[4] = {32, 1, (uint32_t)s0.cout, 1};
  if (!tensor_map_bf16(&L0.A, c->d_act[0], 5, xdims, xbox, 64) ||
      !tensor_map_bf16(&L0.B, c->d_w0p, 4, wdims, wbox, 64))
    return fail(c, GCPSL_E_CUDA, "cuTensorMapEncodeTiled failed for the input layer");
  L0.on = true;
  // its weight gradient: 64-pixel K blocks, split per replica shape only
  L0.whb = 64 / s0.w;
  L0.wbb = 1;
  L0.kb_total = B * (s0.h / L0.whb);
  {
    const int splits = std::max(1, std::min(64, (L0.kb_total + 15) / 16));
    L0.kb_per_split = (L0.kb_total + splits - 1) / splits;
    L0.splits = (L0.kb_total + L0.kb_per_split - 1) / L0.kb_per_split;
  }
  const uint64_t gd[5] = {(uint64_t)s0.cout, (uint64_t)s0.w, (uint64_t)s0.h, (uint64_t)B,
                          (uint64_t)C};
  const uint32_t gb[5] = {(uint32_t)s0.cout, (uint32_t)s0.w, (uint32_t)L0.whb, 1, 1};
  const uint32_t xb[5] = {32, (uint32_t)s0.w, (uint32_t)L0.whb, 1, 1};
  if (!tensor_map_bf16(&L0.wgA, c->gbuf(0), 5, gd, gb, s0.cout * 2) ||
      !tensor_map_bf16(&L0.wgB, c->d_act[0], 5, xdims, xb, 64))
    return fail(c, GCPSL_E_CUDA, "cuTensorMapEncodeTiled failed for the input-layer gradient");
  const int64_t per0 = (int64_t)s0.cout * 27 + s0.cout;
  L0.part = partial_range(c, a.off_w[0], per0, per0, L0.splits);
  if (!L0.part) return fail(c, GCPSL_E_NOMEM, "device allocation failed");
  L0.wg_on = true;
  return GCPSL_OK;
}

void free_all(gcpsl_ctx* c) {
  if (c->stream) cudaStreamSynchronize(c->stream);
  destroy_graphs(c);
  rn_free(c);
  c->timer.destroy();
  for (void* p : c->allocs) cudaFree(p);
  c->allocs.clear();
  if (c->h_images) cudaFreeHost(c->h_images);
  if (c->h_loss) cudaFreeHost(c->h_loss);
  if (c->h_active) cudaFreeHost(c->h_active);
  if (c->h_err) cudaFreeHost(c->h_err);
  if (c->own_stream) cudaStreamDestroy(c->own_stream);
}

gcpsl_status init_impl(gcpsl_ctx* c, const gcpsl_model_desc* desc, int K, int C,
                       const int32_t* assignment, int B, int F, uint64_t seed,
                       const gcpsl_dataset* data, const float* init_params) {
  c->desc = *desc;
  c->K = K; c->C = C; c->B = B; c->F = F; c->seed = seed;
  c->gn_groups = desc->gn_groups ? desc->gn_groups : 32;
  c->bn_momentum = desc->bn_momentum > 0.f ? desc->bn_momentum : 0.1f;
  c->norm_eps = desc->norm_eps > 0.f ? desc->norm_eps : 1e-5f;
  c->bf = desc->operand_dtype == GCPSL_BF16;
  c->esz = c->bf ? 2 : 4;
  c->x0c = c->bf ? 32 : 3;
  const ArchSpec& a = c->a;
  const bool resnet = resnet_classes(desc->arch) != 0;
  c->J = data->num_classes;
  c->P = resnet ? rn_num_params(c->J, GCPSL_CLIENT) + rn_num_params(c->J, GCPSL_SERVER)
                : a.p_total;
  c->n = data->n;

  // clusters: ascending example ids per cluster, r_n, q_n (Eq. 5)
  std::vector<int64_t> nc(C, 0);
  for (int64_t i = 0; i < data->n; ++i) {
    const int k = assignment[data->owner[i]];
    if (k >= 0) nc[k]++;
  }
  int64_t total = 0;
  for (int k = 0; k < C; ++k) {
    if (nc[k] < B)
      return fail(nullptr, GCPSL_E_INVAL, "cluster %d holds %lld examples, fewer than B=%d", k,
                  (long long)nc[k], B);
    total += nc[k];
    c->max_nc = std::max(c->max_nc, nc[k]);
  }
  c->h_off.assign(C + 1, 0);
  for (int k = 0; k < C; ++k) c->h_off[k + 1] = c->h_off[k] + nc[k];
  std::vector<int32_t> ids(total);
  std::vector<int64_t> fill(c->h_off.begin(), c->h_off.end() - 1);
  for (int64_t i = 0; i < data->n; ++i) {
    const int k = assignment[data->owner[i]];
    if (k >= 0) ids[fill[k]++] = (int32_t)i;
  }
  c->h_rounds.resize(C);
  c->h_q.resize(C);
  for (int k = 0; k < C; ++k) {
    c->h_rounds[k] = (int32_t)(nc[k] / B);
    c->h_q[k] = (float)((double)nc[k] / (double)total);
  }

  CK(cudaStreamCreateWithFlags(&c->own_stream, cudaStreamNonBlocking));
  c->stream = c->own_stream;

  // dataset
  const size_t img_bytes = sizeof(float) * (size_t)data->n * 3072;
  if (desc->data_on_host) {
    CK(cudaHostAlloc((void**)&c->h_images, img_bytes, cudaHostAllocMapped | cudaHostAllocPortable));
    std::memcpy(c->h_images, data->images, img_bytes);
    CK(cudaHostGetDevicePointer((void**)&c->d_images, c->h_images, 0));
  } else {
    DALLOC(c->d_images, img_bytes);
    CK(cudaMemcpy(c->d_images, data->images, img_bytes, cudaMemcpyHostToDevice));
  }
  DALLOC(c->d_labels, sizeof(int32_t) * data->n);
  DALLOC(c->d_owner, sizeof(int32_t) * data->n);
  CK(cudaMemcpy(c->d_labels, data->labels, sizeof(int32_t) * data->n, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(c->d_owner, data->owner, sizeof(int32_t) * data->n, cudaMemcpyHostToDevice));
  DALLOC(c->d_off, sizeof(int64_t) * (C + 1));
  DALLOC(c->d_rounds, sizeof(int32_t) * C);
  DALLOC(c->d_q, sizeof(float) * C);
  DALLOC(c->d_ids, sizeof(int32_t) * total);
  DALLOC(c->d_perm, sizeof(int32_t) * total);
  DALLOC(c->d_keys, sizeof(uint64_t) * total);
  CK(cudaMemcpy(c->d_off, c->h_off.data(), sizeof(int64_t) * (C + 1), cudaMemcpyHostToDevice));
  CK(cudaMemcpy(c->d_rounds, c->h_rounds.data(), sizeof(int32_t) * C, cudaMemcpyHostToDevice));
  c->R = 0;
  if (F == -1)
    for (int k = 0; k < C; ++k) c->R = std::max<int64_t>(c->R, c->h_rounds[k]);
  c->h_period.assign(C, 0);
  for (int k = 0; k < C; ++k) c->h_period[k] = c->R ? (int32_t)c->R : c->h_rounds[k];
  DALLOC(c->d_period, sizeof(int32_t) * C);
  DALLOC(c->d_upd, sizeof(int32_t) * C);
  CK(cudaMemcpy(c->d_period, c->h_period.data(), sizeof(int32_t) * C, cudaMemcpyHostToDevice));
  {
    const std::vector<int32_t> ones((size_t)C, 1);
    CK(cudaMemcpy(c->d_upd, ones.data(), sizeof(int32_t) * C, cudaMemcpyHostToDevice));
  }
  CK(cudaMemcpy(c->d_q, c->h_q.data(), sizeof(float) * C, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(c->d_ids, ids.data(), sizeof(int32_t) * total, cudaMemcpyHostToDevice));

  // parameters: C identical replicas
  std::vector<float> can(c->P), ker(c->P);
  if (init_params) std::memcpy(can.data(), init_params, sizeof(float) * c->P);
  else if (resnet) rn_seeded_init(c->J, seed, can.data());
  else seeded_init(a, seed, can.data());
  if (resnet) rn_to_kernel_layout(c->J, can.data(), ker.data());
  else to_kernel_layout(a, can.data(), ker.data());
  c->P_pad = (c->P + 63) / 64 * 64;
  const size_t pb = sizeof(float) * (size_t)(C * c->P_pad);
  DALLOC(c->d_theta, pb);
  DALLOC(c->d_mom, pb);
  DALLOC(c->d_grad, pb);
  CK(cudaMemset(c->d_theta, 0, pb));
  CK(cudaMemset(c->d_mom, 0, pb));
  CK(cudaMemset(c->d_grad, 0, pb));
  for (int k = 0; k < C; ++k)
    CK(cudaMemcpy(c->d_theta + (int64_t)k * c->P_pad, ker.data(), sizeof(float) * c->P,
                  cudaMemcpyHostToDevice));
  DALLOC(c->d_err, sizeof(int));
  CK(cudaMemset(c->d_err, 0, sizeof(int)));
  if (c->bf) {
    DALLOC(c->d_shadow, sizeof(bf16) * (size_t)(C * c->P_pad));
    CK(cudaMemset(c->d_shadow, 0, sizeof(bf16) * (size_t)(C * c->P_pad)));
    std::vector<bf16> sh(c->P);
    for (int64_t p = 0; p < c->P; ++p) sh[p] = __float2bfloat16_rn(ker[p]);
    for (int k = 0; k < C; ++k)
      CK(cudaMemcpy(c->d_shadow + (int64_t)k * c->P_pad, sh.data(), sizeof(bf16) * c->P,
                    cudaMemcpyHostToDevice));
  }

  if (resnet) {
    // shared per-round buffers; the layers' own come from rn_setup
    DALLOC(c->d_act[0], sizeof(bf16) * (size_t)C * B * 1024 * 32);
    DALLOC(c->d_w0p, sizeof(bf16) * (size_t)C * 64 * 32);
    DALLOC(c->d_loss_ex, sizeof(float) * C * B);
    DALLOC(c->d_dlogits, sizeof(float) * C * B * c->J);
    DALLOC(c->d_y, sizeof(int32_t) * C * B);
    DALLOC(c->d_idx, sizeof(int32_t) * C * B);
    DALLOC(c->d_counts, sizeof(int32_t) * (size_t)C * K);
    DALLOC(c->d_active, sizeof(int32_t) * C);
    if (desc->client_average) DALLOC(c->d_cut_scale, sizeof(float) * C * B);
    DALLOC(c->d_loss, sizeof(float) * C);
    DALLOC(c->d_t, sizeof(int64_t));
    CK(cudaMemset(c->d_t, 0, sizeof(int64_t)));
    CK(cudaMemset(c->d_idx, 0, sizeof(int32_t) * C * B));
    CK(cudaMemset(c->d_counts, 0, sizeof(int32_t) * (size_t)C * K));
    CK(cudaHostAlloc((void**)&c->h_loss, sizeof(float) * C, cudaHostAllocDefault));
    CK(cudaHostAlloc((void**)&c->h_active, sizeof(int32_t) * C, cudaHostAllocDefault));
    CK(cudaHostAlloc((void**)&c->h_err, sizeof(int), cudaHostAllocDefault));
    c->w0_off = 0;                                // the stem convolution
    c->w0_cout = 64;
    gcpsl_status st = rn_setup(c);
    if (st != GCPSL_OK) return st;
    st = build_sgd_segments(c);
    if (st != GCPSL_OK) return st;
    st = refresh_derived(c);
    if (st != GCPSL_OK) return st;
    CK(cudaDeviceSynchronize());
    return GCPSL_OK;
  }

  // activations of one round
  int64_t gmax = 0;
  for (int i = 0; i <= a.L(); ++i) {
    DALLOC(c->d_act[i], c->esz * act_elems(c, i));
    DALLOC(c->d_dact[i], c->esz * act_elems(c, i));
  }
  for (int i = 0; i < a.L(); ++i) {
    if (a.conv[i].pool) DALLOC(c->d_code[i], act_elems(c, i + 1));
    gmax = std::max(gmax, (int64_t)C * B * a.conv[i].h * a.conv[i].w * a.conv[i].cout);
  }
  DALLOC(c->d_g, c->esz * gmax);
  DALLOC(c->d_g2, c->esz * gmax);
  DALLOC(c->d_loss_ex, sizeof(float) * C * B);
  DALLOC(c->d_dlogits, sizeof(float) * C * B * a.fc_out);
  DALLOC(c->d_y, sizeof(int32_t) * C * B);
  DALLOC(c->d_idx, sizeof(int32_t) * C * B);
  DALLOC(c->d_counts, sizeof(int32_t) * (size_t)C * K);
  DALLOC(c->d_active, sizeof(int32_t) * C);
  if (desc->client_average) DALLOC(c->d_cut_scale, sizeof(float) * C * B);
  DALLOC(c->d_loss, sizeof(float) * C);
  DALLOC(c->d_t, sizeof(int64_t));
  CK(cudaMemset(c->d_t, 0, sizeof(int64_t)));
  CK(cudaMemset(c->d_idx, 0, sizeof(int32_t) * C * B));
  CK(cudaMemset(c->d_counts, 0, sizeof(int32_t) * (size_t)C * K));
  CK(cudaHostAlloc((void**)&c->h_loss, sizeof(float) * C, cudaHostAllocDefault));
  CK(cudaHostAlloc((void**)&c->h_active, sizeof(int32_t) * C, cudaHostAllocDefault));
  CK(cudaHostAlloc((void**)&c->h_err, sizeof(int), cudaHostAllocDefault));
  // reduction shapes (per replica only, so that the summation order does not
  // depend on C) and the partial-sum scratch
  int64_t bpart = 0;
  for (int i = 0; i < a.L(); ++i) {
    const ConvSpec& s = a.conv[i];
    auto& R = c->red[i];
    R.tr = std::max(1, std::min(s.h, 256 / s.w));
    while (s.h % R.tr) --R.tr;
    const int tiles = B * (s.h / R.tr);
    R.tiles_per_split = std::max(1, (tiles + 127) / 128);
    R.splits = (tiles + R.tiles_per_split - 1) / R.tiles_per_split;
    bpart = std::max(bpart, (int64_t)C * R.splits * ((int64_t)s.cout * 9 * s.cin + s.cout));
  }
  DALLOC(c->d_bpartial, sizeof(float) * bpart);
  c->w0_off = a.off_w[0];
  c->w0_cout = a.conv[0].cout;
  if (c->bf) {
    gcpsl_status st = setup_tensor_core_layers(c);
    if (st != GCPSL_OK) return st;
    st = build_sgd_segments(c);
    if (st != GCPSL_OK) return st;
    st = refresh_derived(c);
    if (st != GCPSL_OK) return st;
  }
  CK(cudaDeviceSynchronize());
  return GCPSL_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" {

int64_t gcpsl_num_params(int arch, int segment) {
  if (resnet_classes(arch)) return rn_num_params(resnet_classes(arch), segment);
  ArchSpec a;
  if (!make_arch(arch, &a)) return -1;
  if (segment == GCPSL_CLIENT) return a.p_client;
  if (segment == GCPSL_SERVER) return a.p_total - a.p_client;
  return -1;
}

gcpsl_status gcpsl_init(const gcpsl_model_desc* desc, int K, int C, const int32_t* assignment,
                        int B, int F, uint64_t seed, const gcpsl_dataset* data,
                        const float* init_params, gcpsl_ctx** out) {
  gcpsl_ctx* c = nullptr;
  if (!out) return fail(nullptr, GCPSL_E_INVAL, "out is NULL");
  *out = nullptr;
  if (!desc || !assignment || !data || !data->images || !data->labels || !data->owner)
    return fail(nullptr, GCPSL_E_INVAL, "NULL argument");
  if (K <= 0 || C <= 0 || B <= 0 || B > 1024 || F < -1 || data->n <= 0 || data->n > INT32_MAX)
    return fail(nullptr, GCPSL_E_INVAL, "bad size (K=%d C=%d B=%d F=%d n=%lld)", K, C, B, F,
                (long long)data->n);
  if (desc->operand_dtype != GCPSL_F32 && desc->operand_dtype != GCPSL_BF16)
    return fail(nullptr, GCPSL_E_INVAL, "unknown operand_dtype %d", desc->operand_dtype);
  if (desc->augment != 0 && desc->augment != 1)
    return fail(nullptr, GCPSL_E_INVAL, "augment must be 0 or 1");
  if (desc->client_average != 0 && desc->client_average != 1)
    return fail(nullptr, GCPSL_E_INVAL, "client_average must be 0 or 1");
  if (desc->gn_groups < 0 || desc->gn_groups > 32 || (desc->gn_groups && 64 % desc->gn_groups) ||
      !(desc->bn_momentum >= 0.f && desc->bn_momentum <= 1.f) ||
      !(desc->norm_eps >= 0.f && desc->norm_eps < 1.f))
    return fail(nullptr, GCPSL_E_INVAL, "bad norm hyper-parameters (groups %d, momentum %g, eps %g)",
                desc->gn_groups, (double)desc->bn_momentum, (double)desc->norm_eps);
  if (!(desc->lr >= 0.f) || !(desc->label_smoothing >= 0.f && desc->label_smoothing < 1.f))
    return fail(nullptr, GCPSL_E_INVAL, "bad lr or label_smoothing");
  ArchSpec a;
  std::memset(&a, 0, sizeof(a));
  if (resnet_classes(desc->arch)) {
    if (desc->operand_dtype != GCPSL_BF16)
      return fail(nullptr, GCPSL_E_UNSUPPORTED, "the ResNet-18 split runs with bf16 operands");
  } else if (!make_arch(desc->arch, &a)) {
    return fail(nullptr, GCPSL_E_UNSUPPORTED, "architecture %d is not built", desc->arch);
  }
  if (data->num_classes != arch_classes(desc->arch))
    return fail(nullptr, GCPSL_E_INVAL, "num_classes=%d, architecture %d has %d", data->num_classes,
                desc->arch, arch_classes(desc->arch));
  for (int k = 0; k < K; ++k)
    if (assignment[k] < -1 || assignment[k] >= C)
      return fail(nullptr, GCPSL_E_INVAL, "assignment[%d]=%d outside [-1, %d)", k, assignment[k], C);
  for (int64_t i = 0; i < data->n; ++i) {
    if (data->owner[i] < 0 || data->owner[i] >= K)
      return fail(nullptr, GCPSL_E_INVAL, "owner[%lld]=%d outside [0, %d)", (long long)i,
                  data->owner[i], K);
    if (data->labels[i] < 0 || data->labels[i] >= data->num_classes)
      return fail(nullptr, GCPSL_E_INVAL, "label[%lld]=%d out of range", (long long)i,
                  data->labels[i]);
  }
  c = new (std::nothrow) gcpsl_ctx();
  if (!c) return fail(nullptr, GCPSL_E_NOMEM, "host allocation failed");
  c->a = a;
  gcpsl_status st = init_impl(c, desc, K, C, assignment, B, F, seed, data, init_params);
  if (st != GCPSL_OK) {
    if (!c->err.empty()) g_init_error = c->err;
    free_all(c);
    delete c;
    return st;
  }
  *out = c;
  return GCPSL_OK;
}

gcpsl_status gcpsl_step(gcpsl_ctx* c, gcpsl_step_stats* stats) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  // the first round runs eagerly (it also sets the kernels' attributes),
  // later rounds replay captured graphs
  if (c->use_graph && c->t > 0) {
    st = run_round_graph(c);
  } else {
    st = c->bf ? enqueue_round<bf16>(c, epoch_boundary(c))
               : enqueue_round<float>(c, epoch_boundary(c));
  }
  if (st != GCPSL_OK) return st;
  c->t++;
  const int64_t every = c->R ? c->R : c->F;       // fusion interval in rounds
  if (every > 0 && c->t % every == 0) {
    st = enqueue_fuse(c);
    if (st != GCPSL_OK) return st;
  }
  if (stats && (stats->loss || stats->active)) {
    CK(cudaMemcpyAsync(c->h_loss, c->d_loss, sizeof(float) * c->C, cudaMemcpyDeviceToHost,
                       c->stream));
    CK(cudaMemcpyAsync(c->h_active, c->d_active, sizeof(int32_t) * c->C, cudaMemcpyDeviceToHost,
                       c->stream));
    // the device error word comes back with the statistics: one synchronisation
    CK(cudaMemcpyAsync(c->h_err, c->d_err, sizeof(int), cudaMemcpyDeviceToHost, c->stream));
    CK(cudaStreamSynchronize(c->stream));
    if (*c->h_err)
      return fail(c, GCPSL_E_TIMEOUT, "device-side wait gave up (error word 0x%x)", *c->h_err);
    // a cluster waiting at the fusion barrier took no update: loss 0
    for (int n = 0; n < c->C; ++n)
      if ((c->t - 1) % c->h_period[n] >= c->h_rounds[n]) c->h_loss[n] = 0.f;
    if (stats->loss) std::memcpy(stats->loss, c->h_loss, sizeof(float) * c->C);
    if (stats->active) std::memcpy(stats->active, c->h_active, sizeof(int32_t) * c->C);
  }
  return GCPSL_OK;
}

gcpsl_status gcpsl_fuse(gcpsl_ctx* c) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  return enqueue_fuse(c);
}

gcpsl_status gcpsl_get_params(gcpsl_ctx* c, int cluster, int segment, float* dst, size_t len,
                              size_t* needed) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (cluster < 0 || cluster >= c->C ||
      (segment != GCPSL_CLIENT && segment != GCPSL_SERVER && !(segment == GCPSL_BN_STATE && c->rn)))
    return fail(c, GCPSL_E_INVAL, "bad cluster %d or segment %d", cluster, segment);
  if (segment == GCPSL_BN_STATE) {
    int64_t S, S_pad;
    const float* bn = rn_bn_state(c, &S, &S_pad);
    if (needed) *needed = (size_t)S;
    if (!dst) return GCPSL_OK;
    if (len < (size_t)S) return fail(c, GCPSL_E_INVAL, "dst too small");
    SYNC_CHECK(c);
    CK(cudaMemcpy(dst, bn + (int64_t)cluster * S_pad, sizeof(float) * S, cudaMemcpyDeviceToHost));
    return GCPSL_OK;
  }
  const int64_t pc = c->rn ? rn_num_params(c->J, GCPSL_CLIENT) : c->a.p_client;
  const int64_t lo = segment == GCPSL_CLIENT ? 0 : pc;
  const int64_t hi = segment == GCPSL_CLIENT ? pc : c->P;
  if (needed) *needed = (size_t)(hi - lo);
  if (!dst) return GCPSL_OK;
  if (len < (size_t)(hi - lo)) return fail(c, GCPSL_E_INVAL, "dst too small");
  std::vector<float> ker(c->P), can(c->P);
  SYNC_CHECK(c);
  CK(cudaMemcpy(ker.data(), c->d_theta + (int64_t)cluster * c->P_pad, sizeof(float) * c->P,
                cudaMemcpyDeviceToHost));
  to_canonical(c, ker.data(), can.data());
  std::memcpy(dst, can.data() + lo, sizeof(float) * (size_t)(hi - lo));
  return GCPSL_OK;
}

gcpsl_status gcpsl_set_params(gcpsl_ctx* c, int cluster, const float* src, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (cluster < 0 || cluster >= c->C || !src || len != (size_t)c->P)
    return fail(c, GCPSL_E_INVAL, "bad cluster, src or len");
  std::vector<float> ker(c->P);
  to_kernel(c, src, ker.data());
  SYNC_CHECK(c);
  CK(cudaMemcpy(c->d_theta + (int64_t)cluster * c->P_pad, ker.data(), sizeof(float) * c->P,
                cudaMemcpyHostToDevice));
  if (c->bf) {
    std::vector<bf16> sh(c->P);
    for (int64_t p = 0; p < c->P; ++p) sh[p] = __float2bfloat16_rn(ker[p]);
    CK(cudaMemcpy(c->d_shadow + (int64_t)cluster * c->P_pad, sh.data(), sizeof(bf16) * c->P,
                  cudaMemcpyHostToDevice));
    return refresh_derived(c);
  }
  return GCPSL_OK;
}

gcpsl_status gcpsl_set_bn_state(gcpsl_ctx* c, int cluster, const float* src, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (!c->rn) return fail(c, GCPSL_E_INVAL, "this architecture has no BatchNorm state");
  int64_t S, S_pad;
  float* bn = rn_bn_state(c, &S, &S_pad);
  if (cluster < 0 || cluster >= c->C || !src || len != (size_t)S)
    return fail(c, GCPSL_E_INVAL, "bad cluster, src or len");
  SYNC_CHECK(c);
  CK(cudaMemcpy(bn + (int64_t)cluster * S_pad, src, sizeof(float) * S, cudaMemcpyHostToDevice));
  return GCPSL_OK;
}

gcpsl_status gcpsl_get_momentum(gcpsl_ctx* c, int cluster, float* dst, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (cluster < 0 || cluster >= c->C || !dst || len != (size_t)c->P)
    return fail(c, GCPSL_E_INVAL, "bad cluster, dst or len");
  std::vector<float> ker(c->P);
  SYNC_CHECK(c);
  CK(cudaMemcpy(ker.data(), c->d_mom + (int64_t)cluster * c->P_pad, sizeof(float) * c->P,
                cudaMemcpyDeviceToHost));
  to_canonical(c, ker.data(), dst);
  return GCPSL_OK;
}

gcpsl_status gcpsl_set_momentum(gcpsl_ctx* c, int cluster, const float* src, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (cluster < 0 || cluster >= c->C || !src || len != (size_t)c->P)
    return fail(c, GCPSL_E_INVAL, "bad cluster, src or len");
  std::vector<float> ker(c->P);
  to_kernel(c, src, ker.data());
  SYNC_CHECK(c);
  CK(cudaMemcpy(c->d_mom + (int64_t)cluster * c->P_pad, ker.data(), sizeof(float) * c->P,
                cudaMemcpyHostToDevice));
  return GCPSL_OK;
}

gcpsl_status gcpsl_get_pool_codes(gcpsl_ctx* c, int layer, uint8_t* dst, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (c->rn || layer < 0 || layer >= c->a.L() || !c->a.conv[layer].pool || !dst)
    return fail(c, GCPSL_E_INVAL, "layer %d has no pooling or dst is NULL", layer);
  const int64_t n = act_elems(c, layer + 1);
  if (len < (size_t)n) return fail(c, GCPSL_E_INVAL, "dst too small");
  std::vector<uint8_t> raw(n);
  SYNC_CHECK(c);
  CK(cudaMemcpy(raw.data(), c->d_code[layer], n, cudaMemcpyDeviceToHost));
  const int ch = c->a.conv[layer].cout, hw = c->a.out_h(layer) * c->a.out_w(layer);
  for (int64_t cb = 0; cb < (int64_t)c->C * c->B; ++cb)
    for (int p = 0; p < hw; ++p)
      for (int k = 0; k < ch; ++k) dst[(cb * ch + k) * hw + p] = raw[(cb * hw + p) * ch + k];
  return GCPSL_OK;
}

gcpsl_status gcpsl_get_relu_masks(gcpsl_ctx* c, uint8_t* dst, size_t len, size_t* needed) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (!c->rn) return fail(c, GCPSL_E_INVAL, "ReLU decisions are kept for the ResNet-18 split");
  return rn_relu_masks(c, dst, len, needed);
}

size_t gcpsl_cut_elems(const gcpsl_ctx* c) {
  if (!c) return 0;
  if (c->rn) return (size_t)c->C * c->B * 64 * 1024;
  return (size_t)act_elems(c, c->a.ncl);
}

gcpsl_status gcpsl_get_cut(gcpsl_ctx* c, int which, float* dst, size_t len) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  const int64_t n = (int64_t)gcpsl_cut_elems(c);
  if (!dst || len < (size_t)n || (which != GCPSL_CUT_ACT && which != GCPSL_CUT_GRAD))
    return fail(c, GCPSL_E_INVAL, "bad dst, len or which");
  const void* src = c->rn ? (const void*)rn_cut(c, which)
                          : (which == GCPSL_CUT_ACT ? c->d_act[c->a.ncl] : c->d_dact[c->a.ncl]);
  std::vector<unsigned char> raw((size_t)n * c->esz);
  SYNC_CHECK(c);
  CK(cudaMemcpy(raw.data(), src, raw.size(), cudaMemcpyDeviceToHost));
  int ch, hw;
  if (c->rn) {
    ch = 64; hw = 1024;
  } else {
    const int l = c->a.ncl - 1;
    ch = c->a.conv[l].cout; hw = c->a.out_h(l) * c->a.out_w(l);
  }
  for (int64_t cb = 0; cb < (int64_t)c->C * c->B; ++cb)
    for (int p = 0; p < hw; ++p)
      for (int k = 0; k < ch; ++k) {
        const int64_t si = (cb * hw + p) * ch + k;
        float v;
        if (c->bf) {
          uint16_t h;
          std::memcpy(&h, raw.data() + 2 * si, 2);
          uint32_t u = (uint32_t)h << 16;
          std::memcpy(&v, &u, 4);
        } else {
          std::memcpy(&v, raw.data() + 4 * si, 4);
        }
        dst[(cb * ch + k) * hw + p] = v;
      }
  return GCPSL_OK;
}

gcpsl_status gcpsl_get_sample(gcpsl_ctx* c, int32_t* idx, int32_t* counts) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  SYNC_CHECK(c);
  if (idx) CK(cudaMemcpy(idx, c->d_idx, sizeof(int32_t) * c->C * c->B, cudaMemcpyDeviceToHost));
  if (counts)
    CK(cudaMemcpy(counts, c->d_counts, sizeof(int32_t) * (size_t)c->C * c->K,
                  cudaMemcpyDeviceToHost));
  return GCPSL_OK;
}

int64_t gcpsl_rounds(const gcpsl_ctx* c) { return c ? c->t : -1; }

gcpsl_status gcpsl_set_stream(gcpsl_ctx* c, void* stream) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  SYNC_CHECK(c);
  c->stream = stream ? (cudaStream_t)stream : c->own_stream;
  return GCPSL_OK;
}

gcpsl_status gcpsl_set_timing(gcpsl_ctx* c, int enable) {
  if (!c) return GCPSL_E_INVAL;
  c->timing = enable != 0;
  return GCPSL_OK;
}

int64_t gcpsl_kernels_launched(const gcpsl_ctx* c) { return c ? c->launched : -1; }

gcpsl_status gcpsl_set_timing_filter(gcpsl_ctx* c, const char* prefix) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  const std::string f = prefix ? prefix : "";
  if (f == c->timer.filter) return GCPSL_OK;
  // the timed graphs hold event nodes for the old selection: rebuild them
  SYNC_CHECK(c);
  account_graph_marks(c);
  for (auto& v : c->graph)
    for (int k = 1; k < 3; ++k) {
      auto& g = v[k];
      if (g.exec) cudaGraphExecDestroy(g.exec);
      g.exec = nullptr;
      for (auto& m : g.marks) { cudaEventDestroy(m.a); cudaEventDestroy(m.b); }
      g.marks.clear();
    }
  c->timer.filter = f;
  return GCPSL_OK;
}

gcpsl_status gcpsl_check_wait_timeout(gcpsl_ctx* c, uint64_t limit_ns) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  if (limit_ns < 1 || limit_ns > 1000000000ull)
    return fail(c, GCPSL_E_INVAL, "limit_ns %llu outside [1, 1e9]", (unsigned long long)limit_ns);
  SYNC_CHECK(c);
  CK(launch_wait_probe(c->stream, c->d_err, limit_ns));
  SYNC_CHECK(c);      // the probe's error word: GCPSL_E_TIMEOUT
  return fail(c, GCPSL_E_CUDA, "the bounded wait did not report its timeout");
}

gcpsl_status gcpsl_set_graph(gcpsl_ctx* c, int enable) {
  gcpsl_status st = check_usable(c);
  if (st != GCPSL_OK) return st;
  SYNC_CHECK(c);
  account_graph_marks(c);
  c->use_graph = enable != 0;
  return GCPSL_OK;
}

int gcpsl_kernel_times(gcpsl_ctx* c, const char** names, int64_t* launches, double* ms, int cap) {
  if (!c) return -1;
  cudaStreamSynchronize(c->stream);
  account_graph_marks(c);
  c->timer.collect();
  const int n = (int)c->timer.names.size();
  for (int i = 0; i < n && i < cap; ++i) {
    if (names) names[i] = c->timer.names[i];
    if (launches) launches[i] = c->timer.launches[i];
    if (ms) ms[i] = c->timer.ms[i];
  }
  return n;
}

void gcpsl_reset_kernel_times(gcpsl_ctx* c) {
  if (!c) return;
  cudaStreamSynchronize(c->stream);
  account_graph_marks(c);
  c->timer.reset();
}

const char* gcpsl_last_error(const gcpsl_ctx* c) {
  return c ? c->err.c_str() : g_init_error.c_str();
}

void gcpsl_destroy(gcpsl_ctx* c) {
  if (!c) return;
  free_all(c);
  delete c;
}

}  // extern "C"
