/*
 * gcpsl_resnet.c -- the CIFAR ResNet-18 split model of the CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY, like gcpsl_oracle.c (which calls into this file
 * for architectures 2 and 3).  Plain fp64 loops in PyTorch's NCHW / OIHW layouts.
 *
 * Model (the workload's split of the CIFAR ResNet-18):
 *   client: stem conv3x3 3->64 (stride 1, pad 1, no bias), GroupNorm, ReLU;
 *           stage 1 = two basic blocks of 64 channels (GroupNorm); 32 groups
 *           unless orn_set_norm chooses another divisor of 64.
 *   server: stages 2-4 (128 / 256 / 512 channels, two basic blocks each, the
 *           first with stride 2 and a 1x1 stride-2 convolution + norm on the
 *           shortcut), train-mode BatchNorm; global average pool over 4x4;
 *           linear 512 -> J with bias (J = 10 classes for architecture 2,
 *           100 for architecture 3, the CIFAR-100 shape of Section V-A).
 *   basic block: out = relu(N2(conv2(relu(N1(conv1(x))))) + s),
 *                s = x, or Ns(conv_s(x)) when the shape changes.
 *   norms: x_hat = (y - mean) / sqrt(var + eps), var biased (eps 1e-5 unless
 *          orn_set_norm sets it), then
 *          gamma * x_hat + beta; GroupNorm over (channels of the group, H, W)
 *          per example, BatchNorm over (B, H, W) per channel.  BatchNorm's
 *          running statistics follow PyTorch: momentum 0.1 (or the one given
 *          to orn_set_norm), the running variance takes the unbiased batch
 *          variance.
 *
 * Canonical parameter blob: PyTorch's named_parameters() order (conv1.weight,
 * bn1.weight, bn1.bias, layer1.0.conv1.weight, ..., shortcut.0.weight,
 * shortcut.1.weight, shortcut.1.bias, ..., linear.weight, linear.bias); the
 * client segment is the stem and stage 1.  The BatchNorm state blob holds,
 * per BatchNorm layer in module order, running_mean[ch] then running_var[ch].
 *
 * bf16 operand mode rounds (to nearest even) every value that the GPU path
 * stores in bf16: the input, the conv / linear weights, every convolution
 * output, every norm(+residual)+ReLU output, the pooled features, the
 * gradient entering the last block, every norm-backward output and every
 * block-input gradient (the sum of its two paths, rounded once).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* norm hyper-parameters: GroupNorm groups, eps of both norms, BatchNorm
 * running-statistics momentum (PyTorch's defaults; orn_set_norm) */
static int RN_GROUPS = 32;
static double RN_EPS = 1e-5;
static double RN_BN_MOMENTUM = 0.1;

/* returns nonzero when the group count does not divide every GroupNorm
 * layer's 64 channels */
int orn_set_norm(int groups, double eps, double momentum) {
  if (groups < 1 || 64 % groups || !(eps > 0.0) || !(momentum > 0.0 && momentum <= 1.0))
    return 1;
  RN_GROUPS = groups;
  RN_EPS = eps;
  RN_BN_MOMENTUM = momentum;
  return 0;
}

typedef struct { int cin, cout, k, stride, hin, win; int64_t w; } rn_conv;
typedef struct { int ch, gn; int64_t g, b; int64_t s; } rn_norm;   /* s: BN state offset */
typedef struct { rn_conv c1, c2, cs; rn_norm n1, n2, ns; int sc; } rn_block;
typedef struct {
  rn_conv stem; rn_norm stem_n; rn_block blk[8];
  int64_t fcw, fcb, p_client, p_total, s_total;
  int J;                                   /* classes: outputs of the linear head */
} rn_net;

static void rn_norm_at(rn_norm* n, int ch, int gn, int64_t* p, int64_t* s) {
  n->ch = ch; n->gn = gn;
  n->g = *p; n->b = *p + ch; *p += 2 * ch;
  n->s = -1;
  if (!gn) { n->s = *s; *s += 2 * ch; }
}

static void rn_build(rn_net* n, int J) {
  int64_t p = 0, s = 0;
  n->J = J;
  n->stem = (rn_conv){3, 64, 3, 1, 32, 32, p}; p += 64 * 3 * 9;
  rn_norm_at(&n->stem_n, 64, 1, &p, &s);
  const int widths[4] = {64, 128, 256, 512};
  int cin = 64, hw = 32;
  for (int st = 0; st < 4; ++st)
    for (int j = 0; j < 2; ++j) {
      rn_block* b = &n->blk[st * 2 + j];
      const int cout = widths[st], stride = (st > 0 && j == 0) ? 2 : 1, gn = st == 0;
      const int ho = hw / stride;
      b->c1 = (rn_conv){cin, cout, 3, stride, hw, hw, p}; p += (int64_t)cout * cin * 9;
      rn_norm_at(&b->n1, cout, gn, &p, &s);
      b->c2 = (rn_conv){cout, cout, 3, 1, ho, ho, p}; p += (int64_t)cout * cout * 9;
      rn_norm_at(&b->n2, cout, gn, &p, &s);
      b->sc = stride != 1 || cin != cout;
      if (b->sc) {
        b->cs = (rn_conv){cin, cout, 1, stride, hw, hw, p}; p += (int64_t)cout * cin;
        rn_norm_at(&b->ns, cout, gn, &p, &s);
      }
      if (st == 0 && j == 1) n->p_client = p;
      cin = cout; hw = ho;
    }
  n->fcw = p; p += (int64_t)J * 512;
  n->fcb = p; p += J;
  n->p_total = p;
  n->s_total = s;
}

int64_t orn_num_params(int J, int segment) {
  rn_net n;
  if (J < 2) return -1;
  rn_build(&n, J);
  if (segment == 0) return n.p_client;
  if (segment == 1) return n.p_total - n.p_client;
  if (segment == 2) return n.s_total;
  return -1;
}

static double rn_bf16(double x) {
  float f = (float)x; uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  u &= 0xFFFF0000u;
  memcpy(&f, &u, 4);
  return (double)f;
}
static void rn_round(double* v, int64_t n, int on) {
  if (!on) return;
  for (int64_t i = 0; i < n; ++i) v[i] = rn_bf16(v[i]);
}

static int out_hw(const rn_conv* c) { return c->hin / c->stride; }

/* y[b,co,oy,ox] = sum_{ci,ky,kx} W[co,ci,ky,kx] x[b,ci,oy*s+ky-p,ox*s+kx-p], p = k/2 */
static void conv_fwd(const rn_conv* c, int B, const double* x, const double* w, double* y) {
  const int Ho = out_hw(c), Wo = Ho, H = c->hin, W = c->win, k = c->k, pad = k / 2, s = c->stride;
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < B; ++b)
    for (int co = 0; co < c->cout; ++co) {
      double* yp = y + ((int64_t)b * c->cout + co) * Ho * Wo;
      for (int i = 0; i < Ho * Wo; ++i) yp[i] = 0.0;
      for (int ci = 0; ci < c->cin; ++ci) {
        const double* xp = x + ((int64_t)b * c->cin + ci) * H * W;
        for (int ky = 0; ky < k; ++ky)
          for (int kx = 0; kx < k; ++kx) {
            const double wv = w[(((int64_t)co * c->cin + ci) * k + ky) * k + kx];
            for (int oy = 0; oy < Ho; ++oy) {
              const int iy = oy * s + ky - pad;
              if (iy < 0 || iy >= H) continue;
              for (int ox = 0; ox < Wo; ++ox) {
                const int ix = ox * s + kx - pad;
                if (ix < 0 || ix >= W) continue;
                yp[oy * Wo + ox] += wv * xp[iy * W + ix];
              }
            }
          }
      }
    }
}

/* dW[co,ci,ky,kx] = sum_{b,oy,ox} dy[b,co,oy,ox] x[b,ci,oy*s+ky-p,ox*s+kx-p] */
static void conv_wgrad(const rn_conv* c, int B, const double* x, const double* dy, double* dw) {
  const int Ho = out_hw(c), Wo = Ho, H = c->hin, W = c->win, k = c->k, pad = k / 2, s = c->stride;
#pragma omp parallel for collapse(2) schedule(static)
  for (int co = 0; co < c->cout; ++co)
    for (int ci = 0; ci < c->cin; ++ci)
      for (int ky = 0; ky < k; ++ky)
        for (int kx = 0; kx < k; ++kx) {
          double acc = 0.0;
          for (int b = 0; b < B; ++b) {
            const double* dp = dy + ((int64_t)b * c->cout + co) * Ho * Wo;
            const double* xp = x + ((int64_t)b * c->cin + ci) * H * W;
            for (int oy = 0; oy < Ho; ++oy) {
              const int iy = oy * s + ky - pad;
              if (iy < 0 || iy >= H) continue;
              for (int ox = 0; ox < Wo; ++ox) {
                const int ix = ox * s + kx - pad;
                if (ix < 0 || ix >= W) continue;
                acc += dp[oy * Wo + ox] * xp[iy * W + ix];
              }
            }
          }
          dw[(((int64_t)co * c->cin + ci) * k + ky) * k + kx] = acc;
        }
}

/* dx[b,ci,iy,ix] = sum over (co, ky, kx, oy, ox) with iy = oy*s+ky-p and
 * ix = ox*s+kx-p of dy[b,co,oy,ox] W[co,ci,ky,kx] (added to dx) */
static void conv_dgrad_add(const rn_conv* c, int B, const double* dy, const double* w, double* dx) {
  const int Ho = out_hw(c), Wo = Ho, H = c->hin, W = c->win, k = c->k, pad = k / 2, s = c->stride;
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < B; ++b)
    for (int ci = 0; ci < c->cin; ++ci) {
      double* xp = dx + ((int64_t)b * c->cin + ci) * H * W;
      for (int co = 0; co < c->cout; ++co) {
        const double* dp = dy + ((int64_t)b * c->cout + co) * Ho * Wo;
        for (int ky = 0; ky < k; ++ky)
          for (int kx = 0; kx < k; ++kx) {
            const double wv = w[(((int64_t)co * c->cin + ci) * k + ky) * k + kx];
            for (int oy = 0; oy < Ho; ++oy) {
              const int iy = oy * s + ky - pad;
              if (iy < 0 || iy >= H) continue;
              for (int ox = 0; ox < Wo; ++ox) {
                const int ix = ox * s + kx - pad;
                if (ix < 0 || ix >= W) continue;
                xp[iy * W + ix] += dp[oy * Wo + ox] * wv;
              }
            }
          }
      }
    }
}

/* Normalisation sets: GroupNorm -> (example b, group g) over its channels
 * and H x W; BatchNorm -> channel c over B x H x W.  set(i) enumerates them. */
typedef struct { int B, C, HW, gn, cpg; } nset;
static int nset_count(const nset* q) { return q->gn ? q->B * RN_GROUPS : q->C; }
static int64_t nset_size(const nset* q) {
  return q->gn ? (int64_t)q->cpg * q->HW : (int64_t)q->B * q->HW;
}
/* element e of set i -> index into [B][C][HW] and its channel */
static int64_t nset_elem(const nset* q, int i, int64_t e, int* ch) {
  if (q->gn) {
    const int b = i / RN_GROUPS, g = i % RN_GROUPS;
    const int c = g * q->cpg + (int)(e / q->HW);
    *ch = c;
    return ((int64_t)b * q->C + c) * q->HW + e % q->HW;
  }
  const int b = (int)(e / q->HW);
  *ch = i;
  return ((int64_t)b * q->C + i) * q->HW + e % q->HW;
}

/* out = gamma * x_hat + beta (+ res), then ReLU when relu; mean / rstd per set */
/* With relu, mask[k] records the decision: bit 0 = the output passes the
 * ReLU (the decision used), bit 1 = the pre-ReLU value is positive (this
 * run's own sign), bit 2 = ambiguous: |value| <= relu_tol * RMS of the
 * layer's pre-ReLU values, bit 3 = |value| <= 5 relu_tol * RMS.  When mask_in is set, its bit 0 replaces the
 * sign test (replaying another run's decisions; the output is then the
 * value wherever the given decision passes). */
static double g_relu_tol = 0.0;
void orn_set_relu_tol(double tol) { g_relu_tol = tol; }

static void norm_fwd(const nset* q, const double* y, const double* gamma, const double* beta,
                     const double* res, int relu, double* out, double* mean, double* rstd,
                     double* var_biased, uint8_t* mask, const uint8_t* mask_in) {
  const int ns = nset_count(q);
  const int64_t n = nset_size(q);
#pragma omp parallel for schedule(static)
  for (int i = 0; i < ns; ++i) {
    int ch;
    double s = 0.0;
    for (int64_t e = 0; e < n; ++e) s += y[nset_elem(q, i, e, &ch)];
    const double mu = s / (double)n;
    double v = 0.0;
    for (int64_t e = 0; e < n; ++e) { const double d = y[nset_elem(q, i, e, &ch)] - mu; v += d * d; }
    v /= (double)n;
    const double r = 1.0 / sqrt(v + RN_EPS);
    mean[i] = mu; rstd[i] = r;
    if (var_biased) var_biased[i] = v;
    for (int64_t e = 0; e < n; ++e) {
      const int64_t k = nset_elem(q, i, e, &ch);
      double o = gamma[ch] * (y[k] - mu) * r + beta[ch];
      if (res) o += res[k];
      out[k] = o;                     /* pre-ReLU value; decisions below */
    }
  }
  if (!relu) return;
  const int64_t total = (int64_t)ns * n;
  double ss = 0.0;
  for (int64_t k = 0; k < total; ++k) ss += out[k] * out[k];
  const double thr = g_relu_tol * sqrt(ss / (double)total);
  for (int64_t k = 0; k < total; ++k) {
    const double o = out[k];
    const uint8_t own = (uint8_t)(o > 0.0);
    const uint8_t pass = mask_in ? (uint8_t)(mask_in[k] & 1u) : own;
    mask[k] = (uint8_t)(pass | (own << 1) | ((fabs(o) <= thr) << 2) | ((fabs(o) <= 5.0 * thr) << 3));
    out[k] = pass ? o : 0.0;
  }
}

/* dy = rstd (dxh - mean(dxh) - x_hat mean(dxh x_hat)), dxh = dz gamma, per set;
 * dgamma[c] = sum dz x_hat, dbeta[c] = sum dz (over all sets holding c) */
static void norm_bwd(const nset* q, const double* y, const double* dz, const double* gamma,
                     const double* mean, const double* rstd, double* dy, double* dgamma,
                     double* dbeta) {
  const int ns = nset_count(q);
  const int64_t n = nset_size(q);
  for (int c = 0; c < q->C; ++c) { dgamma[c] = 0.0; dbeta[c] = 0.0; }
  /* per-channel parameter sums in a fixed order: sets in order, elements in order */
  for (int i = 0; i < ns; ++i)
    for (int64_t e = 0; e < n; ++e) {
      int ch;
      const int64_t k = nset_elem(q, i, e, &ch);
      dgamma[ch] += dz[k] * (y[k] - mean[i]) * rstd[i];
      dbeta[ch] += dz[k];
    }
#pragma omp parallel for schedule(static)
  for (int i = 0; i < ns; ++i) {
    int ch;
    double m1 = 0.0, m2 = 0.0;
    for (int64_t e = 0; e < n; ++e) {
      const int64_t k = nset_elem(q, i, e, &ch);
      const double xh = (y[k] - mean[i]) * rstd[i], g = dz[k] * gamma[ch];
      m1 += g; m2 += g * xh;
    }
    m1 /= (double)n; m2 /= (double)n;
    for (int64_t e = 0; e < n; ++e) {
      const int64_t k = nset_elem(q, i, e, &ch);
      const double xh = (y[k] - mean[i]) * rstd[i];
      dy[k] = rstd[i] * (dz[k] * gamma[ch] - m1 - xh * m2);
    }
  }
}

static nset nset_of(const rn_norm* nm, int B, int HW) {
  nset q = {B, nm->ch, HW, nm->gn, nm->ch / RN_GROUPS};
  return q;
}

/* per-norm saved values of the forward */
typedef struct { double* y; double* mean; double* rstd; double* var; } rn_nsave;
typedef struct {
  double* x;                       /* block input (a view of the previous output) */
  double* y1; double* a1; double* y2; double* ys; double* out;
  uint8_t* m1; uint8_t* m2;        /* ReLU decisions of a1 and out */
  rn_nsave n1, n2, ns;
} rn_bsave;

static void* zal(int64_t n) { return calloc((size_t)(n > 0 ? n : 1), sizeof(double)); }

static void nsave_alloc(rn_nsave* s, const rn_norm* nm, int B) {
  const int sets = nm->gn ? B * RN_GROUPS : nm->ch;
  s->mean = (double*)zal(sets); s->rstd = (double*)zal(sets); s->var = (double*)zal(sets);
}
static void nsave_free(rn_nsave* s) { free(s->mean); free(s->rstd); free(s->var); }

/* BatchNorm running statistics (PyTorch: momentum 0.1, unbiased variance) */
static void bn_running(const rn_norm* nm, const rn_nsave* sv, int64_t count, double* state) {
  if (nm->gn || !state) return;
  double* rm = state + nm->s;
  double* rv = state + nm->s + nm->ch;
  for (int c = 0; c < nm->ch; ++c) {
    rm[c] = (1.0 - RN_BN_MOMENTUM) * rm[c] + RN_BN_MOMENTUM * sv->mean[c];
    rv[c] = (1.0 - RN_BN_MOMENTUM) * rv[c] +
            RN_BN_MOMENTUM * sv->var[c] * (double)count / (double)(count - 1);
  }
}

/* one ReLU's decisions between the per-example records [B][tot] and a
 * [B][per] array (the ReLU's NCHW layout) */
static void mask_gather(const uint8_t* rec, int64_t tot, int64_t off, int64_t per, int B,
                        uint8_t* dst) {
  for (int b = 0; b < B; ++b) memcpy(dst + (int64_t)b * per, rec + (int64_t)b * tot + off, (size_t)per);
}
static void mask_scatter(uint8_t* rec, int64_t tot, int64_t off, int64_t per, int B,
                         const uint8_t* src) {
  for (int b = 0; b < B; ++b) memcpy(rec + (int64_t)b * tot + off, src + (int64_t)b * per, (size_t)per);
}

/* One forward (and, with grad != NULL, backward) pass of the split model on
 * B examples x [B][3][32][32].  bn_state (nullable) is updated with this
 * batch's statistics.  cut_act / cut_grad (nullable) receive the client
 * output [B][64][32][32] and the gradient with respect to it. */
int orn_forward_backward_masks(int J, int bf16, double label_smoothing, const double* params,
                               double* bn_state, int B, const double* x,
                               const int32_t* labels, double* loss_out, double* grad,
                               double* cut_act, double* cut_grad, double* logits_out,
                               const uint8_t* masks_in, uint8_t* masks_out,
                               const double* cut_scale);

int orn_forward_backward(int J, int bf16, double label_smoothing, const double* params,
                         double* bn_state, int B, const double* x, const int32_t* labels,
                         double* loss_out, double* grad, double* cut_act, double* cut_grad,
                         double* logits_out) {
  return orn_forward_backward_masks(J, bf16, label_smoothing, params, bn_state, B, x, labels,
                                    loss_out, grad, cut_act, cut_grad, logits_out, NULL, NULL,
                                    NULL);
}

/* ReLU decisions per example: the stem's then, per block, those of a1 and of
 * the block output, NCHW; returns the byte count per example. */
int64_t orn_mask_elems(void) {
  rn_net n;
  rn_build(&n, 10);   /* the ReLU layers do not depend on the class count */
  int64_t e = 64 * 1024;
  for (int i = 0; i < 8; ++i) {
    const int ho = out_hw(&n.blk[i].c1);
    e += 2 * (int64_t)n.blk[i].c1.cout * ho * ho;
  }
  return e;
}

/* As orn_forward_backward; masks_out (nullable) receives every ReLU
 * decision record ([B][orn_mask_elems()] in the order stem, block 0 a1,
 * block 0 out, ...; bits as in norm_fwd), and masks_in (nullable) replaces
 * the sign tests by the given decisions (bit 0), so that a run can follow
 * another run's (e.g. the GPU's) branches exactly.  cut_scale (nullable,
 * [B]) multiplies each example's gradient at the cut before the client
 * segment's backward (the per-client average of Sec. IV-B's other reading;
 * cut_grad receives the scaled gradient). */
int orn_forward_backward_masks(int J, int bf16, double label_smoothing, const double* params,
                               double* bn_state, int B, const double* x,
                               const int32_t* labels, double* loss_out, double* grad,
                               double* cut_act, double* cut_grad, double* logits_out,
                               const uint8_t* masks_in, uint8_t* masks_out,
                               const double* cut_scale) {
  rn_net n;
  if (B <= 0 || J < 2) return 1;
  rn_build(&n, J);
  for (int b = 0; b < B; ++b)
    if (labels[b] < 0 || labels[b] >= J) return 1;
  const int64_t P = n.p_total;
  double* wr = (double*)malloc(sizeof(double) * (size_t)P);
  if (!wr) return 2;
  memcpy(wr, params, sizeof(double) * (size_t)P);
  /* operand copies of the conv and linear weights; norm affine stays exact */
  {
    const rn_conv* cs[25]; int nc = 0;
    cs[nc++] = &n.stem;
    for (int i = 0; i < 8; ++i) {
      cs[nc++] = &n.blk[i].c1; cs[nc++] = &n.blk[i].c2;
      if (n.blk[i].sc) cs[nc++] = &n.blk[i].cs;
    }
    for (int i = 0; i < nc; ++i)
      rn_round(wr + cs[i]->w, (int64_t)cs[i]->cout * cs[i]->cin * cs[i]->k * cs[i]->k, bf16);
    rn_round(wr + n.fcw, (int64_t)J * 512, bf16);
  }
  const int64_t in_n = (int64_t)B * 3 * 1024;
  double* x0 = (double*)zal(in_n);
  memcpy(x0, x, sizeof(double) * (size_t)in_n);
  rn_round(x0, in_n, bf16);

  /* ---- forward ---- */
  const int64_t stem_n = (int64_t)B * 64 * 1024;
  double* ystem = (double*)zal(stem_n);
  double* astem = (double*)zal(stem_n);
  rn_nsave sstem; nsave_alloc(&sstem, &n.stem_n, B);
  uint8_t* mstem = (uint8_t*)calloc((size_t)stem_n, 1);
  /* offsets of each ReLU's decisions within one example's mask record */
  int64_t moff[17], mper[17];
  {
    int64_t o = 0;
    mper[0] = 64 * 1024; moff[0] = o; o += mper[0];
    for (int i = 0; i < 8; ++i) {
      const int ho = out_hw(&n.blk[i].c1);
      mper[1 + 2 * i] = mper[2 + 2 * i] = (int64_t)n.blk[i].c1.cout * ho * ho;
      moff[1 + 2 * i] = o; o += mper[1 + 2 * i];
      moff[2 + 2 * i] = o; o += mper[2 + 2 * i];
    }
  }
  const int64_t mtot = moff[16] + mper[16];
  /* gather / scatter one ReLU's [B][per] decisions from / to the records */
  uint8_t* mtmp = (uint8_t*)calloc((size_t)B * 512 * 1024, 1);
#define MASK_IN(r, dst)                                                          \
  (masks_in ? (mask_gather(masks_in, mtot, moff[r], mper[r], B, dst), (const uint8_t*)(dst)) \
            : (const uint8_t*)NULL)
  conv_fwd(&n.stem, B, x0, wr + n.stem.w, ystem);
  rn_round(ystem, stem_n, bf16);
  {
    nset q = nset_of(&n.stem_n, B, 1024);
    norm_fwd(&q, ystem, wr + n.stem_n.g, wr + n.stem_n.b, NULL, 1, astem, sstem.mean, sstem.rstd,
             sstem.var, mstem, MASK_IN(0, mtmp));
  }
  rn_round(astem, stem_n, bf16);
  rn_bsave sv[8];
  const double* cur = astem;
  for (int i = 0; i < 8; ++i) {
    const rn_block* bk = &n.blk[i];
    rn_bsave* s = &sv[i];
    memset(s, 0, sizeof(*s));
    const int ho = out_hw(&bk->c1), hw = ho * ho;
    const int64_t on = (int64_t)B * bk->c1.cout * hw;
    s->x = (double*)cur;
    s->y1 = (double*)zal(on); s->a1 = (double*)zal(on); s->y2 = (double*)zal(on);
    s->out = (double*)zal(on);
    s->m1 = (uint8_t*)calloc((size_t)on, 1); s->m2 = (uint8_t*)calloc((size_t)on, 1);
    nsave_alloc(&s->n1, &bk->n1, B); nsave_alloc(&s->n2, &bk->n2, B);
    conv_fwd(&bk->c1, B, cur, wr + bk->c1.w, s->y1);
    rn_round(s->y1, on, bf16);
    nset q1 = nset_of(&bk->n1, B, hw);
    norm_fwd(&q1, s->y1, wr + bk->n1.g, wr + bk->n1.b, NULL, 1, s->a1, s->n1.mean, s->n1.rstd,
             s->n1.var, s->m1, MASK_IN(1 + 2 * i, mtmp));
    rn_round(s->a1, on, bf16);
    conv_fwd(&bk->c2, B, s->a1, wr + bk->c2.w, s->y2);
    rn_round(s->y2, on, bf16);
    double* res = (double*)cur;
    double* scv = NULL;
    if (bk->sc) {
      s->ys = (double*)zal(on);
      nsave_alloc(&s->ns, &bk->ns, B);
      conv_fwd(&bk->cs, B, cur, wr + bk->cs.w, s->ys);
      rn_round(s->ys, on, bf16);
      nset qs = nset_of(&bk->ns, B, hw);
      scv = (double*)zal(on);
      norm_fwd(&qs, s->ys, wr + bk->ns.g, wr + bk->ns.b, NULL, 0, scv, s->ns.mean, s->ns.rstd,
               s->ns.var, NULL, NULL);
      res = scv;
    }
    nset q2 = nset_of(&bk->n2, B, hw);
    norm_fwd(&q2, s->y2, wr + bk->n2.g, wr + bk->n2.b, res, 1, s->out, s->n2.mean, s->n2.rstd,
             s->n2.var, s->m2, MASK_IN(2 + 2 * i, mtmp));
    rn_round(s->out, on, bf16);
    free(scv);
    cur = s->out;
    if (bn_state) {
      bn_running(&bk->n1, &s->n1, (int64_t)B * hw, bn_state);
      bn_running(&bk->n2, &s->n2, (int64_t)B * hw, bn_state);
      if (bk->sc) bn_running(&bk->ns, &s->ns, (int64_t)B * hw, bn_state);
    }
  }
  /* global average pool over 4x4, linear layer, softmax cross-entropy */
  double* h = (double*)zal((int64_t)B * 512);
  for (int b = 0; b < B; ++b)
    for (int c = 0; c < 512; ++c) {
      double s = 0.0;
      for (int p = 0; p < 16; ++p) s += cur[((int64_t)b * 512 + c) * 16 + p];
      h[b * 512 + c] = s / 16.0;
    }
  rn_round(h, (int64_t)B * 512, bf16);
  const double* Wfc = wr + n.fcw;
  const double* bfc = wr + n.fcb;
  double* logits = (double*)zal((int64_t)B * J);
  double* dlog = (double*)zal((int64_t)B * J);
  double loss = 0.0;
  for (int b = 0; b < B; ++b) {
    double* z = logits + b * J;
    for (int j = 0; j < J; ++j) {
      double s = bfc[j];
      for (int k = 0; k < 512; ++k) s += h[b * 512 + k] * Wfc[j * 512 + k];
      z[j] = s;
    }
    double m = z[0];
    for (int j = 1; j < J; ++j) m = z[j] > m ? z[j] : m;
    double se = 0.0;
    for (int j = 0; j < J; ++j) se += exp(z[j] - m);
    const double lse = m + log(se);
    for (int j = 0; j < J; ++j) {
      const double t = (j == labels[b] ? 1.0 - label_smoothing : 0.0) + label_smoothing / J;
      loss += t * (lse - z[j]);
      dlog[b * J + j] = (exp(z[j] - lse) - t) / B;
    }
  }
  *loss_out = loss / B;
  if (masks_out) {
    mask_scatter(masks_out, mtot, moff[0], mper[0], B, mstem);
    for (int i = 0; i < 8; ++i) {
      mask_scatter(masks_out, mtot, moff[1 + 2 * i], mper[1 + 2 * i], B, sv[i].m1);
      mask_scatter(masks_out, mtot, moff[2 + 2 * i], mper[2 + 2 * i], B, sv[i].m2);
    }
  }
  if (logits_out) memcpy(logits_out, logits, sizeof(double) * (size_t)B * J);
  if (cut_act) memcpy(cut_act, sv[1].out, sizeof(double) * (size_t)stem_n);

  int rc = 0;
  if (grad) {
    memset(grad, 0, sizeof(double) * (size_t)P);
    for (int j = 0; j < J; ++j) {
      double sb = 0.0;
      for (int b = 0; b < B; ++b) sb += dlog[b * J + j];
      grad[n.fcb + j] = sb;
      for (int k = 0; k < 512; ++k) {
        double s = 0.0;
        for (int b = 0; b < B; ++b) s += dlog[b * J + j] * h[b * 512 + k];
        grad[n.fcw + j * 512 + k] = s;
      }
    }
    /* gradient entering the last block: dh / 16 at every pooled position */
    const int64_t last_n = (int64_t)B * 512 * 16;
    double* dout = (double*)zal(last_n);
    for (int b = 0; b < B; ++b)
      for (int c = 0; c < 512; ++c) {
        double s = 0.0;
        for (int j = 0; j < J; ++j) s += dlog[b * J + j] * Wfc[j * 512 + c];
        for (int p = 0; p < 16; ++p) dout[((int64_t)b * 512 + c) * 16 + p] = s / 16.0;
      }
    rn_round(dout, last_n, bf16);
    for (int i = 7; i >= 0; --i) {
      const rn_block* bk = &n.blk[i];
      rn_bsave* s = &sv[i];
      const int ho = out_hw(&bk->c1), hw = ho * ho;
      const int64_t on = (int64_t)B * bk->c1.cout * hw;
      const int64_t in_e = (int64_t)B * bk->c1.cin * bk->c1.hin * bk->c1.win;
      /* through the output ReLU */
      double* dz = (double*)zal(on);
      for (int64_t k = 0; k < on; ++k) dz[k] = (s->m2[k] & 1u) ? dout[k] : 0.0;
      double* dy2 = (double*)zal(on);
      nset q2 = nset_of(&bk->n2, B, hw);
      norm_bwd(&q2, s->y2, dz, wr + bk->n2.g, s->n2.mean, s->n2.rstd, dy2, grad + bk->n2.g,
               grad + bk->n2.b);
      rn_round(dy2, on, bf16);
      conv_wgrad(&bk->c2, B, s->a1, dy2, grad + bk->c2.w);
      double* da1 = (double*)zal(on);
      conv_dgrad_add(&bk->c2, B, dy2, wr + bk->c2.w, da1);
      rn_round(da1, on, bf16);
      for (int64_t k = 0; k < on; ++k) if (!(s->m1[k] & 1u)) da1[k] = 0.0;
      double* dy1 = (double*)zal(on);
      nset q1 = nset_of(&bk->n1, B, hw);
      norm_bwd(&q1, s->y1, da1, wr + bk->n1.g, s->n1.mean, s->n1.rstd, dy1, grad + bk->n1.g,
               grad + bk->n1.b);
      rn_round(dy1, on, bf16);
      conv_wgrad(&bk->c1, B, s->x, dy1, grad + bk->c1.w);
      double* dx = (double*)zal(in_e);
      conv_dgrad_add(&bk->c1, B, dy1, wr + bk->c1.w, dx);
      if (bk->sc) {
        double* dys = (double*)zal(on);
        nset qs = nset_of(&bk->ns, B, hw);
        norm_bwd(&qs, s->ys, dz, wr + bk->ns.g, s->ns.mean, s->ns.rstd, dys, grad + bk->ns.g,
                 grad + bk->ns.b);
        rn_round(dys, on, bf16);
        conv_wgrad(&bk->cs, B, s->x, dys, grad + bk->cs.w);
        conv_dgrad_add(&bk->cs, B, dys, wr + bk->cs.w, dx);
        free(dys);
      } else {
        for (int64_t k = 0; k < in_e; ++k) dx[k] += dz[k];
      }
      rn_round(dx, in_e, bf16);
      if (i == 2 && cut_scale) {
        const int64_t per = in_e / B;
        for (int64_t k = 0; k < in_e; ++k) dx[k] *= cut_scale[k / per];
        rn_round(dx, in_e, bf16);
      }
      if (i == 2 && cut_grad) memcpy(cut_grad, dx, sizeof(double) * (size_t)in_e);
      free(dz); free(dy2); free(da1); free(dy1);
      free(dout);
      dout = dx;
    }
    /* stem: through its ReLU and GroupNorm, then the weight gradient */
    double* dz = (double*)zal(stem_n);
    for (int64_t k = 0; k < stem_n; ++k) dz[k] = (mstem[k] & 1u) ? dout[k] : 0.0;
    double* dy = (double*)zal(stem_n);
    nset q = nset_of(&n.stem_n, B, 1024);
    norm_bwd(&q, ystem, dz, wr + n.stem_n.g, sstem.mean, sstem.rstd, dy, grad + n.stem_n.g,
             grad + n.stem_n.b);
    rn_round(dy, stem_n, bf16);
    conv_wgrad(&n.stem, B, x0, dy, grad + n.stem.w);
    free(dz); free(dy); free(dout);
  }
  for (int i = 0; i < 8; ++i) {
    rn_bsave* s = &sv[i];
    free(s->y1); free(s->a1); free(s->y2); free(s->ys); free(s->out); free(s->m1); free(s->m2);
    nsave_free(&s->n1); nsave_free(&s->n2);
    if (n.blk[i].sc) nsave_free(&s->ns);
  }
  nsave_free(&sstem);
  free(mstem); free(mtmp);
#undef MASK_IN
  free(ystem); free(astem); free(x0); free(h); free(logits); free(dlog); free(wr);
  return rc;
}

/* initial BatchNorm state: running_mean 0, running_var 1 (PyTorch) */
void orn_init_bn_state(double* state) {
  rn_net n;
  rn_build(&n, 10);   /* the BatchNorm layers do not depend on the class count */
  const rn_norm* all[3 * 8];
  int k = 0;
  for (int i = 0; i < 8; ++i) {
    all[k++] = &n.blk[i].n1; all[k++] = &n.blk[i].n2;
    if (n.blk[i].sc) all[k++] = &n.blk[i].ns;
  }
  for (int i = 0; i < k; ++i) {
    if (all[i]->gn) continue;
    for (int c = 0; c < all[i]->ch; ++c) {
      state[all[i]->s + c] = 0.0;
      state[all[i]->s + all[i]->ch + c] = 1.0;
    }
  }
}
