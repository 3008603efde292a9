/*
 * gcpsl_oracle.c -- plain, slow CPU oracle of one GCPSL training step.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark load this library; the product path never
 * does.  It shares no code, header or table with the CUDA library.
 *
 * What it computes (Algorithm 2, restricted to a fixed fusion interval of F
 * local rounds):
 *   - cluster-local GPSL sampling of B examples per round (Eq. 1), defined as
 *     an epoch permutation of the cluster's pooled examples drawn from
 *     Philox4x32-10 keys (Salmon et al., SC'11) and sliced into batches; each
 *     example is scheduled once per epoch (Section III-A), the n_c mod B
 *     leftovers are not scheduled in that epoch;
 *   - client-segment forward to the cut, server-segment forward, softmax
 *     cross-entropy averaged over the batch, backward to the cut gradient
 *     and through the client segment (Section III-A, Algorithm 2);
 *   - one client gradient per cluster: the gradient of the batch-mean loss,
 *     i.e. the example-weighted average of the active clients' gradients
 *     (Section IV-B: all client replicas of a cluster share one model);
 *   - SGD with PyTorch's undampened momentum convention, per replica;
 *   - every F rounds, fusion theta_bar = sum_n q_n theta_n with
 *     q_n = |D_{C_n}| / |D| (Eq. 5), broadcast to every replica; momentum
 *     buffers are not fused (Section IV-C).
 *
 * Arithmetic is fp64.  In "bf16 operand" mode every value that the GPU path
 * stores as bf16 (gathered images, weight shadows, layer outputs, the
 * pre-activation gradients and the data gradients) is rounded to bf16
 * (round to nearest even) at that point, so the comparison isolates the
 * accumulation order.
 *
 * Layouts are PyTorch's: activations NCHW, conv weights OIHW, the flatten
 * before the linear layer in (C, H, W) order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* the CIFAR ResNet-18 split model (architectures 2 and 3: 10 and 100
 * classes), gcpsl_resnet.c */
int64_t orn_num_params(int J, int segment);
int orn_forward_backward_masks(int J, int bf16, double label_smoothing, const double* params,
                               double* bn_state, int B, const double* x,
                               const int32_t* labels, double* loss_out, double* grad,
                               double* cut_act, double* cut_grad, double* logits_out,
                               const uint8_t* masks_in, uint8_t* masks_out,
                               const double* cut_scale);
int64_t orn_mask_elems(void);
void orn_init_bn_state(double* state);
int orn_set_norm(int groups, double eps, double momentum);
#define ORC_RESNET18 2
#define ORC_RESNET18_C100 3

#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_ENOMEM 2
#define ORC_EUNSUPPORTED 6

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 counter-based generator (Salmon et al., SC'11, Sec. 3):    */
/* ten rounds of two 32x32->64 multiplications; the key is bumped by the    */
/* Weyl constants between rounds.                                           */
/* ------------------------------------------------------------------------ */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { k0 += W0; k1 += W1; }
    uint64_t p0 = (uint64_t)M0 * c0;
    uint64_t p1 = (uint64_t)M1 * c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* ------------------------------------------------------------------------ */
/* GPSL sampler of one cluster                                              */
/* ------------------------------------------------------------------------ */
typedef struct { uint64_t key; int32_t j; } keyed_t;

static int cmp_keyed(const void* a, const void* b) {
  const keyed_t* x = (const keyed_t*)a; const keyed_t* y = (const keyed_t*)b;
  if (x->key != y->key) return x->key < y->key ? -1 : 1;
  return (x->j > y->j) - (x->j < y->j);
}

/* Epoch permutation: ids[] are the cluster's global example ids.  Each id j
 * gets key Philox(counter=(j, epoch, cluster, 0), key=(seed_lo, seed_hi)),
 * k64 = out0 << 32 | out1; the permutation is the ids sorted by (k64, j). */
void orc_epoch_perm(const int32_t* ids, int64_t n, uint32_t cluster, uint32_t epoch,
                    uint64_t seed, int32_t* perm) {
  keyed_t* t = (keyed_t*)malloc(sizeof(keyed_t) * (size_t)(n > 0 ? n : 1));
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  for (int64_t i = 0; i < n; ++i) {
    uint32_t ctr[4] = {(uint32_t)ids[i], epoch, cluster, 0u}, o[4];
    orc_philox4x32_10(ctr, key, o);
    t[i].key = ((uint64_t)o[0] << 32) | o[1];
    t[i].j = ids[i];
  }
  qsort(t, (size_t)n, sizeof(keyed_t), cmp_keyed);
  for (int64_t i = 0; i < n; ++i) perm[i] = t[i].j;
  free(t);
}

static const int32_t* g_owner_for_sort;
static int cmp_owner_id(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  int32_t ox = g_owner_for_sort[x], oy = g_owner_for_sort[y];
  if (ox != oy) return ox < oy ? -1 : 1;
  return (x > y) - (x < y);
}

/* Round s of an epoch: the B ids perm[sB .. sB+B), ordered by (owner, id);
 * counts[k] = b_{k,t} (Eq. 1); returns |A_{n,t}| = #{k : b_{k,t} > 0}. */
int orc_sample_round(const int32_t* perm, int64_t s, int B, const int32_t* owner, int K,
                     int32_t* idx, int32_t* counts) {
  memcpy(idx, perm + s * B, sizeof(int32_t) * (size_t)B);
  g_owner_for_sort = owner;
  qsort(idx, (size_t)B, sizeof(int32_t), cmp_owner_id);
  for (int k = 0; k < K; ++k) counts[k] = 0;
  for (int b = 0; b < B; ++b) counts[owner[idx[b]]]++;
  int active = 0;
  for (int k = 0; k < K; ++k) active += counts[k] > 0;
  return active;
}

/* ------------------------------------------------------------------------ */
/* Split models                                                             */
/* ------------------------------------------------------------------------ */
typedef struct { int cin, cout, h, w, pool; } conv_l;
typedef struct {
  int ncl, nsv;              /* client / server conv layers */
  conv_l conv[4];
  int fc_in, fc_out;
} arch_t;

static int get_arch(int id, arch_t* a) {
  memset(a, 0, sizeof(*a));
  if (id == 0) {           /* tiny CNN */
    a->ncl = 1; a->nsv = 1;
    a->conv[0] = (conv_l){3, 16, 32, 32, 1};
    a->conv[1] = (conv_l){16, 32, 16, 16, 1};
    a->fc_in = 2048; a->fc_out = 10;
    return 0;
  }
  if (id == 1) {           /* SplitCNN */
    a->ncl = 2; a->nsv = 2;
    a->conv[0] = (conv_l){3, 32, 32, 32, 0};
    a->conv[1] = (conv_l){32, 64, 32, 32, 1};
    a->conv[2] = (conv_l){64, 128, 16, 16, 1};
    a->conv[3] = (conv_l){128, 128, 8, 8, 1};
    a->fc_in = 2048; a->fc_out = 10;
    return 0;
  }
  return -1;
}

/* offsets of conv weight/bias and fc weight/bias in the canonical blob */
typedef struct { int64_t w[4], b[4], fcw, fcb, p_client, p_total; } offs_t;
static void get_offs(const arch_t* a, offs_t* o) {
  int64_t p = 0;
  int L = a->ncl + a->nsv;
  for (int i = 0; i < L; ++i) {
    if (i == a->ncl) o->p_client = p;
    o->w[i] = p; p += (int64_t)a->conv[i].cout * a->conv[i].cin * 9;
    o->b[i] = p; p += a->conv[i].cout;
  }
  o->fcw = p; p += (int64_t)a->fc_out * a->fc_in;
  o->fcb = p; p += a->fc_out;
  o->p_total = p;
}

/* classes of a ResNet-18 architecture id, 0 for any other id */
static int resnet_classes(int arch) {
  return arch == ORC_RESNET18 ? 10 : arch == ORC_RESNET18_C100 ? 100 : 0;
}

int64_t orc_num_params(int arch, int segment) {
  if (resnet_classes(arch)) return orn_num_params(resnet_classes(arch), segment);
  arch_t a; offs_t o;
  if (get_arch(arch, &a)) return -1;
  get_offs(&a, &o);
  return segment == 0 ? o.p_client : o.p_total - o.p_client;
}

static double bf16r(double x) {
  float f = (float)x; uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  u &= 0xFFFF0000u;
  memcpy(&f, &u, 4);
  return (double)f;
}
static void round_buf(double* v, int64_t n, int on) {
  if (!on) return;
  for (int64_t i = 0; i < n; ++i) v[i] = bf16r(v[i]);
}

/* y[b,co,h,w] = bias[co] + sum_{ci,kh,kw} W[co,ci,kh,kw] x[b,ci,h+kh-1,w+kw-1]
 * (3x3 kernel, stride 1, zero padding 1). */
static void conv3x3_fwd(int B, int cin, int cout, int H, int W, const double* x,
                        const double* wt, const double* bias, double* y) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < B; ++b)
    for (int co = 0; co < cout; ++co) {
      double* yp = y + ((int64_t)b * cout + co) * H * W;
      for (int i = 0; i < H * W; ++i) yp[i] = bias[co];
      for (int ci = 0; ci < cin; ++ci)
        for (int kh = 0; kh < 3; ++kh)
          for (int kw = 0; kw < 3; ++kw) {
            double wv = wt[(((int64_t)co * cin + ci) * 3 + kh) * 3 + kw];
            const double* xp = x + ((int64_t)b * cin + ci) * H * W;
            for (int h = 0; h < H; ++h) {
              int ih = h + kh - 1;
              if (ih < 0 || ih >= H) continue;
              for (int w = 0; w < W; ++w) {
                int iw = w + kw - 1;
                if (iw < 0 || iw >= W) continue;
                yp[h * W + w] += wv * xp[ih * W + iw];
              }
            }
          }
    }
}

/* dW[co,ci,kh,kw] = sum_{b,h,w} dy[b,co,h,w] x[b,ci,h+kh-1,w+kw-1];
 * db[co] = sum_{b,h,w} dy[b,co,h,w]. */
static void conv3x3_wgrad(int B, int cin, int cout, int H, int W, const double* x,
                          const double* dy, double* dw, double* db) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int co = 0; co < cout; ++co)
    for (int ci = 0; ci < cin; ++ci)
      for (int kh = 0; kh < 3; ++kh)
        for (int kw = 0; kw < 3; ++kw) {
          double s = 0.0;
          for (int b = 0; b < B; ++b) {
            const double* dyp = dy + ((int64_t)b * cout + co) * H * W;
            const double* xp = x + ((int64_t)b * cin + ci) * H * W;
            for (int h = 0; h < H; ++h) {
              int ih = h + kh - 1;
              if (ih < 0 || ih >= H) continue;
              for (int w = 0; w < W; ++w) {
                int iw = w + kw - 1;
                if (iw < 0 || iw >= W) continue;
                s += dyp[h * W + w] * xp[ih * W + iw];
              }
            }
          }
          dw[(((int64_t)co * cin + ci) * 3 + kh) * 3 + kw] = s;
        }
#pragma omp parallel for schedule(static)
  for (int co = 0; co < cout; ++co) {
    double s = 0.0;
    for (int b = 0; b < B; ++b) {
      const double* dyp = dy + ((int64_t)b * cout + co) * H * W;
      for (int i = 0; i < H * W; ++i) s += dyp[i];
    }
    db[co] = s;
  }
}

/* dx[b,ci,ih,iw] = sum_{co,kh,kw} dy[b,co,ih-kh+1,iw-kw+1] W[co,ci,kh,kw]. */
static void conv3x3_dgrad(int B, int cin, int cout, int H, int W, const double* dy,
                          const double* wt, double* dx) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < B; ++b)
    for (int ci = 0; ci < cin; ++ci) {
      double* dxp = dx + ((int64_t)b * cin + ci) * H * W;
      for (int i = 0; i < H * W; ++i) dxp[i] = 0.0;
      for (int co = 0; co < cout; ++co)
        for (int kh = 0; kh < 3; ++kh)
          for (int kw = 0; kw < 3; ++kw) {
            double wv = wt[(((int64_t)co * cin + ci) * 3 + kh) * 3 + kw];
            const double* dyp = dy + ((int64_t)b * cout + co) * H * W;
            for (int ih = 0; ih < H; ++ih) {
              int h = ih - kh + 1;
              if (h < 0 || h >= H) continue;
              for (int iw = 0; iw < W; ++iw) {
                int w = iw - kw + 1;
                if (w < 0 || w >= W) continue;
                dxp[ih * W + iw] += wv * dyp[h * W + w];
              }
            }
          }
    }
}

/* out = maxpool2x2(relu(y)) or relu(y); arg = first maximum of the window in
 * row-major order (0..3).
 * cand (pooled layers) describes how sharp each window's decision is, for
 * comparisons against an implementation that accumulates in another order:
 * bits 0-3 = the positions q with relu(y_q) >= best - tol*rms(y), rms over
 * the whole layer (the valid maxima), bit 4 = best > 0, bit 5 = the window's
 * largest y lies within tol*rms(y) of zero (the ReLU decision itself is
 * ambiguous).  With tol = 0 only exact ties are candidates. */
static void relu_pool_fwd(int B, int C, int H, int W, int pool, const double* y, double* out,
                          int8_t* arg, uint8_t* cand, double tol) {
  if (!pool) {
    for (int64_t i = 0; i < (int64_t)B * C * H * W; ++i) out[i] = y[i] > 0.0 ? y[i] : 0.0;
    return;
  }
  double rms = 0.0;
  for (int64_t i = 0; i < (int64_t)B * C * H * W; ++i) rms += y[i] * y[i];
  rms = sqrt(rms / ((double)B * C * H * W));
  int Ho = H / 2, Wo = W / 2;
  for (int64_t bc = 0; bc < (int64_t)B * C; ++bc)
    for (int ph = 0; ph < Ho; ++ph)
      for (int pw = 0; pw < Wo; ++pw) {
        const double* yp = y + bc * H * W;
        double v[4], best = 0.0, ymax = 0.0; int bi = 0;
        for (int q = 0; q < 4; ++q) {
          v[q] = yp[(2 * ph + q / 2) * W + 2 * pw + q % 2];
          if (q == 0 || v[q] > ymax) ymax = v[q];
          v[q] = v[q] > 0.0 ? v[q] : 0.0;
          if (q == 0 || v[q] > best) { best = v[q]; bi = q; }
        }
        int64_t o = (bc * Ho + ph) * Wo + pw;
        out[o] = best;
        arg[o] = (int8_t)bi;
        if (cand) {
          uint8_t m = 0;
          for (int q = 0; q < 4; ++q) if (v[q] >= best - tol * rms) m |= (uint8_t)(1u << q);
          if (best > 0.0) m |= 16u;
          if (fabs(ymax) <= tol * rms) m |= 32u;
          cand[o] = m;
        }
      }
}

/* dy = d(out)/dy routed back: through the max-pool to the recorded first
 * maximum, then through ReLU with ReLU'(0) = 0. */
static void relu_pool_bwd(int B, int C, int H, int W, int pool, const double* y,
                          const int8_t* arg, const double* dout, double* dy) {
  int64_t n = (int64_t)B * C * H * W;
  if (!pool) {
    for (int64_t i = 0; i < n; ++i) dy[i] = y[i] > 0.0 ? dout[i] : 0.0;
    return;
  }
  int Ho = H / 2, Wo = W / 2;
  for (int64_t i = 0; i < n; ++i) dy[i] = 0.0;
  for (int64_t bc = 0; bc < (int64_t)B * C; ++bc)
    for (int ph = 0; ph < Ho; ++ph)
      for (int pw = 0; pw < Wo; ++pw) {
        int64_t o = (bc * Ho + ph) * Wo + pw;
        int q = arg[o];
        int64_t yi = bc * H * W + (int64_t)(2 * ph + q / 2) * W + 2 * pw + q % 2;
        dy[yi] = y[yi] > 0.0 ? dout[o] : 0.0;
      }
}

/* One GPSL local round's forward and backward on a batch, for one replica.
 * params: canonical blob (fp64).  x: [B,3,32,32].  Writes the mean
 * cross-entropy, the gradient of it w.r.t. every parameter, the cut
 * activation z and the cut gradient dL/dz (both [B, ch, h, w]), and the
 * logits [B, classes].  Returns 0 or an error code. */
typedef struct {
  double* act[5];     /* act[0] = input, act[i+1] = output of conv i */
  double* pre[4];     /* pre-activation of conv i */
  int8_t* arg[4];
  uint8_t* cand[4];   /* decision sharpness of each pooled window (see relu_pool_fwd) */
  double* dact[5];
  double* dpre;
  double* h;          /* flattened features [B, fc_in] */
  double* logits;
  double* dlogits;
  double* wr;         /* operand copy of the parameters */
} work_t;

static int64_t conv_out_elems(const conv_l* c, int B) {
  return (int64_t)B * c->cout * (c->pool ? c->h * c->w / 4 : c->h * c->w);
}

static void work_free(work_t* w) {
  for (int i = 0; i < 5; ++i) { free(w->act[i]); free(w->dact[i]); }
  for (int i = 0; i < 4; ++i) { free(w->pre[i]); free(w->arg[i]); free(w->cand[i]); }
  free(w->dpre); free(w->h); free(w->logits); free(w->dlogits); free(w->wr);
  memset(w, 0, sizeof(*w));
}

static int work_alloc(work_t* w, const arch_t* a, const offs_t* o, int B) {
  memset(w, 0, sizeof(*w));
  int L = a->ncl + a->nsv;
  int64_t maxpre = 0;
  w->act[0] = (double*)calloc((size_t)B * 3072, sizeof(double));
  w->dact[0] = (double*)calloc((size_t)B * 3072, sizeof(double));
  for (int i = 0; i < L; ++i) {
    int64_t np = (int64_t)B * a->conv[i].cout * a->conv[i].h * a->conv[i].w;
    if (np > maxpre) maxpre = np;
    w->pre[i] = (double*)calloc((size_t)np, sizeof(double));
    w->arg[i] = (int8_t*)calloc((size_t)np, 1);
    w->cand[i] = (uint8_t*)calloc((size_t)np, 1);
    w->act[i + 1] = (double*)calloc((size_t)conv_out_elems(&a->conv[i], B), sizeof(double));
    w->dact[i + 1] = (double*)calloc((size_t)conv_out_elems(&a->conv[i], B), sizeof(double));
  }
  w->dpre = (double*)calloc((size_t)maxpre, sizeof(double));
  w->h = (double*)calloc((size_t)B * a->fc_in, sizeof(double));
  w->logits = (double*)calloc((size_t)B * a->fc_out, sizeof(double));
  w->dlogits = (double*)calloc((size_t)B * a->fc_out, sizeof(double));
  w->wr = (double*)calloc((size_t)o->p_total, sizeof(double));
  if (!w->dpre || !w->h || !w->logits || !w->dlogits || !w->wr) { work_free(w); return ORC_ENOMEM; }
  for (int i = 0; i < L + 1; ++i)
    if (!w->act[i] || !w->dact[i]) { work_free(w); return ORC_ENOMEM; }
  return ORC_OK;
}

/* cut_scale (nullable, [B]): per-example factor on the gradient at the cut
 * before the client segment's backward (see orc_set_client_average) */
static int fwd_bwd(const arch_t* a, const offs_t* o, int bf16, double label_smoothing,
                   const double* params, int B, const int32_t* labels, work_t* w,
                   double* loss_out, double* grad, double tie_tol, const double* cut_scale) {
  int L = a->ncl + a->nsv;
  /* operand copy: bf16(theta) for weights in bf16 mode; biases stay exact */
  memcpy(w->wr, params, sizeof(double) * (size_t)o->p_total);
  for (int i = 0; i < L; ++i)
    round_buf(w->wr + o->w[i], (int64_t)a->conv[i].cout * a->conv[i].cin * 9, bf16);
  round_buf(w->wr + o->fcw, (int64_t)a->fc_out * a->fc_in, bf16);
  round_buf(w->act[0], (int64_t)B * 3072, bf16);

  /* forward through every conv layer */
  for (int i = 0; i < L; ++i) {
    const conv_l* c = &a->conv[i];
    conv3x3_fwd(B, c->cin, c->cout, c->h, c->w, w->act[i], w->wr + o->w[i], w->wr + o->b[i], w->pre[i]);
    relu_pool_fwd(B, c->cout, c->h, c->w, c->pool, w->pre[i], w->act[i + 1], w->arg[i],
                  w->cand[i], tie_tol);
    round_buf(w->act[i + 1], conv_out_elems(c, B), bf16);
  }
  /* flatten (C, H, W) order == NCHW memory order of act[L] */
  memcpy(w->h, w->act[L], sizeof(double) * (size_t)B * a->fc_in);
  const double* Wfc = w->wr + o->fcw;
  const double* bfc = w->wr + o->fcb;
  int J = a->fc_out;
  for (int b = 0; b < B; ++b)
    for (int j = 0; j < J; ++j) {
      double s = bfc[j];
      for (int k = 0; k < a->fc_in; ++k) s += w->h[(int64_t)b * a->fc_in + k] * Wfc[(int64_t)j * a->fc_in + k];
      w->logits[b * J + j] = s;
    }
  /* softmax cross-entropy, mean over the batch; target (1-e) onehot + e/J */
  double loss = 0.0;
  for (int b = 0; b < B; ++b) {
    const double* z = w->logits + b * J;
    double m = z[0];
    for (int j = 1; j < J; ++j) m = z[j] > m ? z[j] : m;
    double se = 0.0;
    for (int j = 0; j < J; ++j) se += exp(z[j] - m);
    double lse = m + log(se);
    for (int j = 0; j < J; ++j) {
      double t = (j == labels[b] ? 1.0 - label_smoothing : 0.0) + label_smoothing / J;
      loss += t * (lse - z[j]);
      w->dlogits[b * J + j] = (exp(z[j] - lse) - t) / B;
    }
  }
  *loss_out = loss / B;
  if (!grad) return ORC_OK;

  /* linear layer backward */
  for (int j = 0; j < J; ++j) {
    double sb = 0.0;
    for (int b = 0; b < B; ++b) sb += w->dlogits[b * J + j];
    grad[o->fcb + j] = sb;
    for (int k = 0; k < a->fc_in; ++k) {
      double s = 0.0;
      for (int b = 0; b < B; ++b) s += w->dlogits[b * J + j] * w->h[(int64_t)b * a->fc_in + k];
      grad[o->fcw + (int64_t)j * a->fc_in + k] = s;
    }
  }
  for (int b = 0; b < B; ++b)
    for (int k = 0; k < a->fc_in; ++k) {
      double s = 0.0;
      for (int j = 0; j < J; ++j) s += w->dlogits[b * J + j] * Wfc[(int64_t)j * a->fc_in + k];
      w->dact[L][(int64_t)b * a->fc_in + k] = s;
    }
  round_buf(w->dact[L], (int64_t)B * a->fc_in, bf16);

  /* conv layers backward, last to first; layer 0 needs no data gradient */
  for (int i = L - 1; i >= 0; --i) {
    const conv_l* c = &a->conv[i];
    if (i == a->ncl - 1 && cut_scale) {
      const int64_t per = conv_out_elems(c, 1), n = per * B;
      for (int64_t k = 0; k < n; ++k) w->dact[i + 1][k] *= cut_scale[k / per];
      round_buf(w->dact[i + 1], n, bf16);
    }
    int64_t np = (int64_t)B * c->cout * c->h * c->w;
    relu_pool_bwd(B, c->cout, c->h, c->w, c->pool, w->pre[i], w->arg[i], w->dact[i + 1], w->dpre);
    round_buf(w->dpre, np, bf16);
    conv3x3_wgrad(B, c->cin, c->cout, c->h, c->w, w->act[i], w->dpre, grad + o->w[i], grad + o->b[i]);
    if (i > 0) {
      conv3x3_dgrad(B, c->cin, c->cout, c->h, c->w, w->dpre, w->wr + o->w[i], w->dact[i]);
      round_buf(w->dact[i], (int64_t)B * c->cin * c->h * c->w, bf16);
    }
  }
  return ORC_OK;
}

/* Standalone forward/backward for the pins: params fp64 canonical blob,
 * x [B,3,32,32] fp64.  grad (nullable) receives dL/dtheta, cut_act and
 * cut_grad (nullable) the cut tensors, logits (nullable) [B, classes]. */
int orc_forward_backward(int arch, int bf16, double label_smoothing, const double* params,
                         int B, const double* x, const int32_t* labels, double* loss,
                         double* grad, double* cut_act, double* cut_grad, double* logits) {
  arch_t a; offs_t o; work_t w;
  if (get_arch(arch, &a)) return ORC_EUNSUPPORTED;
  get_offs(&a, &o);
  if (B <= 0) return ORC_EINVAL;
  if (work_alloc(&w, &a, &o, B)) return ORC_ENOMEM;
  memcpy(w.act[0], x, sizeof(double) * (size_t)B * 3072);
  double* g = grad ? grad : NULL;
  int rc = fwd_bwd(&a, &o, bf16, label_smoothing, params, B, labels, &w, loss, g, 0.0, NULL);
  int64_t ncut = conv_out_elems(&a.conv[a.ncl - 1], B);
  if (cut_act) memcpy(cut_act, w.act[a.ncl], sizeof(double) * (size_t)ncut);
  if (cut_grad && g) memcpy(cut_grad, w.dact[a.ncl], sizeof(double) * (size_t)ncut);
  if (logits) memcpy(logits, w.logits, sizeof(double) * (size_t)B * a.fc_out);
  work_free(&w);
  return rc;
}

/* ------------------------------------------------------------------------ */
/* Fusion (Eq. 5): out[p] = sum_n q[n] theta[n][p], summed in n order.       */
/* ------------------------------------------------------------------------ */
void orc_fuse_arrays(int C, int64_t P, const double* q, const double* theta, double* out) {
  for (int64_t p = 0; p < P; ++p) {
    double s = 0.0;
    for (int n = 0; n < C; ++n) s += q[n] * theta[(int64_t)n * P + p];
    out[p] = s;
  }
}

/* ------------------------------------------------------------------------ */
/* Training context: C cluster workloads stepped in lockstep.               */
/* assignment[k] in [0, C) is client k's cluster; -1 means no cluster of    */
/* this context serves client k (its examples are never sampled here).      */
/* Cluster k draws its permutation keys with cluster id cluster_base + k.   */
/* The images are read in place: the caller keeps them alive.               */
/* ------------------------------------------------------------------------ */
typedef struct {
  int arch, bf16, K, C, B, F, nesterov, cluster_base;
  double lr, momentum, wd, ls;
  uint64_t seed;
  arch_t a; offs_t o;
  int64_t n; const float* images_src; float* images; int32_t* labels; int32_t* owner;
  int32_t** ids; int64_t* nc; int32_t** perm; int64_t* cur_epoch;
  double* q;
  double* theta; double* mom; double* grad;   /* [C][P] */
  int64_t t;                                  /* rounds taken */
  int32_t* idx; int32_t* counts; double* loss; int32_t* active;
  double* cut_act; double* cut_grad;          /* [C][ncut] */
  int64_t ncut;
  work_t w;
  double* xbuf; int32_t* ybuf;
  int resnet;                                 /* architecture 2 or 3 */
  int J;                                      /* classes */
  uint8_t* relu_rec;                          /* [C][B][E] ReLU records of the last round */
  uint8_t* relu_in;                           /* [C][B][E] decisions to replay next round */
  int replay;
  int64_t S;                                  /* BatchNorm state per replica (resnet) */
  double* bn;                                 /* [C][S] running mean / var */
  double tie_tol;                             /* see relu_pool_fwd */
  uint8_t* cand[4];                           /* [C][B][cout][Ho][Wo] of the last round */
  int32_t* ties;                              /* [C][B] ambiguous windows per example */
  int augment;                                /* crop + flip of the sampled images */
  int client_average;                         /* see orc_set_client_average */
  double* cut_scale;                          /* [B] factors of the current cluster */
  int gn_groups;                              /* ResNet norms: GroupNorm groups, */
  double norm_eps, bn_momentum;               /* eps, BatchNorm momentum */
  int64_t R;                                  /* F = -1: rounds per system epoch, else 0 */
  int32_t* upd;                               /* [C] the cluster updated in the last round */
} orc_ctx;

void orc_destroy(orc_ctx* c);

int orc_init(int arch, int bf16, double lr, double momentum, double wd, int nesterov,
             double label_smoothing, int K, int C, const int32_t* assignment, int B, int F,
             uint64_t seed, int cluster_base, const float* images, const int32_t* labels,
             const int32_t* owner, int64_t n, const float* init_params, orc_ctx** out) {
  *out = NULL;
  arch_t a;
  memset(&a, 0, sizeof(a));
  const int resnet = resnet_classes(arch) != 0;
  if (!resnet && get_arch(arch, &a)) return ORC_EUNSUPPORTED;
  const int J = resnet ? resnet_classes(arch) : a.fc_out;
  if (K <= 0 || C <= 0 || B <= 0 || F < -1 || n <= 0 || !assignment || !images || !labels ||
      !owner || !init_params)
    return ORC_EINVAL;
  for (int k = 0; k < K; ++k) if (assignment[k] < -1 || assignment[k] >= C) return ORC_EINVAL;
  for (int64_t i = 0; i < n; ++i)
    if (owner[i] < 0 || owner[i] >= K || labels[i] < 0 || labels[i] >= J) return ORC_EINVAL;
  orc_ctx* c = (orc_ctx*)calloc(1, sizeof(orc_ctx));
  if (!c) return ORC_ENOMEM;
  c->arch = arch; c->bf16 = bf16; c->K = K; c->C = C; c->B = B; c->F = F;
  c->nesterov = nesterov; c->cluster_base = cluster_base;
  c->lr = lr; c->momentum = momentum; c->wd = wd; c->ls = label_smoothing; c->seed = seed;
  c->a = a;
  c->resnet = resnet;
  c->gn_groups = 32; c->norm_eps = 1e-5; c->bn_momentum = 0.1;
  c->J = J;
  if (resnet) {
    memset(&c->o, 0, sizeof(c->o));
    c->o.p_client = orn_num_params(J, 0);
    c->o.p_total = c->o.p_client + orn_num_params(J, 1);
    c->S = orn_num_params(J, 2);
  } else {
    get_offs(&a, &c->o);
  }
  c->n = n;
  c->images_src = images;        /* read-only, caller keeps it alive */
  c->labels = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
  c->owner = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
  memcpy(c->labels, labels, sizeof(int32_t) * (size_t)n);
  memcpy(c->owner, owner, sizeof(int32_t) * (size_t)n);
  c->ids = (int32_t**)calloc((size_t)C, sizeof(int32_t*));
  c->perm = (int32_t**)calloc((size_t)C, sizeof(int32_t*));
  c->nc = (int64_t*)calloc((size_t)C, sizeof(int64_t));
  c->cur_epoch = (int64_t*)calloc((size_t)C, sizeof(int64_t));
  c->q = (double*)calloc((size_t)C, sizeof(double));
  for (int64_t i = 0; i < n; ++i) if (assignment[owner[i]] >= 0) c->nc[assignment[owner[i]]]++;
  int64_t total = 0;
  for (int k = 0; k < C; ++k) {
    if (c->nc[k] < B) { orc_destroy(c); return ORC_EINVAL; }
    c->ids[k] = (int32_t*)malloc(sizeof(int32_t) * (size_t)c->nc[k]);
    c->perm[k] = (int32_t*)malloc(sizeof(int32_t) * (size_t)c->nc[k]);
    c->cur_epoch[k] = -1;
    total += c->nc[k];
  }
  int64_t* fill = (int64_t*)calloc((size_t)C, sizeof(int64_t));
  for (int64_t i = 0; i < n; ++i) {          /* ascending global id per cluster */
    int k = assignment[owner[i]];
    if (k >= 0) c->ids[k][fill[k]++] = (int32_t)i;
  }
  free(fill);
  for (int k = 0; k < C; ++k) c->q[k] = (double)c->nc[k] / (double)total;
  c->upd = (int32_t*)malloc(sizeof(int32_t) * (size_t)C);
  if (!c->upd) { orc_destroy(c); return ORC_ENOMEM; }
  c->R = 0;
  for (int k = 0; k < C; ++k) {
    c->upd[k] = 1;
    if (F == -1 && c->nc[k] / B > c->R) c->R = c->nc[k] / B;
  }
  int64_t P = c->o.p_total;
  c->theta = (double*)malloc(sizeof(double) * (size_t)(C * P));
  c->mom = (double*)calloc((size_t)(C * P), sizeof(double));
  c->grad = (double*)calloc((size_t)(C * P), sizeof(double));
  for (int k = 0; k < C; ++k)
    for (int64_t p = 0; p < P; ++p) c->theta[k * P + p] = (double)init_params[p];
  c->idx = (int32_t*)calloc((size_t)C * B, sizeof(int32_t));
  c->counts = (int32_t*)calloc((size_t)C * K, sizeof(int32_t));
  c->loss = (double*)calloc((size_t)C, sizeof(double));
  c->active = (int32_t*)calloc((size_t)C, sizeof(int32_t));
  c->ncut = resnet ? (int64_t)B * 64 * 1024 : conv_out_elems(&a.conv[a.ncl - 1], B);
  c->cut_act = (double*)calloc((size_t)(C * c->ncut), sizeof(double));
  c->cut_grad = (double*)calloc((size_t)(C * c->ncut), sizeof(double));
  c->ybuf = (int32_t*)calloc((size_t)B, sizeof(int32_t));
  c->tie_tol = 1e-3;
  for (int i = 0; i < a.ncl + a.nsv; ++i)
    if (a.conv[i].pool)
      c->cand[i] = (uint8_t*)calloc((size_t)C * conv_out_elems(&a.conv[i], B), 1);
  c->ties = (int32_t*)calloc((size_t)C * B, sizeof(int32_t));
  if (resnet) {
    c->xbuf = (double*)calloc((size_t)B * 3072, sizeof(double));
    c->bn = (double*)calloc((size_t)(C * c->S > 0 ? C * c->S : 1), sizeof(double));
    const int64_t E = orn_mask_elems();
    c->relu_rec = (uint8_t*)calloc((size_t)(C * B * E), 1);
    c->relu_in = (uint8_t*)calloc((size_t)(C * B * E), 1);
    if (!c->xbuf || !c->bn || !c->relu_rec || !c->relu_in) { orc_destroy(c); return ORC_ENOMEM; }
    for (int k = 0; k < C; ++k) orn_init_bn_state(c->bn + k * c->S);
  }
  if (!c->theta || !c->mom || !c->grad || !c->cut_act || !c->cut_grad ||
      (!resnet && work_alloc(&c->w, &a, &c->o, B))) { orc_destroy(c); return ORC_ENOMEM; }
  *out = c;
  return ORC_OK;
}

void orc_destroy(orc_ctx* c) {
  if (!c) return;
  for (int k = 0; k < c->C; ++k) { if (c->ids) free(c->ids[k]); if (c->perm) free(c->perm[k]); }
  free(c->ids); free(c->perm); free(c->nc); free(c->cur_epoch); free(c->q); free(c->upd);
  free(c->labels); free(c->owner); free(c->theta); free(c->mom); free(c->grad);
  free(c->idx); free(c->counts); free(c->loss); free(c->active);
  free(c->cut_act); free(c->cut_grad); free(c->cut_scale); free(c->ybuf); free(c->ties); free(c->xbuf); free(c->bn); free(c->relu_rec); free(c->relu_in);
  for (int i = 0; i < 4; ++i) free(c->cand[i]);
  work_free(&c->w);
  free(c);
}

/* Fuse every replica's parameters (Eq. 5) and broadcast; momentum untouched. */
int orc_fuse(orc_ctx* c) {
  int64_t P = c->o.p_total;
  double* f = (double*)malloc(sizeof(double) * (size_t)P);
  if (!f) return ORC_ENOMEM;
  orc_fuse_arrays(c->C, P, c->q, c->theta, f);
  for (int k = 0; k < c->C; ++k) memcpy(c->theta + k * P, f, sizeof(double) * (size_t)P);
  free(f);
  if (c->resnet && c->S > 0) {            /* BatchNorm running statistics, same q */
    double* g = (double*)malloc(sizeof(double) * (size_t)c->S);
    if (!g) return ORC_ENOMEM;
    orc_fuse_arrays(c->C, c->S, c->q, c->bn, g);
    for (int k = 0; k < c->C; ++k) memcpy(c->bn + k * c->S, g, sizeof(double) * (size_t)c->S);
    free(g);
  }
  return ORC_OK;
}

/* SGD, PyTorch convention: g += wd theta; v = g on the first round, else
 * v = mu v + g; step g (or g + mu v with Nesterov) when mu != 0. */
static void sgd(orc_ctx* c, int k) {
  int64_t P = c->o.p_total;
  double* th = c->theta + k * P; double* v = c->mom + k * P; const double* g0 = c->grad + k * P;
  for (int64_t p = 0; p < P; ++p) {
    double g = g0[p] + c->wd * th[p];
    if (c->momentum != 0.0) {
      v[p] = c->t == 0 ? g : c->momentum * v[p] + g;
      g = c->nesterov ? g + c->momentum * v[p] : v[p];
    }
    th[p] -= c->lr * g;
  }
}

/* Training augmentation (Section V-A: random crops and horizontal flips),
 * as torchvision's RandomCrop(32, padding=4) followed by
 * RandomHorizontalFlip, with the random draws taken from Philox4x32-10:
 * counter (position in the batch, round, cluster id, 1), key = seed;
 * dy = floor(o0 * 9 / 2^32), dx = floor(o1 * 9 / 2^32) (crop offsets into the
 * 40 x 40 zero-padded image), flip = o2 mod 2.                            */
void orc_augment_params(uint64_t seed, uint32_t t, uint32_t cluster, uint32_t pos,
                        int32_t out[3]) {
  const uint32_t ctr[4] = {pos, t, cluster, 1u};
  const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t o[4];
  orc_philox4x32_10(ctr, key, o);
  out[0] = (int32_t)(((uint64_t)o[0] * 9u) >> 32);
  out[1] = (int32_t)(((uint64_t)o[1] * 9u) >> 32);
  out[2] = (int32_t)(o[2] & 1u);
}

/* dst[ch][y][x] (CHW, 3 x 32 x 32) = the crop of the zero-padded image at
 * rows dy..dy+31, columns dx..dx+31, mirrored left-right when flip:
 * padded[ch][Y][X] = src[ch][Y - 4][X - 4] inside the image, else 0.      */
void orc_augment_image(const float* src, int dy, int dx, int flip, double* dst) {
  for (int ch = 0; ch < 3; ++ch)
    for (int y = 0; y < 32; ++y)
      for (int x = 0; x < 32; ++x) {
        const int cx = flip ? 31 - x : x;             /* column of the crop */
        const int Y = y + dy, X = cx + dx;            /* in the padded image */
        const int sy = Y - 4, sx = X - 4;
        const int in = sy >= 0 && sy < 32 && sx >= 0 && sx < 32;
        dst[(ch * 32 + y) * 32 + x] = in ? (double)src[(ch * 32 + sy) * 32 + sx] : 0.0;
      }
}

void orc_set_augment(orc_ctx* c, int on) { c->augment = on != 0; }

/* Sec. IV-B's "average active client gradients", read as the unweighted
 * mean over the round's active clients of each client's mean-loss
 * gradient: the client segment's gradient then weights example i of client
 * k by 1 / (|A| b_k) instead of 1 / B, i.e. the gradient at the cut is
 * scaled by B / (|A| b_k) before the client backward (0: off, the
 * example-weighted default, the gradient of the batch-mean loss). */
int orc_set_client_average(orc_ctx* c, int on) {
  c->client_average = on != 0;
  if (on && !c->cut_scale) {
    c->cut_scale = (double*)malloc(sizeof(double) * (size_t)c->B);
    if (!c->cut_scale) return ORC_ENOMEM;
  }
  return ORC_OK;
}

/* the ResNet split's norm hyper-parameters (defaults 32, 1e-5, 0.1) */
int orc_set_norm(orc_ctx* c, int groups, double eps, double momentum) {
  if (groups < 1 || 64 % groups || !(eps > 0.0) || !(momentum > 0.0 && momentum <= 1.0))
    return ORC_EINVAL;
  c->gn_groups = groups; c->norm_eps = eps; c->bn_momentum = momentum;
  return ORC_OK;
}

/* the batch's images of cluster k in round t (augmented when set) */
static void batch_images(const orc_ctx* c, int k, const int32_t* idx, double* dst) {
  for (int b = 0; b < c->B; ++b) {
    const float* src = c->images_src + (int64_t)idx[b] * 3072;
    double* d = dst + (int64_t)b * 3072;
    if (c->augment) {
      int32_t a[3];
      orc_augment_params(c->seed, (uint32_t)c->t, (uint32_t)(c->cluster_base + k), (uint32_t)b,
                         a);
      orc_augment_image(src, a[0], a[1], a[2], d);
    } else {
      for (int i = 0; i < 3072; ++i) d[i] = (double)src[i];
    }
  }
}

/* One local round of every cluster, then fusion when (t+1) mod F == 0. */
/* Schedule (Section IV-C; Eq. 6).  Lockstep (F >= 0): every cluster takes
 * a local round every round, its own epoch after r_n = n_c / B of them.
 * Epoch schedule (F = -1): a system epoch is R = max_n r_n rounds; cluster
 * n takes local rounds 0..r_n-1 of it and then waits at the fusion barrier
 * (its batch in a waiting round is its last one, computed but not applied:
 * no padded optimizer step, no normalisation-state update, loss and |A|
 * reported as 0); the replicas are fused after every system epoch.        */
int orc_step(orc_ctx* c) {
  int B = c->B;
  for (int k = 0; k < c->C; ++k) {
    int64_t r = c->nc[k] / B;
    int64_t period = c->R ? c->R : r;
    int64_t e = c->t / period, s = c->t % period;
    c->upd[k] = s < r;
    if (s >= r) s = r - 1;
    if (e != c->cur_epoch[k]) {
      orc_epoch_perm(c->ids[k], c->nc[k], (uint32_t)(c->cluster_base + k), (uint32_t)e, c->seed,
                     c->perm[k]);
      c->cur_epoch[k] = e;
    }
    int32_t* idx = c->idx + (int64_t)k * B;
    c->active[k] = orc_sample_round(c->perm[k], s, B, c->owner, c->K, idx,
                                    c->counts + (int64_t)k * c->K);
    const double* cut_scale = NULL;
    if (c->client_average) {
      /* example b of client k: B / (|A| b_k) */
      const int32_t* cnt = c->counts + (int64_t)k * c->K;
      for (int b = 0; b < B; ++b)
        c->cut_scale[b] = (double)B / ((double)c->active[k] * (double)cnt[c->owner[idx[b]]]);
      cut_scale = c->cut_scale;
    }
    if (c->resnet) {
      orn_set_norm(c->gn_groups, c->norm_eps, c->bn_momentum);
      batch_images(c, k, idx, c->xbuf);
      for (int b = 0; b < B; ++b) c->ybuf[b] = c->labels[idx[b]];
      int64_t P = c->o.p_total;
      const int64_t E = orn_mask_elems();
      /* a waiting cluster keeps its BatchNorm running statistics */
      double* bn_keep = NULL;
      if (!c->upd[k]) {
        bn_keep = (double*)malloc(sizeof(double) * (size_t)c->S);
        if (!bn_keep) return ORC_ENOMEM;
        memcpy(bn_keep, c->bn + k * c->S, sizeof(double) * (size_t)c->S);
      }
      int rc = orn_forward_backward_masks(
          c->J, c->bf16, c->ls, c->theta + k * P, c->bn + k * c->S, B, c->xbuf, c->ybuf, &c->loss[k],
          c->grad + k * P, c->cut_act + k * c->ncut, c->cut_grad + k * c->ncut, NULL,
          c->replay ? c->relu_in + (int64_t)k * B * E : NULL, c->relu_rec + (int64_t)k * B * E,
          cut_scale);
      if (bn_keep) {
        memcpy(c->bn + k * c->S, bn_keep, sizeof(double) * (size_t)c->S);
        free(bn_keep);
      }
      if (rc) return rc;
      continue;
    }
    batch_images(c, k, idx, c->w.act[0]);
    for (int b = 0; b < B; ++b) c->ybuf[b] = c->labels[idx[b]];
    int64_t P = c->o.p_total;
    int rc = fwd_bwd(&c->a, &c->o, c->bf16, c->ls, c->theta + k * P, B, c->ybuf, &c->w,
                     &c->loss[k], c->grad + k * P, c->tie_tol, cut_scale);
    if (rc) return rc;
    for (int b = 0; b < B; ++b) c->ties[(int64_t)k * B + b] = 0;
    for (int i = 0; i < c->a.ncl + c->a.nsv; ++i) {
      if (!c->cand[i]) continue;
      int64_t per = conv_out_elems(&c->a.conv[i], B);
      memcpy(c->cand[i] + k * per, c->w.cand[i], (size_t)per);
      for (int64_t e = 0; e < per; ++e) {
        uint8_t m = c->w.cand[i][e];
        int multi = (m & 15u) != 1u && (m & 15u) != 2u && (m & 15u) != 4u && (m & 15u) != 8u;
        if (((m & 16u) && multi) || (m & 32u)) c->ties[(int64_t)k * B + e / (per / B)]++;
      }
    }
    memcpy(c->cut_act + k * c->ncut, c->w.act[c->a.ncl], sizeof(double) * (size_t)c->ncut);
    memcpy(c->cut_grad + k * c->ncut, c->w.dact[c->a.ncl], sizeof(double) * (size_t)c->ncut);
  }
  for (int k = 0; k < c->C; ++k) {
    if (c->upd[k]) {
      sgd(c, k);
    } else {
      c->loss[k] = 0.0;
      c->active[k] = 0;
    }
  }
  c->replay = 0;
  c->t++;
  const int64_t every = c->R ? c->R : c->F;
  if (every > 0 && c->t % every == 0) return orc_fuse(c);
  return ORC_OK;
}

/* segment 0 = client, 1 = server, 2 = BatchNorm state (resnet); dst gets
 * fp64 canonical-order values */
int orc_get_params(const orc_ctx* c, int cluster, int segment, double* dst) {
  if (cluster < 0 || cluster >= c->C) return ORC_EINVAL;
  if (segment == 2) {
    if (!c->resnet) return ORC_EINVAL;
    memcpy(dst, c->bn + (int64_t)cluster * c->S, sizeof(double) * (size_t)c->S);
    return ORC_OK;
  }
  int64_t P = c->o.p_total, pc = c->o.p_client;
  const double* th = c->theta + (int64_t)cluster * P;
  if (segment == 0) memcpy(dst, th, sizeof(double) * (size_t)pc);
  else if (segment == 1) memcpy(dst, th + pc, sizeof(double) * (size_t)(P - pc));
  else return ORC_EINVAL;
  return ORC_OK;
}

int orc_set_params(orc_ctx* c, int cluster, const double* blob) {
  if (cluster < 0 || cluster >= c->C) return ORC_EINVAL;
  memcpy(c->theta + (int64_t)cluster * c->o.p_total, blob, sizeof(double) * (size_t)c->o.p_total);
  return ORC_OK;
}

int orc_set_bn_state(orc_ctx* c, int cluster, const double* src) {
  if (!c->resnet || cluster < 0 || cluster >= c->C) return ORC_EINVAL;
  memcpy(c->bn + (int64_t)cluster * c->S, src, sizeof(double) * (size_t)c->S);
  return ORC_OK;
}

/* ResNet-18 split: ReLU decisions to replay in the next round ([C][B][E],
 * bit 0 used), and the records of the last round (bits as in
 * gcpsl_resnet.c's norm_fwd); E = orn_mask_elems() */
int orc_set_relu_masks(orc_ctx* c, const uint8_t* src) {
  if (!c->resnet) return ORC_EINVAL;
  memcpy(c->relu_in, src, (size_t)(c->C * c->B * orn_mask_elems()));
  c->replay = 1;
  return ORC_OK;
}
int orc_get_relu_masks(const orc_ctx* c, uint8_t* dst) {
  if (!c->resnet) return ORC_EINVAL;
  memcpy(dst, c->relu_rec, (size_t)(c->C * c->B * orn_mask_elems()));
  return ORC_OK;
}

void orc_get_sample(const orc_ctx* c, int32_t* idx, int32_t* counts) {
  if (idx) memcpy(idx, c->idx, sizeof(int32_t) * (size_t)c->C * c->B);
  if (counts) memcpy(counts, c->counts, sizeof(int32_t) * (size_t)c->C * c->K);
}

void orc_get_stats(const orc_ctx* c, double* loss, int32_t* active) {
  if (loss) memcpy(loss, c->loss, sizeof(double) * (size_t)c->C);
  if (active) memcpy(active, c->active, sizeof(int32_t) * (size_t)c->C);
}

/* which 0 = cut activation, 1 = cut gradient; [C][B][ch][h][w] */
int64_t orc_get_cut(const orc_ctx* c, int which, double* dst) {
  if (dst) memcpy(dst, which ? c->cut_grad : c->cut_act, sizeof(double) * (size_t)(c->C * c->ncut));
  return c->C * c->ncut;
}

/* momentum buffer of one replica, canonical order, both segments */
int orc_get_momentum(const orc_ctx* c, int cluster, double* dst) {
  if (cluster < 0 || cluster >= c->C) return ORC_EINVAL;
  memcpy(dst, c->mom + (int64_t)cluster * c->o.p_total, sizeof(double) * (size_t)c->o.p_total);
  return ORC_OK;
}

int orc_set_momentum(orc_ctx* c, int cluster, const double* src) {
  if (cluster < 0 || cluster >= c->C) return ORC_EINVAL;
  memcpy(c->mom + (int64_t)cluster * c->o.p_total, src, sizeof(double) * (size_t)c->o.p_total);
  return ORC_OK;
}

void orc_set_tie_tol(orc_ctx* c, double tol) { c->tie_tol = tol; }

/* decision sharpness of pooled layer `layer` in the last round,
 * [C][B][cout][Ho][Wo]; returns the element count (0: layer not pooled) */
int64_t orc_get_pool_cand(const orc_ctx* c, int layer, uint8_t* dst) {
  if (layer < 0 || layer >= c->a.ncl + c->a.nsv || !c->cand[layer]) return 0;
  int64_t n = c->C * conv_out_elems(&c->a.conv[layer], c->B);
  if (dst) memcpy(dst, c->cand[layer], (size_t)n);
  return n;
}

/* ambiguous windows per example in the last round, [C][B] */
void orc_get_ties(const orc_ctx* c, int32_t* dst) {
  memcpy(dst, c->ties, sizeof(int32_t) * (size_t)c->C * c->B);
}

void orc_get_q(const orc_ctx* c, double* q) { memcpy(q, c->q, sizeof(double) * (size_t)c->C); }
int64_t orc_rounds(const orc_ctx* c) { return c->t; }

void orc_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}
int orc_get_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
