// GroupNorm / train-mode BatchNorm of the ResNet-18 split, grouped over the C
// replicas, on NHWC bf16 tensors [C][B][HW][ch].
//
//   x_hat = (y - mean) * rstd, rstd = 1 / sqrt(var + 1e-5), var biased;
//   forward  out = relu?(gamma * x_hat + beta + residual)
//   backward dy = rstd * (dz gamma - m1 - x_hat m2), m1 = mean(dz gamma),
//            m2 = mean(dz gamma x_hat) over the normalisation set;
//            dgamma = sum dz x_hat, dbeta = sum dz (per channel).
// Sets: GroupNorm (b, group of ch/32 channels) over the group's channels and
// H x W; BatchNorm one channel over B x H x W.
//
// Both directions go through per-(example, channel) partial sums over the
// pixels (fp32, pixels in a fixed order), combined per set in fp64 by a
// small finalize kernel, then an elementwise apply.  Every sum has a fixed
// order, so results do not depend on C or on launch geometry.
#include "common.cuh"

namespace gcpsl {

namespace {

constexpr int kThreads = 256;
constexpr double kEps = 1e-5;

__device__ __forceinline__ void unpack8(const uint4& u, float* f) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
__device__ __forceinline__ uint4 pack8(const float* f) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    w[i] = *reinterpret_cast<const uint32_t*>(&h);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Per (c, b): 8-channel vectors x pixel lanes.  Lane l takes pixels l,
// l + L, ...; the lanes' sums are added in lane order through shared memory.
// FWD: s1 = sum y, s2 = sum y^2.
// BWD: dz = d (times [mask > 0] when mask is set; written to dz_out when
//      set), s1 = sum dz, s2 = sum dz x_hat with x_hat from y and the stats
//      of its set.
template <bool BWD>
__global__ void __launch_bounds__(kThreads)
k_chan_sums(const bf16* __restrict__ y, const bf16* __restrict__ d, const bf16* __restrict__ mask,
            const float* __restrict__ mean, const float* __restrict__ rstd,
            bf16* __restrict__ dz_out, float* __restrict__ sums, int B, int HW, int ch, int gn) {
  extern __shared__ float red[];                   // [L][V][16]
  pdl_wait();
  pdl_trigger();
  const int cb = blockIdx.x;                       // c * B + b
  const int V = ch / 8;
  const int L = kThreads / V > 0 ? kThreads / V : 1;
  const int v = threadIdx.x % V, l = threadIdx.x / V;
  const int cpg = ch / 32;
  const int64_t base = (int64_t)cb * HW * ch;
  float s1[8] = {0, 0, 0, 0, 0, 0, 0, 0}, s2[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  float mu[8], rs[8];
  if (BWD && l < L && threadIdx.x < L * V) {
    const int c = cb / B, b = cb % B;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int chn = v * 8 + i;
      const int64_t set = gn ? ((int64_t)c * B + b) * 32 + chn / cpg : (int64_t)c * ch + chn;
      mu[i] = mean[set];
      rs[i] = rstd[set];
    }
  }
  if (threadIdx.x < L * V) {
    for (int p = l; p < HW; p += L) {
      const int64_t o = base + (int64_t)p * ch + v * 8;
      float a[8];
      unpack8(*reinterpret_cast<const uint4*>(BWD ? d + o : y + o), a);
      if (!BWD) {
#pragma unroll
        for (int i = 0; i < 8; ++i) { s1[i] += a[i]; s2[i] = fmaf(a[i], a[i], s2[i]); }
      } else {
        if (mask) {
          float m[8];
          unpack8(*reinterpret_cast<const uint4*>(mask + o), m);
#pragma unroll
          for (int i = 0; i < 8; ++i) a[i] = m[i] > 0.f ? a[i] : 0.f;
          if (dz_out) *reinterpret_cast<uint4*>(dz_out + o) = pack8(a);
        }
        float yy[8];
        unpack8(*reinterpret_cast<const uint4*>(y + o), yy);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          s1[i] += a[i];
          s2[i] = fmaf(a[i], (yy[i] - mu[i]) * rs[i], s2[i]);
        }
      }
    }
  }
  float* mine = red + ((int64_t)l * V + v) * 16;
  if (threadIdx.x < L * V) {
#pragma unroll
    for (int i = 0; i < 8; ++i) { mine[i] = s1[i]; mine[8 + i] = s2[i]; }
  }
  __syncthreads();
  for (int q = threadIdx.x; q < V * 16; q += kThreads) {
    const int vv = q / 16, k = q % 16;
    float s = 0.f;
    for (int ll = 0; ll < L; ++ll) s += red[((int64_t)ll * V + vv) * 16 + k];
    const int chn = vv * 8 + (k & 7);
    sums[((int64_t)cb * ch + chn) * 2 + (k >> 3)] = s;
  }
}

// Forward statistics per set from the (b, channel) sums, in fp64; BatchNorm
// also updates its running statistics (momentum 0.1, unbiased variance).
__global__ void k_norm_finalize_fwd(const float* __restrict__ sums, float* __restrict__ mean,
                                    float* __restrict__ rstd, float* __restrict__ run,
                                    int64_t run_rs, int C, int B, int HW, int ch, int gn) {
  pdl_wait();
  pdl_trigger();
  const int sets = gn ? B * 32 : ch;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)C * sets) return;
  const int c = (int)(i / sets), s = (int)(i % sets);
  double s1 = 0.0, s2 = 0.0, n;
  if (gn) {
    const int b = s / 32, g = s % 32, cpg = ch / 32;
    for (int k = 0; k < cpg; ++k) {
      const int64_t o = (((int64_t)c * B + b) * ch + g * cpg + k) * 2;
      s1 += sums[o]; s2 += sums[o + 1];
    }
    n = (double)cpg * HW;
  } else {
    for (int b = 0; b < B; ++b) {
      const int64_t o = (((int64_t)c * B + b) * ch + s) * 2;
      s1 += sums[o]; s2 += sums[o + 1];
    }
    n = (double)B * HW;
  }
  const double mu = s1 / n;
  double var = s2 / n - mu * mu;
  var = var > 0.0 ? var : 0.0;
  mean[i] = (float)mu;
  rstd[i] = (float)(1.0 / sqrt(var + kEps));
  if (!gn && run) {
    float* rm = run + (int64_t)c * run_rs;
    float* rv = rm + ch;
    rm[s] = (float)(0.9 * (double)rm[s] + 0.1 * mu);
    rv[s] = (float)(0.9 * (double)rv[s] + 0.1 * var * n / (n - 1.0));
  }
}

// Backward set constants m1, m2 and the affine gradients.
//   GroupNorm set (b, g): m1 = sum_{c in g} gamma_c S1[b][c] / n,
//                         m2 = sum_{c in g} gamma_c S2[b][c] / n;
//   BatchNorm set c:      m1 = gamma_c sum_b S1[b][c] / n, m2 likewise;
//   dgamma_c = sum_b S2[b][c], dbeta_c = sum_b S1[b][c].
__global__ void k_norm_finalize_bwd(const float* __restrict__ sums,
                                    const float* __restrict__ gamma, int64_t g_rs,
                                    float* __restrict__ m1, float* __restrict__ m2,
                                    float* __restrict__ dgamma, float* __restrict__ dbeta,
                                    int64_t d_rs, int C, int B, int HW, int ch, int gn) {
  pdl_wait();
  pdl_trigger();
  const int sets = gn ? B * 32 : ch;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)C * (sets > ch ? sets : ch);
  if (i >= total) return;
  const int c = (int)(i / (sets > ch ? sets : ch)), s = (int)(i % (sets > ch ? sets : ch));
  const float* gm = gamma + (int64_t)c * g_rs;
  if (s < sets) {
    double a = 0.0, b2 = 0.0, n;
    if (gn) {
      const int b = s / 32, g = s % 32, cpg = ch / 32;
      for (int k = 0; k < cpg; ++k) {
        const int chn = g * cpg + k;
        const int64_t o = (((int64_t)c * B + b) * ch + chn) * 2;
        a += (double)gm[chn] * sums[o];
        b2 += (double)gm[chn] * sums[o + 1];
      }
      n = (double)cpg * HW;
    } else {
      for (int b = 0; b < B; ++b) {
        const int64_t o = (((int64_t)c * B + b) * ch + s) * 2;
        a += sums[o]; b2 += sums[o + 1];
      }
      a *= gm[s]; b2 *= gm[s];
      n = (double)B * HW;
    }
    m1[(int64_t)c * sets + s] = (float)(a / n);
    m2[(int64_t)c * sets + s] = (float)(b2 / n);
  }
  if (s < ch) {
    double dg = 0.0, db = 0.0;
    for (int b = 0; b < B; ++b) {
      const int64_t o = (((int64_t)c * B + b) * ch + s) * 2;
      db += sums[o]; dg += sums[o + 1];
    }
    dgamma[(int64_t)c * d_rs + s] = (float)dg;
    dbeta[(int64_t)c * d_rs + s] = (float)db;
  }
}

// Elementwise, one thread per 8 channels of one pixel.
//   forward: out = relu?(gamma (y - mu) rstd + beta + r), with r = 0, the
//            bf16 tensor res, or a second normalised tensor y2 (its own
//            stats and affine);
//   backward: out = rstd (dz gamma - m1 - x_hat m2), dz = d (times
//            [mask > 0] when mask is set).
struct NormTerm {
  const bf16* y;
  const float* mean;
  const float* rstd;
  const float* gamma;       // replica 0; replica stride g_rs
  const float* beta;
  int64_t g_rs;
};

template <bool BWD>
__global__ void __launch_bounds__(kThreads)
k_norm_apply(NormTerm t, NormTerm t2, const bf16* __restrict__ res, const bf16* __restrict__ d,
             const bf16* __restrict__ mask, bf16* __restrict__ out, int C, int B, int HW, int ch,
             int gn, int relu) {
  pdl_wait();
  pdl_trigger();
  const int V = ch / 8;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)C * B * HW * V) return;
  const int v = (int)(i % V);
  const int64_t pix = i / V;
  const int64_t cb = pix / HW;
  const int c = (int)(cb / B), b = (int)(cb % B);
  const int cpg = ch / 32;
  const int64_t o = pix * ch + v * 8;
  float y[8];
  unpack8(*reinterpret_cast<const uint4*>(t.y + o), y);
  float r[8];
  auto stats = [&](const NormTerm& q, int chn, float& mu, float& rs) {
    const int64_t set = gn ? ((int64_t)c * B + b) * 32 + chn / cpg : (int64_t)c * ch + chn;
    mu = q.mean[set];
    rs = q.rstd[set];
  };
  if (!BWD) {
    if (res) {
      unpack8(*reinterpret_cast<const uint4*>(res + o), r);
    } else if (t2.y) {
      float y2[8];
      unpack8(*reinterpret_cast<const uint4*>(t2.y + o), y2);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int chn = v * 8 + k;
        float mu, rs;
        stats(t2, chn, mu, rs);
        r[k] = fmaf(t2.gamma[(int64_t)c * t2.g_rs + chn], (y2[k] - mu) * rs,
                    t2.beta[(int64_t)c * t2.g_rs + chn]);
      }
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) r[k] = 0.f;
    }
    float o8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int chn = v * 8 + k;
      float mu, rs;
      stats(t, chn, mu, rs);
      float x = fmaf(t.gamma[(int64_t)c * t.g_rs + chn], (y[k] - mu) * rs,
                     t.beta[(int64_t)c * t.g_rs + chn]) + r[k];
      o8[k] = relu ? (x > 0.f ? x : 0.f) : x;
    }
    *reinterpret_cast<uint4*>(out + o) = pack8(o8);
  } else {
    float dz[8];
    unpack8(*reinterpret_cast<const uint4*>(d + o), dz);
    if (mask) {
      float m[8];
      unpack8(*reinterpret_cast<const uint4*>(mask + o), m);
#pragma unroll
      for (int k = 0; k < 8; ++k) dz[k] = m[k] > 0.f ? dz[k] : 0.f;
    }
    float o8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int chn = v * 8 + k;
      float rs, mu;
      stats(t, chn, mu, rs);
      // backward: t.mean / t.rstd are the forward stats, t2.mean / t2.rstd
      // carry m1 / m2 of the same sets
      float m1, m2;
      stats(t2, chn, m1, m2);
      const float xh = (y[k] - mu) * rs;
      o8[k] = rs * (dz[k] * t.gamma[(int64_t)c * t.g_rs + chn] - m1 - xh * m2);
    }
    *reinterpret_cast<uint4*>(out + o) = pack8(o8);
  }
}

// h[c][b][ch] = mean over the HW pixels (fixed order), bf16
__global__ void k_avgpool(const bf16* __restrict__ x, bf16* __restrict__ h, int CB, int HW,
                          int ch) {
  pdl_wait();
  pdl_trigger();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)CB * ch) return;
  const int64_t cb = i / ch;
  const int chn = (int)(i % ch);
  float s = 0.f;
  for (int p = 0; p < HW; ++p) s += __bfloat162float(x[(cb * HW + p) * ch + chn]);
  h[i] = __float2bfloat16_rn(s / (float)HW);
}

inline unsigned nblk(int64_t n, int t) { return (unsigned)((n + t - 1) / t); }

}  // namespace

cudaError_t launch_norm_sums(cudaStream_t s, bool bwd, const bf16* y, const bf16* d,
                             const bf16* mask, const float* mean, const float* rstd, bf16* dz_out,
                             float* sums, int C, int B, int HW, int ch, int gn) {
  if (ch % 32 || ch / 8 > kThreads) return cudaErrorInvalidValue;
  const int V = ch / 8, L = kThreads / V;
  const size_t smem = sizeof(float) * (size_t)L * V * 16;
  if (bwd)
    return launch_k(k_chan_sums<true>, (unsigned)(C * B), kThreads, smem, s, y, d, mask, mean,
                    rstd, dz_out, sums, B, HW, ch, gn);
  return launch_k(k_chan_sums<false>, (unsigned)(C * B), kThreads, smem, s, y, d, mask, mean,
                  rstd, dz_out, sums, B, HW, ch, gn);
}

cudaError_t launch_norm_finalize_fwd(cudaStream_t s, const float* sums, float* mean, float* rstd,
                                     float* run, int64_t run_rs, int C, int B, int HW, int ch,
                                     int gn) {
  const int sets = gn ? B * 32 : ch;
  return launch_k(k_norm_finalize_fwd, nblk((int64_t)C * sets, 128), 128, 0, s, sums, mean, rstd,
                  run, run_rs, C, B, HW, ch, gn);
}

cudaError_t launch_norm_finalize_bwd(cudaStream_t s, const float* sums, const float* gamma,
                                     int64_t g_rs, float* m1, float* m2, float* dgamma,
                                     float* dbeta, int64_t d_rs, int C, int B, int HW, int ch,
                                     int gn) {
  const int sets = gn ? B * 32 : ch;
  const int64_t n = (int64_t)C * (sets > ch ? sets : ch);
  return launch_k(k_norm_finalize_bwd, nblk(n, 128), 128, 0, s, sums, gamma, g_rs, m1, m2,
                  dgamma, dbeta, d_rs, C, B, HW, ch, gn);
}

cudaError_t launch_norm_apply_fwd(cudaStream_t s, const bf16* y, const float* mean,
                                  const float* rstd, const float* gamma, const float* beta,
                                  int64_t g_rs, const bf16* res, const bf16* y2,
                                  const float* mean2, const float* rstd2, const float* gamma2,
                                  const float* beta2, bf16* out, int C, int B, int HW, int ch,
                                  int gn, int relu) {
  const NormTerm t{y, mean, rstd, gamma, beta, g_rs};
  const NormTerm t2{y2, mean2, rstd2, gamma2, beta2, g_rs};
  const int64_t n = (int64_t)C * B * HW * (ch / 8);
  return launch_k(k_norm_apply<false>, nblk(n, kThreads), kThreads, 0, s, t, t2, res,
                  (const bf16*)nullptr, (const bf16*)nullptr, out, C, B, HW, ch, gn, relu);
}

cudaError_t launch_norm_apply_bwd(cudaStream_t s, const bf16* y, const float* mean,
                                  const float* rstd, const float* gamma, int64_t g_rs,
                                  const float* m1, const float* m2, const bf16* d,
                                  const bf16* mask, bf16* out, int C, int B, int HW, int ch,
                                  int gn) {
  const NormTerm t{y, mean, rstd, gamma, nullptr, g_rs};
  const NormTerm t2{nullptr, m1, m2, nullptr, nullptr, g_rs};
  const int64_t n = (int64_t)C * B * HW * (ch / 8);
  return launch_k(k_norm_apply<true>, nblk(n, kThreads), kThreads, 0, s, t, t2,
                  (const bf16*)nullptr, d, mask, out, C, B, HW, ch, gn, 0);
}

cudaError_t launch_avgpool(cudaStream_t s, const bf16* x, bf16* h, int CB, int HW, int ch) {
  return launch_k(k_avgpool, nblk((int64_t)CB * ch, 256), 256, 0, s, x, h, CB, HW, ch);
}

}  // namespace gcpsl
