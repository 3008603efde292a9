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
// pixels (fp32, pixels in a fixed order), combined per set by a small
// finalize kernel (which also folds the normalisation into a per-channel
// affine form), then an elementwise apply.  Every sum has a fixed order, so
// results do not depend on C or on launch geometry.  All of it is fp32: the
// sets combine at most B = 1024 partials, and GB300 executes fp64 at 1/64 of
// the fp32 rate, which made fp64 finalize kernels latency-bound on the fp64
// pipe.
#include "common.cuh"
#include "sm100.cuh"

namespace gcpsl {

namespace {

constexpr int kThreads = 256;
// per-example stride of the GroupNorm mean / rstd arrays: at most 32 groups
constexpr int kMaxGroups = 32;

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
  const int cpg = gn ? ch / gn : 1;
  const int64_t base = (int64_t)cb * HW * ch;
  float s1[8] = {0, 0, 0, 0, 0, 0, 0, 0}, s2[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  float mu[8], rs[8];
  if (BWD && l < L && threadIdx.x < L * V) {
    const int c = cb / B, b = cb % B;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int chn = v * 8 + i;
      const int64_t set =
          gn ? ((int64_t)c * B + b) * kMaxGroups + chn / cpg : (int64_t)c * ch + chn;
      mu[i] = mean[set];
      rs[i] = rstd[set];
    }
  }
  if (threadIdx.x < L * V) {
    // four pixels per step: their loads are issued together, the sums
    // still taken in pixel order
    constexpr int U = 4;
    for (int p0 = l; p0 < HW; p0 += U * L) {
      uint4 ua[U], uy[U], um[U];
#pragma unroll
      for (int j = 0; j < U; ++j) {
        const int p = p0 + j * L;
        if (p < HW) {
          const int64_t o = base + (int64_t)p * ch + v * 8;
          ua[j] = *reinterpret_cast<const uint4*>(BWD ? d + o : y + o);
          if (BWD) {
            uy[j] = *reinterpret_cast<const uint4*>(y + o);
            if (mask) um[j] = *reinterpret_cast<const uint4*>(mask + o);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < U; ++j) {
        const int p = p0 + j * L;
        if (p >= HW) break;
        float a[8];
        unpack8(ua[j], a);
        if (!BWD) {
#pragma unroll
          for (int i = 0; i < 8; ++i) { s1[i] += a[i]; s2[i] = fmaf(a[i], a[i], s2[i]); }
        } else {
          if (mask) {
            float m[8];
            unpack8(um[j], m);
#pragma unroll
            for (int i = 0; i < 8; ++i) a[i] = m[i] > 0.f ? a[i] : 0.f;
            if (dz_out)
              *reinterpret_cast<uint4*>(dz_out + base + (int64_t)p * ch + v * 8) = pack8(a);
          }
          float yy[8];
          unpack8(uy[j], yy);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            s1[i] += a[i];
            s2[i] = fmaf(a[i], (yy[i] - mu[i]) * rs[i], s2[i]);
          }
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

// Per-channel sums over the batch: a block of 8 warps per (replica, chunk of
// 32 channels); lane = channel (coalesced loads of the [b][ch][2] sums), warp
// w takes the examples b = w, w + 8, ... , and the eight warp partials are
// added in warp order.  Fixed order, independent of C.
constexpr int kChanWarps = 8;
__device__ __forceinline__ void batch_sums(const float* __restrict__ sums, int c, int chn, int B,
                                           int ch, float* red, float& s1, float& s2) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  float a = 0.f, q = 0.f;
  for (int b = w; b < B; b += kChanWarps) {
    const float2 v = *reinterpret_cast<const float2*>(sums + (((int64_t)c * B + b) * ch + chn) * 2);
    a += v.x;
    q += v.y;
  }
  red[(w * 32 + lane) * 2] = a;
  red[(w * 32 + lane) * 2 + 1] = q;
  __syncthreads();
  s1 = 0.f;
  s2 = 0.f;
  if (w == 0) {
    for (int k = 0; k < kChanWarps; ++k) {
      s1 += red[(k * 32 + lane) * 2];
      s2 += red[(k * 32 + lane) * 2 + 1];
    }
  }
}

// Forward statistics per set, and per (replica, [example,] channel) the
// affine form of the normalisation: scale = gamma * rstd, shift = beta -
// mean * scale (GroupNorm: per example; BatchNorm: shared over the batch).
// BatchNorm also updates its running statistics (momentum 0.1, unbiased
// variance).  GroupNorm: one thread per (replica, example, group);
// BatchNorm: batch_sums blocks.
__global__ void __launch_bounds__(kChanWarps * 32)
k_norm_finalize_fwd(const float* __restrict__ sums, const float* __restrict__ gamma,
                    const float* __restrict__ beta, int64_t g_rs, float* __restrict__ mean,
                    float* __restrict__ rstd, float2* __restrict__ ss, float* __restrict__ run,
                    int64_t run_rs, int C, int B, int HW, int ch, int gn, float eps,
                    float momentum, const int32_t* __restrict__ upd) {
  __shared__ float red[kChanWarps * 32 * 2];
  pdl_wait();
  pdl_trigger();
  if (gn) {
    const int cpg = ch / gn;
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)C * B * gn) return;
    const int64_t cbv = i / gn;                     // c * B + b
    const int g = (int)(i % gn), c = (int)(cbv / B);
    const int64_t set = cbv * kMaxGroups + g;
    float s1 = 0.f, s2 = 0.f;
    for (int k = 0; k < cpg; ++k) {
      const int64_t o = (cbv * ch + g * cpg + k) * 2;
      s1 += sums[o]; s2 += sums[o + 1];
    }
    const float n = (float)cpg * (float)HW, mu = s1 / n;
    float var = s2 / n - mu * mu;
    var = var > 0.f ? var : 0.f;
    const float r = 1.f / sqrtf(var + eps);
    mean[set] = mu;
    rstd[set] = r;
    const float* gm = gamma + (int64_t)c * g_rs;
    const float* bt = beta + (int64_t)c * g_rs;
    for (int k = 0; k < cpg; ++k) {
      const int chn = g * cpg + k;
      const float sc = gm[chn] * r;
      ss[cbv * ch + chn] = make_float2(sc, bt[chn] - mu * sc);
    }
    return;
  }
  const int chunks = ch / 32;
  const int c = blockIdx.x / chunks, s = (blockIdx.x % chunks) * 32 + (threadIdx.x & 31);
  float s1, s2;
  batch_sums(sums, c, s, B, ch, red, s1, s2);
  if (threadIdx.x >= 32) return;
  const float n = (float)B * (float)HW, mu = s1 / n;
  float var = s2 / n - mu * mu;
  var = var > 0.f ? var : 0.f;
  const float r = 1.f / sqrtf(var + eps);
  const int64_t w = (int64_t)c * ch + s;
  mean[w] = mu;
  rstd[w] = r;
  if (run && (!upd || upd[c])) {          // replicas at the fusion barrier keep theirs
    float* rm = run + (int64_t)c * run_rs;
    float* rv = rm + ch;
    rm[s] = (1.f - momentum) * rm[s] + momentum * mu;
    rv[s] = (1.f - momentum) * rv[s] + momentum * (var * (n / (n - 1.f)));
  }
  const float gsv = gamma[(int64_t)c * g_rs + s], bsv = beta[(int64_t)c * g_rs + s];
  const float sc = gsv * r;
  ss[w] = make_float2(sc, bsv - mu * sc);
}

// Backward: per set m1 = mean(dz gamma), m2 = mean(dz gamma x_hat), and the
// affine form dy = k1 dz + k2 y + k3 with k1 = gamma rstd, k2 = -rstd^2 m2,
// k3 = rstd^2 m2 mean - rstd m1 (GroupNorm per example, BatchNorm shared);
// per channel dgamma = sum_b S2[b][c], dbeta = sum_b S1[b][c].
//   GroupNorm set (b, g): m1 = sum_{c in g} gamma_c S1[b][c] / n (m2 with S2);
//   BatchNorm set c:      m1 = gamma_c sum_b S1[b][c] / n.
// Blocks [0, C ch / 32): batch_sums per channel chunk (dgamma, dbeta and
// the whole BatchNorm set); GroupNorm sets follow, one thread each.
__global__ void __launch_bounds__(kChanWarps * 32)
k_norm_finalize_bwd(const float* __restrict__ sums, const float* __restrict__ gamma,
                    int64_t g_rs, const float* __restrict__ mean, const float* __restrict__ rstd,
                    float4* __restrict__ kk, float* __restrict__ dgamma,
                    float* __restrict__ dbeta, int64_t d_rs, int C, int B, int HW, int ch,
                    int gn) {
  __shared__ float red[kChanWarps * 32 * 2];
  pdl_wait();
  pdl_trigger();
  const int chunks = ch / 32;
  const int nb = C * chunks;
  if ((int)blockIdx.x < nb) {
    const int c = blockIdx.x / chunks, chn = (blockIdx.x % chunks) * 32 + (threadIdx.x & 31);
    float a, b2;
    batch_sums(sums, c, chn, B, ch, red, a, b2);
    if (threadIdx.x >= 32) return;
    dgamma[(int64_t)c * d_rs + chn] = b2;
    dbeta[(int64_t)c * d_rs + chn] = a;
    if (!gn) {
      const int64_t w = (int64_t)c * ch + chn;
      const float g = gamma[(int64_t)c * g_rs + chn];
      const float n = (float)B * (float)HW;
      const float m1 = g * a / n, m2 = g * b2 / n;
      const float mu = mean[w], r = rstd[w];
      kk[w] = make_float4(g * r, -r * r * m2, r * r * m2 * mu - r * m1, 0.f);
    }
    return;
  }
  if (!gn) return;
  const int cpg = ch / gn;
  const int64_t i = (int64_t)(blockIdx.x - nb) * blockDim.x + threadIdx.x;  // set (c, b, g)
  if (i >= (int64_t)C * B * gn) return;
  const int64_t cbv = i / gn;
  const int g = (int)(i % gn), c = (int)(cbv / B);
  const int64_t set = cbv * kMaxGroups + g;
  const float* gm = gamma + (int64_t)c * g_rs;
  float a = 0.f, b2 = 0.f;
  for (int k = 0; k < cpg; ++k) {
    const int chn = g * cpg + k;
    const int64_t o = (cbv * ch + chn) * 2;
    a = fmaf(gm[chn], sums[o], a);
    b2 = fmaf(gm[chn], sums[o + 1], b2);
  }
  const float n = (float)cpg * (float)HW;
  const float m1 = a / n, m2 = b2 / n;
  const float mu = mean[set], r = rstd[set];
  for (int k = 0; k < cpg; ++k) {
    const int chn = g * cpg + k;
    kk[cbv * ch + chn] = make_float4(gm[chn] * r, -r * r * m2, r * r * m2 * mu - r * m1, 0.f);
  }
}

// Elementwise with the per-channel affine forms of the finalize kernels
// (GroupNorm: per example, BatchNorm: shared over the batch).  A block per
// (replica, example, pixel chunk): thread = 8 channels x a pixel lane, so
// each thread loads its affine coefficients once.
//   forward:  out = relu?(y scale + shift + r), r = res (bf16), or
//             y2 scale2 + shift2 (the shortcut's norm), or 0;
//   backward: out = k1 dz + k2 y + k3, dz = d (times [mask > 0]).
constexpr int kApplyPixels = 256;        // pixels per block at most
template <bool BWD>
__global__ void __launch_bounds__(kThreads)
k_norm_apply(const bf16* __restrict__ y, const void* __restrict__ aff, int aff_gn,
             const bf16* __restrict__ y2, const float2* __restrict__ aff2, int aff2_gn,
             const bf16* __restrict__ res, const bf16* __restrict__ d,
             const bf16* __restrict__ mask, bf16* __restrict__ out, int C, int B, int HW, int ch,
             int relu) {
  pdl_wait();
  pdl_trigger();
  const int V = ch / 8;
  const int L = kThreads / V;
  const int chunks = (HW + kApplyPixels - 1) / kApplyPixels;
  const int64_t cb = blockIdx.x / chunks;
  const int p0 = (int)(blockIdx.x % chunks) * kApplyPixels;
  const int p1 = p0 + kApplyPixels < HW ? p0 + kApplyPixels : HW;
  const int c = (int)(cb / B);
  const int v = threadIdx.x % V, l = threadIdx.x / V;
  if (l >= L) return;
  const int64_t arow = (aff_gn ? cb : (int64_t)c) * ch + v * 8;
  if (!BWD) {
    float sc[8], sh[8], sc2[8], sh2[8];
    const float4* a4 = reinterpret_cast<const float4*>(reinterpret_cast<const float2*>(aff) + arow);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float4 q = a4[k];
      sc[2 * k] = q.x; sh[2 * k] = q.y; sc[2 * k + 1] = q.z; sh[2 * k + 1] = q.w;
    }
    if (y2) {
      const float4* b4 =
          reinterpret_cast<const float4*>(aff2 + (aff2_gn ? cb : (int64_t)c) * ch + v * 8);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float4 q = b4[k];
        sc2[2 * k] = q.x; sh2[2 * k] = q.y; sc2[2 * k + 1] = q.z; sh2[2 * k + 1] = q.w;
      }
    }
#pragma unroll 4
    for (int p = p0 + l; p < p1; p += L) {
      const int64_t o = (cb * HW + p) * ch + v * 8;
      float yy[8], r[8] = {0, 0, 0, 0, 0, 0, 0, 0}, o8[8];
      unpack8(*reinterpret_cast<const uint4*>(y + o), yy);
      if (res) {
        unpack8(*reinterpret_cast<const uint4*>(res + o), r);
      } else if (y2) {
        float z[8];
        unpack8(*reinterpret_cast<const uint4*>(y2 + o), z);
#pragma unroll
        for (int k = 0; k < 8; ++k) r[k] = fmaf(z[k], sc2[k], sh2[k]);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float x = fmaf(yy[k], sc[k], sh[k]) + r[k];
        o8[k] = relu ? (x > 0.f ? x : 0.f) : x;
      }
      *reinterpret_cast<uint4*>(out + o) = pack8(o8);
    }
  } else {
    float k1[8], k2[8], k3[8];
    const float4* k4 = reinterpret_cast<const float4*>(aff) + arow;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 q = k4[k];
      k1[k] = q.x; k2[k] = q.y; k3[k] = q.z;
    }
#pragma unroll 4
    for (int p = p0 + l; p < p1; p += L) {
      const int64_t o = (cb * HW + p) * ch + v * 8;
      float yy[8], dz[8], o8[8];
      unpack8(*reinterpret_cast<const uint4*>(y + o), yy);
      unpack8(*reinterpret_cast<const uint4*>(d + o), dz);
      if (mask) {
        float m[8];
        unpack8(*reinterpret_cast<const uint4*>(mask + o), m);
#pragma unroll
        for (int k = 0; k < 8; ++k) dz[k] = m[k] > 0.f ? dz[k] : 0.f;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) o8[k] = fmaf(k1[k], dz[k], fmaf(k2[k], yy[k], k3[k]));
      *reinterpret_cast<uint4*>(out + o) = pack8(o8);
    }
  }
}

// GroupNorm of one example in one kernel: a GroupNorm set (example, group)
// never leaves its example, so one block per (replica, example) computes the
// statistics and applies them, with the example's tensor (y forward, dz
// backward; HW x ch bf16 <= 128 KB) staged in shared memory between the two
// passes: one block per SM, 512 threads.  The staged tensor (y, or d) comes
// in by one bulk copy.
//   FWD: per-channel fp32 sums (pixels in lane order, lanes combined by a
//        fixed shuffle tree and then in warp order), per group mean / rstd
//        in fp64 (written for the backward), then
//        out = relu?(gamma x_hat + beta + res).
//   BWD: dz = d [mask > 0] (kept in dz_out when set), per-channel S1 = sum
//        dz and S2 = sum dz x_hat (written to sums for dgamma / dbeta), per
//        group m1, m2 and the affine form, then dy = k1 dz + k2 y + k3.
// Threads: V = ch / 8 channel vectors x L pixel lanes (thread = l V + v).
constexpr int kGnThreads = 512, kGnStageBytes = 128 * 1024;
template <bool BWD>
__global__ void __launch_bounds__(kGnThreads, 1)
k_gn_fused(const bf16* __restrict__ y, const bf16* __restrict__ d, const bf16* __restrict__ mask,
           const bf16* __restrict__ res, const float* __restrict__ gamma,
           const float* __restrict__ beta, int64_t g_rs, float* __restrict__ mean,
           float* __restrict__ rstd, float* __restrict__ sums, bf16* __restrict__ dz_out,
           bf16* __restrict__ out, int B, int HW, int ch, int relu, int G, float eps, int* err) {
  extern __shared__ uint4 gsm4[];
  __shared__ uint64_t bar;
  uint8_t* stage = reinterpret_cast<uint8_t*>(gsm4);             // HW x ch bf16
  float* red = reinterpret_cast<float*>(stage + kGnStageBytes);  // [warps][V][16]
  const int V = ch / 8, L = kGnThreads / V;
  const int nw = kGnThreads / 32;
  float* csum = red + nw * V * 16;                               // [ch][2]
  float4* aff = reinterpret_cast<float4*>(csum + 2 * ch);        // [ch]
  const int64_t cb = blockIdx.x;                     // c * B + b
  if (threadIdx.x == 0) {
    sm100::mbar_init(&bar, 1);
    sm100::fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x == 0) {
    const uint32_t bytes = (uint32_t)(HW * ch * 2);
    sm100::mbar_arrive_expect_tx(&bar, bytes);
    sm100::bulk_load(stage, (BWD ? d : y) + cb * HW * ch, bytes, &bar);
  }
  const int c = (int)(cb / B);
  const int v = threadIdx.x % V, l = threadIdx.x / V;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int cpg = ch / G;
  const int64_t base = cb * HW * ch + v * 8;
  const float* gm = gamma + (int64_t)c * g_rs;
  float mu[8], rs[8];
  if (BWD) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int64_t set = cb * kMaxGroups + (v * 8 + i) / cpg;
      mu[i] = mean[set];
      rs[i] = rstd[set];
    }
  }
  if (!sm100::mbar_wait(&bar, 0) && threadIdx.x == 0) atomicOr(err, 64);
  // pass 1: per-lane channel sums; the backward turns the staged d into dz
  float s1[8] = {0, 0, 0, 0, 0, 0, 0, 0}, s2[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll 4
  for (int p = l; p < HW; p += L) {
    const int64_t o = base + (int64_t)p * ch;
    uint4* st = reinterpret_cast<uint4*>(stage + ((int64_t)p * ch + v * 8) * 2);
    float a[8];
    if (!BWD) {
      unpack8(*st, a);
#pragma unroll
      for (int i = 0; i < 8; ++i) { s1[i] += a[i]; s2[i] = fmaf(a[i], a[i], s2[i]); }
    } else {
      unpack8(*st, a);
      if (mask) {
        float m[8];
        unpack8(*reinterpret_cast<const uint4*>(mask + o), m);
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = m[i] > 0.f ? a[i] : 0.f;
      }
      const uint4 dzr = pack8(a);
      *st = dzr;
      if (dz_out) *reinterpret_cast<uint4*>(dz_out + o) = dzr;
      unpack8(dzr, a);                                 // the stored (bf16) dz
      float yy[8];
      unpack8(*reinterpret_cast<const uint4*>(y + o), yy);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        s1[i] += a[i];
        s2[i] = fmaf(a[i], (yy[i] - mu[i]) * rs[i], s2[i]);
      }
    }
  }
  // lanes of a warp with the same v (32 / V of them) by a fixed xor tree,
  // then the warps in order
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    for (int o = 16; o >= V; o >>= 1) {
      s1[i] += __shfl_xor_sync(0xffffffffu, s1[i], o);
      s2[i] += __shfl_xor_sync(0xffffffffu, s2[i], o);
    }
  }
  if (lane < V) {
    float* mine = red + ((int64_t)warp * V + v) * 16;
#pragma unroll
    for (int i = 0; i < 8; ++i) { mine[i] = s1[i]; mine[8 + i] = s2[i]; }
  }
  __syncthreads();
  for (int q = threadIdx.x; q < V * 16; q += kGnThreads) {
    const int vv = q / 16, k = q % 16;
    float t = 0.f;
    for (int w = 0; w < nw; ++w) t += red[((int64_t)w * V + vv) * 16 + k];
    const int chn = vv * 8 + (k & 7);
    csum[chn * 2 + (k >> 3)] = t;
    if (BWD) sums[(cb * ch + chn) * 2 + (k >> 3)] = t;
  }
  __syncthreads();
  if (threadIdx.x < G) {
    const int g = threadIdx.x;
    const float n = (float)cpg * (float)HW;
    if (!BWD) {
      float a = 0.f, q2 = 0.f;
      for (int k = 0; k < cpg; ++k) { a += csum[(g * cpg + k) * 2]; q2 += csum[(g * cpg + k) * 2 + 1]; }
      const float m = a / n;
      float var = q2 / n - m * m;
      var = var > 0.f ? var : 0.f;
      const float r = 1.f / sqrtf(var + eps);
      mean[cb * kMaxGroups + g] = m;
      rstd[cb * kMaxGroups + g] = r;
      const float* bt = beta + (int64_t)c * g_rs;
      for (int k = 0; k < cpg; ++k) {
        const int chn = g * cpg + k;
        const float sc = gm[chn] * r;
        aff[chn] = make_float4(sc, bt[chn] - m * sc, 0.f, 0.f);
      }
    } else {
      float a = 0.f, b2 = 0.f;
      for (int k = 0; k < cpg; ++k) {
        const int chn = g * cpg + k;
        a = fmaf(gm[chn], csum[chn * 2], a);
        b2 = fmaf(gm[chn], csum[chn * 2 + 1], b2);
      }
      const float m1 = a / n, m2 = b2 / n;
      const float m = mean[cb * kMaxGroups + g], r = rstd[cb * kMaxGroups + g];
      for (int k = 0; k < cpg; ++k) {
        const int chn = g * cpg + k;
        aff[chn] = make_float4(gm[chn] * r, -r * r * m2, r * r * m2 * m - r * m1, 0.f);
      }
    }
  }
  __syncthreads();
  // pass 2 from the staged tensor
  float k1[8], k2[8], k3[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 q = aff[v * 8 + i];
    k1[i] = q.x; k2[i] = q.y; k3[i] = q.z;
  }
#pragma unroll 4
  for (int p = l; p < HW; p += L) {
    const int64_t o = base + (int64_t)p * ch;
    const uint4 sv = *reinterpret_cast<const uint4*>(stage + ((int64_t)p * ch + v * 8) * 2);
    float o8[8];
    if (!BWD) {
      float yy[8], r8[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      unpack8(sv, yy);
      if (res) unpack8(*reinterpret_cast<const uint4*>(res + o), r8);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float x = fmaf(yy[i], k1[i], k2[i]) + r8[i];
        o8[i] = relu ? (x > 0.f ? x : 0.f) : x;
      }
    } else {
      float dz[8], yy[8];
      unpack8(sv, dz);
      unpack8(*reinterpret_cast<const uint4*>(y + o), yy);
#pragma unroll
      for (int i = 0; i < 8; ++i) o8[i] = fmaf(k1[i], dz[i], fmaf(k2[i], yy[i], k3[i]));
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

// gn: GroupNorm's group count (it divides ch, at most kMaxGroups), 0 for BatchNorm
static bool groups_ok(int gn, int ch) { return gn == 0 || (gn > 0 && gn <= kMaxGroups && ch % gn == 0); }

cudaError_t launch_norm_sums(cudaStream_t s, bool bwd, const bf16* y, const bf16* d,
                             const bf16* mask, const float* mean, const float* rstd, bf16* dz_out,
                             float* sums, int C, int B, int HW, int ch, int gn) {
  if (ch % 32 || ch / 8 > kThreads || !groups_ok(gn, ch)) return cudaErrorInvalidValue;
  const int V = ch / 8, L = kThreads / V;
  const size_t smem = sizeof(float) * (size_t)L * V * 16;
  if (bwd)
    return launch_k(k_chan_sums<true>, (unsigned)(C * B), kThreads, smem, s, y, d, mask, mean,
                    rstd, dz_out, sums, B, HW, ch, gn);
  return launch_k(k_chan_sums<false>, (unsigned)(C * B), kThreads, smem, s, y, d, mask, mean,
                  rstd, dz_out, sums, B, HW, ch, gn);
}

cudaError_t launch_norm_finalize_fwd(cudaStream_t s, const float* sums, const float* gamma,
                                     const float* beta, int64_t g_rs, float* mean, float* rstd,
                                     float2* ss, float* run, int64_t run_rs, int C, int B, int HW,
                                     int ch, int gn, float eps, float momentum,
                                     const int32_t* upd) {
  if (ch % 32 || !groups_ok(gn, ch)) return cudaErrorInvalidValue;
  const unsigned blocks = gn ? nblk((int64_t)C * B * gn, 256) : (unsigned)(C * (ch / 32));
  return launch_k(k_norm_finalize_fwd, blocks, 256, 0, s, sums, gamma, beta, g_rs,
                  mean, rstd, ss, run, run_rs, C, B, HW, ch, gn, eps, momentum, upd);
}

cudaError_t launch_norm_finalize_bwd(cudaStream_t s, const float* sums, const float* gamma,
                                     int64_t g_rs, const float* mean, const float* rstd,
                                     float4* kk, float* dgamma, float* dbeta, int64_t d_rs, int C,
                                     int B, int HW, int ch, int gn) {
  if (ch % 32 || !groups_ok(gn, ch)) return cudaErrorInvalidValue;
  const unsigned blocks = (unsigned)(C * (ch / 32)) + (gn ? nblk((int64_t)C * B * gn, 256) : 0u);
  return launch_k(k_norm_finalize_bwd, blocks, 256, 0, s, sums, gamma, g_rs, mean,
                  rstd, kk, dgamma, dbeta, d_rs, C, B, HW, ch, gn);
}

cudaError_t launch_norm_apply_fwd(cudaStream_t s, const bf16* y, const float2* ss, int gn,
                                  const bf16* res, const bf16* y2, const float2* ss2, int gn2,
                                  bf16* out, int C, int B, int HW, int ch, int relu) {
  if (ch % 8 || ch / 8 > kThreads) return cudaErrorInvalidValue;
  const int64_t n = (int64_t)C * B * ((HW + kApplyPixels - 1) / kApplyPixels);
  return launch_k(k_norm_apply<false>, (unsigned)n, kThreads, 0, s, y, (const void*)ss, gn,
                  y2, ss2, gn2, res, (const bf16*)nullptr, (const bf16*)nullptr, out, C, B, HW,
                  ch, relu);
}

cudaError_t launch_norm_apply_bwd(cudaStream_t s, const bf16* y, const float4* kk, int gn,
                                  const bf16* d, const bf16* mask, bf16* out, int C, int B, int HW,
                                  int ch) {
  if (ch % 8 || ch / 8 > kThreads) return cudaErrorInvalidValue;
  const int64_t n = (int64_t)C * B * ((HW + kApplyPixels - 1) / kApplyPixels);
  return launch_k(k_norm_apply<true>, (unsigned)n, kThreads, 0, s, y, (const void*)kk, gn,
                  (const bf16*)nullptr, (const float2*)nullptr, 0, (const bf16*)nullptr, d, mask,
                  out, C, B, HW, ch, 0);
}

static size_t gn_smem(int ch) {
  const int V = ch / 8;
  return kGnStageBytes + sizeof(float) * ((size_t)(kGnThreads / 32) * V * 16 + 2 * ch) +
         sizeof(float4) * ch;
}

template <bool BWD>
static bool gn_attr() {
  static bool done = false;
  if (!done)
    done = cudaFuncSetAttribute(k_gn_fused<BWD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)gn_smem(256)) == cudaSuccess;
  return done;
}

static bool gn_shape_ok(int HW, int ch) {
  // V = ch / 8 lanes of a warp share the xor tree: V divides 32
  return ch % 32 == 0 && ch <= 256 && (int64_t)HW * ch * 2 <= kGnStageBytes;
}

cudaError_t launch_gn_fused_fwd(cudaStream_t s, const bf16* y, const bf16* res,
                                const float* gamma, const float* beta, int64_t g_rs, float* mean,
                                float* rstd, bf16* out, int C, int B, int HW, int ch, int relu,
                                int groups, float eps, int* err) {
  if (!gn_shape_ok(HW, ch) || groups < 1 || !groups_ok(groups, ch) || !gn_attr<false>())
    return cudaErrorInvalidValue;
  return launch_k(k_gn_fused<false>, (unsigned)(C * B), kGnThreads, gn_smem(ch), s, y,
                  (const bf16*)nullptr, (const bf16*)nullptr, res, gamma, beta, g_rs, mean, rstd,
                  (float*)nullptr, (bf16*)nullptr, out, B, HW, ch, relu, groups, eps, err);
}

cudaError_t launch_gn_fused_bwd(cudaStream_t s, const bf16* y, const bf16* d, const bf16* mask,
                                bf16* dz_out, const float* gamma, int64_t g_rs, const float* mean,
                                const float* rstd, float* sums, bf16* out, int C, int B, int HW,
                                int ch, int groups, int* err) {
  if (!gn_shape_ok(HW, ch) || groups < 1 || !groups_ok(groups, ch) || (dz_out && !mask) ||
      !gn_attr<true>())
    return cudaErrorInvalidValue;
  return launch_k(k_gn_fused<true>, (unsigned)(C * B), kGnThreads, gn_smem(ch), s, y, d, mask,
                  (const bf16*)nullptr, gamma, (const float*)nullptr, g_rs,
                  const_cast<float*>(mean), const_cast<float*>(rstd), sums, dz_out, out, B, HW,
                  ch, 0, groups, 0.f, err);
}

cudaError_t launch_norm_finalize_bwd_channels(cudaStream_t s, const float* sums, float* dgamma,
                                              float* dbeta, int64_t d_rs, int C, int B, int ch) {
  if (ch % 32) return cudaErrorInvalidValue;
  // the channel blocks of k_norm_finalize_bwd only (gn = 1: no BatchNorm
  // form; the GroupNorm sets are left to the caller)
  return launch_k(k_norm_finalize_bwd, (unsigned)(C * (ch / 32)), 256, 0, s, sums,
                  (const float*)nullptr, (int64_t)0, (const float*)nullptr, (const float*)nullptr,
                  (float4*)nullptr, dgamma, dbeta, d_rs, C, B, 1, ch, 1);
}

cudaError_t launch_avgpool(cudaStream_t s, const bf16* x, bf16* h, int CB, int HW, int ch) {
  return launch_k(k_avgpool, nblk((int64_t)CB * ch, 256), 256, 0, s, x, h, CB, HW, ch);
}

}  // namespace gcpsl
