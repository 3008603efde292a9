// Grouped 3x3 convolutions (stride 1, zero padding 1) on CUDA cores, over C
// replicas at once; the replica index is part of every grid.  fp32
// accumulation; storage T = float (fp32 path) or bf16.
//
// Layouts: activations NHWC [C][B][H][W][ch]; weights [C][cout][3][3][cin]
// (replica stride w_rs elements); the gradient w.r.t. the pre-activation
// g = dL/dy is NHWC [C][B][H][W][cout].
//
// Forward (Section III-A, client f_theta_c and server g_theta_s segments):
//   y[b,h,w,co] = bias[co] + sum_{kh,kw,ci} x[b,h+kh-1,w+kw-1,ci] W[co,kh,kw,ci]
//   out = relu(y) or maxpool2x2(relu(y)); for a pooled layer the byte code
//   records the first maximum of the window in row-major order (bits 0-1)
//   and whether that maximum is positive (bit 2), decided on the fp32 y.
// Backward: g = route(dout) through the pool and ReLU (ReLU'(0) = 0);
//   dx[b,ih,iw,ci] = sum_{kh,kw,co} g[b,ih-kh+1,iw-kw+1,co] W[co,kh,kw,ci];
//   dW[co,kh,kw,ci] = sum_{b,h,w} g[b,h,w,co] x[b,h+kh-1,w+kw-1,ci];
//   db[co] = sum_{b,h,w} g[b,h,w,co].
#include "common.cuh"

namespace gcpsl {

namespace {

template <typename T>
__global__ void k_conv_fwd(const T* __restrict__ x, const T* __restrict__ w, int64_t w_rs,
                           const float* __restrict__ bias, int64_t b_rs, T* __restrict__ out,
                           uint8_t* __restrict__ code, int C, int B, int cin, int cout, int H,
                           int W, int pool) {
  pdl_wait();
  pdl_trigger();
  const int Ho = pool ? H / 2 : H, Wo = pool ? W / 2 : W;
  const int64_t total = (int64_t)C * B * Ho * Wo * cout;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int co = (int)(i % cout);
  int64_t r = i / cout;
  const int ow = (int)(r % Wo); r /= Wo;
  const int oh = (int)(r % Ho); r /= Ho;
  const int b = (int)(r % B);
  const int c = (int)(r / B);
  const T* xb = x + ((int64_t)c * B + b) * H * W * cin;
  const T* wc = w + (int64_t)c * w_rs + (int64_t)co * 9 * cin;
  const int np = pool ? 4 : 1;
  const int h0 = pool ? 2 * oh : oh, w0 = pool ? 2 * ow : ow;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int kh = 0; kh < 3; ++kh)
    for (int kw = 0; kw < 3; ++kw) {
      const T* wk = wc + (kh * 3 + kw) * cin;
      for (int q = 0; q < np; ++q) {
        const int ih = h0 + (q >> 1) + kh - 1, iw = w0 + (q & 1) + kw - 1;
        if (ih < 0 || ih >= H || iw < 0 || iw >= W) continue;
        const T* xp = xb + ((int64_t)ih * W + iw) * cin;
        float s = acc[q];
        for (int ci = 0; ci < cin; ++ci) s = fmaf(to_f(xp[ci]), to_f(wk[ci]), s);
        acc[q] = s;
      }
    }
  const float bv = bias[(int64_t)c * b_rs + co];
  if (!pool) {
    const float v = acc[0] + bv;
    out[i] = from_f<T>(v > 0.f ? v : 0.f);
    return;
  }
  float best = acc[0] + bv;
  int arg = 0;
  for (int q = 1; q < 4; ++q) {
    const float v = acc[q] + bv;
    if (v > best) { best = v; arg = q; }
  }
  out[i] = from_f<T>(best > 0.f ? best : 0.f);
  code[i] = (uint8_t)(arg | (best > 0.f ? 4 : 0));
}

// g = dL/dy from dL/d(out).  One thread per (output pixel, group of V
// channels), V = 16 bytes of T: for a pooled layer it reads the pooled
// gradient and codes once and writes the whole 2x2 window (the gradient at
// the recorded first maximum when it is positive, zero elsewhere); without
// pooling g = dout where the ReLU output is positive.
template <typename T>
__global__ void k_relu_pool_bwd(const T* __restrict__ dout, const uint8_t* __restrict__ code,
                                const T* __restrict__ act, T* __restrict__ g, int C, int B,
                                int cout, int H, int W, int pool) {
  pdl_wait();
  pdl_trigger();
  constexpr int V = 16 / sizeof(T);
  const int Ho = pool ? H / 2 : H, Wo = pool ? W / 2 : W;
  const int groups = cout / V;
  const int64_t total = (int64_t)C * B * Ho * Wo * groups;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int grp = (int)(i % groups);
  const int64_t opix = i / groups;                    // output pixel (pooled grid)
  const int64_t o = opix * cout + grp * V;
  const uint4 dv = *reinterpret_cast<const uint4*>(dout + o);
  const T* d = reinterpret_cast<const T*>(&dv);
  if (!pool) {
    const uint4 av = *reinterpret_cast<const uint4*>(act + o);
    const T* av_ = reinterpret_cast<const T*>(&av);
    __align__(16) T out[V];
#pragma unroll
    for (int k = 0; k < V; ++k) out[k] = to_f(av_[k]) > 0.f ? d[k] : from_f<T>(0.f);
    *reinterpret_cast<uint4*>(g + o) = *reinterpret_cast<const uint4*>(out);
    return;
  }
  uint8_t cd[V];
  if (V == 8) {
    const uint2 cv = *reinterpret_cast<const uint2*>(code + o);
    *reinterpret_cast<uint2*>(cd) = cv;
  } else {
    const uint32_t cv = *reinterpret_cast<const uint32_t*>(code + o);
    *reinterpret_cast<uint32_t*>(cd) = cv;
  }
  const int pw = (int)(opix % Wo);
  const int ph = (int)((opix / Wo) % Ho);
  const int64_t cb = opix / ((int64_t)Wo * Ho);
#pragma unroll
  for (int qd = 0; qd < 4; ++qd) {
    __align__(16) T out[V];
#pragma unroll
    for (int k = 0; k < V; ++k) out[k] = ((cd[k] & 4) && (cd[k] & 3) == qd) ? d[k] : from_f<T>(0.f);
    const int64_t gi = ((cb * H + 2 * ph + (qd >> 1)) * W + 2 * pw + (qd & 1)) * cout + grp * V;
    *reinterpret_cast<uint4*>(g + gi) = *reinterpret_cast<const uint4*>(out);
  }
}

// Weight and bias gradient partials of an input layer with CIN <= 4 channels
// (x padded to xc channels per pixel): thread = (4-channel output group q,
// input channel ci, pixel lane); for each of its pixels it loads g for four
// output channels and x for nine taps and does 36 FMAs.  The lanes' sums are
// then added in lane order.  Layout of the partial as in k_wgrad_partial.
template <typename T, int CIN>
__global__ void __launch_bounds__(256, 2)
k_wgrad_small_cin(const T* __restrict__ x, int xc, const T* __restrict__ g,
                  float* __restrict__ partial, int B, int cout, int H, int W, int tr,
                  int tiles_per_split) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  const int c = blockIdx.y, split = blockIdx.x;
  const int per_w = cout * 9 * CIN, per = per_w + cout;
  const int combos = (cout / 4) * CIN, lanes = 256 / combos;
  const int t = threadIdx.x, combo = t % combos, lane = t / combos;
  const bool worker = lane < lanes;
  const int q = combo / CIN, ci = combo % CIN;
  float* gs = sm;                                   // [tr*W][cout]
  float* xs = sm + tr * W * cout;                   // [(tr+2)][(W+2)][CIN]
  float acc[36], bacc[4];
#pragma unroll
  for (int k = 0; k < 36; ++k) acc[k] = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) bacc[k] = 0.f;
  const int tiles_img = H / tr, tiles = B * tiles_img;
  const int t0 = split * tiles_per_split, t1 = min(t0 + tiles_per_split, tiles);
  for (int tile = t0; tile < t1; ++tile) {
    const int b = tile / tiles_img, h0 = (tile % tiles_img) * tr;
    const T* gb = g + (((int64_t)c * B + b) * H + h0) * W * cout;
    for (int i = t; i < tr * W * cout; i += blockDim.x) gs[i] = to_f(gb[i]);
    const T* xb = x + ((int64_t)c * B + b) * H * W * xc;
    for (int i = t; i < (tr + 2) * (W + 2) * CIN; i += blockDim.x) {
      const int cc = i % CIN, ww = (i / CIN) % (W + 2) - 1, hh = i / (CIN * (W + 2)) + h0 - 1;
      xs[i] = (hh >= 0 && hh < H && ww >= 0 && ww < W) ? to_f(xb[((int64_t)hh * W + ww) * xc + cc])
                                                      : 0.f;
    }
    __syncthreads();
    if (worker) {
      for (int p = lane; p < tr * W; p += lanes) {
        const int r = p / W, w = p % W;
        const float4 gv = *reinterpret_cast<const float4*>(gs + p * cout + 4 * q);
        const float gq[4] = {gv.x, gv.y, gv.z, gv.w};
#pragma unroll
        for (int kh = 0; kh < 3; ++kh)
#pragma unroll
          for (int kw = 0; kw < 3; ++kw) {
            const float xv = xs[((r + kh) * (W + 2) + w + kw) * CIN + ci];
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[(kh * 3 + kw) * 4 + j] = fmaf(gq[j], xv, acc[(kh * 3 + kw) * 4 + j]);
          }
#pragma unroll
        for (int j = 0; j < 4; ++j) bacc[j] += gq[j];
      }
    }
    __syncthreads();
  }
  // red[lane][combo][40]: 36 weight sums + 4 bias sums
  float* red = sm;
  if (worker) {
    float* dst = red + ((int64_t)lane * combos + combo) * 40;
#pragma unroll
    for (int k = 0; k < 36; ++k) dst[k] = acc[k];
#pragma unroll
    for (int k = 0; k < 4; ++k) dst[36 + k] = bacc[k];
  }
  __syncthreads();
  float* out = partial + ((int64_t)c * gridDim.x + split) * per;
  for (int o = t; o < per; o += blockDim.x) {
    int cmb, k;
    if (o < per_w) {
      const int cc = o % CIN, tap = (o / CIN) % 9, co = o / (9 * CIN);
      cmb = (co / 4) * CIN + cc;
      k = tap * 4 + co % 4;
    } else {
      const int co = o - per_w;
      cmb = (co / 4) * CIN;                       // the ci == 0 threads hold the bias sums
      k = 36 + co % 4;
    }
    float s = 0.f;
    for (int l = 0; l < lanes; ++l) s += red[((int64_t)l * combos + cmb) * 40 + k];
    out[o] = s;
  }
}

template <typename T>
__global__ void k_conv_dgrad(const T* __restrict__ g, const T* __restrict__ w, int64_t w_rs,
                             T* __restrict__ dx, int C, int B, int cin, int cout, int H, int W) {
  pdl_wait();
  pdl_trigger();
  const int64_t total = (int64_t)C * B * H * W * cin;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int ci = (int)(i % cin);
  int64_t r = i / cin;
  const int iw = (int)(r % W); r /= W;
  const int ih = (int)(r % H); r /= H;
  const int b = (int)(r % B);
  const int c = (int)(r / B);
  const T* gb = g + ((int64_t)c * B + b) * H * W * cout;
  const T* wc = w + (int64_t)c * w_rs + ci;
  float acc = 0.f;
  for (int kh = 0; kh < 3; ++kh)
    for (int kw = 0; kw < 3; ++kw) {
      const int h = ih - kh + 1, ww = iw - kw + 1;
      if (h < 0 || h >= H || ww < 0 || ww >= W) continue;
      const T* gp = gb + ((int64_t)h * W + ww) * cout;
      const T* wk = wc + (kh * 3 + kw) * cin;
      for (int co = 0; co < cout; ++co) acc = fmaf(to_f(gp[co]), to_f(wk[(int64_t)co * 9 * cin]), acc);
    }
  dx[i] = from_f<T>(acc);
}

// Weight and bias gradient partial sums over a range of image-row tiles,
// staged in shared memory: outputs o < cout*9*cin are dW[co][tap][ci],
// outputs cout*9*cin + co are db[co] (the bias follows the weight in the
// parameter store, so one reduction writes both).  Block = 256 threads,
// grid = (splits, C); partial[c][split][o].  Each thread sums its outputs
// over the block's pixels in a fixed order.
constexpr int kWgOut = 32;   // outputs per thread (per <= 256 * kWgOut)

template <typename T>
__global__ void __launch_bounds__(256)
k_wgrad_partial(const T* __restrict__ x, const T* __restrict__ g, float* __restrict__ partial,
                int B, int cin, int xc, int cout, int H, int W, int tr, int tiles_per_split) {
  pdl_wait();
  pdl_trigger();
  // xc = channels per pixel of x in memory (>= cin; the padded input layer)
  extern __shared__ float sm[];
  const int c = blockIdx.y, split = blockIdx.x;
  const int per_w = cout * 9 * cin, per = per_w + cout;
  float* gs = sm;                                   // [tr*W][cout]
  float* xs = sm + tr * W * cout;                   // [(tr+2)][(W+2)][cin]
  float acc[kWgOut];
#pragma unroll
  for (int j = 0; j < kWgOut; ++j) acc[j] = 0.f;
  const int tiles_img = H / tr, tiles = B * tiles_img;
  const int t0 = split * tiles_per_split, t1 = min(t0 + tiles_per_split, tiles);
  for (int tile = t0; tile < t1; ++tile) {
    const int b = tile / tiles_img, h0 = (tile % tiles_img) * tr;
    const T* gb = g + (((int64_t)c * B + b) * H + h0) * W * cout;
    for (int i = threadIdx.x; i < tr * W * cout; i += blockDim.x) gs[i] = to_f(gb[i]);
    const T* xb = x + ((int64_t)c * B + b) * H * W * xc;
    for (int i = threadIdx.x; i < (tr + 2) * (W + 2) * cin; i += blockDim.x) {
      const int ci = i % cin, ww = (i / cin) % (W + 2) - 1, hh = i / (cin * (W + 2)) + h0 - 1;
      xs[i] = (hh >= 0 && hh < H && ww >= 0 && ww < W) ? to_f(xb[((int64_t)hh * W + ww) * xc + ci])
                                                      : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kWgOut; ++j) {
      const int o = threadIdx.x + j * 256;
      if (o >= per) break;
      float s = acc[j];
      if (o < per_w) {
        const int ci = o % cin, tap = (o / cin) % 9, co = o / (9 * cin);
        const int kh = tap / 3, kw = tap % 3;
        for (int r = 0; r < tr; ++r)
          for (int w = 0; w < W; ++w)
            s = fmaf(gs[(r * W + w) * cout + co], xs[((r + kh) * (W + 2) + w + kw) * cin + ci], s);
      } else {
        const int co = o - per_w;
        for (int q = 0; q < tr * W; ++q) s += gs[q * cout + co];
      }
      acc[j] = s;
    }
    __syncthreads();
  }
  float* dst = partial + ((int64_t)c * gridDim.x + split) * per;
#pragma unroll
  for (int j = 0; j < kWgOut; ++j) {
    const int o = threadIdx.x + j * 256;
    if (o < per) dst[o] = acc[j];
  }
}

inline unsigned blocks(int64_t n, int t) { return (unsigned)((n + t - 1) / t); }

}  // namespace

template <typename T>
cudaError_t launch_conv_fwd_simt(cudaStream_t s, const T* x, const T* w, int64_t w_rs,
                                 const float* bias, int64_t b_rs, T* out, uint8_t* code, int C,
                                 int B, const ConvSpec& cs) {
  const int Ho = cs.pool ? cs.h / 2 : cs.h, Wo = cs.pool ? cs.w / 2 : cs.w;
  const int64_t n = (int64_t)C * B * Ho * Wo * cs.cout;
  return launch_k(k_conv_fwd<T>, blocks(n, 256), 256, 0, s, x, w, w_rs, bias, b_rs, out, code, C,
                  B, cs.cin, cs.cout, cs.h, cs.w, cs.pool);
}

template <typename T>
cudaError_t launch_relu_pool_bwd(cudaStream_t s, const T* dout, const uint8_t* code,
                                 const T* act, T* g, int C, int B, const ConvSpec& cs) {
  constexpr int V = 16 / sizeof(T);
  if (cs.cout % V) return cudaErrorInvalidValue;
  const int64_t opix = (int64_t)C * B * (cs.pool ? cs.h * cs.w / 4 : cs.h * cs.w);
  const int64_t n = opix * (cs.cout / V);
  return launch_k(k_relu_pool_bwd<T>, blocks(n, 256), 256, 0, s, dout, code, act, g, C, B,
                  cs.cout, cs.h, cs.w, cs.pool);
}

template <typename T>
cudaError_t launch_conv_dgrad_simt(cudaStream_t s, const T* g, const T* w, int64_t w_rs, T* dx,
                                   int C, int B, const ConvSpec& cs) {
  const int64_t n = (int64_t)C * B * cs.h * cs.w * cs.cin;
  return launch_k(k_conv_dgrad<T>, blocks(n, 256), 256, 0, s, g, w, w_rs, dx, C, B, cs.cin,
                  cs.cout, cs.h, cs.w);
}

template <typename T>
cudaError_t launch_wgrad_simt(cudaStream_t s, const T* x, int xc, const T* g, float* partial,
                              int C, int B, const ConvSpec& cs, int tr, int splits,
                              int tiles_per_split) {
  if (cs.cin <= 4 && cs.cout % 4 == 0 && (cs.cout / 4) * cs.cin <= 256) {
    const int stage = (tr * cs.w * cs.cout + (tr + 2) * (cs.w + 2) * cs.cin) * (int)sizeof(float);
    const int red = 256 * 40 * (int)sizeof(float);
    const int sm = stage > red ? stage : red;
#define GCPSL_SMALL_CIN(CI)                                                                   \
  if (cs.cin == CI) {                                                                         \
    static bool attr = false;                                                                 \
    if (!attr) {                                                                              \
      cudaError_t e = cudaFuncSetAttribute(k_wgrad_small_cin<T, CI>,                          \
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, 96 << 10); \
      if (e != cudaSuccess) return e;                                                         \
      attr = true;                                                                            \
    }                                                                                         \
    if (sm > (96 << 10)) return cudaErrorInvalidValue;                                        \
    return launch_k(k_wgrad_small_cin<T, CI>, dim3(splits, C), 256, sm, s, x, xc, g, partial, \
                    B, cs.cout, cs.h, cs.w, tr, tiles_per_split);                             \
  }
    GCPSL_SMALL_CIN(1)
    GCPSL_SMALL_CIN(2)
    GCPSL_SMALL_CIN(3)
    GCPSL_SMALL_CIN(4)
#undef GCPSL_SMALL_CIN
  }
  const int smem = (tr * cs.w * cs.cout + (tr + 2) * (cs.w + 2) * cs.cin) * (int)sizeof(float);
  if ((int64_t)cs.cout * 9 * cs.cin + cs.cout > 256 * kWgOut) return cudaErrorInvalidValue;
  static int attr_set = 0;
  if (smem > 48 * 1024 && attr_set < smem) {
    cudaError_t e = cudaFuncSetAttribute(k_wgrad_partial<T>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = smem;
  }
  return launch_k(k_wgrad_partial<T>, dim3(splits, C), 256, smem, s, x, g, partial, B, cs.cin, xc,
                  cs.cout, cs.h, cs.w, tr, tiles_per_split);
}

#define GCPSL_INST(T)                                                                          \
  template cudaError_t launch_conv_fwd_simt<T>(cudaStream_t, const T*, const T*, int64_t,      \
                                               const float*, int64_t, T*, uint8_t*, int, int,  \
                                               const ConvSpec&);                               \
  template cudaError_t launch_relu_pool_bwd<T>(cudaStream_t, const T*, const uint8_t*,         \
                                               const T*, T*, int, int, const ConvSpec&);       \
  template cudaError_t launch_conv_dgrad_simt<T>(cudaStream_t, const T*, const T*, int64_t,    \
                                                 T*, int, int, const ConvSpec&);               \
  template cudaError_t launch_wgrad_simt<T>(cudaStream_t, const T*, int, const T*, float*, int, \
                                            int, const ConvSpec&, int, int, int);
GCPSL_INST(float)
GCPSL_INST(bf16)
#undef GCPSL_INST

}  // namespace gcpsl
