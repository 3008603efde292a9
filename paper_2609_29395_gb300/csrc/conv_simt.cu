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

template <typename T>
__global__ void k_relu_pool_bwd(const T* __restrict__ dout, const uint8_t* __restrict__ code,
                                const T* __restrict__ act, T* __restrict__ g, int C, int B,
                                int cout, int H, int W, int pool) {
  const int64_t total = (int64_t)C * B * H * W * cout;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  if (!pool) {
    g[i] = to_f(act[i]) > 0.f ? dout[i] : from_f<T>(0.f);
    return;
  }
  const int co = (int)(i % cout);
  int64_t r = i / cout;
  const int w = (int)(r % W); r /= W;
  const int h = (int)(r % H);
  const int64_t cb = r / H;
  const int64_t o = ((cb * (H / 2) + h / 2) * (W / 2) + w / 2) * cout + co;
  const int cd = code[o];
  const bool hit = (cd & 4) && (cd & 3) == ((h & 1) * 2 + (w & 1));
  g[i] = hit ? dout[o] : from_f<T>(0.f);
}

template <typename T>
__global__ void k_conv_dgrad(const T* __restrict__ g, const T* __restrict__ w, int64_t w_rs,
                             T* __restrict__ dx, int C, int B, int cin, int cout, int H, int W) {
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
                int B, int cin, int cout, int H, int W, int tr, int tiles_per_split) {
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
    const T* xb = x + ((int64_t)c * B + b) * H * W * cin;
    for (int i = threadIdx.x; i < (tr + 2) * (W + 2) * cin; i += blockDim.x) {
      const int ci = i % cin, ww = (i / cin) % (W + 2) - 1, hh = i / (cin * (W + 2)) + h0 - 1;
      xs[i] = (hh >= 0 && hh < H && ww >= 0 && ww < W) ? to_f(xb[((int64_t)hh * W + ww) * cin + ci])
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

// Bias-gradient partials: partial[c][chunk][co] = sum of g over the chunk's
// `chunk_px` pixels (consecutive threads read consecutive channels).
template <typename T>
__global__ void k_bias_partial(const T* __restrict__ g, float* __restrict__ partial, int64_t npix,
                               int cout, int chunk_px) {
  const int c = blockIdx.y, chunk = blockIdx.x;
  const int64_t p0 = (int64_t)chunk * chunk_px;
  const int64_t p1 = min(p0 + chunk_px, npix);
  const T* gc = g + (int64_t)c * npix * cout;
  for (int co = threadIdx.x; co < cout; co += blockDim.x) {
    float s = 0.f;
    for (int64_t p = p0; p < p1; ++p) s += to_f(gc[p * cout + co]);
    partial[((int64_t)c * gridDim.x + chunk) * cout + co] = s;
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
  k_conv_fwd<T><<<blocks(n, 256), 256, 0, s>>>(x, w, w_rs, bias, b_rs, out, code, C, B, cs.cin,
                                                cs.cout, cs.h, cs.w, cs.pool);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_relu_pool_bwd(cudaStream_t s, const T* dout, const uint8_t* code,
                                 const T* act, T* g, int C, int B, const ConvSpec& cs) {
  const int64_t n = (int64_t)C * B * cs.h * cs.w * cs.cout;
  k_relu_pool_bwd<T><<<blocks(n, 256), 256, 0, s>>>(dout, code, act, g, C, B, cs.cout, cs.h,
                                                     cs.w, cs.pool);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_conv_dgrad_simt(cudaStream_t s, const T* g, const T* w, int64_t w_rs, T* dx,
                                   int C, int B, const ConvSpec& cs) {
  const int64_t n = (int64_t)C * B * cs.h * cs.w * cs.cin;
  k_conv_dgrad<T><<<blocks(n, 256), 256, 0, s>>>(g, w, w_rs, dx, C, B, cs.cin, cs.cout, cs.h,
                                                  cs.w);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_wgrad_simt(cudaStream_t s, const T* x, const T* g, float* partial, int C,
                              int B, const ConvSpec& cs, int tr, int splits, int tiles_per_split) {
  const int smem = (tr * cs.w * cs.cout + (tr + 2) * (cs.w + 2) * cs.cin) * (int)sizeof(float);
  if ((int64_t)cs.cout * 9 * cs.cin + cs.cout > 256 * kWgOut) return cudaErrorInvalidValue;
  static int attr_set = 0;
  if (smem > 48 * 1024 && attr_set < smem) {
    cudaError_t e = cudaFuncSetAttribute(k_wgrad_partial<T>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = smem;
  }
  k_wgrad_partial<T><<<dim3(splits, C), 256, smem, s>>>(x, g, partial, B, cs.cin, cs.cout, cs.h,
                                                        cs.w, tr, tiles_per_split);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_bias_partial(cudaStream_t s, const T* g, float* partial, int C, int B,
                                const ConvSpec& cs, int chunks, int chunk_px) {
  const int64_t npix = (int64_t)B * cs.h * cs.w;
  const int threads = cs.cout < 256 ? cs.cout : 256;
  k_bias_partial<T><<<dim3(chunks, C), threads, 0, s>>>(g, partial, npix, cs.cout, chunk_px);
  return cudaGetLastError();
}

#define GCPSL_INST(T)                                                                          \
  template cudaError_t launch_conv_fwd_simt<T>(cudaStream_t, const T*, const T*, int64_t,      \
                                               const float*, int64_t, T*, uint8_t*, int, int,  \
                                               const ConvSpec&);                               \
  template cudaError_t launch_relu_pool_bwd<T>(cudaStream_t, const T*, const uint8_t*,         \
                                               const T*, T*, int, int, const ConvSpec&);       \
  template cudaError_t launch_conv_dgrad_simt<T>(cudaStream_t, const T*, const T*, int64_t,    \
                                                 T*, int, int, const ConvSpec&);               \
  template cudaError_t launch_wgrad_simt<T>(cudaStream_t, const T*, const T*, float*, int, int, \
                                            const ConvSpec&, int, int, int);                   \
  template cudaError_t launch_bias_partial<T>(cudaStream_t, const T*, float*, int, int,        \
                                              const ConvSpec&, int, int);
GCPSL_INST(float)
GCPSL_INST(bf16)
#undef GCPSL_INST

}  // namespace gcpsl
