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

template <typename T>
__global__ void k_conv_wgrad(const T* __restrict__ x, const T* __restrict__ g,
                             float* __restrict__ dw, int64_t dw_rs, int C, int B, int cin,
                             int cout, int H, int W) {
  const int64_t per = (int64_t)cout * 9 * cin;
  const int64_t total = (int64_t)C * per;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int c = (int)(i / per);
  int64_t r = i % per;
  const int ci = (int)(r % cin); r /= cin;
  const int tap = (int)(r % 9);
  const int co = (int)(r / 9);
  const int kh = tap / 3, kw = tap % 3;
  float acc = 0.f;
  for (int b = 0; b < B; ++b) {
    const T* gb = g + ((int64_t)c * B + b) * H * W * cout + co;
    const T* xb = x + ((int64_t)c * B + b) * H * W * cin + ci;
    for (int h = 0; h < H; ++h) {
      const int ih = h + kh - 1;
      if (ih < 0 || ih >= H) continue;
      for (int w = 0; w < W; ++w) {
        const int iw = w + kw - 1;
        if (iw < 0 || iw >= W) continue;
        acc = fmaf(to_f(gb[((int64_t)h * W + w) * cout]), to_f(xb[((int64_t)ih * W + iw) * cin]), acc);
      }
    }
  }
  dw[(int64_t)c * dw_rs + (int64_t)co * 9 * cin + tap * cin + ci] = acc;
}

// db[c][co] = sum over (b, h, w) of g; one warp per (c, co), fixed order:
// lane l sums pixels l, l+32, ...; then a fixed shuffle tree.
template <typename T>
__global__ void k_bias_grad(const T* __restrict__ g, float* __restrict__ db, int64_t db_rs,
                            int C, int B, int cout, int HW) {
  const int warp = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (warp >= C * cout) return;
  const int c = warp / cout, co = warp % cout;
  const int64_t npix = (int64_t)B * HW;
  const T* gc = g + (int64_t)c * npix * cout + co;
  float s = 0.f;
  for (int64_t p = lane; p < npix; p += 32) s += to_f(gc[p * cout]);
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) db[(int64_t)c * db_rs + co] = s;
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
cudaError_t launch_conv_wgrad_simt(cudaStream_t s, const T* x, const T* g, float* dw,
                                   int64_t dw_rs, int C, int B, const ConvSpec& cs) {
  const int64_t n = (int64_t)C * cs.cout * 9 * cs.cin;
  k_conv_wgrad<T><<<blocks(n, 128), 128, 0, s>>>(x, g, dw, dw_rs, C, B, cs.cin, cs.cout, cs.h,
                                                  cs.w);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_bias_grad(cudaStream_t s, const T* g, float* db, int64_t db_rs, int C, int B,
                             const ConvSpec& cs) {
  const int64_t warps = (int64_t)C * cs.cout;
  k_bias_grad<T><<<blocks(warps * 32, 256), 256, 0, s>>>(g, db, db_rs, C, B, cs.cout,
                                                          cs.h * cs.w);
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
  template cudaError_t launch_conv_wgrad_simt<T>(cudaStream_t, const T*, const T*, float*,     \
                                                 int64_t, int, int, const ConvSpec&);          \
  template cudaError_t launch_bias_grad<T>(cudaStream_t, const T*, float*, int64_t, int, int,  \
                                           const ConvSpec&);
GCPSL_INST(float)
GCPSL_INST(bf16)
#undef GCPSL_INST

}  // namespace gcpsl
