// Server head: linear layer, softmax cross-entropy averaged over the batch,
// and the linear layer's backward, grouped over the C replicas.
//
// h is the last conv layer's pooled output read as [C][B][fin] (NHWC flatten;
// the linear weight is stored in the same (h, w, ch) order, so it equals
// PyTorch's (ch, h, w) flatten of an NCHW tensor with permuted weights).
//   logits[b,j] = b_fc[j] + sum_k h[b,k] W[j,k]
//   loss = (1/B) sum_b ( lse(logits_b) - sum_j t_bj logits_bj ),
//     t = (1-e) onehot(y) + e/J   (label smoothing e, 0 by default)
//   dlogits[b,j] = (softmax(logits_b)_j - t_bj) / B
//   dW[j,k] = sum_b dlogits[b,j] h[b,k];  db[j] = sum_b dlogits[b,j]
//   dh[b,k] = sum_j dlogits[b,j] W[j,k]
#include "common.cuh"

namespace gcpsl {

namespace {

// one warp per (c, b, j); lanes stride over k; fixed shuffle tree
template <typename T>
__global__ void k_fc_fwd(const T* __restrict__ h, const T* __restrict__ w, int64_t w_rs,
                         const float* __restrict__ bias, int64_t b_rs, float* __restrict__ logits,
                         int C, int B, int fin, int fout) {
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= (int64_t)C * B * fout) return;
  const int j = (int)(warp % fout);
  const int64_t cb = warp / fout;
  const int c = (int)(cb / B);
  const T* hp = h + cb * fin;
  const T* wp = w + (int64_t)c * w_rs + (int64_t)j * fin;
  float s = 0.f;
  for (int k = lane; k < fin; k += 32) s = fmaf(to_f(hp[k]), to_f(wp[k]), s);
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) logits[warp] = s + bias[(int64_t)c * b_rs + j];
}

// one block per replica, one thread per example (B <= 1024)
__global__ void k_softmax_ce(const float* __restrict__ logits, const int32_t* __restrict__ y,
                             float* __restrict__ loss, float* __restrict__ dlogits, int B,
                             int fout, float eps) {
  extern __shared__ float red[];
  const int c = blockIdx.x, b = threadIdx.x;
  const float* z = logits + ((int64_t)c * B + b) * fout;
  float* dz = dlogits + ((int64_t)c * B + b) * fout;
  const int yb = y[(int64_t)c * B + b];
  float m = z[0];
  for (int j = 1; j < fout; ++j) m = fmaxf(m, z[j]);
  float se = 0.f;
  for (int j = 0; j < fout; ++j) se += expf(z[j] - m);
  const float lse = m + logf(se);
  float l = 0.f;
  const float invB = 1.f / (float)B;
  for (int j = 0; j < fout; ++j) {
    const float t = (j == yb ? 1.f - eps : 0.f) + eps / (float)fout;
    l += t * (lse - z[j]);
    dz[j] = (expf(z[j] - lse) - t) * invB;
  }
  // deterministic tree over a power-of-two padded block
  int n2 = 1;
  while (n2 < blockDim.x) n2 <<= 1;
  red[b] = l;
  for (int q = b + blockDim.x; q < n2; q += blockDim.x) red[q] = 0.f;
  __syncthreads();
  for (int st = n2 >> 1; st > 0; st >>= 1) {
    for (int q = b; q < st; q += blockDim.x) red[q] += red[q + st];
    __syncthreads();
  }
  if (b == 0) loss[c] = red[0] * invB;
}

// dW and db: one thread per (c, j, k) (k == fin means the bias), summed over b
template <typename T>
__global__ void k_fc_bwd_w(const float* __restrict__ dlogits, const T* __restrict__ h,
                           float* __restrict__ dw, float* __restrict__ db, int64_t g_rs, int C,
                           int B, int fin, int fout) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t per = (int64_t)fout * (fin + 1);
  if (i >= (int64_t)C * per) return;
  const int c = (int)(i / per);
  const int64_t r = i % per;
  const int j = (int)(r / (fin + 1));
  const int k = (int)(r % (fin + 1));
  const float* dz = dlogits + (int64_t)c * B * fout + j;
  float s = 0.f;
  if (k == fin) {
    for (int b = 0; b < B; ++b) s += dz[(int64_t)b * fout];
    db[(int64_t)c * g_rs + j] = s;
    return;
  }
  const T* hp = h + (int64_t)c * B * fin + k;
  for (int b = 0; b < B; ++b) s = fmaf(dz[(int64_t)b * fout], to_f(hp[(int64_t)b * fin]), s);
  dw[(int64_t)c * g_rs + (int64_t)j * fin + k] = s;
}

// dh: one thread per (c, b, k)
template <typename T>
__global__ void k_fc_bwd_x(const float* __restrict__ dlogits, const T* __restrict__ w,
                           int64_t w_rs, T* __restrict__ dh, int C, int B, int fin, int fout) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)C * B * fin) return;
  const int k = (int)(i % fin);
  const int64_t cb = i / fin;
  const int c = (int)(cb / B);
  const float* dz = dlogits + cb * fout;
  const T* wp = w + (int64_t)c * w_rs + k;
  float s = 0.f;
  for (int j = 0; j < fout; ++j) s = fmaf(dz[j], to_f(wp[(int64_t)j * fin]), s);
  dh[i] = from_f<T>(s);
}

inline unsigned blocks(int64_t n, int t) { return (unsigned)((n + t - 1) / t); }

}  // namespace

template <typename T>
cudaError_t launch_fc_fwd(cudaStream_t s, const T* h, const T* w, int64_t w_rs, const float* b,
                          int64_t b_rs, float* logits, int C, int B, int fin, int fout) {
  const int64_t warps = (int64_t)C * B * fout;
  k_fc_fwd<T><<<blocks(warps * 32, 256), 256, 0, s>>>(h, w, w_rs, b, b_rs, logits, C, B, fin,
                                                       fout);
  return cudaGetLastError();
}

cudaError_t launch_softmax_ce(cudaStream_t s, const float* logits, const int32_t* y, float* loss,
                              float* dlogits, int C, int B, int fout, float label_smoothing) {
  int n2 = 1;
  while (n2 < B) n2 <<= 1;
  k_softmax_ce<<<C, B, n2 * sizeof(float), s>>>(logits, y, loss, dlogits, B, fout,
                                                 label_smoothing);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fc_bwd(cudaStream_t s, const float* dlogits, const T* h, const T* w,
                          int64_t w_rs, float* dw, float* db, int64_t g_rs, T* dh, int C, int B,
                          int fin, int fout) {
  const int64_t nw = (int64_t)C * fout * (fin + 1);
  k_fc_bwd_w<T><<<blocks(nw, 256), 256, 0, s>>>(dlogits, h, dw, db, g_rs, C, B, fin, fout);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t nx = (int64_t)C * B * fin;
  k_fc_bwd_x<T><<<blocks(nx, 256), 256, 0, s>>>(dlogits, w, w_rs, dh, C, B, fin, fout);
  return cudaGetLastError();
}

template cudaError_t launch_fc_fwd<float>(cudaStream_t, const float*, const float*, int64_t,
                                          const float*, int64_t, float*, int, int, int, int);
template cudaError_t launch_fc_fwd<bf16>(cudaStream_t, const bf16*, const bf16*, int64_t,
                                         const float*, int64_t, float*, int, int, int, int);
template cudaError_t launch_fc_bwd<float>(cudaStream_t, const float*, const float*, const float*,
                                          int64_t, float*, float*, int64_t, float*, int, int, int,
                                          int);
template cudaError_t launch_fc_bwd<bf16>(cudaStream_t, const float*, const bf16*, const bf16*,
                                         int64_t, float*, float*, int64_t, bf16*, int, int, int,
                                         int);

}  // namespace gcpsl
