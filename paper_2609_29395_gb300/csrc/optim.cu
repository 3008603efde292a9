// Per-replica SGD and split-model fusion, both elementwise over the [C][P]
// fp32 parameter store, refreshing the bf16 operand shadow when present.
//
// SGD (PyTorch convention, Section V-A optimiser): g' = g + wd*theta;
//   v = mu*v + g' (v starts at 0, so round one takes v = g');
//   theta -= lr * (nesterov ? g' + mu*v : v), or theta -= lr*g' when mu = 0.
// Fusion (Eq. 5): theta_bar = sum_n q_n theta_n, written to every replica
//   (Section IV-C broadcast; momentum is not fused).  Since sum_n q_n = 1 it
//   is evaluated as theta_0 + sum_{n>=1} q_n (theta_n - theta_0) in fp32,
//   which returns theta exactly when all replicas are equal.
#include "common.cuh"

namespace gcpsl {

namespace {

__global__ void k_sgd(float* __restrict__ theta, float* __restrict__ mom,
                      const float* __restrict__ grad, bf16* __restrict__ shadow, int64_t n,
                      float lr, float mu, float wd, int nesterov, int64_t* __restrict__ d_t) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    float th = theta[i];
    float g = grad[i];
    if (wd != 0.f) g = fmaf(wd, th, g);
    if (mu != 0.f) {
      const float v = fmaf(mu, mom[i], g);
      mom[i] = v;
      g = nesterov ? fmaf(mu, v, g) : v;
    }
    th = fmaf(-lr, g, th);
    theta[i] = th;
    if (shadow) shadow[i] = __float2bfloat16_rn(th);
  }
  // the round counter advances once the update of this round is enqueued;
  // nothing later in the round reads it
  if (blockIdx.x == 0 && threadIdx.x == 0) *d_t += 1;
}

__global__ void k_fuse(float* __restrict__ theta, bf16* __restrict__ shadow,
                       const float* __restrict__ q, int C, int64_t P) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P; p += stride) {
    const float base = theta[p];
    float acc = 0.f;
    for (int n = 1; n < C; ++n) acc = fmaf(q[n], theta[(int64_t)n * P + p] - base, acc);
    const float f = base + acc;
    for (int n = 0; n < C; ++n) {
      theta[(int64_t)n * P + p] = f;
      if (shadow) shadow[(int64_t)n * P + p] = __float2bfloat16_rn(f);
    }
  }
}

unsigned grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  const int64_t cap = 152 * 16;
  return (unsigned)(b < cap ? (b > 0 ? b : 1) : cap);
}

}  // namespace

cudaError_t launch_sgd(cudaStream_t s, float* theta, float* mom, const float* grad,
                       bf16* shadow, int64_t n, float lr, float momentum, float wd,
                       int nesterov, int64_t* d_t) {
  return launch_k(k_sgd, grid_for(n, 256), 256, 0, s, theta, mom, grad, shadow, n, lr, momentum,
                  wd, nesterov, d_t);
}

cudaError_t launch_fuse(cudaStream_t s, float* theta, bf16* shadow, const float* q, int C,
                        int64_t P) {
  return launch_k(k_fuse, grid_for(P, 256), 256, 0, s, theta, shadow, q, C, P);
}

}  // namespace gcpsl
