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
#include "sm100.cuh"

namespace gcpsl {

namespace {

__global__ void k_sgd(float* __restrict__ theta, float* __restrict__ mom,
                      const float* __restrict__ grad, bf16* __restrict__ shadow, int64_t n,
                      int64_t P_pad, float lr, float mu, float wd, int nesterov,
                      const int32_t* __restrict__ upd, int64_t* __restrict__ d_t) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    if (upd && !upd[i / P_pad]) continue;          // waiting at the fusion barrier
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

// k_sgd over parameter segments (see SgdSeg): the split partials of a
// weight gradient are summed here, in split order, instead of in a separate
// reduction pass.  Everything is in units of 4 parameters (segment offsets,
// counts, strides and the replica stride are multiples of 4), 32-bit
// indices.  Block b takes blocks[b] = {segment, first quad, quads}: fewer
// quads per block where a segment has more splits, so that every block
// reads about the same number of bytes; a thread keeps the loads of its
// kSgdPer quads in flight together.
__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float sgd1(float& th, float& m, float g, float lr, float mu, float wd,
                                      int nesterov) {
  if (wd != 0.f) g = fmaf(wd, th, g);
  if (mu != 0.f) {
    const float v = fmaf(mu, m, g);
    m = v;
    g = nesterov ? fmaf(mu, v, g) : v;
  }
  th = fmaf(-lr, g, th);
  return th;
}

__global__ void __launch_bounds__(kSgdThreads)
k_sgd_seg(float4* __restrict__ theta, float4* __restrict__ mom, uint2* __restrict__ shadow,
          const SgdSeg* __restrict__ segs, const int4* __restrict__ blocks, uint32_t P4,
          float lr, float mu, float wd, int nesterov, const int32_t* __restrict__ upd,
          int64_t* __restrict__ d_t) {
  pdl_wait();
  pdl_trigger();
  const int4 bk = blocks[blockIdx.x];
  const SgdSeg& sq = segs[bk.x];
  const float4* src = reinterpret_cast<const float4*>(sq.src);
  const uint32_t cnt4 = (uint32_t)(sq.count >> 2), per4 = (uint32_t)(sq.per >> 2);
  const uint32_t off4 = (uint32_t)(sq.off >> 2);
  const int splits = sq.splits;
  float4 g[kSgdPer];
  uint32_t at[kSgdPer], sa[kSgdPer];
  bool ok[kSgdPer];
#pragma unroll
  for (int k = 0; k < kSgdPer; ++k) {
    const uint32_t r = (uint32_t)(k * kSgdThreads) + threadIdx.x;
    const uint32_t local = (uint32_t)bk.y + r;
    const uint32_t c = local / cnt4, j = local - c * cnt4;
    ok[k] = r < (uint32_t)bk.z && (!upd || upd[c]);   // skip replicas at the fusion barrier
    at[k] = c * P4 + off4 + j;
    sa[k] = c * (uint32_t)splits * per4 + j;
    g[k] = ok[k] ? src[sa[k]] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int sp = 1; sp < splits; ++sp) {
#pragma unroll
    for (int k = 0; k < kSgdPer; ++k)
      if (ok[k]) g[k] = f4add(g[k], src[sa[k] + (uint32_t)sp * per4]);
  }
#pragma unroll
  for (int k = 0; k < kSgdPer; ++k) {
    if (!ok[k]) continue;
    float4 th = theta[at[k]];
    float4 m = mu != 0.f ? mom[at[k]] : make_float4(0.f, 0.f, 0.f, 0.f);
    sgd1(th.x, m.x, g[k].x, lr, mu, wd, nesterov);
    sgd1(th.y, m.y, g[k].y, lr, mu, wd, nesterov);
    sgd1(th.z, m.z, g[k].z, lr, mu, wd, nesterov);
    sgd1(th.w, m.w, g[k].w, lr, mu, wd, nesterov);
    theta[at[k]] = th;
    if (mu != 0.f) mom[at[k]] = m;
    if (shadow) {
      const __nv_bfloat162 lo = __floats2bfloat162_rn(th.x, th.y);
      const __nv_bfloat162 hi = __floats2bfloat162_rn(th.z, th.w);
      shadow[at[k]] = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                                 *reinterpret_cast<const uint32_t*>(&hi));
    }
    if (sq.w0p) {
      // element j of the input layer's weights [co][27] -> w0p[c][co][j % 27]
      const uint32_t local = (uint32_t)bk.y + (uint32_t)(k * kSgdThreads) + threadIdx.x;
      const uint32_t c = local / cnt4, j0 = (local - c * cnt4) * 4;
      const uint32_t n27 = (uint32_t)sq.w0_cout * 27;
      const float t4[4] = {th.x, th.y, th.z, th.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t j = j0 + e;
        if (j < n27) {
          const uint32_t co = j / 27;
          sq.w0p[((int64_t)c * sq.w0_cout + co) * 32 + (j - co * 27)] = __float2bfloat16_rn(t4[e]);
        }
      }
    }
  }
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
                       bf16* shadow, int64_t n, int64_t P_pad, float lr, float momentum, float wd,
                       int nesterov, const int32_t* upd, int64_t* d_t) {
  return launch_k(k_sgd, grid_for(n, 256), 256, 0, s, theta, mom, grad, shadow, n, P_pad, lr,
                  momentum, wd, nesterov, upd, d_t);
}

cudaError_t launch_sgd_seg(cudaStream_t s, float* theta, float* mom, bf16* shadow,
                           const SgdSeg* segs, const int4* blocks, int nblocks, int64_t P_pad,
                           float lr, float momentum, float wd, int nesterov, const int32_t* upd,
                           int64_t* d_t) {
  if (nblocks < 1 || P_pad % 4 || (uintptr_t)theta % 16 || (uintptr_t)mom % 16 ||
      (uintptr_t)shadow % 8)
    return cudaErrorInvalidValue;
  return launch_k(k_sgd_seg, (unsigned)nblocks, kSgdThreads, 0, s,
                  reinterpret_cast<float4*>(theta), reinterpret_cast<float4*>(mom),
                  reinterpret_cast<uint2*>(shadow), segs, blocks, (uint32_t)(P_pad / 4), lr,
                  momentum, wd, nesterov, upd, d_t);
}

cudaError_t launch_fuse(cudaStream_t s, float* theta, bf16* shadow, const float* q, int C,
                        int64_t P) {
  return launch_k(k_fuse, grid_for(P, 256), 256, 0, s, theta, shadow, q, C, P);
}

// The failure path of the bounded waits: one thread waits on an mbarrier
// that expects one arrival which never comes, gives up after limit_ns and
// records bit 256 in the error word.
namespace {
__global__ void k_wait_probe(int* err, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  sm100::mbar_init(&bar, 1);
  sm100::fence_mbar_init();
  if (!sm100::mbar_wait(&bar, 0, limit_ns)) atomicOr(err, 256);
}
}  // namespace

cudaError_t launch_wait_probe(cudaStream_t s, int* err, uint64_t limit_ns) {
  k_wait_probe<<<1, 1, 0, s>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace gcpsl
