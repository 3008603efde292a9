// GPSL global sampling inside each cluster (Eq. 1; epoch rule of
// Section III-A) and the gather of the sampled images (with bf16 operands,
// straight into the input layer's im2col), optionally with the crop and
// flip augmentation of Section V-A (see AugArgs).
//
// Epoch permutation of cluster n: every example id j of the cluster gets the
// 64-bit key (o0 << 32 | o1) of Philox4x32-10(counter = (j, epoch, n', 0),
// key = seed), n' = cluster_base + n, and the epoch order is the ids sorted by
// (key, j).  Round s of the epoch takes positions [sB, sB + B) and orders them
// by (owner, j).  The sort is a rank count: rank(i) = #{m : (k_m, j_m) <
// (k_i, j_i)}, which is exact, deterministic and needs no scratch; it runs
// once per epoch per cluster (every n_c / B rounds).
//
// The round counter t lives in device memory so that a captured step can be
// replayed: cluster n is in epoch t / r_n, round t % r_n.
#include "common.cuh"

namespace gcpsl {

namespace {

constexpr int kRankThreads = 256;

__global__ void k_epoch_keys(const int32_t* __restrict__ ids, const int64_t* __restrict__ off,
                             const int32_t* __restrict__ period, const int64_t* __restrict__ d_t,
                             int cluster_base, uint32_t s0, uint32_t s1,
                             uint64_t* __restrict__ keys) {
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y;
  const int64_t t = *d_t;
  const int64_t r = period[c];
  if (t % r != 0) return;                       // not an epoch boundary
  const uint32_t epoch = (uint32_t)(t / r);
  const int64_t base = off[c], n = off[c + 1] - base;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  uint32_t ctr[4] = {(uint32_t)ids[base + i], epoch, (uint32_t)(cluster_base + c), 0u};
  philox4x32_10(ctr, s0, s1);
  keys[base + i] = ((uint64_t)ctr[0] << 32) | ctr[1];
}

__device__ __forceinline__ bool key_less(uint64_t ka, int32_t ja, uint64_t kb, int32_t jb) {
  return ka < kb || (ka == kb && ja < jb);
}

__global__ void __launch_bounds__(kRankThreads)
k_epoch_rank(const int32_t* __restrict__ ids, const int64_t* __restrict__ off,
             const int32_t* __restrict__ period, const int64_t* __restrict__ d_t,
             const uint64_t* __restrict__ keys, int32_t* __restrict__ perm) {
  __shared__ uint64_t sk[kRankThreads];
  __shared__ int32_t sj[kRankThreads];
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y;
  const int64_t t = *d_t;
  if (t % period[c] != 0) return;
  const int64_t base = off[c], n = off[c + 1] - base;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if ((int64_t)blockIdx.x * blockDim.x >= n) return;      // whole block idle
  const bool mine = i < n;
  const uint64_t ki = mine ? keys[base + i] : 0;
  const int32_t ji = mine ? ids[base + i] : 0;
  int64_t rank = 0;
  for (int64_t t0 = 0; t0 < n; t0 += kRankThreads) {
    const int64_t m = t0 + threadIdx.x;
    if (m < n) { sk[threadIdx.x] = keys[base + m]; sj[threadIdx.x] = ids[base + m]; }
    __syncthreads();
    const int lim = (n - t0) < kRankThreads ? (int)(n - t0) : kRankThreads;
    for (int q = 0; q < lim; ++q) rank += key_less(sk[q], sj[q], ki, ji);
    __syncthreads();
  }
  if (mine) perm[base + rank] = ji;
}

// One block per cluster, one thread per batch slot (B <= 1024).
__global__ void k_sample(const int32_t* __restrict__ perm, const int64_t* __restrict__ off,
                         const int32_t* __restrict__ rounds, const int32_t* __restrict__ period,
                         const int64_t* __restrict__ d_t, const int32_t* __restrict__ owner,
                         const int32_t* __restrict__ labels, int K, int B,
                         int32_t* __restrict__ idx, int32_t* __restrict__ counts,
                         int32_t* __restrict__ active, int32_t* __restrict__ y,
                         int32_t* __restrict__ upd, float* __restrict__ cut_scale) {
  extern __shared__ int32_t sm[];
  int32_t* sid = sm;          // [B] ids of the round
  int32_t* sown = sm + B;     // [B] their owners
  int32_t* sorted_own = sm + 2 * B;
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.x;
  const int b = threadIdx.x;
  int64_t s = *d_t % period[c];
  const bool updates = s < rounds[c];          // else waiting at the fusion barrier
  if (!updates) s = rounds[c] - 1;
  int32_t* cnt = counts + (int64_t)c * K;
  for (int k = b; k < K; k += blockDim.x) cnt[k] = 0;
  const int32_t id = perm[off[c] + s * B + b];
  const int32_t own = owner[id];
  sid[b] = id;
  sown[b] = own;
  __syncthreads();
  int rank = 0;
  for (int q = 0; q < B; ++q)
    rank += (sown[q] < own) || (sown[q] == own && sid[q] < id);
  idx[(int64_t)c * B + rank] = id;
  y[(int64_t)c * B + rank] = labels[id];
  sorted_own[rank] = own;
  atomicAdd(&cnt[own], 1);
  __syncthreads();
  const int first = __syncthreads_count(rank == 0 || sorted_own[rank - 1] != own);
  if (b == 0) {
    active[c] = updates ? first : 0;
    if (upd) upd[c] = updates;
  }
  if (cut_scale)   // B / (|A| b_k): the counts are complete after the barrier above
    cut_scale[(int64_t)c * B + rank] = (float)B / ((float)first * (float)cnt[own]);
}

// crop offsets and flip of sampled image cb = c * B + b (see AugArgs)
__device__ __forceinline__ void aug_params(const AugArgs& a, int64_t cb, int& dy, int& dx,
                                           int& flip) {
  dy = dx = 4;
  flip = 0;
  if (!a.on) return;
  const int c = (int)(cb / a.B), b = (int)(cb % a.B);
  uint32_t ctr[4] = {(uint32_t)b, (uint32_t)*a.d_t, (uint32_t)(a.cluster_base + c), 1u};
  philox4x32_10(ctr, a.s0, a.s1);
  dy = (int)(((uint64_t)ctr[0] * 9u) >> 32);
  dx = (int)(((uint64_t)ctr[1] * 9u) >> 32);
  flip = (int)(ctr[2] & 1u);
}

// fp32 storage: x0[c][b][h][w][ch] = images[idx[c][b]][ch][h][w] (3 channels).
__global__ void k_gather_f32(const float* __restrict__ images, const int32_t* __restrict__ idx,
                             int CB, float* __restrict__ x0, const AugArgs aug) {
  pdl_wait();
  pdl_trigger();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)CB * 1024) return;
  const int64_t cb = i >> 10;
  const int p = (int)(i & 1023), y = p >> 5, x = p & 31;
  int dy, dx, flip;
  aug_params(aug, cb, dy, dx, flip);
  const int sy = y + dy - 4, sx = (flip ? 31 - x : x) + dx - 4;
  const bool in = sy >= 0 && sy < 32 && sx >= 0 && sx < 32;
  const float* src = images + (int64_t)idx[cb] * 3072 + (in ? sy * 32 + sx : 0);
  float* dst = x0 + i * 3;
  dst[0] = in ? src[0] : 0.f;
  dst[1] = in ? src[1024] : 0.f;
  dst[2] = in ? src[2048] : 0.f;
}

// bf16 storage: the input layer's im2col, x0[c][b][y][x][32] with column
// k = tap * 3 + ch (tap = 3 ky + kx) = image[ch][y + ky - 1][x + kx - 1]
// (0 outside the image), k = 27 = 1 (its weight-gradient column is the
// bias gradient) and k = 28..31 = 0.  A block per (sampled image, band of
// kIm2colRows output rows): the band's rows of the image and their one-row
// halo are staged with a zero border in shared memory, then every thread
// writes 16-byte groups of 8 columns (a warp writes 512 contiguous bytes).
constexpr int kIm2colThreads = 256, kIm2colRows = 8;
__global__ void __launch_bounds__(kIm2colThreads)
k_gather_im2col(const float* __restrict__ images, const int32_t* __restrict__ idx,
                bf16* __restrict__ x0, const AugArgs aug) {
  constexpr int TR = kIm2colRows + 2;              // staged rows (padded rows r0 .. r0 + TR - 1)
  __shared__ float tile[3][TR][34];
  pdl_wait();
  pdl_trigger();
  constexpr int bands = 32 / kIm2colRows;
  const int64_t cb = blockIdx.x / bands;
  const int r0 = (int)(blockIdx.x % bands) * kIm2colRows;   // first output row of the band
  const float* src = images + (int64_t)idx[cb] * 3072;
  int dy, dx, flip;
  aug_params(aug, cb, dy, dx, flip);
  for (int i = threadIdx.x; i < 3 * TR * 34; i += kIm2colThreads) {
    const int ch = i / (TR * 34), t = (i / 34) % TR, xx = i % 34;
    // padded pixel (r0 + t, xx) = the augmented image's (r0 + t - 1, xx - 1),
    // zero around it
    const int y = r0 + t - 1, x = xx - 1;
    const int sy = y + dy - 4, sx = (flip ? 31 - x : x) + dx - 4;
    const bool in = y >= 0 && y < 32 && x >= 0 && x < 32 && sy >= 0 && sy < 32 && sx >= 0 &&
                    sx < 32;
    tile[ch][t][xx] = in ? src[ch * 1024 + sy * 32 + sx] : 0.f;
  }
  __syncthreads();
  uint4* dst = reinterpret_cast<uint4*>(x0 + (cb * 1024 + r0 * 32) * 32);
  for (int q = threadIdx.x; q < kIm2colRows * 32 * 4; q += kIm2colThreads) {
    const int pix = q >> 2, g = q & 3, yl = pix >> 5, x = pix & 31;
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int k = 8 * g + e;
      const int tap = k / 3, ch = k - 3 * tap;
      v[e] = k < 27 ? tile[ch][yl + tap / 3][x + tap % 3] : (k == 27 ? 1.f : 0.f);
    }
    __align__(16) bf16 h[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) h[e] = __float2bfloat16_rn(v[e]);
    dst[q] = *reinterpret_cast<const uint4*>(h);
  }
}

// The per-client average of Sec. IV-B's other reading: example cb's gradient
// at the cut is multiplied by scale[cb] = B / (|A| b_k) (written by the
// sampler) before the client segment's backward.  Grid (chunks of
// kScaleThreads x 8 elements, C B examples); a and b (nullable) are
// [C B][per] tensors scaled in place, 8 elements per thread.
constexpr int kScaleThreads = 256;
template <typename T>
__global__ void __launch_bounds__(kScaleThreads)
k_client_avg_scale(T* __restrict__ a, T* __restrict__ b2, int64_t per_a, int64_t per_b,
                   const float* __restrict__ scale) {
  pdl_wait();
  pdl_trigger();
  const int64_t cb = blockIdx.y;
  const float sc = scale[cb];
  const int64_t e = ((int64_t)blockIdx.x * kScaleThreads + threadIdx.x) * 8;
  for (int t = 0; t < 2; ++t) {
    T* p = t == 0 ? a : b2;
    const int64_t per = t == 0 ? per_a : per_b;
    if (!p || e >= per) continue;
    T* q = p + cb * per + e;
#pragma unroll
    for (int i = 0; i < 8; ++i) q[i] = from_f<T>(to_f(q[i]) * sc);
  }
}

}  // namespace

cudaError_t launch_epoch_keys(cudaStream_t s, const int32_t* ids, const int64_t* off,
                              const int32_t* period, const int64_t* d_t, int cluster_base,
                              uint64_t seed, uint64_t* keys, int C, int64_t max_nc) {
  dim3 grid((unsigned)((max_nc + 255) / 256), (unsigned)C);
  return launch_k(k_epoch_keys, grid, 256, 0, s, ids, off, period, d_t, cluster_base,
                  (uint32_t)seed, (uint32_t)(seed >> 32), keys);
}

cudaError_t launch_epoch_rank(cudaStream_t s, const int32_t* ids, const int64_t* off,
                              const int32_t* period, const int64_t* d_t, const uint64_t* keys,
                              int32_t* perm, int C, int64_t max_nc) {
  dim3 grid((unsigned)((max_nc + kRankThreads - 1) / kRankThreads), (unsigned)C);
  return launch_k(k_epoch_rank, grid, kRankThreads, 0, s, ids, off, period, d_t, keys, perm);
}

cudaError_t launch_sample(cudaStream_t s, const int32_t* perm, const int64_t* off,
                          const int32_t* rounds, const int32_t* period, const int64_t* d_t,
                          const int32_t* owner, const int32_t* labels, int K, int B, int C,
                          int32_t* idx, int32_t* counts, int32_t* active, int32_t* y,
                          int32_t* upd, float* cut_scale) {
  return launch_k(k_sample, C, B, 3 * B * sizeof(int32_t), s, perm, off, rounds, period, d_t,
                  owner, labels, K, B, idx, counts, active, y, upd, cut_scale);
}

template <>
cudaError_t launch_gather<float>(cudaStream_t s, const float* images, const int32_t* idx, int CB,
                                 float* x0, const AugArgs& aug) {
  const int64_t n = (int64_t)CB * 1024;
  return launch_k(k_gather_f32, (unsigned)((n + 255) / 256), 256, 0, s, images, idx, CB, x0,
                  aug);
}
template <>
cudaError_t launch_gather<bf16>(cudaStream_t s, const float* images, const int32_t* idx, int CB,
                                bf16* x0, const AugArgs& aug) {
  return launch_k(k_gather_im2col, (unsigned)(CB * (32 / kIm2colRows)), kIm2colThreads, 0, s,
                  images, idx, x0, aug);
}

template <typename T>
cudaError_t launch_client_avg_scale(cudaStream_t s, T* a, int64_t per_a, T* b, int64_t per_b,
                                    const float* scale, int CB) {
  if (per_a % 8 || per_b % 8 || (uintptr_t)a % 16 || (uintptr_t)b % 16 || CB > 65535)
    return cudaErrorInvalidValue;
  const int64_t per = per_a > per_b ? per_a : per_b;
  const dim3 grid((unsigned)((per / 8 + kScaleThreads - 1) / kScaleThreads), (unsigned)CB);
  return launch_k(k_client_avg_scale<T>, grid, kScaleThreads, 0, s, a, b, per_a, per_b, scale);
}
template cudaError_t launch_client_avg_scale<float>(cudaStream_t, float*, int64_t, float*, int64_t,
                                                    const float*, int);
template cudaError_t launch_client_avg_scale<bf16>(cudaStream_t, bf16*, int64_t, bf16*, int64_t,
                                                   const float*, int);

}  // namespace gcpsl
