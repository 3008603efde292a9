// Server head: linear layer, softmax cross-entropy averaged over the batch,
// and the linear layer's backward, grouped over the C replicas.
//
// h is the last conv layer's pooled output read as [C][B][fin] (NHWC flatten;
// the linear weight is stored in the same (h, w, ch) order, so it equals
// PyTorch's (ch, h, w) flatten of an NCHW tensor with permuted weights).
//   logits[b,j] = b_fc[j] + sum_k h[b,k] W[j,k]
//   loss = (1/B) sum_b l_b,  l_b = lse(logits_b) - sum_j t_bj logits_bj,
//     t = (1-e) onehot(y) + e/J   (label smoothing e, 0 by default)
//   dlogits[b,j] = (softmax(logits_b)_j - t_bj) / B
//   dW[j,k] = sum_b dlogits[b,j] h[b,k];  db[j] = sum_b dlogits[b,j]
//   dh[b,k] = sum_j dlogits[b,j] W[j,k]
//
// Two launches: the forward with the per-example softmax (a block per four
// examples, its warps on feature slices, 16-byte loads of h and W), and the
// backward (lanes on feature pairs, warps on example chunks, all J classes
// in registers), which also sums the per-example losses and the bias
// gradient in a fixed order, and can hand dh straight through the last conv
// layer's max-pool / ReLU backward.
#include "common.cuh"

namespace gcpsl {

namespace {

constexpr int kFwdSlices = 8;      // warps (feature slices) per forward block
constexpr int kBwdPairs = 32;      // feature pairs per backward block (one per lane)
constexpr int kBwdChunks = 8;      // example chunks per backward block (one per warp)

// VEC consecutive elements starting at p, as floats (16-byte load for VEC > 1)
template <typename T, int VEC> struct VecLoad;
template <> struct VecLoad<bf16, 8> {
  __device__ static void run(const bf16* p, float* o) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      o[2 * i] = __uint_as_float(w[i] << 16);
      o[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
};
template <> struct VecLoad<float, 4> {
  __device__ static void run(const float* p, float* o) {
    const float4 u = *reinterpret_cast<const float4*>(p);
    o[0] = u.x; o[1] = u.y; o[2] = u.z; o[3] = u.w;
  }
};
template <> struct VecLoad<bf16, 2> {
  __device__ static void run(const bf16* p, float* o) {
    const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
    o[0] = __uint_as_float(u << 16);
    o[1] = __uint_as_float(u & 0xffff0000u);
  }
};
template <> struct VecLoad<float, 2> {
  __device__ static void run(const float* p, float* o) {
    const float2 u = *reinterpret_cast<const float2*>(p);
    o[0] = u.x; o[1] = u.y;
  }
};
template <typename T> struct VecLoad<T, 1> {
  __device__ static void run(const T* p, float* o) { o[0] = to_f(p[0]); }
};

// Block = (replica c, EX consecutive examples); warp w takes the k
// slices w, w + kFwdSlices, ... of VEC * 32 features (one slice each when
// fin = kFwdSlices * 32 * VEC), so every load of the block is issued at
// once.  The classes are taken JC at a time (JC weight rows in registers);
// lane partial sums are reduced by a fixed xor tree, the warps' sums in
// warp order; then one warp per example takes the softmax: with J <= 32
// every lane reads all J logits, otherwise lane l holds the logits
// l, l + 32, ... and max, sum and loss are xor-tree warp reductions.
template <typename T, int VEC, int J, int JC, int EX>
__global__ void __launch_bounds__(kFwdSlices * 32)
k_fc_fwd_ce(const T* __restrict__ h, const T* __restrict__ w, int64_t w_rs,
            const float* __restrict__ bias, int64_t b_rs, const int32_t* __restrict__ y,
            float* __restrict__ loss_ex, float* __restrict__ dlogits, int C, int B, int fin,
            float eps) {
  static_assert(J % JC == 0, "class chunks must tile J");
  __shared__ float part[kFwdSlices][EX * J];
  __shared__ float logit[EX][J];
  pdl_wait();
  pdl_trigger();
  const int per_c = (B + EX - 1) / EX;
  const int c = blockIdx.x / per_c, e0 = (blockIdx.x % per_c) * EX;
  const int ne = B - e0 < EX ? B - e0 : EX;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* hp = h + ((int64_t)c * B + e0) * fin;
  const T* wp = w + (int64_t)c * w_rs;
  for (int j0 = 0; j0 < J; j0 += JC) {
    float acc[EX][JC];
#pragma unroll
    for (int e = 0; e < EX; ++e)
#pragma unroll
      for (int j = 0; j < JC; ++j) acc[e][j] = 0.f;
    for (int k = (warp * 32 + lane) * VEC; k < fin; k += kFwdSlices * 32 * VEC) {
      float hv[EX][VEC], wv[JC][VEC];
#pragma unroll
      for (int e = 0; e < EX; ++e) {
        if (e < ne) VecLoad<T, VEC>::run(hp + (int64_t)e * fin + k, hv[e]);
        else
#pragma unroll
          for (int v = 0; v < VEC; ++v) hv[e][v] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < JC; ++j) VecLoad<T, VEC>::run(wp + (int64_t)(j0 + j) * fin + k, wv[j]);
#pragma unroll
      for (int e = 0; e < EX; ++e)
#pragma unroll
        for (int j = 0; j < JC; ++j)
#pragma unroll
          for (int v = 0; v < VEC; ++v) acc[e][j] = fmaf(hv[e][v], wv[j][v], acc[e][j]);
    }
#pragma unroll
    for (int e = 0; e < EX; ++e)
#pragma unroll
      for (int j = 0; j < JC; ++j) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[e][j] += __shfl_xor_sync(0xffffffffu, acc[e][j], o);
        if (lane == 0) part[warp][e * J + j0 + j] = acc[e][j];
      }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < EX * J; i += kFwdSlices * 32) {
    const int e = i / J, j = i % J;
    float z = 0.f;
#pragma unroll
    for (int q = 0; q < kFwdSlices; ++q) z += part[q][i];
    logit[e][j] = z + bias[(int64_t)c * b_rs + j];
  }
  __syncthreads();
  if (warp >= ne) return;
  const int64_t cb = (int64_t)c * B + e0 + warp;
  const int yb = y[cb];
  const float invB = 1.f / (float)B;
  if constexpr (J <= 32) {
    // softmax of example e0 + warp: every lane reads the J logits
    float z[J];
#pragma unroll
    for (int j = 0; j < J; ++j) z[j] = logit[warp][j];
    float m = z[0];
#pragma unroll
    for (int j = 1; j < J; ++j) m = fmaxf(m, z[j]);
    float se = 0.f;
#pragma unroll
    for (int j = 0; j < J; ++j) se += expf(z[j] - m);
    const float lse = m + logf(se);
    float l = 0.f;
#pragma unroll
    for (int j = 0; j < J; ++j) {
      const float t = (j == yb ? 1.f - eps : 0.f) + eps / (float)J;
      l += t * (lse - z[j]);
      if (lane == j) dlogits[cb * J + j] = (expf(z[j] - lse) - t) * invB;
    }
    if (lane == 0) loss_ex[cb] = l;
  } else {
    constexpr int NJ = (J + 31) / 32;
    float z[NJ];
    float m = -INFINITY;
#pragma unroll
    for (int i = 0; i < NJ; ++i) {
      const int j = lane + 32 * i;
      z[i] = j < J ? logit[warp][j] : -INFINITY;
      m = fmaxf(m, z[i]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float se = 0.f;
#pragma unroll
    for (int i = 0; i < NJ; ++i)
      if (lane + 32 * i < J) se += expf(z[i] - m);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
    const float lse = m + logf(se);
    float l = 0.f;
#pragma unroll
    for (int i = 0; i < NJ; ++i) {
      const int j = lane + 32 * i;
      if (j < J) {
        const float t = (j == yb ? 1.f - eps : 0.f) + eps / (float)J;
        l += t * (lse - z[i]);
        dlogits[cb * J + j] = (expf(z[i] - lse) - t) * invB;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (lane == 0) loss_ex[cb] = l;
  }
}

// two consecutive features as floats
template <typename T> __device__ __forceinline__ float2 load2(const T* p);
template <> __device__ __forceinline__ float2 load2<float>(const float* p) {
  return *reinterpret_cast<const float2*>(p);
}
template <> __device__ __forceinline__ float2 load2<bf16>(const bf16* p) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
}
template <typename T> __device__ __forceinline__ void store2(T* p, float a, float b);
template <> __device__ __forceinline__ void store2<float>(float* p, float a, float b) {
  *reinterpret_cast<float2*>(p) = make_float2(a, b);
}
template <> __device__ __forceinline__ void store2<bf16>(bf16* p, float a, float b) {
  *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(a, b);
}

// Where dh goes: stored as is, or routed straight into the previous conv
// layer's g (the gradient w.r.t. its pre-activation) through that layer's
// 2x2 max-pool (codes: position | positive << 2) or its ReLU (act > 0).
struct HeadRoute {
  int mode;                 // FC_DH_STORE, FC_DH_POOL, FC_DH_RELU
  const uint8_t* code;      // FC_DH_POOL: codes, layout of h
  const void* act;          // FC_DH_RELU: ReLU output, layout of h
  int Ho, Wo, ch;           // h viewed as [Ho][Wo][ch]; g is [2Ho][2Wo][ch] for FC_DH_POOL
};

// dh of features (k, k+1) of example cb into dh or the routed g
template <typename T>
__device__ __forceinline__ void put_dh(T* __restrict__ out, const HeadRoute& rt, int64_t cb,
                                       int fin, int k, float d0, float d1) {
  const int64_t o = cb * fin + k;
  if (rt.mode == FC_DH_STORE) {
    store2<T>(out + o, d0, d1);
  } else if (rt.mode == FC_DH_AVG) {
    const int hw = rt.Ho * rt.Wo;
    const float inv = 1.f / (float)hw;
    for (int p = 0; p < hw; ++p) store2<T>(out + (cb * hw + p) * rt.ch + k, d0 * inv, d1 * inv);
  } else if (rt.mode == FC_DH_RELU) {
    const float2 a = load2<T>(reinterpret_cast<const T*>(rt.act) + o);
    store2<T>(out + o, a.x > 0.f ? d0 : 0.f, a.y > 0.f ? d1 : 0.f);
  } else {
    const uint8_t c0 = rt.code[o], c1 = rt.code[o + 1];
    const int cc = k % rt.ch, pix = k / rt.ch;
    const int x = pix % rt.Wo, y = pix / rt.Wo;
#pragma unroll
    for (int qd = 0; qd < 4; ++qd) {
      const int64_t go =
          ((cb * (2 * rt.Ho) + 2 * y + (qd >> 1)) * (2 * rt.Wo) + 2 * x + (qd & 1)) * rt.ch + cc;
      store2<T>(out + go, c0 == (4 | qd) ? d0 : 0.f, c1 == (4 | qd) ? d1 : 0.f);
    }
  }
}

// grid (ceil(fin / (2 * kBwdPairs)), C, J / JC).  Lane = feature pair
// (k, k+1), warp = chunk of ceil(B / kBwdChunks) consecutive examples,
// blockIdx.z = the classes j0 .. j0 + JC - 1; the warps' dW partial sums are
// added in warp order through shared memory.  Blocks with x == 0 also write
// db of their classes (warp 0); block (0, c, 0) writes loss[c] (warp 1).
// With DH (only when JC = J) the block also forms dh, all J classes of a
// feature pair being in its registers; otherwise k_fc_bwd_dh does.
template <typename T, int JC, bool DH>
__global__ void __launch_bounds__(kBwdPairs * kBwdChunks)
k_fc_bwd(const float* __restrict__ dlogits, const float* __restrict__ loss_ex,
         const T* __restrict__ h, const T* __restrict__ w, int64_t w_rs, float* __restrict__ dw,
         float* __restrict__ db, int64_t g_rs, T* __restrict__ dh, float* __restrict__ loss,
         int B, int fin, int J, const HeadRoute rt) {
  extern __shared__ float sm[];
  float* sdz = sm;                                 // [B][JC]
  float* red = sm + B * JC;                        // [kBwdChunks][kBwdPairs][2JC]
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y, j0 = blockIdx.z * JC;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* dz = dlogits + (int64_t)c * B * J;
  for (int i = threadIdx.x; i < B * JC; i += kBwdPairs * kBwdChunks)
    sdz[i] = dz[(i / JC) * J + j0 + i % JC];
  __syncthreads();
  const int k = 2 * (blockIdx.x * kBwdPairs + lane);
  const int bc = (B + kBwdChunks - 1) / kBwdChunks;
  const int b_lo = warp * bc, b_hi = b_lo + bc < B ? b_lo + bc : B;
  float a0[JC], a1[JC];
#pragma unroll
  for (int j = 0; j < JC; ++j) a0[j] = a1[j] = 0.f;
  if (k < fin) {
    float w0[JC], w1[JC];
    if constexpr (DH) {
      const T* wp = w + (int64_t)c * w_rs + k;
#pragma unroll
      for (int j = 0; j < JC; ++j) {
        const float2 v = load2<T>(wp + (int64_t)j * fin);
        w0[j] = v.x; w1[j] = v.y;
      }
    }
    const T* hp = h + (int64_t)c * B * fin + k;
    constexpr int U = 4;
    for (int b0 = b_lo; b0 < b_hi; b0 += U) {
      float2 hv[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        hv[u] = b0 + u < b_hi ? load2<T>(hp + (int64_t)(b0 + u) * fin) : make_float2(0.f, 0.f);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (b0 + u < b_hi) {
          const float* g = sdz + (b0 + u) * JC;
          float d0 = 0.f, d1 = 0.f;
#pragma unroll
          for (int j = 0; j < JC; ++j) {
            a0[j] = fmaf(g[j], hv[u].x, a0[j]);
            a1[j] = fmaf(g[j], hv[u].y, a1[j]);
            if constexpr (DH) {
              d0 = fmaf(g[j], w0[j], d0);
              d1 = fmaf(g[j], w1[j], d1);
            }
          }
          if constexpr (DH) put_dh<T>(dh, rt, (int64_t)c * B + b0 + u, fin, k, d0, d1);
        }
      }
    }
  }
  float* mine = red + (warp * kBwdPairs + lane) * 2 * JC;
#pragma unroll
  for (int j = 0; j < JC; ++j) { mine[2 * j] = a0[j]; mine[2 * j + 1] = a1[j]; }
  __syncthreads();
  // dW[j0 + j][k0 + pair*2 + x] = sum over chunks (in order) of the partials
  for (int o = threadIdx.x; o < kBwdPairs * 2 * JC; o += kBwdPairs * kBwdChunks) {
    const int pr = o / (2 * JC), jj = o % (2 * JC);
    const int kk = 2 * (blockIdx.x * kBwdPairs + pr) + (jj & 1);
    if (kk >= fin) continue;
    float sum = 0.f;
#pragma unroll
    for (int q = 0; q < kBwdChunks; ++q) sum += red[(q * kBwdPairs + pr) * 2 * JC + jj];
    dw[(int64_t)c * g_rs + (int64_t)(j0 + (jj >> 1)) * fin + kk] = sum;
  }
  if (blockIdx.x != 0) return;
  if (warp == 0 && lane < JC) {
    float sum = 0.f;
    for (int b = 0; b < B; ++b) sum += sdz[b * JC + lane];
    db[(int64_t)c * g_rs + j0 + lane] = sum;
  } else if (warp == 1 && blockIdx.z == 0) {
    float sum = 0.f;
    for (int b = lane; b < B; b += 32) sum += loss_ex[(int64_t)c * B + b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) loss[c] = sum / (float)B;
  }
}

// dh[b][k] = sum_j dlogits[b][j] W[j][k] for heads too wide for k_fc_bwd's
// registers.  grid (ceil(fin / (2 * kBwdPairs)), C, ceil(B / kDhExamples)):
// the block stages its J x 2 kBwdPairs slice of W in shared memory as fp32;
// lane = feature pair, warp = kDhExamples / kBwdChunks consecutive examples
// of the block's chunk, each dlogits row read as float4 (a broadcast: every
// lane reads the same row), classes summed in order 0 .. J-1.
constexpr int kDhExamples = 16;   // examples per k_fc_bwd_dh block

template <typename T, int J>
__global__ void __launch_bounds__(kBwdPairs * kBwdChunks)
k_fc_bwd_dh(const float* __restrict__ dlogits, const T* __restrict__ w, int64_t w_rs,
            T* __restrict__ dh, int B, int fin, const HeadRoute rt) {
  static_assert(J % 4 == 0, "dlogits rows are read as float4");
  __shared__ float2 ws[J][kBwdPairs];
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < J * kBwdPairs; i += kBwdPairs * kBwdChunks) {
    const int j = i / kBwdPairs, pr = i % kBwdPairs;
    const int kk = 2 * (blockIdx.x * kBwdPairs + pr);
    ws[j][pr] = kk < fin ? load2<T>(w + (int64_t)c * w_rs + (int64_t)j * fin + kk)
                         : make_float2(0.f, 0.f);
  }
  __syncthreads();
  const int k = 2 * (blockIdx.x * kBwdPairs + lane);
  if (k >= fin) return;
  constexpr int per_warp = kDhExamples / kBwdChunks;
  const int b_lo = blockIdx.z * kDhExamples + warp * per_warp;
  const int b_hi = b_lo + per_warp < B ? b_lo + per_warp : B;
  for (int b = b_lo; b < b_hi; ++b) {
    const float4* g4 = reinterpret_cast<const float4*>(dlogits + ((int64_t)c * B + b) * J);
    float d0 = 0.f, d1 = 0.f;
#pragma unroll 5
    for (int q = 0; q < J / 4; ++q) {
      const float4 g = g4[q];
      const float gv[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float2 wv = ws[4 * q + u][lane];
        d0 = fmaf(gv[u], wv.x, d0);
        d1 = fmaf(gv[u], wv.y, d1);
      }
    }
    put_dh<T>(dh, rt, (int64_t)c * B + b, fin, k, d0, d1);
  }
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15) == 0; }

}  // namespace

// The class count is a compile-time constant of the kernels: 10 and 100 are
// built.  The 100-way head takes its classes 10 at a time in the forward and
// the weight gradient and forms dh in k_fc_bwd_dh.
constexpr int kClassChunk = 10;

bool fc_bwd_split_dh(int fout) { return fout > kClassChunk; }

template <typename T>
cudaError_t launch_fc_fwd_ce(cudaStream_t s, const T* h, const T* w, int64_t w_rs,
                             const float* b, int64_t b_rs, const int32_t* y, float* loss_ex,
                             float* dlogits, int C, int B, int fin, int fout,
                             float label_smoothing) {
  if (fout != 10 && fout != 100) return cudaErrorInvalidValue;
  constexpr int VEC = 16 / (int)sizeof(T);
  // two examples per block for the 10-way head (more blocks), four for the
  // 100-way head (each block reads its W chunks once for more examples)
  const int ex = fout == 10 ? 2 : 4;
  const unsigned grid = (unsigned)((int64_t)C * ((B + ex - 1) / ex));
  // 16-byte loads need every row of h and of each replica's W on a 16-byte boundary
  const bool vec = fin % VEC == 0 && (w_rs * (int64_t)sizeof(T)) % 16 == 0 && aligned16(h) &&
                   aligned16(w);
#define FWD_ARGS s, h, w, w_rs, b, b_rs, y, loss_ex, dlogits, C, B, fin, label_smoothing
  if (fout == 10)
    return vec ? launch_k(k_fc_fwd_ce<T, VEC, 10, 10, 2>, grid, kFwdSlices * 32, 0, FWD_ARGS)
               : launch_k(k_fc_fwd_ce<T, 1, 10, 10, 2>, grid, kFwdSlices * 32, 0, FWD_ARGS);
  // the 100-way head loads pairs, so that all eight warps share fin = 512
  const bool vec2 = fin % 2 == 0 && w_rs % 2 == 0 && (uintptr_t)h % (2 * sizeof(T)) == 0 &&
                    (uintptr_t)w % (2 * sizeof(T)) == 0;
  return vec2 ? launch_k(k_fc_fwd_ce<T, 2, 100, kClassChunk, 4>, grid, kFwdSlices * 32, 0,
                         FWD_ARGS)
              : launch_k(k_fc_fwd_ce<T, 1, 100, kClassChunk, 4>, grid, kFwdSlices * 32, 0,
                         FWD_ARGS);
#undef FWD_ARGS
}

namespace {

bool head_route(int route, const uint8_t* code, const void* act, int Ho, int Wo, int ch, int fin,
                HeadRoute* rt) {
  if (route == FC_DH_AVG && (ch != fin || Ho * Wo < 1)) return false;
  if (route != FC_DH_STORE && route != FC_DH_AVG &&
      (ch % 2 || (int64_t)Ho * Wo * ch != fin || (route == FC_DH_POOL && !code) ||
       (route == FC_DH_RELU && !act)))
    return false;
  *rt = HeadRoute{route, code, act, Ho, Wo, ch};
  return true;
}

}  // namespace

template <typename T>
cudaError_t launch_fc_bwd(cudaStream_t s, const float* dlogits, const float* loss_ex,
                          const T* h, const T* w, int64_t w_rs, float* dw, float* db,
                          int64_t g_rs, T* dh, float* loss, int C, int B, int fin, int fout,
                          int route, const uint8_t* code, const T* act, int Ho, int Wo, int ch) {
  // feature pairs: even fin and 2-element alignment of every row
  if ((fout != 10 && fout != 100) || fin % 2 || w_rs % 2 || g_rs % 2 ||
      ((uintptr_t)w % (2 * sizeof(T))) || ((uintptr_t)dw % (2 * sizeof(float))))
    return cudaErrorInvalidValue;
  HeadRoute rt;
  if (!head_route(route, code, act, Ho, Wo, ch, fin, &rt)) return cudaErrorInvalidValue;
  const int JC = fout == 10 ? 10 : kClassChunk;
  const dim3 grid((unsigned)((fin / 2 + kBwdPairs - 1) / kBwdPairs), (unsigned)C,
                  (unsigned)(fout / JC));
  const size_t smem = sizeof(float) * ((size_t)B * JC + (size_t)kBwdChunks * kBwdPairs * 2 * JC);
  auto kern = fc_bwd_split_dh(fout) ? k_fc_bwd<T, kClassChunk, false> : k_fc_bwd<T, 10, true>;
  if (smem > 48 * 1024) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  return launch_k(kern, grid, kBwdPairs * kBwdChunks, smem, s, dlogits, loss_ex, h, w, w_rs, dw,
                  db, g_rs, dh, loss, B, fin, fout, rt);
}

template <typename T>
cudaError_t launch_fc_bwd_dh(cudaStream_t s, const float* dlogits, const T* w, int64_t w_rs,
                             T* dh, int C, int B, int fin, int fout, int route,
                             const uint8_t* code, const T* act, int Ho, int Wo, int ch) {
  if (fout != 100 || fin % 2 || w_rs % 2 || ((uintptr_t)w % (2 * sizeof(T))) ||
      !aligned16(dlogits))
    return cudaErrorInvalidValue;
  HeadRoute rt;
  if (!head_route(route, code, act, Ho, Wo, ch, fin, &rt)) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)((fin / 2 + kBwdPairs - 1) / kBwdPairs), (unsigned)C,
                  (unsigned)((B + kDhExamples - 1) / kDhExamples));
  return launch_k(k_fc_bwd_dh<T, 100>, grid, kBwdPairs * kBwdChunks, 0, s, dlogits, w, w_rs, dh,
                  B, fin, rt);
}

template cudaError_t launch_fc_fwd_ce<float>(cudaStream_t, const float*, const float*, int64_t,
                                             const float*, int64_t, const int32_t*, float*,
                                             float*, int, int, int, int, float);
template cudaError_t launch_fc_fwd_ce<bf16>(cudaStream_t, const bf16*, const bf16*, int64_t,
                                            const float*, int64_t, const int32_t*, float*, float*,
                                            int, int, int, int, float);
template cudaError_t launch_fc_bwd<float>(cudaStream_t, const float*, const float*, const float*,
                                          const float*, int64_t, float*, float*, int64_t, float*,
                                          float*, int, int, int, int, int, const uint8_t*,
                                          const float*, int, int, int);
template cudaError_t launch_fc_bwd<bf16>(cudaStream_t, const float*, const float*, const bf16*,
                                         const bf16*, int64_t, float*, float*, int64_t, bf16*,
                                         float*, int, int, int, int, int, const uint8_t*,
                                         const bf16*, int, int, int);

template cudaError_t launch_fc_bwd_dh<float>(cudaStream_t, const float*, const float*, int64_t,
                                             float*, int, int, int, int, int, const uint8_t*,
                                             const float*, int, int, int);
template cudaError_t launch_fc_bwd_dh<bf16>(cudaStream_t, const float*, const bf16*, int64_t,
                                            bf16*, int, int, int, int, int, const uint8_t*,
                                            const bf16*, int, int, int);

}  // namespace gcpsl
