// Grouped 3x3 convolutions (stride 1, zero padding 1) on the 5th-generation
// tensor cores: tcgen05.mma with bf16 operands staged in shared memory by
// TMA and fp32 accumulators in TMEM.  The replica index is gridDim.z, so one
// launch covers all C cluster replicas.
//
// Implicit GEMM.  Activations are NHWC [C][B][H][W][ch] bf16 and are read as
// 5-D TMA boxes (ch, W, rows, images, 1).  For kernel tap (kh, kw) the box
// origin is shifted by (kh-1, kw-1); out-of-range rows and columns are
// zero-filled by the TMA unit, which is exactly the convolution's padding.
//
//  k_conv_tc (fprop and dgrad):  D[m][n] = sum_{tap, c} A[m][tap, c] B[n][tap, c]
//    m = output pixel (one M tile = 128 pixels: whole image rows),
//    A = shifted input activation (K-major, 32 or 64 channels per stage),
//    B = weights [n][tap][c] (K-major, the bf16 shadow).
//    fprop: n = cout, B = W[co][tap][ci]; epilogue bias + ReLU (+ 2x2 max-pool
//      with the first-maximum code, decided on the fp32 values).
//    dgrad: input = g (gradient w.r.t. the pre-activation), n = cin, B = the
//      transposed, tap-flipped shadow Wt[ci][8-tap][co]; epilogue stores dx.
//  k_wgrad_tc: dW[co][tap][ci] = sum_p g[p][co] x[p + shift(tap)][ci]
//    M = co, N = ci, K = pixels.  Both operands are MN-major tiles (pixels are
//    rows, channels contiguous), loaded as 64-pixel boxes.  The pixel range is
//    split across CTAs; each writes an fp32 partial tile and k_wgrad_reduce
//    sums the partials in split order (deterministic).
//
// Warp roles (192 threads): warp 0 issues TMA, warp 1 allocates TMEM and
// issues MMAs, warps 2-5 run the epilogue (warp w reads TMEM lanes
// 32*(w%4) .. +31).  Every mbarrier wait is bounded; on expiry the CTA sets
// the context's error word and unwinds.
#include <cuda.h>

#include "common.cuh"
#include "sm100.cuh"

namespace gcpsl {

using namespace sm100;

namespace {

constexpr int kThreads = 192;
constexpr int BM = 128;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return (uint8_t*)(((uintptr_t)p + 1023) & ~(uintptr_t)1023);
}

__device__ __forceinline__ void epi_bar() {   // the four epilogue warps only
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

template <int BN, int BKC>
struct ConvCfg {
  static constexpr int A_BYTES = BM * BKC * 2;
  static constexpr int B_BYTES = BN * BKC * 2;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int S = STAGE >= 24576 ? 3 : (STAGE >= 12288 ? 4 : 6);
  static constexpr int PIPE = S * STAGE;
  static constexpr int STAGING = BM * (BN + 1) * 4;      // pooled epilogue
  static constexpr int SMEM = 1024 + (PIPE > STAGING ? PIPE : STAGING);
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
};

template <int BN, int BKC, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
k_conv_tc(const __grid_constant__ CUtensorMap tA, const __grid_constant__ CUtensorMap tB,
          const ConvTcArgs p) {
  using Cfg = ConvCfg<BN, BKC>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], done;
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x, c = blockIdx.z;
  const int n0 = blockIdx.y * BN;
  const int b0 = (mt / p.tiles_h) * p.bb, h0 = (mt % p.tiles_h) * p.hb;
  const int kper = p.kch / BKC;
  const int KB = 9 * kper;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(&done, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tA);
    tma_prefetch_desc(&tB);
  }
  if (warp == 1) { tmem_alloc(&tbase, Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    if (elect_one()) {
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % S;
        if (kb >= S && !mbar_wait(&empty[s], ((kb / S) & 1) ^ 1)) { atomicOr(p.err, 1); break; }
        uint8_t* sa = sm + s * Cfg::STAGE;
        const int tap = kb / kper, ch = (kb % kper) * BKC;
        mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
        tma_load_5d(sa, &tA, &full[s], ch, tap % 3 - 1, h0 + tap / 3 - 1, b0, c);
        tma_load_4d(sa + Cfg::A_BYTES, &tB, &full[s], ch, tap, n0, c);
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, 0, 0);
      constexpr uint32_t swz = BKC == 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t sbo = BKC * 2 * 8;
      bool ok = true;
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % S;
        if (!mbar_wait(&full[s], (kb / S) & 1)) { atomicOr(p.err, 2); ok = false; break; }
        tc_fence_after();
        const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
        for (int k = 0; k < BKC / 16; ++k)
          mma_f16(tmem, smem_desc(a + k * 32, 16, sbo, swz), smem_desc(b + k * 32, 16, sbo, swz),
                  idesc, (kb | k) != 0);
        mma_commit(&empty[s]);
      }
      (void)ok;
      mma_commit(&done);
    }
  } else {
    // ---------------- epilogue: warps 2..5 ----------------
    const int q = warp & 3;                     // TMEM lane quarter of this warp
    const int r = q * 32 + lane;                // M row = pixel of the tile
    const bool ok = mbar_wait(&done, 0);
    if (!ok) atomicOr(p.err, 4);
    tc_fence_after();
    const int W = p.W, H = p.H;
    const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
    if (EPI == EPI_POOL) {
      float* st = reinterpret_cast<float*>(sm);
      const float* bias = p.bias + (int64_t)c * p.bias_rs + n0;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) st[r * (BN + 1) + c0 + i] = v[i] + bias[c0 + i];
      }
      epi_bar();
      const int Wo = W / 2, hbo = p.hb / 2, Ho = H / 2;
      const int te = threadIdx.x - 64;
#pragma unroll 1
      for (int idx = te; idx < 32 * BN; idx += 128) {
        const int pp = idx / BN, co = idx % BN;
        const int pw = pp % Wo, ph = (pp / Wo) % hbo, bb = pp / (Wo * hbo);
        if (b0 + bb >= p.B) continue;
        const int r00 = (bb * p.hb + 2 * ph) * W + 2 * pw;
        const float* s0 = st + r00 * (BN + 1) + co;
        float best = s0[0];
        int arg = 0;
        const float v1 = s0[BN + 1], v2 = s0[W * (BN + 1)], v3 = s0[(W + 1) * (BN + 1)];
        if (v1 > best) { best = v1; arg = 1; }
        if (v2 > best) { best = v2; arg = 2; }
        if (v3 > best) { best = v3; arg = 3; }
        const int64_t o =
            ((((int64_t)c * p.B + b0 + bb) * Ho + h0 / 2 + ph) * Wo + pw) * p.n_total + n0 + co;
        p.out[o] = __float2bfloat16_rn(best > 0.f ? best : 0.f);
        p.code[o] = (uint8_t)(arg | (best > 0.f ? 4 : 0));
      }
    } else {
      const int w = r % W, hh = (r / W) % p.hb, bb = r / (W * p.hb);
      const bool valid = b0 + bb < p.B;
      const int64_t o = ((((int64_t)c * p.B + b0 + bb) * H + h0 + hh) * W + w) * p.n_total + n0;
      const float* bias = EPI == EPI_RELU ? p.bias + (int64_t)c * p.bias_rs + n0 : nullptr;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        tmem_ld_wait();
        if (!valid) continue;
        __align__(16) bf16 h[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float x = v[i];
          if (EPI == EPI_RELU) { x += bias[c0 + i]; x = x > 0.f ? x : 0.f; }
          h[i] = __float2bfloat16_rn(x);
        }
        uint4* dst = reinterpret_cast<uint4*>(p.out + o + c0);
        dst[0] = reinterpret_cast<uint4*>(h)[0];
        dst[1] = reinterpret_cast<uint4*>(h)[1];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, Cfg::TCOLS);
}

// ---------------------------------------------------------------------------
// weight gradient
// ---------------------------------------------------------------------------
template <int BN>
struct WgCfg {
  static constexpr int BKP = 64;                         // pixels per stage
  static constexpr int A_BYTES = 2 * 64 * BKP * 2;       // 128 co (two 64-wide blocks)
  static constexpr int B_BYTES = BN * BKP * 2;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int S = STAGE >= 32768 ? 4 : 5;
  static constexpr int SMEM = 1024 + S * STAGE;
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : 128;
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
k_wgrad_tc(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tX,
           const WgradTcArgs p) {
  using Cfg = WgCfg<BN>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], done;
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, c = blockIdx.z;
  const int ci_tiles = p.cin / BN;
  const int co_tiles = (p.cout + 127) / 128;
  int t = blockIdx.y;
  const int ci0 = (t % ci_tiles) * BN; t /= ci_tiles;
  const int co0 = (t % co_tiles) * 128; t /= co_tiles;
  const int tap = t;                                 // 0..8
  const int kh = tap / 3, kw = tap % 3;
  const int kb_begin = split * p.kb_per_split;
  const int kb_end = min(kb_begin + p.kb_per_split, p.kb_total);
  const int nkb = kb_end > kb_begin ? kb_end - kb_begin : 0;
  const int rows_blocks = p.H / p.hb;               // pixel blocks per image group

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(&done, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tG);
    tma_prefetch_desc(&tX);
  }
  if (warp == 1) { tmem_alloc(&tbase, Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    if (elect_one()) {
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (i >= S && !mbar_wait(&empty[s], ((i / S) & 1) ^ 1)) { atomicOr(p.err, 8); break; }
        const int kb = kb_begin + i;
        const int b = (kb / rows_blocks) * p.bb, h = (kb % rows_blocks) * p.hb;
        uint8_t* sa = sm + s * Cfg::STAGE;
        uint8_t* sb = sa + Cfg::A_BYTES;
        mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
        tma_load_5d(sa, &tG, &full[s], co0, 0, h, b, c);
        // rows 64..127 of the M tile: the next 64 channels, or (cout <= 64) a
        // second copy of the first block whose results the epilogue drops
        tma_load_5d(sa + 64 * Cfg::BKP * 2, &tG, &full[s], p.cout > co0 + 64 ? co0 + 64 : co0, 0,
                    h, b, c);
#pragma unroll
        for (int j = 0; j < (BN + 63) / 64; ++j)
          tma_load_5d(sb + j * 64 * Cfg::BKP * 2, &tX, &full[s], ci0 + 64 * j, kw - 1, h + kh - 1,
                      b, c);
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, 1, 1);
      // A: two 64-co blocks of BKP rows x 128 B; B: 64-ci blocks (SW128) or
      // one 32-ci block of 64-byte rows (SW64)
      constexpr uint32_t a_lbo = 64 * Cfg::BKP * 2;
      constexpr uint32_t b_swz = BN >= 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t b_row = BN >= 64 ? 128 : 64;
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (!mbar_wait(&full[s], (i / S) & 1)) { atomicOr(p.err, 16); break; }
        tc_fence_after();
        const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
        for (int k = 0; k < Cfg::BKP / 16; ++k)
          mma_f16(tmem, smem_desc(a + k * 16 * 128, a_lbo, 1024, SWZ_128),
                  smem_desc(b + k * 16 * b_row, a_lbo, 8 * b_row, b_swz), idesc, (i | k) != 0);
        mma_commit(&empty[s]);
      }
      mma_commit(&done);
    }
  } else {
    const int q = warp & 3;
    const int co = co0 + q * 32 + lane;
    const bool ok = mbar_wait(&done, 0);
    if (!ok) atomicOr(p.err, 32);
    tc_fence_after();
    float* dst = p.partial + (((int64_t)c * p.splits + split) * p.cout + co) * 9 * p.cin +
                 (int64_t)tap * p.cin + ci0;
    const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(trow + c0, v);
      tmem_ld_wait();
      if (co < p.cout) {
        float4* d4 = reinterpret_cast<float4*>(dst + c0);
#pragma unroll
        for (int i = 0; i < 4; ++i)
          d4[i] = nkb ? make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3])
                      : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, Cfg::TCOLS);
}

// dw[c][i] = sum over splits (in order) of partial[c][s][i]
__global__ void k_wgrad_reduce(const float* __restrict__ partial, float* __restrict__ dw,
                               int64_t dw_rs, int splits, int64_t per) {
  const int c = blockIdx.y;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < per;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float* src = partial + (int64_t)c * splits * per + i;
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += src[(int64_t)k * per];
    dw[(int64_t)c * dw_rs + i] = s;
  }
}

// Wt[c][ci][8 - tap][co] = W[c][co][tap][ci] (bf16 shadow, conv weights only)
__global__ void k_flip_shadow(const bf16* __restrict__ w, bf16* __restrict__ wt, int64_t rs,
                              int cout, int cin) {
  const int c = blockIdx.y;
  const int64_t per = (int64_t)cout * 9 * cin;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < per;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int ci = (int)(i % cin);
    const int tap = (int)((i / cin) % 9);
    const int co = (int)(i / (9 * (int64_t)cin));
    wt[(int64_t)c * rs + ((int64_t)ci * 9 + (8 - tap)) * cout + co] = w[(int64_t)c * rs + i];
  }
}

template <int BN, int BKC, int EPI>
cudaError_t launch_conv_inst(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                             const ConvTcArgs& p, dim3 grid) {
  using Cfg = ConvCfg<BN, BKC>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv_tc<BN, BKC, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_conv_tc<BN, BKC, EPI><<<grid, kThreads, Cfg::SMEM, s>>>(a, b, p);
  return cudaGetLastError();
}

template <int BN>
cudaError_t launch_wgrad_inst(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                              const WgradTcArgs& p, dim3 grid) {
  using Cfg = WgCfg<BN>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_wgrad_tc<BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_wgrad_tc<BN><<<grid, kThreads, Cfg::SMEM, s>>>(g, x, p);
  return cudaGetLastError();
}

}  // namespace

// ---------------------------------------------------------------------------
// host: tensor maps
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool tensor_map_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                     const uint32_t* box, int swizzle_bytes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  uint64_t stride = 2;
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i > 0) gs[i - 1] = stride;
    stride *= dims[i];
  }
  const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                      : CU_TENSOR_MAP_SWIZZLE_NONE;
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), gd, gs,
            bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// same as tensor_map_bf16 but with an explicit byte stride for the outermost
// dimension (the replica stride of the [C][P] weight shadow)
bool tensor_map_bf16_strided(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                             uint64_t outer_stride_bytes, const uint32_t* box,
                             int swizzle_bytes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  uint64_t stride = 2;
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i > 0) gs[i - 1] = (i == rank - 1) ? outer_stride_bytes : stride;
    stride *= dims[i];
  }
  const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                      : CU_TENSOR_MAP_SWIZZLE_NONE;
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), gd, gs,
            bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
cudaError_t launch_conv_tc(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                           const ConvTcArgs& p, int bn, int bkc, int epi, int C) {
  const int tiles_m = p.tiles_h * ((p.B + p.bb - 1) / p.bb);
  dim3 grid(tiles_m, p.n_total / bn, C);
#define GCPSL_CONV_CASE(BN_, BKC_, EPI_) \
  if (bn == BN_ && bkc == BKC_ && epi == EPI_) return launch_conv_inst<BN_, BKC_, EPI_>(s, a, b, p, grid);
#define GCPSL_CONV_EPIS(BN_, BKC_)          \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_POOL)      \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_RELU)      \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_STORE)
  GCPSL_CONV_EPIS(32, 64)
  GCPSL_CONV_EPIS(64, 32)
  GCPSL_CONV_EPIS(64, 64)
  GCPSL_CONV_EPIS(128, 32)
  GCPSL_CONV_EPIS(128, 64)
  GCPSL_CONV_EPIS(256, 64)
#undef GCPSL_CONV_EPIS
#undef GCPSL_CONV_CASE
  return cudaErrorInvalidValue;
}

cudaError_t launch_wgrad_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                            const WgradTcArgs& p, int bn, int C) {
  const int tiles = 9 * (p.cin / bn) * ((p.cout + 127) / 128);
  dim3 grid(p.splits, tiles, C);
  if (bn == 32) return launch_wgrad_inst<32>(s, g, x, p, grid);
  if (bn == 64) return launch_wgrad_inst<64>(s, g, x, p, grid);
  if (bn == 128) return launch_wgrad_inst<128>(s, g, x, p, grid);
  return cudaErrorInvalidValue;
}

cudaError_t launch_wgrad_reduce(cudaStream_t s, const float* partial, float* dw, int64_t dw_rs,
                                int splits, int64_t per, int C) {
  const int threads = 256;
  int64_t blocks = (per + threads - 1) / threads;
  if (blocks > 1024) blocks = 1024;
  k_wgrad_reduce<<<dim3((unsigned)blocks, C), threads, 0, s>>>(partial, dw, dw_rs, splits, per);
  return cudaGetLastError();
}

cudaError_t launch_flip_shadow(cudaStream_t s, const bf16* w, bf16* wt, int64_t rs, int cout,
                               int cin, int C) {
  const int64_t per = (int64_t)cout * 9 * cin;
  int64_t blocks = (per + 255) / 256;
  if (blocks > 512) blocks = 512;
  k_flip_shadow<<<dim3((unsigned)blocks, C), 256, 0, s>>>(w, wt, rs, cout, cin);
  return cudaGetLastError();
}

}  // namespace gcpsl
