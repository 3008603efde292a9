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
//    dgrad: input = g (gradient w.r.t. the pre-activation), n = cin,
//      B[ci][tap][co] = W[co][8-tap][ci], read MN-major from the same shadow;
//      epilogue stores dx.
//  k_conv0_tc: the input layer (<= 8 channels, images padded to 8): two taps
//    per K=16 MMA step through the unswizzled layout.
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

// Epilogue of a 128-pixel x BN-channel accumulator tile, run by the four
// epilogue warps; the thread of TMEM row r owns pixel (bb, hh, ww) of the
// tile (r = (bb*hb + hh)*bw + ww, tiles are bw <= 16 pixels wide, so a warp
// holds whole 2x2 windows: partners at lane^1 and lane^bw).
//  EPI_POOL : + bias; 2x2 max-pool decided on the fp32 values (the larger
//             value wins, ties go to the earlier position in row-major
//             order, i.e. the first maximum); the window's top-left thread
//             stores relu(max) in bf16 and the code (position | positive<<2).
//  EPI_RELU : + bias, relu, bf16 store;   EPI_STORE: bf16 store.
// 16 channels per TMEM load; stores are 16-byte vectors.
template <int BN, int EPI>
__device__ __forceinline__ void conv_epilogue_drain(uint32_t trow, int r, int n0, int b0, int h0,
                                                    int w0, int c, const ConvTcArgs& p) {
  const int W = p.W, H = p.H, bw = p.bw;
  const int ww = r % bw, hh = (r / bw) % p.hb, bb = r / (bw * p.hb);
  const bool valid = b0 + bb < p.B;
  const float* bias = EPI != EPI_STORE ? p.bias + (int64_t)c * p.bias_rs + n0 : nullptr;
  int64_t o;
  bool owner = valid;
  if (EPI == EPI_POOL) {
    o = ((((int64_t)c * p.B + b0 + bb) * (H / 2) + (h0 + hh) / 2) * (W / 2) + (w0 + ww) / 2) *
            p.n_total + n0;
    owner = valid && !(hh & 1) && !(ww & 1);
  } else {
    o = ((((int64_t)c * p.B + b0 + bb) * H + h0 + hh) * W + w0 + ww) * p.n_total + n0;
  }
  const int mypos = (hh & 1) * 2 + (ww & 1);
#pragma unroll 1
  for (int c0 = 0; c0 < BN; c0 += 16) {
    float v[16];
    tmem_ld16(trow + c0, v);
    tmem_ld_wait();
    __align__(16) bf16 h[16];
    if (EPI == EPI_POOL) {
      __align__(16) uint8_t code[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        float val = v[i] + bias[c0 + i];
        int pos = mypos;
#pragma unroll
        for (int step = 0; step < 2; ++step) {
          const int x = step == 0 ? 1 : bw;
          const float pv = __shfl_xor_sync(0xffffffffu, val, x);
          const int pp = __shfl_xor_sync(0xffffffffu, pos, x);
          if (pv > val || (pv == val && pp < pos)) { val = pv; pos = pp; }
        }
        h[i] = __float2bfloat16_rn(val > 0.f ? val : 0.f);
        code[i] = (uint8_t)(pos | (val > 0.f ? 4 : 0));
      }
      if (owner) {
        uint4* dst = reinterpret_cast<uint4*>(p.out + o + c0);
        dst[0] = reinterpret_cast<uint4*>(h)[0];
        dst[1] = reinterpret_cast<uint4*>(h)[1];
        *reinterpret_cast<uint4*>(p.code + o + c0) = *reinterpret_cast<uint4*>(code);
      }
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        float x = v[i];
        if (EPI == EPI_RELU) { x += bias[c0 + i]; x = x > 0.f ? x : 0.f; }
        h[i] = __float2bfloat16_rn(x);
      }
      if (owner) {
        uint4* dst = reinterpret_cast<uint4*>(p.out + o + c0);
        dst[0] = reinterpret_cast<uint4*>(h)[0];
        dst[1] = reinterpret_cast<uint4*>(h)[1];
      }
    }
  }
}

template <int BN, int BKC, int EPI>
struct ConvCfg {
  static constexpr int A_BYTES = BM * BKC * 2;
  static constexpr int B_BYTES = BN * BKC * 2;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  // two CTAs per SM when both fit in TMEM (2 x 2 x TCOLS <= 512 columns)
  static constexpr int CTAS = 2 * TCOLS <= 256 ? 2 : 1;
  static constexpr int BUDGET = CTAS == 2 ? 100 * 1024 : 200 * 1024;
  static constexpr int S0 = BUDGET / STAGE;
  static constexpr int S = S0 > 8 ? 8 : (S0 < 2 ? 2 : S0);
  static constexpr int PIPE = S * STAGE;
  static constexpr int SMEM = 1024 + PIPE;
};

// (b0, h0, w0) of M tile mt
__device__ __forceinline__ void tile_origin(int mt, const ConvTcArgs& p, int& b0, int& h0,
                                            int& w0) {
  const int wt = mt % p.tiles_w, ht = (mt / p.tiles_w) % p.tiles_h, bt = mt / (p.tiles_w * p.tiles_h);
  b0 = bt * p.bb;
  h0 = ht * p.hb;
  w0 = wt * p.bw;
}

// Persistent implicit-GEMM convolution.  CTA b takes work items b, b + G,
// ... of the (replica, M tile, N tile) list (N fastest).  The TMA warp runs
// ahead through an S-stage ring across item boundaries; the MMA warp
// alternates between two TMEM accumulators (2 x TCOLS columns), so the
// epilogue of one item overlaps the MMAs of the next: tfull[b] (MMA ->
// epilogue) and tempty[b] (epilogue -> MMA, 128 arrivals) hand a buffer over.
// BMN = 0: B tile is K-major [n][tap][k] (fprop: W[co][tap][ci]).
// BMN = 1: B tile is read MN-major from W[co][tap][ci] itself (dgrad: n = ci,
//   k = co, tap flipped), as 64-wide (or one 32-wide) N blocks of BKC rows.
template <int BN, int BKC, int EPI, int BMN>
__global__ void __launch_bounds__(kThreads, 1)
k_conv_tc(const __grid_constant__ CUtensorMap tA, const __grid_constant__ CUtensorMap tB,
          const ConvTcArgs p, int tiles_m, int tiles_n, int items) {
  using Cfg = ConvCfg<BN, BKC, EPI>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], tfull[2], tempty[2];
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kper = p.kch / BKC;
  const int KB = 9 * kper;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&tfull[b], 1); mbar_init(&tempty[b], 128); }
    fence_mbar_init();
    tma_prefetch_desc(&tA);
    tma_prefetch_desc(&tB);
  }
  if (warp == 1) { tmem_alloc(&tbase, 2 * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    if (elect_one()) {
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < items && ok; t += gridDim.x) {
        const int c = t / (tiles_m * tiles_n), r = t % (tiles_m * tiles_n);
        const int mt = r / tiles_n, n0 = (r % tiles_n) * BN;
        int b0, h0, w0;
        tile_origin(mt, p, b0, h0, w0);
        for (int kb = 0; kb < KB; ++kb, ++it) {
          const int s = it % S;
          if (it >= S && !mbar_wait(&empty[s], ((it / S) & 1) ^ 1)) {
            atomicOr(p.err, 1);
            ok = false;
            break;
          }
          uint8_t* sa = sm + s * Cfg::STAGE;
          const int tap = kb / kper, ch = (kb % kper) * BKC;
          mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
          tma_load_5d(sa, &tA, &full[s], ch, w0 + tap % 3 - 1, h0 + tap / 3 - 1, b0, c);
          if (!BMN) {
            tma_load_4d(sa + Cfg::A_BYTES, &tB, &full[s], ch, tap, n0, c);
          } else {
            constexpr int NBW = BN < 64 ? BN : 64;           // N block width
#pragma unroll
            for (int j = 0; j < BN / NBW; ++j)
              tma_load_4d(sa + Cfg::A_BYTES + j * NBW * BKC * 2, &tB, &full[s], n0 + j * NBW,
                          8 - tap, ch, c);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, 0, BMN);
      constexpr uint32_t swz = BKC == 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t sbo = BKC * 2 * 8;
      // MN-major B: rows of NBW*2 bytes along K, N blocks BKC rows apart
      constexpr int NBW = BN < 64 ? BN : 64;
      constexpr uint32_t b_row = NBW * 2;
      constexpr uint32_t b_swz = NBW == 64 ? SWZ_128 : SWZ_64;
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < items && ok; t += gridDim.x, ++tl) {
        const int buf = tl & 1;
        if (tl >= 2 && !mbar_wait(&tempty[buf], ((tl >> 1) & 1) ^ 1)) {
          atomicOr(p.err, 2);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * Cfg::TCOLS;
        for (int kb = 0; kb < KB; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (it / S) & 1)) {
            atomicOr(p.err, 2);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
          for (int k = 0; k < BKC / 16; ++k) {
            const uint64_t bd = BMN ? smem_desc(b + k * 16 * b_row, NBW * BKC * 2, 8 * b_row, b_swz)
                                    : smem_desc(b + k * 32, 16, sbo, swz);
            mma_f16(d, smem_desc(a + k * 32, 16, sbo, swz), bd, idesc, (kb | k) != 0);
          }
          mma_commit(&empty[s]);
        }
        mma_commit(&tfull[buf]);
      }
    }
  } else {
    // ---------------- epilogue: warps 2..5 ----------------
    const int q = warp & 3;                     // TMEM lane quarter of this warp
    const int r = q * 32 + lane;                // M row = pixel of the tile
    int tl = 0;
    for (int t = blockIdx.x; t < items; t += gridDim.x, ++tl) {
      const int buf = tl & 1;
      // warp-uniform decision: the epilogue shuffles need the whole warp
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl >> 1) & 1))) {
        if (lane == 0) atomicOr(p.err, 4);
        break;
      }
      tc_fence_after();
      const int c = t / (tiles_m * tiles_n), rr = t % (tiles_m * tiles_n);
      const int mt = rr / tiles_n, n0 = (rr % tiles_n) * BN;
      int b0, h0, w0;
      tile_origin(mt, p, b0, h0, w0);
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16);
      conv_epilogue_drain<BN, EPI>(trow, r, n0, b0, h0, w0, c, p);
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * Cfg::TCOLS);
}

// ---------------------------------------------------------------------------
// input layer: at most 8 input channels (the gathered images, padded to 8)
// ---------------------------------------------------------------------------
// A K=16 MMA step takes two taps: with the unswizzled K-major layout a K=16
// slice is two 8-element core-matrix columns whose distance is the leading
// byte offset, so tap t's 128 x 16 B box and tap t+1's box can sit 2 KB apart.
// Ten tap slots are loaded (slot 9 repeats tap 8); the packed weights
// [tap][co][8] have zeros for tap 9 and for channels >= cin.
template <int BN, int EPI>
struct Conv0Cfg {
  static constexpr int SLOT_A = BM * 16;                 // one tap: 128 px x 8 ch
  static constexpr int A_BYTES = 10 * SLOT_A;
  static constexpr int B_BYTES = 10 * BN * 16;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int S = 3;
  static constexpr int PIPE = S * STAGE;
  static constexpr int SMEM = 1024 + PIPE;
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  static constexpr int CTAS = 2;                          // 2 x 2 x TCOLS <= 512 for BN <= 64
};

// Persistent like k_conv_tc: one ring stage holds one work item (ten tap
// slots and the packed weights), two TMEM accumulators alternate.
template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
k_conv0_tc(const __grid_constant__ CUtensorMap tA, const __grid_constant__ CUtensorMap tB,
           const ConvTcArgs p, int tiles_m, int items) {
  using Cfg = Conv0Cfg<BN, EPI>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], tfull[2], tempty[2];
  __shared__ uint32_t tbase;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&tfull[b], 1); mbar_init(&tempty[b], 128); }
    fence_mbar_init();
  }
  if (warp == 1) { tmem_alloc(&tbase, 2 * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  if (warp == 0) {
    if (elect_one()) {
      int it = 0;
      for (int t = blockIdx.x; t < items; t += gridDim.x, ++it) {
        const int c = t / tiles_m, mt = t % tiles_m;
        int b0, h0, w0;
        tile_origin(mt, p, b0, h0, w0);
        const int s = it % S;
        if (it >= S && !mbar_wait(&empty[s], ((it / S) & 1) ^ 1)) { atomicOr(p.err, 64); break; }
        uint8_t* st = sm + s * Cfg::STAGE;
        mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
#pragma unroll
        for (int j = 0; j < 10; ++j) {
          const int tap = j < 9 ? j : 8;
          tma_load_5d(st + j * Cfg::SLOT_A, &tA, &full[s], 0, w0 + tap % 3 - 1, h0 + tap / 3 - 1,
                      b0, c);
        }
        tma_load_4d(st + Cfg::A_BYTES, &tB, &full[s], 0, 0, 0, c);
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, 0, 0);
      int tl = 0;
      for (int t = blockIdx.x; t < items; t += gridDim.x, ++tl) {
        const int buf = tl & 1, s = tl % S;
        if (tl >= 2 && !mbar_wait(&tempty[buf], ((tl >> 1) & 1) ^ 1)) {
          atomicOr(p.err, 64);
          break;
        }
        if (!mbar_wait(&full[s], (tl / S) & 1)) { atomicOr(p.err, 64); break; }
        tc_fence_after();
        const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
        const uint32_t d = tmem + buf * Cfg::TCOLS;
#pragma unroll
        for (int k = 0; k < 5; ++k)
          mma_f16(d, smem_desc(a + 2 * k * Cfg::SLOT_A, Cfg::SLOT_A, 128, SWZ_NONE),
                  smem_desc(b + 2 * k * BN * 16, BN * 16, 128, SWZ_NONE), idesc, k != 0);
        mma_commit(&empty[s]);
        mma_commit(&tfull[buf]);
      }
    }
  } else {
    const int q = warp & 3, r = q * 32 + lane;
    int tl = 0;
    for (int t = blockIdx.x; t < items; t += gridDim.x, ++tl) {
      const int buf = tl & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl >> 1) & 1))) {
        if (lane == 0) atomicOr(p.err, 128);
        break;
      }
      tc_fence_after();
      const int c = t / tiles_m, mt = t % tiles_m;
      int b0, h0, w0;
      tile_origin(mt, p, b0, h0, w0);
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16);
      conv_epilogue_drain<BN, EPI>(trow, r, 0, b0, h0, w0, c, p);
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * Cfg::TCOLS);
}

// packed input-layer weights: w0p[c][tap][co][8] = W[co][tap][ci] for
// tap < 9 and ci < cin, else 0
__global__ void k_pack_w0(const bf16* __restrict__ w, bf16* __restrict__ w0p, int64_t rs,
                          int cout, int cin) {
  const int c = blockIdx.y;
  const int per = 10 * cout * 8;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < per; i += gridDim.x * blockDim.x) {
    const int ch = i % 8, co = (i / 8) % cout, tap = i / (8 * cout);
    bf16 v = __float2bfloat16_rn(0.f);
    if (tap < 9 && ch < cin) v = w[(int64_t)c * rs + ((int64_t)co * 9 + tap) * cin + ch];
    w0p[(int64_t)c * per + i] = v;
  }
}

// ---------------------------------------------------------------------------
// weight gradient
// ---------------------------------------------------------------------------
// One CTA owns a group of up to TG = 256/BN slots of a (128-co, BN-ci) tile:
// per K block the g tile is loaded once and multiplied, in one N <= 256 MMA,
// against the group's tap-shifted x tiles (consecutive N blocks).  Group 0
// holds taps 0..TG-2 and, in its last slot, a block of ones (written once
// into every ring stage), so its accumulator also yields the bias gradient
// sum_p g[p][co]; groups g >= 1 hold TG taps each.  The fp32 partial of a
// split is laid out like the parameters, [cout][9][cin] then [cout].
template <int BN>
struct WgCfg {
  static constexpr int BKP = 64;                         // pixels per stage
  static constexpr int TG = 256 / BN;                    // taps per CTA
  static constexpr int A_BYTES = 2 * 64 * BKP * 2;       // 128 co (two 64-wide blocks)
  static constexpr int TAP_BYTES = BN * BKP * 2;         // one tap's x tile
  static constexpr int STAGE = A_BYTES + TG * TAP_BYTES;
  static constexpr int S = 4;
  static constexpr int SMEM = 1024 + S * STAGE;
  static constexpr uint32_t TCOLS = 256;
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
k_wgrad_tc(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tX,
           const WgradTcArgs p) {
  using Cfg = WgCfg<BN>;
  constexpr int S = Cfg::S, TG = Cfg::TG;
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
  const int grp = t;                                 // tap group
  const bool bias_grp = grp == 0;
  const int tap0 = bias_grp ? 0 : (TG - 1) + (grp - 1) * TG;
  const int ntaps = bias_grp ? TG - 1 : (9 - tap0 < TG ? 9 - tap0 : TG);
  const int nslots = bias_grp ? TG : ntaps;          // N = nslots * BN
  const int per = p.cout * 9 * p.cin + p.cout;       // partial length per split
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
  if (bias_grp) {
    // the ones block (bf16 1.0 everywhere, so the swizzle does not matter)
    const uint4 ones = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    for (int s = 0; s < S; ++s) {
      uint4* dst = reinterpret_cast<uint4*>(sm + s * Cfg::STAGE + Cfg::A_BYTES +
                                            (TG - 1) * Cfg::TAP_BYTES);
      for (int i = threadIdx.x; i < Cfg::TAP_BYTES / 16; i += blockDim.x) dst[i] = ones;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
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
        mbar_arrive_expect_tx(&full[s], Cfg::A_BYTES + ntaps * Cfg::TAP_BYTES);
        tma_load_5d(sa, &tG, &full[s], co0, 0, h, b, c);
        // rows 64..127 of the M tile: the next 64 channels, or (cout <= 64) a
        // second copy of the first block whose results the epilogue drops
        tma_load_5d(sa + 64 * Cfg::BKP * 2, &tG, &full[s], p.cout > co0 + 64 ? co0 + 64 : co0, 0,
                    h, b, c);
        for (int tj = 0; tj < ntaps; ++tj) {
          const int tap = tap0 + tj, kh = tap / 3, kw = tap % 3;
#pragma unroll
          for (int j = 0; j < (BN + 63) / 64; ++j)
            tma_load_5d(sb + tj * Cfg::TAP_BYTES + j * 64 * Cfg::BKP * 2, &tX, &full[s],
                        ci0 + 64 * j, kw - 1, h + kh - 1, b, c);
        }
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      // one MMA per k step with N = ntaps*BN: the taps' x tiles are the
      // consecutive MN-major N blocks of one B operand (64-ci blocks, SW128,
      // or 32-ci blocks of 64-byte rows, SW64), `b_blk` bytes apart
      const uint32_t idesc = idesc_bf16(BM, nslots * BN, 1, 1);
      constexpr uint32_t a_lbo = 64 * Cfg::BKP * 2;
      constexpr uint32_t b_swz = BN >= 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t b_row = BN >= 64 ? 128 : 64;
      constexpr uint32_t b_blk = b_row * Cfg::BKP;
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (!mbar_wait(&full[s], (i / S) & 1)) { atomicOr(p.err, 16); break; }
        tc_fence_after();
        const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
        for (int k = 0; k < Cfg::BKP / 16; ++k)
          mma_f16(tmem, smem_desc(a + k * 16 * 128, a_lbo, 1024, SWZ_128),
                  smem_desc(b + k * 16 * b_row, b_blk, 8 * b_row, b_swz), idesc, (i | k) != 0);
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
    const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
    float* part = p.partial + ((int64_t)c * p.splits + split) * per;
    if (bias_grp && ci0 == 0) {
      float v[16];
      tmem_ld16(trow + (TG - 1) * BN, v);
      tmem_ld_wait();
      if (co < p.cout) part[p.cout * 9 * p.cin + co] = nkb ? v[0] : 0.f;
    }
    for (int tj = 0; tj < ntaps; ++tj) {
      float* dst = part + (int64_t)co * 9 * p.cin + (int64_t)(tap0 + tj) * p.cin + ci0;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + tj * BN + c0, v);
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
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, Cfg::TCOLS);
}

// Weight and bias gradient of the input layer (x padded to 8 channels, cout
// 32 or 64): D[co][slot*8 + ch] = sum_p g[p][co] B[p][slot*8 + ch] with slots
// 0..8 the tap-shifted x tiles (64 pixels x 16 bytes, unswizzled MN-major
// N blocks 1 KB apart) and slot 9 a block of ones (bias).  The g tile
// (cout channels, swizzled MN-major) fills the 128 MMA rows 128/cout times;
// the epilogue keeps rows < cout.  Partial layout as in k_wgrad_tc.
template <int COUT>
struct Wg0Cfg {
  static constexpr int BKP = 64;
  static constexpr int A_BLK = COUT * BKP * 2;           // one copy of the g tile
  static constexpr int A_BYTES = 128 * BKP * 2;
  static constexpr int SLOT = BKP * 16;
  static constexpr int B_BYTES = 10 * SLOT;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int S = 4;
  static constexpr int SMEM = 1024 + S * STAGE;
};

template <int COUT>
__global__ void __launch_bounds__(kThreads, 1)
k_wgrad0_tc(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tX,
            const WgradTcArgs p) {
  using Cfg = Wg0Cfg<COUT>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], done;
  __shared__ uint32_t tbase;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, c = blockIdx.z;
  const int per = COUT * 9 * p.cin + COUT;
  const int kb_begin = split * p.kb_per_split;
  const int kb_end = min(kb_begin + p.kb_per_split, p.kb_total);
  const int nkb = kb_end > kb_begin ? kb_end - kb_begin : 0;
  const int rows_blocks = p.H / p.hb;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(&done, 1);
    fence_mbar_init();
  }
  {
    const uint4 ones = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    for (int s = 0; s < S; ++s) {
      uint4* dst = reinterpret_cast<uint4*>(sm + s * Cfg::STAGE + Cfg::A_BYTES + 9 * Cfg::SLOT);
      for (int i = threadIdx.x; i < Cfg::SLOT / 16; i += blockDim.x) dst[i] = ones;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) { tmem_alloc(&tbase, 128); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  if (warp == 0) {
    if (elect_one()) {
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (i >= S && !mbar_wait(&empty[s], ((i / S) & 1) ^ 1)) { atomicOr(p.err, 256); break; }
        const int kb = kb_begin + i;
        const int b = (kb / rows_blocks) * p.bb, h = (kb % rows_blocks) * p.hb;
        uint8_t* sa = sm + s * Cfg::STAGE;
        uint8_t* sb = sa + Cfg::A_BYTES;
        mbar_arrive_expect_tx(&full[s], Cfg::A_BYTES + 9 * Cfg::SLOT);
#pragma unroll
        for (int j = 0; j < 128 / COUT; ++j) tma_load_5d(sa + j * Cfg::A_BLK, &tG, &full[s], 0, 0, h, b, c);
#pragma unroll
        for (int tap = 0; tap < 9; ++tap)
          tma_load_5d(sb + tap * Cfg::SLOT, &tX, &full[s], 0, tap % 3 - 1, h + tap / 3 - 1, b, c);
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, 80, 1, 1);
      constexpr uint32_t a_row = COUT * 2;
      constexpr uint32_t a_swz = COUT == 64 ? SWZ_128 : SWZ_64;
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (!mbar_wait(&full[s], (i / S) & 1)) { atomicOr(p.err, 256); break; }
        tc_fence_after();
        const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
        for (int k = 0; k < Cfg::BKP / 16; ++k)
          mma_f16(tmem, smem_desc(a + k * 16 * a_row, Cfg::A_BLK, 8 * a_row, a_swz),
                  smem_desc(b + k * 16 * 16, 128, Cfg::SLOT, SWZ_NONE), idesc, (i | k) != 0);
        mma_commit(&empty[s]);
      }
      mma_commit(&done);
    }
  } else {
    const int q = warp & 3;
    const int co = q * 32 + lane;
    if (!mbar_wait(&done, 0)) atomicOr(p.err, 512);
    tc_fence_after();
    if (q * 32 < COUT) {                        // warp-uniform
      const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
      float* part = p.partial + ((int64_t)c * p.splits + split) * per;
#pragma unroll 1
      for (int c0 = 0; c0 < 80; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int col = c0 + i, slot = col / 8, ch = col % 8;
          const float x = nkb ? v[i] : 0.f;
          if (slot < 9 && ch < p.cin) part[(co * 9 + slot) * p.cin + ch] = x;
          else if (slot == 9 && ch == 0) part[COUT * 9 * p.cin + co] = x;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 128);
}

// dw[c][i] = sum_s partial[c][s][i].  A block of 8 warps covers 32 * 8/G
// consecutive columns; the G warps of a column group split the s range
// (warp g takes s = g, g+G, ...) and their sums are added in warp order, so
// the order depends on `splits` only.
template <int G>
__global__ void __launch_bounds__(256)
k_wgrad_reduce(const float* __restrict__ partial, float* __restrict__ dw, int64_t dw_rs,
               int splits, int64_t per) {
  __shared__ float red[8][32];
  const int c = blockIdx.y;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int grp = w / G, sub = w % G;
  const int64_t i = ((int64_t)blockIdx.x * (8 / G) + grp) * 32 + lane;
  float s = 0.f;
  if (i < per) {
    const float* src = partial + (int64_t)c * splits * per + i;
    for (int k = sub; k < splits; k += G) s += src[(int64_t)k * per];
  }
  if (G == 1) {
    if (i < per) dw[(int64_t)c * dw_rs + i] = s;
    return;
  }
  red[w][lane] = s;
  __syncthreads();
  if (sub == 0 && i < per) {
    float t = red[w][lane];
#pragma unroll
    for (int q = 1; q < G; ++q) t += red[w + q][lane];
    dw[(int64_t)c * dw_rs + i] = t;
  }
}

// SMs of the current device (persistent grids use one CTA per SM)
int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
  }
  return n;
}

template <int BN, int BKC, int EPI, int BMN>
cudaError_t launch_conv_inst(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                             const ConvTcArgs& p, int tiles_m, int tiles_n, int items) {
  using Cfg = ConvCfg<BN, BKC, EPI>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv_tc<BN, BKC, EPI, BMN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int cap = sm_count() * Cfg::CTAS;
  const int grid = items < cap ? items : cap;
  k_conv_tc<BN, BKC, EPI, BMN><<<grid, kThreads, Cfg::SMEM, s>>>(a, b, p, tiles_m, tiles_n,
                                                                  items);
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
  const int tiles_m = p.tiles_w * p.tiles_h * ((p.B + p.bb - 1) / p.bb);
  const int tiles_n = p.n_total / bn;
  const int items = tiles_m * tiles_n * C;
  // fprop epilogues read a K-major B; the data gradient (EPI_STORE) reads
  // the same weights MN-major
#define GCPSL_CONV_CASE(BN_, BKC_, EPI_, BMN_)             \
  if (bn == BN_ && bkc == BKC_ && epi == EPI_)             \
    return launch_conv_inst<BN_, BKC_, EPI_, BMN_>(s, a, b, p, tiles_m, tiles_n, items);
#define GCPSL_CONV_EPIS(BN_, BKC_)          \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_POOL, 0)   \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_RELU, 0)   \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_STORE, 1)
  GCPSL_CONV_EPIS(32, 64)
  GCPSL_CONV_EPIS(64, 32)
  GCPSL_CONV_EPIS(64, 64)
  GCPSL_CONV_EPIS(128, 32)
  GCPSL_CONV_EPIS(128, 64)
  GCPSL_CONV_CASE(256, 64, EPI_RELU, 0)     // no staging tile for 256 channels
  GCPSL_CONV_CASE(256, 64, EPI_STORE, 1)
#undef GCPSL_CONV_EPIS
#undef GCPSL_CONV_CASE
  return cudaErrorInvalidValue;
}

template <int BN, int EPI>
static cudaError_t launch_conv0_inst(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                                     const ConvTcArgs& p, int tiles_m, int items) {
  using Cfg = Conv0Cfg<BN, EPI>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv0_tc<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int cap = sm_count() * Cfg::CTAS;
  const int grid = items < cap ? items : cap;
  k_conv0_tc<BN, EPI><<<grid, kThreads, Cfg::SMEM, s>>>(a, b, p, tiles_m, items);
  return cudaGetLastError();
}

cudaError_t launch_conv0_tc(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                            const ConvTcArgs& p, int epi, int C) {
  const int tiles_m = p.tiles_w * p.tiles_h * ((p.B + p.bb - 1) / p.bb);
  const int items = tiles_m * C;
  const int bn = p.n_total;
#define GCPSL_CONV0_CASE(BN_, EPI_) \
  if (bn == BN_ && epi == EPI_) return launch_conv0_inst<BN_, EPI_>(s, a, b, p, tiles_m, items);
  GCPSL_CONV0_CASE(16, EPI_POOL)
  GCPSL_CONV0_CASE(16, EPI_RELU)
  GCPSL_CONV0_CASE(32, EPI_POOL)
  GCPSL_CONV0_CASE(32, EPI_RELU)
  GCPSL_CONV0_CASE(64, EPI_POOL)
  GCPSL_CONV0_CASE(64, EPI_RELU)
#undef GCPSL_CONV0_CASE
  return cudaErrorInvalidValue;
}

cudaError_t launch_pack_w0(cudaStream_t s, const bf16* w, bf16* w0p, int64_t rs, int cout,
                           int cin, int C) {
  const int per = 10 * cout * 8;
  k_pack_w0<<<dim3((unsigned)((per + 255) / 256), C), 256, 0, s>>>(w, w0p, rs, cout, cin);
  return cudaGetLastError();
}

cudaError_t launch_wgrad_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                            const WgradTcArgs& p, int bn, int C) {
  const int tg = 256 / bn;                            // slots per CTA
  const int groups = 1 + (9 - (tg - 1) + tg - 1) / tg;
  const int tiles = groups * (p.cin / bn) * ((p.cout + 127) / 128);
  dim3 grid(p.splits, tiles, C);
  if (bn == 32) return launch_wgrad_inst<32>(s, g, x, p, grid);
  if (bn == 64) return launch_wgrad_inst<64>(s, g, x, p, grid);
  if (bn == 128) return launch_wgrad_inst<128>(s, g, x, p, grid);
  return cudaErrorInvalidValue;
}

cudaError_t launch_wgrad0_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                             const WgradTcArgs& p, int C) {
#define GCPSL_WG0(CO)                                                                        \
  if (p.cout == CO) {                                                                        \
    static bool attr = false;                                                                \
    if (!attr) {                                                                             \
      cudaError_t e = cudaFuncSetAttribute(k_wgrad0_tc<CO>,                                  \
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,      \
                                           Wg0Cfg<CO>::SMEM);                                \
      if (e != cudaSuccess) return e;                                                        \
      attr = true;                                                                           \
    }                                                                                        \
    k_wgrad0_tc<CO><<<dim3(p.splits, 1, C), kThreads, Wg0Cfg<CO>::SMEM, s>>>(g, x, p);       \
    return cudaGetLastError();                                                               \
  }
  GCPSL_WG0(32)
  GCPSL_WG0(64)
#undef GCPSL_WG0
  return cudaErrorInvalidValue;
}

cudaError_t launch_wgrad_reduce(cudaStream_t s, const float* partial, float* dw, int64_t dw_rs,
                                int splits, int64_t per, int C) {
  const int G = splits <= 2 ? 1 : splits <= 8 ? 2 : splits <= 32 ? 4 : 8;
  const int64_t cols_per_block = 32 * (8 / G);
  const dim3 grid((unsigned)((per + cols_per_block - 1) / cols_per_block), C);
  if (G == 1) k_wgrad_reduce<1><<<grid, 256, 0, s>>>(partial, dw, dw_rs, splits, per);
  else if (G == 2) k_wgrad_reduce<2><<<grid, 256, 0, s>>>(partial, dw, dw_rs, splits, per);
  else if (G == 4) k_wgrad_reduce<4><<<grid, 256, 0, s>>>(partial, dw, dw_rs, splits, per);
  else k_wgrad_reduce<8><<<grid, 256, 0, s>>>(partial, dw, dw_rs, splits, per);
  return cudaGetLastError();
}


}  // namespace gcpsl
