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
//      the epilogue stores dx, or routes it through the previous layer's
//      max-pool / ReLU backward into that layer's g.
//    The input layer runs through it with one tap over its im2col (K = 32).
//  k_wgrad_tc: dW[co][tap][ci] = sum_p g[p][co] x[p + shift(tap)][ci]
//    M = co, N = ci, K = pixels.  Both operands are MN-major tiles (pixels are
//    rows, channels contiguous), loaded as 64-pixel boxes.  Persistent: a
//    CTA works through a contiguous range of (replica, tile, pixel split)
//    items; a single split writes the gradient, several write fp32 partials
//    that k_wgrad_reduce sums in split order (deterministic).
//  k_wgrad_halo: the same for 3x3 stride-1 layers from one halo box of x per
//    K block.
//  k_conv_halo: 3x3 stride-1 fprop / dgrad from one halo box per K block,
//    weights resident in shared memory.
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

// Epilogue scratch of the pooling epilogue: per epilogue warp a 32 x 16
// fp32 tile, rows padded to 20 words (16-byte accesses conflict-free)
constexpr int kXsRow = 20;
constexpr int kEpiScratch = 4 * 32 * kXsRow * 4;
__host__ __device__ constexpr int epi_scratch(int epi) { return epi == EPI_POOL ? kEpiScratch : 0; }

// wait for this thread's outstanding TMEM loads; the values pass through
// the asm so that no use of them can be scheduled before the wait
__device__ __forceinline__ void tmem_wait_regs(float (&v)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+f"(v[0]), "+f"(v[1]), "+f"(v[2]), "+f"(v[3]), "+f"(v[4]), "+f"(v[5]),
                 "+f"(v[6]), "+f"(v[7]), "+f"(v[8]), "+f"(v[9]), "+f"(v[10]), "+f"(v[11]),
                 "+f"(v[12]), "+f"(v[13]), "+f"(v[14]), "+f"(v[15])
               :
               : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Epilogue of a 128-pixel x BN-channel accumulator tile, run by the four
// epilogue warps; the thread of TMEM row r owns pixel (bb, hh, ww) of the
// tile (r = (bb*hb + hh)*bw + ww; tiles are bw <= 16 pixels wide and an even
// number of rows high, so a warp holds whole 2x2 windows).  TMEM is read 16
// columns at a time, the next load in flight while a chunk is processed.
//  EPI_POOL : + bias, 2x2 max-pool decided on the fp32 values (the larger
//             value wins, ties go to the earlier position in row-major
//             order, i.e. the first maximum), bf16 relu(max) and the code
//             (position | positive << 2).  The warp transposes each chunk
//             through shared memory so that the window's four threads each
//             decide 4 of the 16 channels from all four positions.
//  EPI_RELU : + bias, relu, bf16 store.
//  EPI_STORE / EPI_DSTORE: bf16 store (bias-free forward / data gradient).
//  EPI_DPOOL: data gradient routed through the previous layer's max-pool:
//             the four pixels of the previous layer's 2x2 window get the
//             bf16 gradient where the code names that position and the
//             maximum was positive, else 0 (out, if set, also gets the
//             gradient itself: the cut).
//  EPI_DRELU: data gradient times the previous layer's ReLU mask (act > 0),
//             written to gout (and to out if set).
//  EPI_ADD  : bf16(acc + res) (a data gradient plus the residual path's).
//  Outside EPI_POOL the output pixel is mapped by (osy, ooy, osx, oox).
template <int BN, int EPI>
__device__ __forceinline__ void conv_epilogue_drain(uint32_t trow, int r, int n0, int b0, int h0,
                                                    int w0, int c, const ConvTcArgs& p,
                                                    float* xs) {
  const int W = p.W, H = p.H, bw = p.bw;
  const int lane = r & 31;
  const int ww = r % bw, hh = (r / bw) % p.hb, bb = r / (bw * p.hb);
  const bool valid = b0 + bb < p.B;
  const int64_t img = (int64_t)c * p.B + b0 + bb;
  float v[16];
  tmem_ld16(trow, v);
  if (EPI == EPI_POOL) {
    const int pos = (hh & 1) * 2 + (ww & 1);        // my position in the window
    const int l0 = lane - (ww & 1) - (hh & 1) * bw;  // lane of position 0
    const int64_t o =
        ((img * (H / 2) + (h0 + hh) / 2) * (W / 2) + (w0 + ww) / 2) * p.n_total + n0 + 4 * pos;
    const float* bias = p.bias + (int64_t)c * p.bias_rs + n0 + 4 * pos;
    float4* mine = reinterpret_cast<float4*>(xs + lane * kXsRow);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float b4[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) b4[i] = bias[c0 + i];
      tmem_wait_regs(v);
#pragma unroll
      for (int j = 0; j < 4; ++j) mine[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
      __syncwarp();
      if (c0 + 16 < BN) tmem_ld16(trow + c0 + 16, v);
      float4 wq[4];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        wq[q] = *reinterpret_cast<const float4*>(xs + (l0 + (q & 1) + (q >> 1) * bw) * kXsRow +
                                                 4 * pos);
      __syncwarp();
      float best[4] = {wq[0].x + b4[0], wq[0].y + b4[1], wq[0].z + b4[2], wq[0].w + b4[3]};
      int at[4] = {0, 0, 0, 0};
#pragma unroll
      for (int q = 1; q < 4; ++q) {
        const float x4[4] = {wq[q].x + b4[0], wq[q].y + b4[1], wq[q].z + b4[2], wq[q].w + b4[3]};
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (x4[i] > best[i]) { best[i] = x4[i]; at[i] = q; }
      }
      uint32_t code = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) code |= (uint32_t)(at[i] | (best[i] > 0.f ? 4 : 0)) << (8 * i);
      if (valid) {
        uint2 hv;
        float rl[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) rl[i] = best[i] > 0.f ? best[i] : 0.f;
        hv.x = pack_bf16x2(rl[0], rl[1]);
        hv.y = pack_bf16x2(rl[2], rl[3]);
        *reinterpret_cast<uint2*>(p.out + o + c0) = hv;
        *reinterpret_cast<uint32_t*>(p.code + o + c0) = code;
      }
    }
    return;
  }
  const int oH = p.out_H ? p.out_H : H, oW = p.out_W ? p.out_W : W;
  const int64_t o = ((img * oH + (h0 + hh) * p.osy + p.ooy) * oW + (w0 + ww) * p.osx + p.oox) *
                        p.n_total + n0;
  const float* bias = EPI == EPI_RELU ? p.bias + (int64_t)c * p.bias_rs + n0 : nullptr;
#pragma unroll 1
  for (int c0 = 0; c0 < BN; c0 += 16) {
    float b16[16];
    if (EPI == EPI_RELU) {
#pragma unroll
      for (int i = 0; i < 16; i += 4) {
        const float4 t = *reinterpret_cast<const float4*>(bias + c0 + i);
        b16[i] = t.x; b16[i + 1] = t.y; b16[i + 2] = t.z; b16[i + 3] = t.w;
      }
    }
    uint4 cd;
    uint4 am[2];
    if (EPI == EPI_DPOOL && valid) cd = *reinterpret_cast<const uint4*>(p.code + o + c0);
    if (EPI == EPI_ADD && valid) {
      am[0] = *reinterpret_cast<const uint4*>(p.res + o + c0);
      am[1] = *reinterpret_cast<const uint4*>(p.res + o + c0 + 8);
    }
    if (EPI == EPI_DRELU && valid) {
      am[0] = *reinterpret_cast<const uint4*>(p.act + o + c0);
      am[1] = *reinterpret_cast<const uint4*>(p.act + o + c0 + 8);
    }
    tmem_wait_regs(v);
    uint32_t hw[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float x0 = v[2 * i], x1 = v[2 * i + 1];
      if (EPI == EPI_RELU) {
        x0 += b16[2 * i];
        x1 += b16[2 * i + 1];
        x0 = x0 > 0.f ? x0 : 0.f;
        x1 = x1 > 0.f ? x1 : 0.f;
      }
      if (EPI == EPI_ADD) {
        const uint32_t r = (&am[0].x)[i];
        x0 += __uint_as_float(r << 16);
        x1 += __uint_as_float(r & 0xffff0000u);
      }
      hw[i] = pack_bf16x2(x0, x1);
    }
    if (c0 + 16 < BN) tmem_ld16(trow + c0 + 16, v);
    if (!valid) continue;
    if (EPI != EPI_DPOOL && EPI != EPI_DRELU) {
      uint4* dst = reinterpret_cast<uint4*>(p.out + o + c0);
      dst[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
      dst[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
      continue;
    }
    if (p.out) {
      uint4* dst = reinterpret_cast<uint4*>(p.out + o + c0);
      dst[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
      dst[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
    }
    if (EPI == EPI_DRELU) {
      // act > 0 <=> its bf16 bits are > 0 as a signed 16-bit integer
      const uint32_t a[8] = {am[0].x, am[0].y, am[0].z, am[0].w, am[1].x, am[1].y, am[1].z, am[1].w};
      uint32_t gw[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) gw[i] = hw[i] & __vcmpgts2(a[i], 0u);
      uint4* dst = reinterpret_cast<uint4*>(p.gout + o + c0);
      dst[0] = make_uint4(gw[0], gw[1], gw[2], gw[3]);
      dst[1] = make_uint4(gw[4], gw[5], gw[6], gw[7]);
    } else {
      // byte k of the codes selects the window position that gets channel k
      const uint32_t cw[4] = {cd.x & 0x07070707u, cd.y & 0x07070707u, cd.z & 0x07070707u,
                              cd.w & 0x07070707u};
      const int y = h0 + hh, x = w0 + ww;
#pragma unroll
      for (int qd = 0; qd < 4; ++qd) {
        const uint32_t want = (uint32_t)(4 | qd) * 0x01010101u;
        uint32_t gw[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t m = __vcmpeq4(cw[j], want);           // 0xff per selected channel
          gw[2 * j] = hw[2 * j] & __byte_perm(m, 0, 0x1100);
          gw[2 * j + 1] = hw[2 * j + 1] & __byte_perm(m, 0, 0x3322);
        }
        const int64_t go =
            ((img * (2 * H) + 2 * y + (qd >> 1)) * (2 * W) + 2 * x + (qd & 1)) * p.n_total + n0 + c0;
        uint4* dst = reinterpret_cast<uint4*>(p.gout + go);
        dst[0] = make_uint4(gw[0], gw[1], gw[2], gw[3]);
        dst[1] = make_uint4(gw[4], gw[5], gw[6], gw[7]);
      }
    }
  }
}

// 32 lanes x 32 consecutive columns, waited for in one go (the values pass
// through the wait so that no use is scheduled before it)
__device__ __forceinline__ void tmem_ld32_wait(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Epilogue of the non-pooling kinds over NC columns (a multiple of 16), in
// groups of G = min(32, NC) columns: the operands the epilogue reads (res,
// act, codes) of the first group are loaded before the accumulator is
// waited for, and those of the next group while the current one is
// processed; each group's TMEM columns come in one load and one wait.
// Results are those of conv_epilogue_drain.  Returns false if the wait for
// the accumulator gave up.
template <int NC, int EPI>
__device__ __forceinline__ bool conv_epilogue_stream(uint64_t* tfull, uint32_t parity,
                                                     uint32_t trow, int r, int n0, int b0, int h0,
                                                     int w0, int c, const ConvTcArgs& p) {
  static_assert(EPI != EPI_POOL, "pooling epilogue: conv_epilogue_drain");
  constexpr int G = NC < 32 ? NC : 32;
  constexpr int NA = G / 8;                        // uint4 of bf16 aux per group
  const int W = p.W, H = p.H, bw = p.bw;
  const int ww = r % bw, hh = (r / bw) % p.hb, bb = r / (bw * p.hb);
  const bool valid = b0 + bb < p.B;
  const int64_t img = (int64_t)c * p.B + b0 + bb;
  const int oH = p.out_H ? p.out_H : H, oW = p.out_W ? p.out_W : W;
  const int64_t o = ((img * oH + (h0 + hh) * p.osy + p.ooy) * oW + (w0 + ww) * p.osx + p.oox) *
                        p.n_total + n0;
  const float* bias = EPI == EPI_RELU ? p.bias + (int64_t)c * p.bias_rs + n0 : nullptr;
  const bf16* aux_src = EPI == EPI_ADD ? p.res : EPI == EPI_DRELU ? p.act : nullptr;
  uint4 aux[NA];
  uint4 cd[(G + 15) / 16];
  auto load_aux = [&](int g0) {
    if (!valid) return;
    if (aux_src) {
#pragma unroll
      for (int i = 0; i < NA; ++i) aux[i] = *reinterpret_cast<const uint4*>(aux_src + o + g0 + 8 * i);
    }
    if (EPI == EPI_DPOOL) {
#pragma unroll
      for (int i = 0; i < (G + 15) / 16; ++i)
        cd[i] = *reinterpret_cast<const uint4*>(p.code + o + g0 + 16 * i);
    }
  };
  load_aux(0);
  if (!__all_sync(0xffffffffu, mbar_wait(tfull, parity))) return false;
  tc_fence_after();
#pragma unroll 1
  for (int g0 = 0; g0 < NC; g0 += G) {
    float v[32];
    if (G == 32) {
      tmem_ld32_wait(trow + g0, v);
    } else {
      float h[16];
      tmem_ld16(trow + g0, h);
      tmem_wait_regs(h);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = h[i];
    }
    uint4 am[NA];
    uint4 cw[(G + 15) / 16];
#pragma unroll
    for (int i = 0; i < NA; ++i) am[i] = aux[i];
#pragma unroll
    for (int i = 0; i < (G + 15) / 16; ++i) cw[i] = cd[i];
    if (g0 + G < NC) load_aux(g0 + G);
    if (!valid) continue;
    uint32_t hw[G / 2];
#pragma unroll
    for (int i = 0; i < G / 2; ++i) {
      float x0 = v[2 * i], x1 = v[2 * i + 1];
      if (EPI == EPI_RELU) {
        x0 += bias[g0 + 2 * i];
        x1 += bias[g0 + 2 * i + 1];
        x0 = x0 > 0.f ? x0 : 0.f;
        x1 = x1 > 0.f ? x1 : 0.f;
      }
      if (EPI == EPI_ADD) {
        const uint32_t rr = (&am[0].x)[i];
        x0 += __uint_as_float(rr << 16);
        x1 += __uint_as_float(rr & 0xffff0000u);
      }
      hw[i] = pack_bf16x2(x0, x1);
    }
    if (EPI != EPI_DPOOL && EPI != EPI_DRELU) {
      uint4* dst = reinterpret_cast<uint4*>(p.out + o + g0);
#pragma unroll
      for (int i = 0; i < G / 8; ++i)
        dst[i] = make_uint4(hw[4 * i], hw[4 * i + 1], hw[4 * i + 2], hw[4 * i + 3]);
      continue;
    }
    if (p.out) {
      uint4* dst = reinterpret_cast<uint4*>(p.out + o + g0);
#pragma unroll
      for (int i = 0; i < G / 8; ++i)
        dst[i] = make_uint4(hw[4 * i], hw[4 * i + 1], hw[4 * i + 2], hw[4 * i + 3]);
    }
    if (EPI == EPI_DRELU) {
      // act > 0 <=> its bf16 bits are > 0 as a signed 16-bit integer
      uint32_t gw[G / 2];
#pragma unroll
      for (int i = 0; i < G / 2; ++i) gw[i] = hw[i] & __vcmpgts2((&am[0].x)[i], 0u);
      uint4* dst = reinterpret_cast<uint4*>(p.gout + o + g0);
#pragma unroll
      for (int i = 0; i < G / 8; ++i)
        dst[i] = make_uint4(gw[4 * i], gw[4 * i + 1], gw[4 * i + 2], gw[4 * i + 3]);
    } else {
      // byte k of the codes selects the window position that gets channel k
      const int y = h0 + hh, x = w0 + ww;
#pragma unroll
      for (int qd = 0; qd < 4; ++qd) {
        const uint32_t want = (uint32_t)(4 | qd) * 0x01010101u;
        uint32_t gw[G / 2];
#pragma unroll
        for (int j = 0; j < G / 4; ++j) {
          const uint32_t m = __vcmpeq4((&cw[0].x)[j] & 0x07070707u, want);
          gw[2 * j] = hw[2 * j] & __byte_perm(m, 0, 0x1100);
          gw[2 * j + 1] = hw[2 * j + 1] & __byte_perm(m, 0, 0x3322);
        }
        const int64_t go =
            ((img * (2 * H) + 2 * y + (qd >> 1)) * (2 * W) + 2 * x + (qd & 1)) * p.n_total + n0 + g0;
        uint4* dst = reinterpret_cast<uint4*>(p.gout + go);
#pragma unroll
        for (int i = 0; i < G / 8; ++i)
          dst[i] = make_uint4(gw[4 * i], gw[4 * i + 1], gw[4 * i + 2], gw[4 * i + 3]);
      }
    }
  }
  return true;
}

template <int BN, int BKC, int EPI>
struct ConvCfg {
  static constexpr int A_BYTES = BM * BKC * 2;
  static constexpr int B_BYTES = BN * BKC * 2;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  // two CTAs per SM when both fit in TMEM (2 x 2 x TCOLS <= 512 columns)
  static constexpr int CTAS = 2 * TCOLS <= 256 ? 2 : 1;
  static constexpr int XS = epi_scratch(EPI);
  static constexpr int BUDGET = (CTAS == 2 ? 100 * 1024 : 200 * 1024) - XS;
  static constexpr int S0 = BUDGET / STAGE;
  static constexpr int S = S0 > 8 ? 8 : (S0 < 2 ? 2 : S0);
  static constexpr int PIPE = S * STAGE;
  static constexpr int SMEM = 1024 + PIPE + XS;
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
          const __grid_constant__ CUtensorMap tA2, const __grid_constant__ CUtensorMap tB2,
          const ConvTcArgs p, int tiles_m, int tiles_n, int items) {
  using Cfg = ConvCfg<BN, BKC, EPI>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  __shared__ uint64_t full[S], empty[S], tfull[2], tempty[2];
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kper = p.kch / BKC;
  const int KB = p.ntaps * kper;
  bool two = false;                              // a second operand pair in the tap list
  for (int t = 0; t < p.ntaps; ++t) two |= p.tsrc[t] != 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&tfull[b], 1); mbar_init(&tempty[b], 128); }
    fence_mbar_init();
    tma_prefetch_desc(&tA);
    tma_prefetch_desc(&tB);
    if (two) { tma_prefetch_desc(&tA2); tma_prefetch_desc(&tB2); }
  }
  if (warp == 1) { tmem_alloc(&tbase, 2 * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  pdl_wait();
  pdl_trigger();

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
          const CUtensorMap* ma = p.tsrc[tap] ? &tA2 : &tA;
          const CUtensorMap* mb = p.tsrc[tap] ? &tB2 : &tB;
          mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
          tma_load_5d(sa, ma, &full[s], ch, w0 * p.stride + p.tdx[tap],
                      h0 * p.stride + p.tdy[tap], b0, c);
          if (!BMN) {
            tma_load_4d(sa + Cfg::A_BYTES, mb, &full[s], ch, p.tw[tap], n0, c);
          } else {
            constexpr int NBW = BN < 64 ? BN : 64;           // N block width
#pragma unroll
            for (int j = 0; j < BN / NBW; ++j)
              tma_load_4d(sa + Cfg::A_BYTES + j * NBW * BKC * 2, mb, &full[s], n0 + j * NBW,
                          p.tw[tap], ch, c);
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
      const int c = t / (tiles_m * tiles_n), rr = t % (tiles_m * tiles_n);
      const int mt = rr / tiles_n, n0 = (rr % tiles_n) * BN;
      int b0, h0, w0;
      tile_origin(mt, p, b0, h0, w0);
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16);
      if (EPI == EPI_POOL) {
        // warp-uniform decision: the epilogue shuffles need the whole warp
        if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl >> 1) & 1))) {
          if (lane == 0) atomicOr(p.err, 4);
          break;
        }
        tc_fence_after();
        conv_epilogue_drain<BN, EPI>(trow, r, n0, b0, h0, w0, c, p,
                                     reinterpret_cast<float*>(sm + Cfg::PIPE) + q * 32 * kXsRow);
      } else if (!conv_epilogue_stream<BN, EPI == EPI_POOL ? EPI_STORE : EPI>(
                     &tfull[buf], (tl >> 1) & 1, trow, r, n0, b0, h0, w0, c, p)) {
        if (lane == 0) atomicOr(p.err, 4);
        break;
      }
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * Cfg::TCOLS);
}

// ---------------------------------------------------------------------------
// Halo-tiled 3x3 stride-1 convolution (forward or data gradient) with the
// weights resident in shared memory.
//
// An M tile is 8 columns x 16 rows of one image.  Per K block of BKC channels
// the TMA warp loads ONE box of (8+2) x (16+2) pixels around it (zero fill
// outside the image is the padding), and the nine taps read it in place: the
// tap with shift (sy, sx) is the K-major operand that starts (sy+1)*10 +
// (sx+1) pixel rows into the box, its 16 groups of 8 pixels 10 rows apart.
// (The operand swizzle is a function of the shared-memory address, so a
// start that is not aligned to the swizzle repeat reads the TMA-written
// rows correctly.)  The weights of the current (replica, N tile) -- 9 taps x
// K blocks, loaded once -- stay in shared memory while the CTA works through
// a contiguous range of items (replica, N tile, M tile; M fastest), and are
// reloaded only when the replica or N tile changes.  Accumulators, epilogue
// and TMEM double buffering as in k_conv_tc.
// ---------------------------------------------------------------------------
constexpr int kHaloW = 10, kHaloH = 18, kHaloMaxStages = 8;
// warps: 0 TMA, 1 MMA, 2..9 epilogue (two per TMEM lane quarter, each
// draining half of the N columns)
constexpr int kHaloThreads = 320, kHaloEpiThreads = 256;
template <int BN, int BKC, int EPI>
struct HaloCfg {
  static constexpr int ROWB = BKC * 2;                        // bytes per pixel row
  static constexpr int A_RAW = kHaloW * kHaloH * ROWB;        // bytes of one halo box
  static constexpr int A_BYTES = (A_RAW + 1023) / 1024 * 1024;
  static constexpr int B_TILE = BN * BKC * 2;                 // one (tap, K block) weight tile
  static constexpr uint32_t TCOLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  static constexpr int XS = 2 * epi_scratch(EPI);            // eight epilogue warps
  // dynamic shared memory at most: the opt-in maximum per CTA (227 KB) less
  // 1 KB for the static barriers
  static constexpr int SMEM_MAX = 232448 - 1024;
};
__host__ __device__ inline int halo_item_begin(int cta, int ctas, int items) {
  return (int)((int64_t)items * cta / ctas);
}

template <int BN, int BKC, int EPI, int BMN>
__global__ void __launch_bounds__(kHaloThreads, 1)
k_conv_halo(const __grid_constant__ CUtensorMap tA, const __grid_constant__ CUtensorMap tB,
            const ConvTcArgs p, int tiles_m, int tiles_n, int items, int S) {
  using Cfg = HaloCfg<BN, BKC, EPI>;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  const int kper = p.kch / BKC;
  uint8_t* sB = sm;                                           // 9 * kper weight tiles
  uint8_t* sA = sm + 9 * kper * Cfg::B_TILE;                  // S halo stages
  float* xs = reinterpret_cast<float*>(sA + S * Cfg::A_BYTES);
  __shared__ uint64_t full[kHaloMaxStages], empty[kHaloMaxStages], tfull[2], tempty[2];
  __shared__ uint64_t wfull, wempty;
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t_begin = halo_item_begin(blockIdx.x, gridDim.x, items);
  const int t_end = halo_item_begin(blockIdx.x + 1, gridDim.x, items);
  const int per_c = tiles_m * tiles_n;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kHaloEpiThreads);
    }
    mbar_init(&wfull, 1);
    mbar_init(&wempty, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tA);
    tma_prefetch_desc(&tB);
  }
  if (warp == 1) { tmem_alloc(&tbase, 2 * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (elect_one()) {
      int it = 0, wl = 0, prev = -1;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t) {
        const int c = t / per_c, r = t % per_c;
        const int nt = r / tiles_m, mt = r % tiles_m;
        const int key = c * tiles_n + nt, n0 = nt * BN;
        if (key != prev) {
          // new (replica, N tile): its weights, once the MMAs on the old ones are done
          if (wl > 0 && !mbar_wait(&wempty, (wl - 1) & 1)) { atomicOr(p.err, 1); break; }
          mbar_arrive_expect_tx(&wfull, 9 * kper * Cfg::B_TILE);
          for (int tap = 0; tap < 9; ++tap)
            for (int kb = 0; kb < kper; ++kb) {
              uint8_t* dst = sB + (tap * kper + kb) * Cfg::B_TILE;
              if (!BMN) {
                tma_load_4d(dst, &tB, &wfull, kb * BKC, p.tw[tap], n0, c);
              } else {
                constexpr int NBW = BN < 64 ? BN : 64;
#pragma unroll
                for (int j = 0; j < BN / NBW; ++j)
                  tma_load_4d(dst + j * NBW * BKC * 2, &tB, &wfull, n0 + j * NBW, p.tw[tap],
                              kb * BKC, c);
              }
            }
          ++wl;
          prev = key;
        }
        int b0, h0, w0;
        tile_origin(mt, p, b0, h0, w0);
        for (int kb = 0; kb < kper; ++kb, ++it) {
          const int s = it % S;
          if (it >= S && !mbar_wait(&empty[s], ((it / S) & 1) ^ 1)) {
            atomicOr(p.err, 1);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], Cfg::A_RAW);
          tma_load_5d(sA + s * Cfg::A_BYTES, &tA, &full[s], kb * BKC, w0 - 1, h0 - 1, b0, c);
        }
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, 0, BMN);
      constexpr uint32_t swz = BKC == 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t a_sbo = kHaloW * Cfg::ROWB;           // 8-pixel groups one row apart
      constexpr int NBW = BN < 64 ? BN : 64;
      constexpr uint32_t b_row = NBW * 2;
      constexpr uint32_t b_swz = NBW == 64 ? SWZ_128 : SWZ_64;
      // descriptors are built once; an operand at byte offset o from its base
      // is the base descriptor plus o >> 4 (the start-address field)
      uint32_t aoff[9];
#pragma unroll
      for (int tap = 0; tap < 9; ++tap)
        aoff[tap] = (uint32_t)(((p.tdy[tap] + 1) * kHaloW + p.tdx[tap] + 1) * Cfg::ROWB) >> 4;
      const uint64_t a_desc0 = smem_desc(smem_u32(sA), 16, a_sbo, swz);
      const uint64_t b_desc0 = BMN ? smem_desc(smem_u32(sB), NBW * BKC * 2, 8 * b_row, b_swz)
                                   : smem_desc(smem_u32(sB), 16, BKC * 2 * 8, swz);
      constexpr uint32_t b_kstep = (BMN ? 16 * b_row : 32) >> 4;   // per K = 16 step
      const uint32_t b_tapstep = (uint32_t)(kper * Cfg::B_TILE) >> 4;
      int it = 0, tl = 0, wl = 0, prev = -1;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t, ++tl) {
        const int c = t / per_c, nt = (t % per_c) / tiles_m;
        const int key = c * tiles_n + nt;
        if (key != prev) {
          if (!mbar_wait(&wfull, wl & 1)) { atomicOr(p.err, 2); break; }
          ++wl;
          prev = key;
        }
        const int buf = tl & 1;
        if (tl >= 2 && !mbar_wait(&tempty[buf], ((tl >> 1) & 1) ^ 1)) {
          atomicOr(p.err, 2);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * Cfg::TCOLS;
        for (int kb = 0; kb < kper; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (it / S) & 1)) {
            atomicOr(p.err, 2);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = a_desc0 + (uint32_t)((s * Cfg::A_BYTES) >> 4);
          const uint64_t db = b_desc0 + (uint32_t)((kb * Cfg::B_TILE) >> 4);
#pragma unroll
          for (int tap = 0; tap < 9; ++tap) {
#pragma unroll
            for (int k = 0; k < BKC / 16; ++k)
              mma_f16(d, da + aoff[tap] + 2 * k, db + tap * b_tapstep + k * b_kstep, idesc,
                      (kb | tap | k) != 0);
          }
          mma_commit(&empty[s]);
        }
        mma_commit(&tfull[buf]);
        // the last item on these weights: release them to the TMA warp
        const int nx = t + 1;
        const int nkey = nx < t_end ? (nx / per_c) * tiles_n + (nx % per_c) / tiles_m : -1;
        if (nkey != key) mma_commit(&wempty);
      }
    }
  } else {
    // ---------------- epilogue: warps 2..9 ----------------
    const int q = warp & 3;                      // TMEM lane quarter
    const int half = (warp - 2) >> 2;            // columns [half * BN/2, (half + 1) * BN/2)
    const int r = q * 32 + lane;
    constexpr int NH = BN / 2;
    int tl = 0;
    for (int t = t_begin; t < t_end; ++t, ++tl) {
      const int buf = tl & 1;
      const int c = t / per_c, rr = t % per_c;
      const int n0 = (rr / tiles_m) * BN, mt = rr % tiles_m;
      int b0, h0, w0;
      tile_origin(mt, p, b0, h0, w0);
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16) + half * NH;
      if (EPI == EPI_POOL) {
        if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl >> 1) & 1))) {
          if (lane == 0) atomicOr(p.err, 4);
          break;
        }
        tc_fence_after();
        conv_epilogue_drain<NH, EPI>(trow, r, n0 + half * NH, b0, h0, w0, c, p,
                                     xs + (warp - 2) * 32 * kXsRow);
      } else if (!conv_epilogue_stream<NH, EPI == EPI_POOL ? EPI_STORE : EPI>(
                     &tfull[buf], (tl >> 1) & 1, trow, r, n0 + half * NH, b0, h0, w0, c, p)) {
        if (lane == 0) atomicOr(p.err, 4);
        break;
      }
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * Cfg::TCOLS);
}

// ---------------------------------------------------------------------------
// input layer (3 channels): with bf16 operands the gather writes its im2col,
// x0[p][k] with k = tap * 3 + ch (27 columns), a ones column (k = 27) and
// zero padding to 32; the forward is then k_conv_tc with one tap and K = 32
// against weights packed as w0p[c][co][32].
// ---------------------------------------------------------------------------
// packed input-layer weights: w0p[c][co][k] = W[co][tap][ci] at k = tap * 3 + ci
// (k < 27), else 0
__global__ void k_pack_w0(const bf16* __restrict__ w, bf16* __restrict__ w0p, int64_t rs,
                          int cout) {
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y;
  const int per = cout * 32;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < per; i += gridDim.x * blockDim.x) {
    const int k = i % 32, co = i / 32;
    w0p[(int64_t)c * per + i] =
        k < 27 ? w[(int64_t)c * rs + (int64_t)co * 27 + k] : __float2bfloat16_rn(0.f);
  }
}

// ---------------------------------------------------------------------------
// weight gradient (persistent)
// ---------------------------------------------------------------------------
// A work item is (replica, tile, split): one tile of dW over one K range (a
// split of the output pixels).  CTA b of G takes the contiguous item range
// [b items / G, (b+1) items / G) (splits fastest).  The TMA warp runs
// through an S-stage ring across items; the MMA warp alternates between
// NBUF TMEM accumulators, so one item's epilogue overlaps the next item's
// MMAs.  An item's fp32 result goes to the gradient itself (one split) or
// to its split's partial, laid out like the parameters ([cout][taps][cin]
// then [cout]), summed in split order by k_wgrad_reduce.  The bias gradient
// sum_p g[p][co] is one extra N = 32 MMA per K step against a block of
// ones, in the items of the last tap group with ci0 = 0.  MT = 128 output
// channels per tile (two 64-wide g blocks), or MT = 64 for layers with 64
// output channels (M = 64 MMAs: row r of the accumulator is TMEM lane
// 32 * (r / 16) + r % 16).
constexpr int kOnesBytes = 16 * 64;            // 16 K rows x 32 ones (64-byte rows)

struct WgItem {
  int c, tile, split, kb0, nkb;
};
__device__ __forceinline__ WgItem wg_item(int t, int tiles, const WgradTcArgs& p) {
  WgItem it;
  it.c = t / (tiles * p.splits);
  const int r = t % (tiles * p.splits);
  it.tile = r / p.splits;
  it.split = r % p.splits;
  it.kb0 = it.split * p.kb_per_split;
  const int kb1 = min(it.kb0 + p.kb_per_split, p.kb_total);
  it.nkb = kb1 > it.kb0 ? kb1 - it.kb0 : 0;
  return it;
}

// Drain one accumulator (rows = output channels co0 + row) to the fp32
// store of its replica and split: columns [0, ncols) in chunks of 16 that
// stay inside one (tap, channel block); dst_col(col) gives the offset of a
// column in a row ([tap][cin] order) and bias_col (if >= 0) the column that
// holds the bias.
template <int MT, typename ColFn>
__device__ __forceinline__ void wgrad_drain(uint32_t trow, int q, int lane, int co0, int ncols,
                                            int bias_col, bool zero, float* dst, int row_len,
                                            int cout, ColFn dst_col) {
  const int co = co0 + (MT == 128 ? q * 32 + lane : q * 16 + lane);
  const bool mine = (MT == 128 || lane < 16) && co < cout;
#pragma unroll 1
  for (int c0 = 0; c0 < ncols; c0 += 16) {
    float v[16];
    tmem_ld16(trow + c0, v);
    tmem_wait_regs(v);
    if (!mine) continue;
    if (c0 == bias_col) {
      dst[(int64_t)cout * row_len + co] = zero ? 0.f : v[0];
      continue;
    }
    if (bias_col >= 0 && c0 > bias_col) continue;
    float4* d4 = reinterpret_cast<float4*>(dst + (int64_t)co * row_len + dst_col(c0));
#pragma unroll
    for (int i = 0; i < 4; ++i)
      d4[i] = zero ? make_float4(0.f, 0.f, 0.f, 0.f)
                   : make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
  }
}

__device__ __forceinline__ float* wgrad_dst(const WgradTcArgs& p, const WgItem& it, int per) {
  return p.out ? p.out + (int64_t)it.c * p.out_rs
               : p.partial + ((int64_t)it.c * p.splits + it.split) * per;
}

// k_wgrad_tc: any 3x3 / 1x1 layer (stride 1 or 2).  A tile is a group of up
// to TG = 256/BN taps of a (MT-co, BN-ci) block: per K block the g tile is
// loaded once and multiplied, in one N <= 256 MMA, against the group's
// tap-shifted x tiles (consecutive MN-major N blocks).
template <int BN, int MT>
struct WgCfg {
  static constexpr int BKP = 64;                         // pixels per stage
  static constexpr int TG = 256 / BN;                    // taps per tile
  static constexpr int A_BYTES = MT * BKP * 2;           // MT co (64-wide blocks)
  static constexpr int TAP_BYTES = BN * BKP * 2;         // one tap's x tile
  static constexpr int STAGE = A_BYTES + TG * TAP_BYTES;
  static constexpr int S0 = 200 * 1024 / STAGE;
  static constexpr int S = S0 > 6 ? 6 : S0;
  static constexpr int SMEM = 1024 + S * STAGE + kOnesBytes;
  static constexpr uint32_t TCOLS = 256;                 // per accumulator; two of them
  static_assert(BN + 32 <= TCOLS, "last tap group and bias exceed the accumulator");
  // all 512 TMEM columns per CTA: one CTA per SM
  static_assert(SMEM > 116 * 1024, "a second CTA per SM would wait for TMEM");
};

template <int BN, int MT>
__global__ void __launch_bounds__(kThreads, 1)
k_wgrad_tc(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tX,
           const WgradTcArgs p, int C) {
  using Cfg = WgCfg<BN, MT>;
  constexpr int S = Cfg::S, TG = Cfg::TG;
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  uint8_t* ones = sm + S * Cfg::STAGE;
  __shared__ uint64_t full[S], empty[S], tfull[2], tempty[2];
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ci_tiles = p.cin / BN;
  const int co_tiles = (p.cout + MT - 1) / MT;
  const int groups = (p.taps + TG - 1) / TG;
  const int tiles = groups * ci_tiles * co_tiles;
  const int items = C * tiles * p.splits;
  const int t_begin = (int)((int64_t)items * blockIdx.x / gridDim.x);
  const int t_end = (int)((int64_t)items * (blockIdx.x + 1) / gridDim.x);
  const int ksz = p.taps == 9 ? 3 : 1;
  const int per = p.cout * p.taps * p.cin + (p.bias ? p.cout : 0);
  const int rows_blocks = p.H / p.hb;               // pixel blocks per image group
  // tile -> (tap group, ci0, co0); the bias rides on the last group at ci0 = 0
  auto tile_of = [&](int tile, int& g, int& ci0, int& co0) {
    ci0 = (tile % ci_tiles) * BN; tile /= ci_tiles;
    co0 = (tile % co_tiles) * MT; tile /= co_tiles;
    g = tile;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&tfull[b], 1); mbar_init(&tempty[b], 128); }
    fence_mbar_init();
    tma_prefetch_desc(&tG);
    tma_prefetch_desc(&tX);
  }
  {
    const uint4 one = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    for (int i = threadIdx.x; i < kOnesBytes / 16; i += blockDim.x)
      reinterpret_cast<uint4*>(ones)[i] = one;
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) { tmem_alloc(&tbase, 2 * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (elect_one()) {
      int it = 0;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t) {
        const WgItem w = wg_item(t, tiles, p);
        int g, ci0, co0;
        tile_of(w.tile, g, ci0, co0);
        const int tap0 = g * TG, ntaps = min(TG, p.taps - tap0);
        for (int i = 0; i < w.nkb; ++i, ++it) {
          const int s = it % S;
          if (it >= S && !mbar_wait(&empty[s], ((it / S) & 1) ^ 1)) {
            atomicOr(p.err, 8);
            ok = false;
            break;
          }
          const int kb = w.kb0 + i;
          const int b = (kb / rows_blocks) * p.bb, h = (kb % rows_blocks) * p.hb;
          uint8_t* sa = sm + s * Cfg::STAGE;
          uint8_t* sb = sa + Cfg::A_BYTES;
          mbar_arrive_expect_tx(&full[s], Cfg::A_BYTES + ntaps * Cfg::TAP_BYTES);
          tma_load_5d(sa, &tG, &full[s], co0, 0, h, b, w.c);
          // rows 64..127 of an MT = 128 tile: the next 64 channels, or (cout
          // < co0 + 128) a second copy of the first block whose results the
          // epilogue drops
          if (MT == 128)
            tma_load_5d(sa + 64 * Cfg::BKP * 2, &tG, &full[s], p.cout > co0 + 64 ? co0 + 64 : co0,
                        0, h, b, w.c);
          for (int tj = 0; tj < ntaps; ++tj) {
            const int tap = tap0 + tj, kh = tap / ksz, kw = tap % ksz;
#pragma unroll
            for (int j = 0; j < (BN + 63) / 64; ++j)
              tma_load_5d(sb + tj * Cfg::TAP_BYTES + j * 64 * Cfg::BKP * 2, &tX, &full[s],
                          ci0 + 64 * j, kw - p.pad, h * p.stride + kh - p.pad, b, w.c);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      // MN-major B: the taps' x tiles are consecutive N blocks (64-ci blocks,
      // SW128, or 32-ci blocks of 64-byte rows, SW64), `b_blk` bytes apart
      constexpr uint32_t a_lbo = 64 * Cfg::BKP * 2;
      constexpr uint32_t b_swz = BN >= 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t b_row = BN >= 64 ? 128 : 64;
      constexpr uint32_t b_blk = b_row * Cfg::BKP;
      const uint32_t idesc_b = idesc_bf16(MT, 32, 1, 1);
      const uint64_t ones_desc = smem_desc(smem_u32(ones), 64 * 16, 8 * 64, SWZ_64);
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t, ++tl) {
        const WgItem w = wg_item(t, tiles, p);
        int g, ci0, co0;
        tile_of(w.tile, g, ci0, co0);
        const int ntaps = min(TG, p.taps - g * TG);
        const bool bias = p.bias && ci0 == 0 && g == groups - 1;
        const uint32_t idesc = idesc_bf16(MT, ntaps * BN, 1, 1);
        const int buf = tl & 1;
        if (tl >= 2 && !mbar_wait(&tempty[buf], ((tl >> 1) & 1) ^ 1)) { atomicOr(p.err, 16); break; }
        tc_fence_after();
        const uint32_t d = tmem + buf * Cfg::TCOLS;
        for (int i = 0; i < w.nkb; ++i, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (it / S) & 1)) { atomicOr(p.err, 16); ok = false; break; }
          tc_fence_after();
          const uint32_t a = smem_u32(sm + s * Cfg::STAGE), b = a + Cfg::A_BYTES;
#pragma unroll
          for (int k = 0; k < Cfg::BKP / 16; ++k) {
            const uint64_t ad = smem_desc(a + k * 16 * 128, a_lbo, 1024, SWZ_128);
            mma_f16(d, ad, smem_desc(b + k * 16 * b_row, b_blk, 8 * b_row, b_swz), idesc,
                    (i | k) != 0);
            if (bias) mma_f16(d + ntaps * BN, ad, ones_desc, idesc_b, (i | k) != 0);
          }
          mma_commit(&empty[s]);
        }
        mma_commit(&tfull[buf]);
      }
    }
  } else {
    const int q = warp & 3;
    int tl = 0;
    for (int t = t_begin; t < t_end; ++t, ++tl) {
      const int buf = tl & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl >> 1) & 1))) {
        if (lane == 0) atomicOr(p.err, 32);
        break;
      }
      tc_fence_after();
      const WgItem w = wg_item(t, tiles, p);
      int g, ci0, co0;
      tile_of(w.tile, g, ci0, co0);
      const int tap0 = g * TG, ntaps = min(TG, p.taps - tap0);
      const bool bias = p.bias && ci0 == 0 && g == groups - 1;
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16);
      const int cin = p.cin;
      wgrad_drain<MT>(trow, q, lane, co0, ntaps * BN + (bias ? 32 : 0), bias ? ntaps * BN : -1,
                      w.nkb == 0, wgrad_dst(p, w, per), p.taps * p.cin, p.cout,
                      [&](int col) { return (tap0 + col / BN) * cin + ci0 + col % BN; });
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * Cfg::TCOLS);
}

// k_wgrad_halo: 3x3 stride-1 layers from halo tiles.
//
// Per K block (64 output pixels: hb rows x W columns of one image, W = 8,
// 16 or 32) the TMA warp loads the g tile and ONE box of x around the
// block: (W + 2) columns x (hb + 2) rows (ND = 3: all three kernel rows dy
// per tile) or hb rows shifted by dy (ND = 1: one kernel row per tile; the
// instantiated form).  For a K step of 16
// pixels (two 8-pixel groups: in one image row, or for W = 8 in two rows,
// one halo row apart) and a kernel row dy, the three taps dx =
// -1, 0, 1 are one MN-major B operand of N = 3 CB: its N blocks of CB
// channels start one pixel row apart (LBO = row bytes), so block j reads
// the x rows of block 0 shifted by j pixels.  A K step is ND MMAs of
// N = 3 CB, with no per-tap loads.  Accumulator columns: [dy][dx][ci], then
// the bias.  Tiles: (dy group, ci block, co block), dy fastest.
template <int CB, int MT, int ND>
struct WhCfg {
  static constexpr int ROWB = CB * 2;
  static constexpr int A_BYTES = MT * 64 * 2;               // MT co x 64 pixels
  // halo rows at most: (hb + 2)(W + 2) <= 3 * 66 (ND = 3), hb (W + 2) <= 8 * 10 (ND = 1)
  static constexpr int HMAX = ND == 3 ? 3 * 66 : 8 * 10;
  static constexpr int H_BYTES = (HMAX * ROWB + 1023) / 1024 * 1024;
  static constexpr int STAGE = A_BYTES + H_BYTES;
  static constexpr int NT = ND * 3 * CB;                     // tap columns
  static constexpr int S0 = (NT + 32 <= 256 ? 110 : 200) * 1024 / STAGE;
  static constexpr int S = S0 > 8 ? 8 : S0;
  // one accumulator per CTA; with at most 256 columns two CTAs share an SM
  // (one's epilogue overlaps the other's MMAs), else one CTA holds all 512
  static constexpr int NBUF = 1;
  static constexpr uint32_t TCOLS = NT + 32 <= 256 ? 256 : 512;
  static constexpr int CTAS = TCOLS == 256 ? 2 : 1;
  static constexpr int SMEM0 = 1024 + S * STAGE + kOnesBytes;
  // a lone CTA keeps at least 116 KB so that no second one lands on its SM
  static constexpr int SMEM = CTAS == 2 ? SMEM0 : (SMEM0 > 116 * 1024 ? SMEM0 : 116 * 1024);
  static_assert(CTAS == 1 || SMEM0 <= 113 * 1024, "two CTAs per SM do not fit");
};

template <int CB, int MT, int ND>
__global__ void __launch_bounds__(kThreads, 1)
k_wgrad_halo(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tX,
             const WgradTcArgs p, int C) {
  using Cfg = WhCfg<CB, MT, ND>;
  constexpr int S = Cfg::S, NT = Cfg::NT, NBUF = Cfg::NBUF;
  constexpr int DG = 3 / ND;                                 // dy groups
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = align1024(smraw);
  uint8_t* ones = sm + S * Cfg::STAGE;
  __shared__ uint64_t full[S], empty[S], tfull[2], tempty[2];
  __shared__ uint32_t tbase;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ci_tiles = p.cin / CB;
  const int tiles = ((p.cout + MT - 1) / MT) * ci_tiles * DG;
  const int items = C * tiles * p.splits;
  const int t_begin = (int)((int64_t)items * blockIdx.x / gridDim.x);
  const int t_end = (int)((int64_t)items * (blockIdx.x + 1) / gridDim.x);
  const int per = p.cout * 9 * p.cin + (p.bias ? p.cout : 0);
  const int rows_blocks = p.H / p.hb;
  const int HW2 = p.W + 2;
  const int hrows = ND == 3 ? p.hb + 2 : p.hb;
  const uint32_t h_tx = (uint32_t)(HW2 * hrows * Cfg::ROWB);
  auto tile_of = [&](int tile, int& dyg, int& ci0, int& co0) {
    dyg = tile % DG; tile /= DG;
    ci0 = (tile % ci_tiles) * CB; tile /= ci_tiles;
    co0 = tile * MT;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(&tfull[b], 1); mbar_init(&tempty[b], 128); }
    fence_mbar_init();
    tma_prefetch_desc(&tG);
    tma_prefetch_desc(&tX);
  }
  {
    const uint4 one = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    for (int i = threadIdx.x; i < kOnesBytes / 16; i += blockDim.x)
      reinterpret_cast<uint4*>(ones)[i] = one;
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) { tmem_alloc(&tbase, NBUF * Cfg::TCOLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (elect_one()) {
      int it = 0;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t) {
        const WgItem w = wg_item(t, tiles, p);
        int dyg, ci0, co0;
        tile_of(w.tile, dyg, ci0, co0);
        for (int i = 0; i < w.nkb; ++i, ++it) {
          const int s = it % S;
          if (it >= S && !mbar_wait(&empty[s], ((it / S) & 1) ^ 1)) {
            atomicOr(p.err, 8);
            ok = false;
            break;
          }
          const int kb = w.kb0 + i;
          const int b = kb / rows_blocks, h = (kb % rows_blocks) * p.hb;
          uint8_t* sa = sm + s * Cfg::STAGE;
          mbar_arrive_expect_tx(&full[s], Cfg::A_BYTES + h_tx);
          tma_load_5d(sa, &tG, &full[s], co0, 0, h, b, w.c);
          if (MT == 128)
            tma_load_5d(sa + 64 * 64 * 2, &tG, &full[s], p.cout > co0 + 64 ? co0 + 64 : co0, 0, h,
                        b, w.c);
          tma_load_5d(sa + Cfg::A_BYTES, &tX, &full[s], ci0, -1, ND == 3 ? h - 1 : h + dyg - 1, b,
                      w.c);
        }
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t swz = CB == 64 ? SWZ_128 : SWZ_64;
      constexpr uint32_t idesc = idesc_bf16(MT, 3 * CB, 1, 1);
      constexpr uint32_t idesc_b = idesc_bf16(MT, 32, 1, 1);
      constexpr uint32_t a_lbo = 64 * 64 * 2;                 // the two 64-co blocks (MT = 128)
      const uint64_t ones_desc = smem_desc(smem_u32(ones), 64 * 16, 8 * 64, SWZ_64);
      const uint32_t b_sbo = (uint32_t)((p.W >= 16 ? 8 : HW2) * Cfg::ROWB);
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok; ++t, ++tl) {
        const WgItem w = wg_item(t, tiles, p);
        int dyg, ci0, co0;
        tile_of(w.tile, dyg, ci0, co0);
        const bool bias = p.bias && ci0 == 0 && dyg == 0;
        const int buf = tl % NBUF;
        if (tl >= NBUF && !mbar_wait(&tempty[buf], ((tl / NBUF) & 1) ^ 1)) {
          atomicOr(p.err, 16);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * Cfg::TCOLS;
        for (int i = 0; i < w.nkb; ++i, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (it / S) & 1)) { atomicOr(p.err, 16); ok = false; break; }
          tc_fence_after();
          const uint32_t a = smem_u32(sm + s * Cfg::STAGE), hb0 = a + Cfg::A_BYTES;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            // a K step of 16 pixels: two 8-pixel groups, consecutive in one
            // image row (W >= 16) or the same columns of two rows (W = 8)
            const int y = (16 * k) / p.W, x0 = (16 * k) % p.W;
            const uint64_t ad = smem_desc(a + k * 16 * 128, a_lbo, 1024, SWZ_128);
#pragma unroll
            for (int dd = 0; dd < ND; ++dd) {
              const uint32_t start = hb0 + (uint32_t)(((y + dd) * HW2 + x0) * Cfg::ROWB);
              mma_f16(d + dd * 3 * CB, ad, smem_desc(start, Cfg::ROWB, b_sbo, swz), idesc,
                      (i | k) != 0);
            }
            if (bias) mma_f16(d + NT, ad, ones_desc, idesc_b, (i | k) != 0);
          }
          mma_commit(&empty[s]);
        }
        mma_commit(&tfull[buf]);
      }
    }
  } else {
    const int q = warp & 3;
    int tl = 0;
    for (int t = t_begin; t < t_end; ++t, ++tl) {
      const int buf = tl % NBUF;
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull[buf], (tl / NBUF) & 1))) {
        if (lane == 0) atomicOr(p.err, 32);
        break;
      }
      tc_fence_after();
      const WgItem w = wg_item(t, tiles, p);
      int dyg, ci0, co0;
      tile_of(w.tile, dyg, ci0, co0);
      const bool bias = p.bias && ci0 == 0 && dyg == 0;
      const uint32_t trow = tmem + buf * Cfg::TCOLS + ((uint32_t)(q * 32) << 16);
      const int cin = p.cin;
      wgrad_drain<MT>(trow, q, lane, co0, NT + (bias ? 32 : 0), bias ? NT : -1, w.nkb == 0,
                      wgrad_dst(p, w, per), 9 * p.cin, p.cout, [&](int col) {
                        const int dd = col / (3 * CB), j = (col % (3 * CB)) / CB;
                        return ((ND == 3 ? dd : dyg) * 3 + j) * cin + ci0 + col % CB;
                      });
      tc_fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, NBUF * Cfg::TCOLS);
}

// Weight and bias gradient of the input layer from its im2col (cout 32 or
// 64): D[co][k] = sum_p g[p][co] x0[p][k], a plain GEMM over the pixels;
// column k < 27 is W[co][tap][ci] (k = tap * 3 + ci), column 27 (the ones
// column) the bias.  The g tile (cout channels, swizzled MN-major) fills
// the 128 MMA rows 128/cout times; the epilogue keeps rows < cout.  The x0
// tile is one MN-major 64-pixel x 32-column box.  Partial layout as in
// k_wgrad_tc: [cout][27] then [cout].
template <int COUT>
struct Wg0Cfg {
  static constexpr int BKP = 64;
  static constexpr int A_BLK = COUT * BKP * 2;           // one copy of the g tile
  static constexpr int A_BYTES = 128 * BKP * 2;
  static constexpr int B_BYTES = BKP * 32 * 2;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int S = 6;
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
  const int per = COUT * 27 + COUT;
  const int kb_begin = split * p.kb_per_split;
  const int kb_end = min(kb_begin + p.kb_per_split, p.kb_total);
  const int nkb = kb_end > kb_begin ? kb_end - kb_begin : 0;
  const int rows_blocks = p.H / p.hb;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(&done, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tG);
    tma_prefetch_desc(&tX);
  }
  if (warp == 1) { tmem_alloc(&tbase, 32); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tbase;
  pdl_wait();
  pdl_trigger();
  if (warp == 0) {
    if (elect_one()) {
      for (int i = 0; i < nkb; ++i) {
        const int s = i % S;
        if (i >= S && !mbar_wait(&empty[s], ((i / S) & 1) ^ 1)) { atomicOr(p.err, 256); break; }
        const int kb = kb_begin + i;
        const int b = (kb / rows_blocks) * p.bb, h = (kb % rows_blocks) * p.hb;
        uint8_t* sa = sm + s * Cfg::STAGE;
        mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
#pragma unroll
        for (int j = 0; j < 128 / COUT; ++j)
          tma_load_5d(sa + j * Cfg::A_BLK, &tG, &full[s], 0, 0, h, b, c);
        tma_load_5d(sa + Cfg::A_BYTES, &tX, &full[s], 0, 0, h, b, c);
      }
    }
  } else if (warp == 1) {
    if (elect_one()) {
      constexpr uint32_t idesc = idesc_bf16(BM, 32, 1, 1);
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
                  smem_desc(b + k * 16 * 64, Cfg::B_BYTES, 8 * 64, SWZ_64), idesc, (i | k) != 0);
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
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int k = c0 + i;
          const float x = nkb ? v[i] : 0.f;
          if (k < 27) part[co * 27 + k] = x;
          else if (k == 27) part[COUT * 27 + co] = x;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 32);
}

// dw[c][i] = sum_s partial[c][s][i] for i < count (partials `per` apart).  A block of 8 warps covers 32 * 8/G
// consecutive columns; the G warps of a column group split the s range
// (warp g takes s = g, g+G, ...) and their sums are added in warp order, so
// the order depends on `splits` only.
template <int G>
__global__ void __launch_bounds__(256)
k_wgrad_reduce(const float* __restrict__ partial, float* __restrict__ dw, int64_t dw_rs,
               int splits, int64_t per, int64_t count) {
  __shared__ float red[8][32];
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.y;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int grp = w / G, sub = w % G;
  const int64_t i = ((int64_t)blockIdx.x * (8 / G) + grp) * 32 + lane;
  float s = 0.f;
  if (i < count) {
    const float* src = partial + (int64_t)c * splits * per + i;
    for (int k = sub; k < splits; k += G) s += src[(int64_t)k * per];
  }
  if (G == 1) {
    if (i < count) dw[(int64_t)c * dw_rs + i] = s;
    return;
  }
  red[w][lane] = s;
  __syncthreads();
  if (sub == 0 && i < count) {
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
                             const CUtensorMap& a2, const CUtensorMap& b2, const ConvTcArgs& p,
                             int tiles_m, int tiles_n, int items) {
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
  return launch_k(k_conv_tc<BN, BKC, EPI, BMN>, grid, kThreads, Cfg::SMEM, s, a, b, a2, b2, p,
                  tiles_m, tiles_n, items);
}

// persistent weight-gradient launch: one CTA per SM at most
template <typename KernelT>
cudaError_t launch_wgrad_persistent(KernelT* kernel, int smem, int ctas, bool& attr,
                                    cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                                    const WgradTcArgs& p, int C, int tiles) {
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int items = C * tiles * p.splits;
  const int cap = ctas * sm_count();
  const int grid = items < cap ? items : cap;
  return launch_k(kernel, grid, kThreads, smem, s, g, x, p, C);
}

template <int BN, int MT>
cudaError_t launch_wgrad_inst(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                              const WgradTcArgs& p, int C, int tiles) {
  static bool attr = false;
  return launch_wgrad_persistent(k_wgrad_tc<BN, MT>, WgCfg<BN, MT>::SMEM, 1, attr, s, g, x, p, C,
                                 tiles);
}

template <int CB, int MT, int ND>
cudaError_t launch_wgrad_halo_inst(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                                   const WgradTcArgs& p, int C, int tiles) {
  static bool attr = false;
  using Cfg = WhCfg<CB, MT, ND>;
  return launch_wgrad_persistent(k_wgrad_halo<CB, MT, ND>, Cfg::SMEM, Cfg::CTAS, attr, s, g, x,
                                 p, C, tiles);
}

template <int BN, int BKC, int EPI, int BMN>
cudaError_t launch_halo_inst(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                             const ConvTcArgs& p, int tiles_m, int tiles_n, int items) {
  using Cfg = HaloCfg<BN, BKC, EPI>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv_halo<BN, BKC, EPI, BMN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Cfg::SMEM_MAX);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int kper = p.kch / BKC;
  const int fixed = 1024 + 9 * kper * Cfg::B_TILE + Cfg::XS;
  int S = (Cfg::SMEM_MAX - fixed) / Cfg::A_BYTES;
  if (S > 6) S = 6;
  if (S < 2) return cudaErrorInvalidValue;
  const int smem = fixed + S * Cfg::A_BYTES;
  const int grid = items < sm_count() ? items : sm_count();
  return launch_k(k_conv_halo<BN, BKC, EPI, BMN>, grid, kHaloThreads, smem, s, a, b, p, tiles_m,
                  tiles_n, items, S);
}

}  // namespace

// ---------------------------------------------------------------------------
// host: tap tables
// ---------------------------------------------------------------------------
void conv_taps_fwd3(ConvTcArgs& p) {
  p.ntaps = 9;
  for (int t = 0; t < 9; ++t) {
    p.tdy[t] = (int8_t)(t / 3 - 1);
    p.tdx[t] = (int8_t)(t % 3 - 1);
    p.tw[t] = (int8_t)t;
    p.tsrc[t] = 0;
  }
}

void conv_taps_one(ConvTcArgs& p) {
  p.ntaps = 1;
  p.tdy[0] = p.tdx[0] = p.tw[0] = p.tsrc[0] = 0;
}

// dx[y][x] = sum_{sy,sx} g[y+sy][x+sx] W[1-sy][1-sx] (correlation with the
// flipped kernel)
void conv_taps_dgrad3(ConvTcArgs& p) {
  p.ntaps = 9;
  for (int t = 0; t < 9; ++t) {
    const int sy = t / 3 - 1, sx = t % 3 - 1;
    p.tdy[t] = (int8_t)sy;
    p.tdx[t] = (int8_t)sx;
    p.tw[t] = (int8_t)((1 - sy) * 3 + (1 - sx));
    p.tsrc[t] = 0;
  }
}

// input pixel (2Y+py, 2X+px) of a stride-2 3x3 convolution receives
// g[Y + (py+1-ky)/2][X + (px+1-kx)/2] W[ky][kx] for the taps with py+1-ky
// and px+1-kx even
void conv_taps_dgrad3_s2(ConvTcArgs& p, int py, int px, bool with_sc) {
  int n = 0;
  for (int ky = 0; ky < 3; ++ky)
    for (int kx = 0; kx < 3; ++kx) {
      if ((py + 1 - ky) % 2 != 0 || (px + 1 - kx) % 2 != 0) continue;
      p.tdy[n] = (int8_t)((py + 1 - ky) / 2);
      p.tdx[n] = (int8_t)((px + 1 - kx) / 2);
      p.tw[n] = (int8_t)(ky * 3 + kx);
      p.tsrc[n] = 0;
      ++n;
    }
  if (with_sc && py == 0 && px == 0) {
    p.tdy[n] = p.tdx[n] = p.tw[n] = 0;
    p.tsrc[n] = 1;
    ++n;
  }
  p.ntaps = n;
  p.stride = 1;
  p.osy = p.osx = 2;
  p.ooy = py;
  p.oox = px;
}

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
                     const uint32_t* box, int swizzle_bytes, const uint32_t* elem_strides) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  uint64_t stride = 2;
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = elem_strides ? elem_strides[i] : 1;
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
                           const ConvTcArgs& p, int bn, int bkc, int epi, int C,
                           const CUtensorMap* a2, const CUtensorMap* b2) {
  if (p.ntaps < 1 || p.ntaps > 9 || p.stride < 1) return cudaErrorInvalidValue;
  for (int t = 0; t < p.ntaps; ++t)
    if (p.tsrc[t] && (!a2 || !b2)) return cudaErrorInvalidValue;
  const CUtensorMap& A2 = a2 ? *a2 : a;
  const CUtensorMap& B2 = b2 ? *b2 : b;
  const int tiles_m = p.tiles_w * p.tiles_h * ((p.B + p.bb - 1) / p.bb);
  const int tiles_n = p.n_total / bn;
  const int items = tiles_m * tiles_n * C;
  // forward epilogues read a K-major B; the data-gradient epilogues read
  // the same weights MN-major
#define GCPSL_CONV_CASE(BN_, BKC_, EPI_, BMN_)             \
  if (bn == BN_ && bkc == BKC_ && epi == EPI_)             \
    return launch_conv_inst<BN_, BKC_, EPI_, BMN_>(s, a, b, A2, B2, p, tiles_m, tiles_n, items);
// EPI_STORE: the bias-free forward (pre-norm output, K-major B);
// EPI_DSTORE: the same store for a data gradient (MN-major B)
#define GCPSL_CONV_EPIS(BN_, BKC_)           \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_POOL, 0)    \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_RELU, 0)    \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_STORE, 0)   \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_DSTORE, 1)  \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_DPOOL, 1)   \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_DRELU, 1)   \
  GCPSL_CONV_CASE(BN_, BKC_, EPI_ADD, 1)
  GCPSL_CONV_CASE(32, 32, EPI_POOL, 0)      // the input layer (im2col, K = 32)
  GCPSL_CONV_CASE(32, 32, EPI_RELU, 0)
  GCPSL_CONV_EPIS(32, 64)
  GCPSL_CONV_EPIS(64, 32)
  GCPSL_CONV_EPIS(64, 64)
  GCPSL_CONV_EPIS(128, 32)
  GCPSL_CONV_EPIS(128, 64)
  GCPSL_CONV_CASE(256, 64, EPI_RELU, 0)
  GCPSL_CONV_CASE(256, 64, EPI_STORE, 0)
  GCPSL_CONV_CASE(256, 64, EPI_DSTORE, 1)
  GCPSL_CONV_CASE(256, 64, EPI_DPOOL, 1)
  GCPSL_CONV_CASE(256, 64, EPI_DRELU, 1)
  GCPSL_CONV_CASE(256, 64, EPI_ADD, 1)
#undef GCPSL_CONV_EPIS
#undef GCPSL_CONV_CASE
  return cudaErrorInvalidValue;
}

cudaError_t launch_pack_w0(cudaStream_t s, const bf16* w, bf16* w0p, int64_t rs, int cout,
                           int C) {
  const int per = cout * 32;
  return launch_k(k_pack_w0, dim3((unsigned)((per + 255) / 256), C), 256, 0, s, w, w0p, rs, cout);
}

// the instantiated (BN, BKC, epilogue) combinations of k_conv_halo
static const int kHaloKinds[][3] = {{64, 64, EPI_STORE}, {64, 64, EPI_DRELU}, {64, 64, EPI_ADD},
                                    {64, 32, EPI_POOL},  {128, 64, EPI_POOL}, {32, 64, EPI_DRELU},
                                    {64, 64, EPI_DPOOL}};

bool halo_supported(int H, int W, int kch, int bn, int bkc, int epi) {
  if (H % 16 || W % 8 || kch % bkc) return false;
  // resident weights and at least two halo stages within the shared memory
  const int a_bytes = ((kHaloW * kHaloH * bkc * 2) + 1023) / 1024 * 1024;
  const int need = 1024 + 9 * kch * bn * 2 + (epi == EPI_POOL ? 2 * kEpiScratch : 0) + 2 * a_bytes;
  if (need > 232448 - 1024) return false;
  for (const auto& k : kHaloKinds)
    if (k[0] == bn && k[1] == bkc && k[2] == epi) return true;
  return false;
}

cudaError_t launch_conv_halo(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                             const ConvTcArgs& p, int bn, int bkc, int epi, int C) {
  if (p.ntaps != 9 || p.stride != 1 || p.bw != 8 || p.hb != 16 || p.bb != 1 ||
      !halo_supported(p.H, p.W, p.kch, bn, bkc, epi) || p.tiles_w * 8 != p.W ||
      p.tiles_h * 16 != p.H ||
      p.n_total % bn)
    return cudaErrorInvalidValue;
  for (int t = 0; t < 9; ++t)
    if (p.tsrc[t] || p.tdy[t] < -1 || p.tdy[t] > 1 || p.tdx[t] < -1 || p.tdx[t] > 1)
      return cudaErrorInvalidValue;
  const int tiles_m = p.tiles_w * p.tiles_h * p.B;
  const int tiles_n = p.n_total / bn;
  const int items = C * tiles_m * tiles_n;
#define GCPSL_HALO(BN_, BKC_, EPI_, BMN_)                                                  \
  if (bn == BN_ && bkc == BKC_ && epi == EPI_ && (BMN_ == (epi >= EPI_DPOOL)))            \
    return launch_halo_inst<BN_, BKC_, EPI_, BMN_>(s, a, b, p, tiles_m, tiles_n, items);
  GCPSL_HALO(64, 64, EPI_STORE, 0)
  GCPSL_HALO(64, 64, EPI_DRELU, 1)
  GCPSL_HALO(64, 64, EPI_ADD, 1)
  GCPSL_HALO(64, 32, EPI_POOL, 0)
  GCPSL_HALO(128, 64, EPI_POOL, 0)
  GCPSL_HALO(32, 64, EPI_DRELU, 1)
  GCPSL_HALO(64, 64, EPI_DPOOL, 1)
#undef GCPSL_HALO
  return cudaErrorInvalidValue;
}

// one kernel row per tile: at most 3 x 64 + 32 accumulator columns, so two
// CTAs share an SM and the partials stay few
int wgrad_halo_rows(int) { return 1; }

bool wgrad_halo_supported(int H, int W, int cin, int cout, int taps, int stride) {
  // hb (W + 2) <= 80 halo rows: W = 8, 16 or 32
  const bool w_ok = W == 8 || W == 16 || W == 32;
  return taps == 9 && stride == 1 && w_ok && H % (64 / W) == 0 &&
         (cin == 32 || cin % 64 == 0) && (cout == 64 || cout % 128 == 0);
}

int wgrad_halo_tiles(int cin, int cout) {
  const int cb = cin == 32 ? 32 : 64;
  const int mt = cout % 128 == 0 ? 128 : 64;
  return (cout / mt) * (cin / cb) * (3 / wgrad_halo_rows(cin));
}

int wgrad_splits(int tiles, int kb_total, int64_t per) {
  // about 64 items per replica (a few per SM once several replicas are
  // grouped), at least 8 K blocks each, and at most 16 MB of partials per
  // replica; the per-replica shape alone decides the split, hence the
  // summation order, so C grouped replicas reproduce C one-replica runs bit
  // for bit
  int splits = (64 + tiles - 1) / tiles;
  splits = std::min(splits, std::max(1, kb_total / 8));
  splits = (int)std::min<int64_t>(splits, std::max<int64_t>(1, (4 << 20) / per));
  return std::max(1, splits);
}

static cudaError_t check_wgrad_out(const WgradTcArgs& p) {
  if (p.out && (p.splits != 1 || (uintptr_t)p.out % 16 || p.out_rs % 4))
    return cudaErrorInvalidValue;
  return cudaSuccess;
}

cudaError_t launch_wgrad_halo(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                              const WgradTcArgs& p, int C) {
  if (!wgrad_halo_supported(p.H, p.W, p.cin, p.cout, p.taps, p.stride) || p.hb * p.W != 64 ||
      p.bb != 1 || p.pad != 1 || check_wgrad_out(p) != cudaSuccess)
    return cudaErrorInvalidValue;
  const int tiles = wgrad_halo_tiles(p.cin, p.cout);
  const bool m64 = p.cout % 128 != 0;
  if (p.cin == 32)
    return m64 ? launch_wgrad_halo_inst<32, 64, 1>(s, g, x, p, C, tiles)
               : launch_wgrad_halo_inst<32, 128, 1>(s, g, x, p, C, tiles);
  return m64 ? launch_wgrad_halo_inst<64, 64, 1>(s, g, x, p, C, tiles)
             : launch_wgrad_halo_inst<64, 128, 1>(s, g, x, p, C, tiles);
}

int wgrad_tc_tiles(int cin, int cout, int taps, int bn) {
  const int tg = 256 / bn;
  const int mt = cout % 128 == 0 ? 128 : 64;
  return ((taps + tg - 1) / tg) * (cin / bn) * ((cout + mt - 1) / mt);
}

cudaError_t launch_wgrad_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                            const WgradTcArgs& p, int bn, int C) {
  if ((p.taps != 9 && p.taps != 1) || (p.taps == 1 && p.pad != 0) ||
      check_wgrad_out(p) != cudaSuccess)
    return cudaErrorInvalidValue;
  const int tiles = wgrad_tc_tiles(p.cin, p.cout, p.taps, bn);
  if (p.cout % 128 != 0) {
    if (bn == 32) return launch_wgrad_inst<32, 64>(s, g, x, p, C, tiles);
    if (bn == 64) return launch_wgrad_inst<64, 64>(s, g, x, p, C, tiles);
    if (bn == 128) return launch_wgrad_inst<128, 64>(s, g, x, p, C, tiles);
    return cudaErrorInvalidValue;
  }
  if (bn == 32) return launch_wgrad_inst<32, 128>(s, g, x, p, C, tiles);
  if (bn == 64) return launch_wgrad_inst<64, 128>(s, g, x, p, C, tiles);
  if (bn == 128) return launch_wgrad_inst<128, 128>(s, g, x, p, C, tiles);
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
    return launch_k(k_wgrad0_tc<CO>, dim3(p.splits, 1, C), kThreads, Wg0Cfg<CO>::SMEM, s, g, x, \
                    p);                                                                      \
  }
  GCPSL_WG0(32)
  GCPSL_WG0(64)
#undef GCPSL_WG0
  return cudaErrorInvalidValue;
}

cudaError_t launch_wgrad_reduce(cudaStream_t s, const float* partial, float* dw, int64_t dw_rs,
                                int splits, int64_t per, int C, int64_t count) {
  if (count < 0) count = per;
  const int G = splits <= 2 ? 1 : splits <= 8 ? 2 : splits <= 32 ? 4 : 8;
  const int64_t cols_per_block = 32 * (8 / G);
  const dim3 grid((unsigned)((count + cols_per_block - 1) / cols_per_block), C);
  if (G == 1)
    return launch_k(k_wgrad_reduce<1>, grid, 256, 0, s, partial, dw, dw_rs, splits, per, count);
  if (G == 2)
    return launch_k(k_wgrad_reduce<2>, grid, 256, 0, s, partial, dw, dw_rs, splits, per, count);
  if (G == 4)
    return launch_k(k_wgrad_reduce<4>, grid, 256, 0, s, partial, dw, dw_rs, splits, per, count);
  return launch_k(k_wgrad_reduce<8>, grid, 256, 0, s, partial, dw, dw_rs, splits, per, count);
}


}  // namespace gcpsl
