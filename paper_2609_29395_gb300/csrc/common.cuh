// Internal declarations of libgcpsl.so (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace gcpsl {

typedef __nv_bfloat16 bf16;

// ---------------------------------------------------------------------------
// Split-model description.  Conv layers: 3x3, stride 1, pad 1, bias, ReLU,
// optional 2x2/2 max-pool.  Activations are NHWC with the replica index
// outermost: [C][B][H][W][ch].
// ---------------------------------------------------------------------------
struct ConvSpec { int cin, cout, h, w, pool; };
struct ArchSpec {
  int ncl, nsv;          // client / server conv layers (ncl + nsv <= 4)
  ConvSpec conv[4];
  int fc_in, fc_out;
  // parameter offsets within one replica, same order as the PyTorch
  // state_dict: conv{i}.weight, conv{i}.bias, ..., fc.weight, fc.bias
  int64_t off_w[4], off_b[4], off_fcw, off_fcb, p_client, p_total;
  int L() const { return ncl + nsv; }
  int out_h(int i) const { return conv[i].pool ? conv[i].h / 2 : conv[i].h; }
  int out_w(int i) const { return conv[i].pool ? conv[i].w / 2 : conv[i].w; }
};
bool make_arch(int id, ArchSpec* a);

// message returned by gcpsl_last_error(NULL) for calls without a context
void set_global_error(const char* msg);

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11): ten rounds, two 32x32 -> 64-bit
// products per round, key bumped by the Weyl increments between rounds.
// ---------------------------------------------------------------------------
__host__ __device__ inline void philox4x32_10(uint32_t c[4], uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { k0 += W0; k1 += W1; }
    uint64_t p0 = (uint64_t)M0 * c[0];
    uint64_t p1 = (uint64_t)M1 * c[2];
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ c[1] ^ k0;
    uint32_t n2 = (uint32_t)(p0 >> 32) ^ c[3] ^ k1;
    c[1] = (uint32_t)p1;
    c[3] = (uint32_t)p0;
    c[0] = n0;
    c[2] = n2;
  }
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  Every kernel of the library is launched
// with programmatic stream serialisation, so it may be scheduled while the
// previous kernel on the stream drains.  Each kernel therefore runs only
// set-up that touches no global memory (barrier init, TMEM allocation,
// descriptor prefetch) before pdl_wait(), which returns once the previous
// grid has completed and its writes are visible; it then calls
// pdl_trigger() so that the next kernel can be scheduled in turn.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------------------
// Element conversions for the two storage types
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// ---------------------------------------------------------------------------
// Kernel launchers (each enqueues on `s`; return the launch error)
// ---------------------------------------------------------------------------
// sampler.cu
// period[n]: rounds per epoch of cluster n's sampler (r_n in lockstep, the
// system epoch's max_m r_m under the epoch schedule); the permutation of
// epoch t / period[n] is built when t % period[n] == 0.
cudaError_t launch_epoch_keys(cudaStream_t s, const int32_t* ids, const int64_t* off,
                              const int32_t* period, const int64_t* d_t, int cluster_base,
                              uint64_t seed, uint64_t* keys, int C, int64_t max_nc);
cudaError_t launch_epoch_rank(cudaStream_t s, const int32_t* ids, const int64_t* off,
                              const int32_t* period, const int64_t* d_t, const uint64_t* keys,
                              int32_t* perm, int C, int64_t max_nc);
// The round's batch of every cluster: local round s = t % period[n] of its
// epoch when s < rounds[n]; a cluster past its r_n rounds (epoch schedule)
// waits at the fusion barrier: upd[n] = 0 (nullable), its batch is its last
// one (s = r_n - 1) and active[n] = 0.  cut_scale (nullable, [C][B]):
// B / (|A| b_k) of every batch position (|A| of the batch itself, also for a
// waiting cluster), the per-client average's factor.
cudaError_t launch_sample(cudaStream_t s, const int32_t* perm, const int64_t* off,
                          const int32_t* rounds, const int32_t* period, const int64_t* d_t,
                          const int32_t* owner, const int32_t* labels, int K, int B, int C,
                          int32_t* idx, int32_t* counts, int32_t* active, int32_t* y,
                          int32_t* upd, float* cut_scale = nullptr);
// Training augmentation of the gathered images (Sec. V-A: random crops and
// horizontal flips): sampled image b of cluster n in round t is cropped
// from its 4-pixel zero-padded version at offset (dy, dx) in [0, 8]^2 and
// then mirrored when flip = 1, i.e. out[ch][y][x] = img[ch][y + dy - 4]
// [x' + dx - 4] with x' = flip ? 31 - x : x (0 outside).  With Philox4x32-10
// (counter = (b, t, n', 1), key = seed), n' = cluster_base + n:
// dy = (o0 * 9) >> 32, dx = (o1 * 9) >> 32, flip = o2 & 1.  Off: dy = dx = 4,
// flip = 0 (the image itself).
struct AugArgs {
  int on;
  uint32_t s0, s1;              // the seed's low and high words
  const int64_t* d_t;           // the device round counter
  int cluster_base, B;
};
// fp32: x0 = the sampled images, NHWC with 3 channels; bf16: x0 = the input
// layer's im2col [CB][32][32][32] (27 tap x channel columns, a ones column
// for the bias gradient, zero padding)
template <typename T>
cudaError_t launch_gather(cudaStream_t s, const float* images, const int32_t* idx, int CB, T* x0,
                          const AugArgs& aug);
template <>
cudaError_t launch_gather<float>(cudaStream_t s, const float* images, const int32_t* idx, int CB,
                                 float* x0, const AugArgs& aug);
template <>
cudaError_t launch_gather<bf16>(cudaStream_t s, const float* images, const int32_t* idx, int CB,
                                bf16* x0, const AugArgs& aug);
// per-client average (Sec. IV-B, the unweighted reading): a ([C B][per_a])
// and b ([C B][per_b], nullable) scaled in place, example cb by scale[cb]
// (the sampler's cut_scale); per_* multiples of 8
template <typename T>
cudaError_t launch_client_avg_scale(cudaStream_t s, T* a, int64_t per_a, T* b, int64_t per_b,
                                    const float* scale, int CB);

// conv_simt.cu
template <typename T>
cudaError_t launch_conv_fwd_simt(cudaStream_t s, const T* x, const T* w, int64_t w_rs,
                                 const float* bias, int64_t b_rs, T* out, uint8_t* code, int C,
                                 int B, const ConvSpec& cs);
template <typename T>
cudaError_t launch_relu_pool_bwd(cudaStream_t s, const T* dout, const uint8_t* code,
                                 const T* act, T* g, int C, int B, const ConvSpec& cs);
template <typename T>
cudaError_t launch_conv_dgrad_simt(cudaStream_t s, const T* g, const T* w, int64_t w_rs, T* dx,
                                   int C, int B, const ConvSpec& cs);
// weight+bias gradient partials of a CUDA-core layer over `splits` pixel
// ranges (tiles of `tr` image rows): partial[c][split][cout*9*cin + cout]
template <typename T>
cudaError_t launch_wgrad_simt(cudaStream_t s, const T* x, int xc, const T* g, float* partial,
                              int C, int B, const ConvSpec& cs, int tr, int splits,
                              int tiles_per_split);

// head.cu
// forward of the linear layer with the per-example softmax cross-entropy:
// loss_ex[c][b] = l_b, dlogits[c][b][j]
template <typename T>
cudaError_t launch_fc_fwd_ce(cudaStream_t s, const T* h, const T* w, int64_t w_rs,
                             const float* b, int64_t b_rs, const int32_t* y, float* loss_ex,
                             float* dlogits, int C, int B, int fin, int fout,
                             float label_smoothing);
// backward of the linear layer (dW, db, dh) and loss[c] = mean_b loss_ex[c][b];
// fout = 10 or 100 classes.  When fc_bwd_split_dh(fout), this launch writes
// dW, db and loss only, and launch_fc_bwd_dh (same route arguments) writes dh.
// route: FC_DH_STORE writes dh; FC_DH_POOL writes the last conv layer's g
// (2Ho x 2Wo x ch) through its max-pool codes; FC_DH_RELU writes g = dh where
// act > 0; FC_DH_AVG writes dh / (Ho Wo) to every pixel of an Ho x Wo x ch
// map (global average pool backward, h = [ch]).  Otherwise h is [Ho][Wo][ch].
enum { FC_DH_STORE = 0, FC_DH_POOL = 1, FC_DH_RELU = 2, FC_DH_AVG = 3 };
template <typename T>
cudaError_t launch_fc_bwd(cudaStream_t s, const float* dlogits, const float* loss_ex,
                          const T* h, const T* w, int64_t w_rs, float* dw, float* db,
                          int64_t g_rs, T* dh, float* loss, int C, int B, int fin, int fout,
                          int route, const uint8_t* code, const T* act, int Ho, int Wo, int ch);
bool fc_bwd_split_dh(int fout);
template <typename T>
cudaError_t launch_fc_bwd_dh(cudaStream_t s, const float* dlogits, const T* w, int64_t w_rs,
                             T* dh, int C, int B, int fin, int fout, int route,
                             const uint8_t* code, const T* act, int Ho, int Wo, int ch);

// conv_tc.cu (tensor-core convolutions, bf16 operands)
enum {
  EPI_POOL = 0, EPI_RELU = 1, EPI_STORE = 2, EPI_DPOOL = 3, EPI_DRELU = 4, EPI_ADD = 5,
  EPI_DSTORE = 6
};
struct ConvTcArgs {
  int H, W, B;          // M grid (the GEMM's output pixels) and batch per replica
  int kch;              // channels of the activation operand (multiple of the stage width)
  int bw, hb, bb;       // M tile of 128 pixels: bw columns x hb rows x bb images
  int tiles_w, tiles_h; // W / bw, H / hb
  int n_total;          // output channels (row length of `out`)
  const float* bias;    // fp32 bias of replica 0 (EPI_POOL / EPI_RELU)
  int64_t bias_rs;      // replica stride of the bias
  bf16* out;            // NHWC output, [C][B][H'][W'][n_total] (may be null for EPI_D*)
  uint8_t* code;        // max-pool codes, same layout as out (EPI_POOL writes, EPI_DPOOL reads)
  int* err;             // error word: bounded waits that gave up
  const bf16* act;      // EPI_DRELU: the previous layer's ReLU output, layout of out
  bf16* gout;           // EPI_DPOOL / EPI_DRELU: the previous layer's g (2H x 2W for DPOOL)
  // K taps: A box origin = (M pixel) * stride + (tdy, tdx); B tap index tw;
  // tsrc selects the operand pair (0: a/b, 1: a2/b2).  Filled by the
  // conv_taps_* helpers.
  int stride = 1;
  int ntaps = 9;
  int8_t tdy[9] = {}, tdx[9] = {}, tw[9] = {}, tsrc[9] = {};
  // output pixel of M pixel (y, x): (y * osy + ooy, x * osx + oox) in an
  // out_H x out_W grid (0: the M grid) -- EPI_STORE / EPI_ADD / EPI_DRELU
  int out_H = 0, out_W = 0, osy = 1, osx = 1, ooy = 0, oox = 0;
  const bf16* res = nullptr;  // EPI_ADD: out = bf16(acc + res), layout of out
};
// 3x3 forward taps (kernel row/col ky, kx -> shift (ky-1, kx-1), tap ky*3+kx)
void conv_taps_fwd3(ConvTcArgs& p);
// one tap without shift (1x1 convolutions, the im2col input layer)
void conv_taps_one(ConvTcArgs& p);
// 3x3 stride-1 data gradient: shift (sy, sx), weight tap (1-sy)*3 + (1-sx)
void conv_taps_dgrad3(ConvTcArgs& p);
// 3x3 stride-2 data gradient for the input pixels of parity (py, px): the
// taps with (p+1-k) even, shift (p+1-k)/2; with_sc adds the 1x1 stride-2
// shortcut (operand pair 1) to parity (0, 0)
void conv_taps_dgrad3_s2(ConvTcArgs& p, int py, int px, bool with_sc);
struct WgradTcArgs {
  int H, W, B, cout, cin;   // H, W: the output grid (g)
  int hb, bb;           // image rows / images per 64-pixel K block (W * hb * bb == 64)
  int kb_total;         // K blocks per replica
  int kb_per_split, splits;
  float* partial;       // [C][splits][cout][taps][cin] (+ [cout] bias)
  int* err;
  int taps = 9;         // 9 (3x3) or 1 (1x1)
  int bias = 1;         // also the bias gradient (a block of ones)
  int stride = 1, pad = 1;  // x pixel of output pixel p and tap (kh, kw): p*stride + k - pad
  // non-null (one split only): the gradient is written to out[c * out_rs +
  // ...] directly (same layout as a partial; 16-byte aligned) and `partial`
  // is unused
  float* out = nullptr;
  int64_t out_rs = 0;
};
// splits of a weight gradient with `tiles` tiles and kb_total K blocks per
// replica (a function of the per-replica shape only)
int wgrad_splits(int tiles, int kb_total, int64_t per);
int wgrad_tc_tiles(int cin, int cout, int taps, int bn);
// elem_strides (nullable): traversal stride per dimension; a box then
// loads ceil(box[i] / elem_strides[i]) elements along dimension i
bool tensor_map_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                     const uint32_t* box, int swizzle_bytes,
                     const uint32_t* elem_strides = nullptr);
bool tensor_map_bf16_strided(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                             uint64_t outer_stride_bytes, const uint32_t* box, int swizzle_bytes);
cudaError_t launch_conv_tc(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                           const ConvTcArgs& p, int bn, int bkc, int epi, int C,
                           const CUtensorMap* a2 = nullptr, const CUtensorMap* b2 = nullptr);
cudaError_t launch_wgrad_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                            const WgradTcArgs& p, int bn, int C);
// 3x3 stride-1 convolution (forward, or data gradient with the dgrad3 tap
// table) on 8 x 16-pixel M tiles of one image, weights resident in shared
// memory: `a` maps the activation operand with a box of BKC channels x 10
// x 18 pixels, `b` the weights as for launch_conv_tc with an N box of
// min(bn, 64).  p.bw = 8, p.hb = 16, p.bb = 1.
// weight gradient of a 3x3 stride-1 convolution from halo tiles of x:
// `x` maps the input with a box of CB = (cin == 32 ? 32 : 64) channels x
// (W + 2) columns x (hb + 2) rows (cin == 32) or hb rows (otherwise); `g`
// as for launch_wgrad_tc.  p.hb * W == 64, p.bb == 1; tiles per replica
// from wgrad_halo_tiles.
bool wgrad_halo_supported(int H, int W, int cin, int cout, int taps, int stride);
int wgrad_halo_rows(int cin);     // kernel rows per CTA (3 or 1)
int wgrad_halo_tiles(int cin, int cout);
cudaError_t launch_wgrad_halo(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                              const WgradTcArgs& p, int C);
bool halo_supported(int H, int W, int kch, int bn, int bkc, int epi);
cudaError_t launch_conv_halo(cudaStream_t s, const CUtensorMap& a, const CUtensorMap& b,
                             const ConvTcArgs& p, int bn, int bkc, int epi, int C);
// input layer: b = packed weights w0p[C][cout][32] (k = tap * 3 + ci < 27, else 0)
cudaError_t launch_pack_w0(cudaStream_t s, const bf16* w, bf16* w0p, int64_t rs, int cout, int C);
// input-layer weight and bias gradient partials from its im2col (cout 32 or
// 64), partial layout [C][splits][cout*27 + cout]
cudaError_t launch_wgrad0_tc(cudaStream_t s, const CUtensorMap& g, const CUtensorMap& x,
                             const WgradTcArgs& p, int C);
// dw[c * dw_rs + i] = sum over s (in order) of partial[c][s][i], i < count
// (partials `per` apart)
cudaError_t launch_wgrad_reduce(cudaStream_t s, const float* partial, float* dw, int64_t dw_rs,
                                int splits, int64_t per, int C, int64_t count = -1);

// norm.cu (GroupNorm / train-mode BatchNorm on [C][B][HW][ch] bf16 tensors;
// statistics per set: GroupNorm (c, b, group), BatchNorm (c, ch)).  gn is the
// GroupNorm group count (a divisor of ch, at most 32; the per-example mean /
// rstd arrays keep a stride of 32), 0 for BatchNorm.
// per-(c, b, ch) pixel sums: forward (sum y, sum y^2); backward (sum dz,
// sum dz x_hat) with dz = d (times [mask > 0], written to dz_out if set)
cudaError_t launch_norm_sums(cudaStream_t s, bool bwd, const bf16* y, const bf16* d,
                             const bf16* mask, const float* mean, const float* rstd, bf16* dz_out,
                             float* sums, int C, int B, int HW, int ch, int gn);
// per set: mean, rstd, and per (c, [b,] ch) the affine form ss = (gamma rstd,
// beta - mean gamma rstd) (GroupNorm per example, BatchNorm shared over the
// batch); BatchNorm also updates run ([C] x run_rs: mean[ch], var[ch]) of the
// replicas with upd[c] (upd nullable: all)
cudaError_t launch_norm_finalize_fwd(cudaStream_t s, const float* sums, const float* gamma,
                                     const float* beta, int64_t g_rs, float* mean, float* rstd,
                                     float2* ss, float* run, int64_t run_rs, int C, int B, int HW,
                                     int ch, int gn, float eps, float momentum,
                                     const int32_t* upd = nullptr);
// backward affine form kk = (k1, k2, k3, 0): dy = k1 dz + k2 y + k3 per
// (c, [b,] ch); per channel dgamma, dbeta
cudaError_t launch_norm_finalize_bwd(cudaStream_t s, const float* sums, const float* gamma,
                                     int64_t g_rs, const float* mean, const float* rstd,
                                     float4* kk, float* dgamma, float* dbeta, int64_t d_rs, int C,
                                     int B, int HW, int ch, int gn);
// out = relu?(y scale + shift + r): r = res (bf16), or y2 scale2 + shift2, or 0
cudaError_t launch_norm_apply_fwd(cudaStream_t s, const bf16* y, const float2* ss, int gn,
                                  const bf16* res, const bf16* y2, const float2* ss2, int gn2,
                                  bf16* out, int C, int B, int HW, int ch, int relu);
// out = k1 dz + k2 y + k3, dz = d (times [mask > 0])
cudaError_t launch_norm_apply_bwd(cudaStream_t s, const bf16* y, const float4* kk, int gn,
                                  const bf16* d, const bf16* mask, bf16* out, int C, int B, int HW,
                                  int ch);
// GroupNorm (`groups` groups) of one example per block, statistics and apply in
// one launch: forward out = relu?(norm(y) + res) (res nullable), writing the
// per-set mean / rstd; backward dy from d (times [mask > 0], kept in dz_out
// when set) with the per-(example, channel) sums for dgamma / dbeta, which
// launch_norm_finalize_bwd_channels then reduces over the batch.
cudaError_t launch_gn_fused_fwd(cudaStream_t s, const bf16* y, const bf16* res,
                                const float* gamma, const float* beta, int64_t g_rs, float* mean,
                                float* rstd, bf16* out, int C, int B, int HW, int ch, int relu,
                                int groups, float eps, int* err);
cudaError_t launch_gn_fused_bwd(cudaStream_t s, const bf16* y, const bf16* d, const bf16* mask,
                                bf16* dz_out, const float* gamma, int64_t g_rs, const float* mean,
                                const float* rstd, float* sums, bf16* out, int C, int B, int HW,
                                int ch, int groups, int* err);
cudaError_t launch_norm_finalize_bwd_channels(cudaStream_t s, const float* sums, float* dgamma,
                                              float* dbeta, int64_t d_rs, int C, int B, int ch);
cudaError_t launch_avgpool(cudaStream_t s, const bf16* x, bf16* h, int CB, int HW, int ch);

// optim.cu
// A range of every replica's parameters [off, off + count) whose gradient
// the update reads from src: element j of replica c is the sum over s <
// splits of src[(c * splits + s) * per + j] (split partials of a weight
// gradient), or src[c * per + j] with splits = 1 (the gradient store).
// total = C * count elements, in (replica, element) order.
struct SgdSeg {
  const float* src;
  int64_t off, count, per, total;
  int splits;
  // the input layer's weights: also written packed as w0p[c][co][32]
  // (column k = tap * 3 + ci < 27) for its one-tap forward; else null
  bf16* w0p;
  int w0_cout;
};
constexpr int kSgdThreads = 256, kSgdPer = 2;
// quads (4 parameters) per update block of a segment with `splits` sources:
// about the same bytes per block whatever the split count
inline int sgd_chunk(int splits) {
  const int n = kSgdThreads * kSgdPer * 2 / (splits + 1);
  return n < kSgdThreads ? kSgdThreads : n;
}
// SGD over the segments (they tile [0, P_pad) of each replica; offsets,
// counts and strides multiples of 4), then the bf16 shadow; one launch for
// all replicas.  blocks[b] = {segment, first quad of the block in it, quads
// (<= kSgdThreads * kSgdPer), 0}.
cudaError_t launch_sgd_seg(cudaStream_t s, float* theta, float* mom, bf16* shadow,
                           const SgdSeg* segs, const int4* blocks, int nblocks, int64_t P_pad,
                           float lr, float momentum, float wd, int nesterov, const int32_t* upd,
                           int64_t* d_t);
// upd (nullable): replica c = i / P_pad takes the update only when upd[c]
cudaError_t launch_sgd(cudaStream_t s, float* theta, float* mom, const float* grad,
                       bf16* shadow, int64_t n, int64_t P_pad, float lr, float momentum, float wd,
                       int nesterov, const int32_t* upd, int64_t* d_t);
cudaError_t launch_fuse(cudaStream_t s, float* theta, bf16* shadow, const float* q, int C,
                        int64_t P);

// one block waiting, bounded by limit_ns, on an mbarrier nothing arrives on:
// sets bit 256 of err (the library's bounded-wait failure path)
cudaError_t launch_wait_probe(cudaStream_t s, int* err, uint64_t limit_ns);

}  // namespace gcpsl
