// Host-side context of libgcpsl.so, shared by the translation units of the
// C ABI (ctx.cu: sampler, SplitCNN rounds, fusion, accessors; resnet.cu: the
// ResNet-18 split's rounds).  Not part of the C ABI.
#pragma once

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "common.cuh"
#include "gcpsl.h"

namespace gcpsl {

// ---------------------------------------------------------------------------
// Kernel timing with CUDA events on the context's stream
// ---------------------------------------------------------------------------
struct KernelTimer {
  std::vector<const char*> names;
  std::vector<int64_t> launches;
  std::vector<double> ms;
  struct Pending { int kind; cudaEvent_t a, b; };
  std::vector<Pending> pending;
  std::vector<cudaEvent_t> pool;
  int cur_kind = -1;
  cudaEvent_t cur_a = nullptr;
  // while a round is being captured into a graph, the event pairs become
  // external event-record nodes of that graph and are listed here
  std::vector<Pending>* capture = nullptr;
  // only kernels whose name starts with this prefix are timed (empty: all)
  std::string filter;

  bool wants(const char* name) const {
    return filter.empty() || std::strncmp(name, filter.c_str(), filter.size()) == 0;
  }

  int kind(const char* name) {
    for (size_t i = 0; i < names.size(); ++i)
      if (names[i] == name || std::strcmp(names[i], name) == 0) return (int)i;
    names.push_back(name); launches.push_back(0); ms.push_back(0.0);
    return (int)names.size() - 1;
  }
  cudaEvent_t get() {
    if (!pool.empty()) { cudaEvent_t e = pool.back(); pool.pop_back(); return e; }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  void record(cudaEvent_t e, cudaStream_t s) {
    if (capture) cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
    else cudaEventRecord(e, s);
  }
  void begin(const char* name, cudaStream_t s) {
    cur_kind = kind(name);
    cur_a = get();
    record(cur_a, s);
  }
  void end(cudaStream_t s) {
    cudaEvent_t b = get();
    record(b, s);
    (capture ? *capture : pending).push_back({cur_kind, cur_a, b});
  }
  // add the elapsed times of recorded pairs (waits for each pair's end)
  void account(const std::vector<Pending>& v) {
    for (auto& p : v) {
      float t = 0.f;
      if (cudaEventSynchronize(p.b) == cudaSuccess && cudaEventElapsedTime(&t, p.a, p.b) == cudaSuccess) {
        ms[p.kind] += t;
        launches[p.kind] += 1;
      }
    }
  }
  void collect() {
    account(pending);
    for (auto& p : pending) { pool.push_back(p.a); pool.push_back(p.b); }
    pending.clear();
  }
  void reset() {
    collect();
    std::fill(launches.begin(), launches.end(), 0);
    std::fill(ms.begin(), ms.end(), 0.0);
  }
  void destroy() {
    collect();
    for (auto e : pool) cudaEventDestroy(e);
    pool.clear();
  }
};

struct RnState;    // the ResNet-18 split's buffers and layers (resnet.cu)

}  // namespace gcpsl

using gcpsl::ArchSpec;
using gcpsl::bf16;
using gcpsl::KernelTimer;

struct gcpsl_ctx {
  gcpsl_model_desc desc{};
  ArchSpec a{};
  int K = 0, C = 0, B = 0, F = 0;
  int J = 10;                       // classes (outputs of the linear head)
  // ResNet norms: GroupNorm groups, eps of both norms, BatchNorm momentum
  int gn_groups = 32;
  float norm_eps = 1e-5f, bn_momentum = 0.1f;
  uint64_t seed = 0;
  bool bf = false;
  size_t esz = 4;
  cudaStream_t own_stream = nullptr, stream = nullptr;

  int64_t n = 0;
  float* d_images = nullptr;       // device copy, or device view of h_images
  float* h_images = nullptr;       // pinned mapped host copy (data_on_host)
  int32_t* d_labels = nullptr;
  int32_t* d_owner = nullptr;

  std::vector<int64_t> h_off;      // [C+1] offsets of the clusters' id lists
  std::vector<int32_t> h_rounds;   // r_n = n_c / B
  // schedule: lockstep (F >= 0): period_n = r_n; epoch schedule (F = -1):
  // period_n = R = max_n r_n, fuse every R rounds, cluster n updates in the
  // first r_n rounds of each system epoch (d_upd[n] of the current round)
  std::vector<int32_t> h_period;
  int64_t R = 0;
  int32_t* d_period = nullptr;
  int32_t* d_upd = nullptr;
  std::vector<float> h_q;          // fusion weights
  int64_t max_nc = 0;
  int64_t* d_off = nullptr;
  int32_t* d_rounds = nullptr;
  int32_t* d_ids = nullptr;
  int32_t* d_perm = nullptr;
  uint64_t* d_keys = nullptr;
  float* d_q = nullptr;

  int64_t P = 0;
  int64_t P_pad = 0;               // replica stride of every [C][P] array (multiple of 64)
  float* d_theta = nullptr;        // [C][P_pad] fp32 master, kernel layout
  float* d_mom = nullptr;
  float* d_grad = nullptr;
  bf16* d_shadow = nullptr;        // [C][P_pad] bf16 operand copy (bf16 mode)
  int* d_err = nullptr;            // device error word (bounded waits that gave up)

  // tensor-core layers (bf16 mode): tile shapes and TMA descriptors
  struct TcLayer {
    bool on = false;
    int bw, hb, bb, tiles_w, tiles_h;   // 128-pixel M tile
    int whb, wbb;                  // 64-pixel K block of the weight gradient
    int bn_f, bkc_f, bn_d, bkc_d, bn_w;
    int splits, kb_total, kb_per_split;
    CUtensorMap fwdA, fwdB, dgrA, dgrB, wgA, wgB;
    // halo-tiled forward / data gradient (3x3 stride 1, resident weights)
    bool halo_f = false, halo_d = false;
    CUtensorMap hfA, hdA;
    bool wg_halo = false;          // weight gradient from halo tiles of x
    CUtensorMap wgH;
    float* part = nullptr;         // its split partials (null: written to the gradient)
  } tc[4];
  // input layer on the tensor cores (bf16 mode): the gather writes its
  // im2col, x0c = 32 columns per pixel; packed weights [C][cout][32]
  struct Tc0Layer {
    bool on = false;
    int bw, hb, bb, tiles_w, tiles_h;
    CUtensorMap A, B;
    bool wg_on = false;            // its weight gradient on the tensor cores too
    int whb, wbb, kb_total, kb_per_split, splits;
    CUtensorMap wgA, wgB;
    float* part = nullptr;         // its split partials
  } tc0;
  int x0c = 3;
  // the ResNet-18 split (architecture 2), else null
  gcpsl::RnState* rn = nullptr;
  // the input layer's packed weights: offset and output channels
  int64_t w0_off = 0;
  int w0_cout = 0;
  bf16* d_w0p = nullptr;
  // weight-gradient split partials of the tensor-core layers, one buffer
  // per layer ([C][splits][per]), summed by the update itself (k_sgd_seg);
  // the update's segments tile [0, P_pad) with these ranges and the
  // gradient store
  struct PartialRange { int64_t off, count, per; int splits; float* buf; };
  std::vector<PartialRange> pranges;
  gcpsl::SgdSeg* d_sgd_segs = nullptr;
  int4* d_sgd_blocks = nullptr;    // per update block: {segment, first element, count, 0}
  int n_sgd_blocks = 0;
  bool sgd_packs_w0 = false;       // the update also writes d_w0p
  // CUDA-core weight+bias gradient partials of the layers not on the tensor
  // cores (tiles of tr image rows, tiles_per_split tiles per block)
  struct RedLayer { int tr, splits, tiles_per_split; } red[4];
  float* d_bpartial = nullptr;

  void* d_x0 = nullptr;
  void* d_act[5] = {};             // d_act[i+1] = output of conv i
  void* d_dact[5] = {};
  uint8_t* d_code[4] = {};
  // g_i, the gradient w.r.t. layer i's pre-activation: layers alternate
  // between two buffers, since layer i's data gradient reads g_i while its
  // epilogue writes g_{i-1}
  void* d_g = nullptr;
  void* d_g2 = nullptr;
  void* gbuf(int i) const { return (i & 1) ? d_g2 : d_g; }
  float* d_loss_ex = nullptr;     // [C][B] per-example loss
  float* d_dlogits = nullptr;
  int32_t* d_y = nullptr;
  int32_t* d_idx = nullptr;
  int32_t* d_counts = nullptr;
  int32_t* d_active = nullptr;
  float* d_cut_scale = nullptr;    // [C][B] B / (|A| b_k), with client_average only
  int* h_err = nullptr;            // pinned copy of d_err (read back with the step statistics)
  float* d_loss = nullptr;
  int64_t* d_t = nullptr;
  float* h_loss = nullptr;         // pinned staging
  int32_t* h_active = nullptr;

  int64_t t = 0;
  gcpsl_status sticky = GCPSL_OK;
  std::string err;
  std::vector<void*> allocs;
  bool timing = false;
  KernelTimer timer;

  // CUDA graphs of one round: [epoch boundary or not][untimed, timed A, timed B].
  // The two timed copies alternate so that one copy's event pairs are read
  // while the other runs.
  int64_t launched = 0;            // kernels launched so far (eager or graph nodes)
  int64_t enqueued = 0;            // kernels passed through LAUNCH (eager or captured)
  bool capturing = false;          // a round is being captured into a graph
  struct RoundGraph {
    cudaGraphExec_t exec = nullptr;
    int64_t kernels = 0;          // kernel nodes of the captured round
    std::vector<KernelTimer::Pending> marks;
    bool unread = false;          // marks of the last launch not yet added to the timer
  };
  bool use_graph = true;
  RoundGraph graph[2][3];
  int timed_phase = 0;
};


namespace gcpsl {

gcpsl_status fail(gcpsl_ctx* c, gcpsl_status st, const char* fmt, ...);

// resnet.cu: the ResNet-18 split (architecture 2)
// the ResNet-18 split with a J-way linear head (J = 10: GCPSL_RESNET18, 100: GCPSL_RESNET18_C100)
int64_t rn_num_params(int J, int segment);       // GCPSL_CLIENT / SERVER / BN_STATE
void rn_to_kernel_layout(int J, const float* can, float* ker);
void rn_to_canonical_layout(int J, const float* ker, float* can);
void rn_seeded_init(int J, uint64_t seed, float* can);
gcpsl_status rn_setup(gcpsl_ctx* c);
void rn_free(gcpsl_ctx* c);
gcpsl_status rn_enqueue_round(gcpsl_ctx* c);
const bf16* rn_cut(const gcpsl_ctx* c, int which);
gcpsl_status rn_relu_masks(gcpsl_ctx* c, uint8_t* dst, size_t len, size_t* needed);
float* rn_bn_state(const gcpsl_ctx* c, int64_t* S, int64_t* S_pad);
gcpsl_status check_device_error(gcpsl_ctx* c);
gcpsl_status check_usable(gcpsl_ctx* c);
// 128-pixel M tile of a W x H image: bw <= 16 columns, hb rows, bb images
bool m_tile(int W, int H, int& bw, int& hb, int& bb);

#define CK(call)                                                                           \
  do {                                                                                     \
    cudaError_t _e = (call);                                                               \
    if (_e != cudaSuccess)                                                                 \
      return fail(c, _e == cudaErrorMemoryAllocation ? GCPSL_E_NOMEM : GCPSL_E_CUDA,       \
                  "%s failed: %s (%s:%d)", #call, cudaGetErrorString(_e), __FILE__, __LINE__); \
  } while (0)

// launch through the timer when enabled
#define LAUNCH(name, call)                                                                 \
  do {                                                                                     \
    const bool _t = c->timing && c->timer.wants(name);                                     \
    ++c->enqueued;                                                                         \
    if (!c->capturing) ++c->launched;                                                      \
    if (_t) c->timer.begin(name, c->stream);                                               \
    cudaError_t _e = (call);                                                               \
    if (_t) c->timer.end(c->stream);                                                       \
    if (_e != cudaSuccess)                                                                 \
      return fail(c, GCPSL_E_CUDA, "kernel %s: %s", name, cudaGetErrorString(_e));        \
  } while (0)

// synchronise the stream, then fail on a device-side timeout
#define SYNC_CHECK(c)                                        \
  do {                                                       \
    CK(cudaStreamSynchronize((c)->stream));                  \
    gcpsl_status _d = check_device_error(c);                 \
    if (_d != GCPSL_OK) return _d;                           \
  } while (0)

template <typename P>
gcpsl_status dalloc(gcpsl_ctx* c, P** p, size_t bytes) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes ? bytes : 16);
  if (e != cudaSuccess)
    return fail(c, GCPSL_E_NOMEM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  c->allocs.push_back(q);
  *p = (P*)q;
  return GCPSL_OK;
}
// a [C][splits][per] partial buffer for parameters [off, off + count) of
// every replica, summed by the update (null on allocation failure)
float* partial_range(gcpsl_ctx* c, int64_t off, int64_t count, int64_t per, int splits);
// the update's segments from the partial ranges (after every setup)
gcpsl_status build_sgd_segments(gcpsl_ctx* c);

#define DALLOC(p, bytes)                                   \
  do {                                                     \
    gcpsl_status _s = dalloc(c, &(p), (size_t)(bytes));    \
    if (_s != GCPSL_OK) return _s;                         \
  } while (0)

}  // namespace gcpsl
