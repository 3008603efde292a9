// gcpsl_sample_round_noalloc: the GPSL round sampler for callers that cannot
// allocate device memory.  The sampler's working storage (one 64-bit key and
// one permutation slot per example, plus the per-cluster offsets, round
// counts and the round number) lives in a fixed-size file-scope __device__
// array instead of memory from cudaMalloc.  Every GPU that loads the library
// holds this array (kScratchBytes, about 3.2 MB) until the process exits.
//
// The entry point computes, for round `round` of every cluster, the same
// batch that gcpsl_step draws: the epoch permutation of the cluster's
// examples (Philox4x32-10 keys, exact rank sort), the slice of round
// round mod r_n, its (owner, id) order, the per-client counts and |A|.
// Unlike the context, it rebuilds the epoch permutation on every call.
#include <cstring>
#include <vector>

#include "common.cuh"
#include "gcpsl.h"

namespace gcpsl {

namespace {

constexpr int64_t kMaxExamples = 1 << 18;   // examples over all clusters of one call
constexpr int kMaxClusters = 1024;
constexpr int kMaxDevices = 64;

// byte layout of the scratch array
constexpr int64_t kKeysOff = 0;                                   // uint64 [kMaxExamples]
constexpr int64_t kPermOff = kKeysOff + 8 * kMaxExamples;         // int32 [kMaxExamples]
constexpr int64_t kOffOff = kPermOff + 4 * kMaxExamples;          // int64 [kMaxClusters + 1]
constexpr int64_t kRoundsOff = kOffOff + 8 * (kMaxClusters + 1);  // int32 [kMaxClusters]
constexpr int64_t kTOff = (kRoundsOff + 4 * kMaxClusters + 7) / 8 * 8;   // int64
constexpr int64_t kScratchBytes = kTOff + 8;

static __device__ __align__(256) unsigned char g_sample_scratch[kScratchBytes];

// Host-side cache of the scratch array's device address, one per device.  In
// host code `g_sample_scratch` is only a stand-in symbol, so the address must
// come from cudaGetSymbolAddress with the device current.
unsigned char* g_scratch_addr[kMaxDevices] = {};

// keys of every example of every cluster for the epoch that contains `round`
__global__ void k_keys_any_round(const int32_t* __restrict__ ids, const int64_t* __restrict__ off,
                                 const int32_t* __restrict__ rounds, const int64_t* __restrict__ t,
                                 int cluster_base, uint32_t s0, uint32_t s1,
                                 uint64_t* __restrict__ keys) {
  const int c = blockIdx.y;
  const uint32_t epoch = (uint32_t)(*t / rounds[c]);
  const int64_t base = off[c], n = off[c + 1] - base;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  uint32_t ctr[4] = {(uint32_t)ids[base + i], epoch, (uint32_t)(cluster_base + c), 0u};
  philox4x32_10(ctr, s0, s1);
  keys[base + i] = ((uint64_t)ctr[0] << 32) | ctr[1];
}

// perm[base + rank] = id, rank = #{m : (k_m, id_m) < (k_i, id_i)}
__global__ void __launch_bounds__(256)
k_rank_any_round(const int32_t* __restrict__ ids, const int64_t* __restrict__ off,
                 const uint64_t* __restrict__ keys, int32_t* __restrict__ perm) {
  __shared__ uint64_t sk[256];
  __shared__ int32_t sj[256];
  const int c = blockIdx.y;
  const int64_t base = off[c], n = off[c + 1] - base;
  if ((int64_t)blockIdx.x * blockDim.x >= n) return;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const bool mine = i < n;
  const uint64_t ki = mine ? keys[base + i] : 0;
  const int32_t ji = mine ? ids[base + i] : 0;
  int64_t rank = 0;
  for (int64_t t0 = 0; t0 < n; t0 += 256) {
    const int64_t m = t0 + threadIdx.x;
    if (m < n) { sk[threadIdx.x] = keys[base + m]; sj[threadIdx.x] = ids[base + m]; }
    __syncthreads();
    const int lim = (n - t0) < 256 ? (int)(n - t0) : 256;
    for (int q = 0; q < lim; ++q) rank += sk[q] < ki || (sk[q] == ki && sj[q] < ji);
    __syncthreads();
  }
  if (mine) perm[base + rank] = ji;
}

unsigned char* scratch_for_current_device(gcpsl_status* st) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *st = GCPSL_E_CUDA;
    return nullptr;
  }
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_sample_scratch) != cudaSuccess || !p) {
      *st = GCPSL_E_CUDA;
      return nullptr;
    }
    g_scratch_addr[dev] = static_cast<unsigned char*>(p);
  }
  *st = GCPSL_OK;
  return g_scratch_addr[dev];
}

}  // namespace

}  // namespace gcpsl

using namespace gcpsl;

extern "C" gcpsl_status gcpsl_sample_round_noalloc(
    const int32_t* ids, const int64_t* cluster_offsets, const int32_t* owner,
    const int32_t* labels, int K, int C, int B, int64_t round, int cluster_id_base, uint64_t seed,
    int32_t* idx, int32_t* counts, int32_t* active, int32_t* batch_labels, void* stream) {
  if (!ids || !cluster_offsets || !owner || !labels || !idx || !counts || !active ||
      !batch_labels) {
    set_global_error("gcpsl_sample_round_noalloc: NULL pointer");
    return GCPSL_E_INVAL;
  }
  if (C < 1 || C > kMaxClusters || K < 1 || B < 1 || B > 1024 || round < 0) {
    set_global_error("gcpsl_sample_round_noalloc: need 1 <= C <= 1024, K >= 1, "
                     "1 <= B <= 1024 and round >= 0");
    return GCPSL_E_INVAL;
  }
  if (cluster_offsets[0] != 0) {
    set_global_error("gcpsl_sample_round_noalloc: cluster_offsets[0] must be 0");
    return GCPSL_E_INVAL;
  }
  std::vector<int32_t> r(C);
  int64_t max_nc = 0;
  for (int c = 0; c < C; ++c) {
    const int64_t nc = cluster_offsets[c + 1] - cluster_offsets[c];
    if (nc < B) {
      set_global_error("gcpsl_sample_round_noalloc: a cluster holds fewer than B examples");
      return GCPSL_E_INVAL;
    }
    r[c] = (int32_t)(nc / B);
    if (nc > max_nc) max_nc = nc;
  }
  if (cluster_offsets[C] > kMaxExamples) {
    set_global_error("gcpsl_sample_round_noalloc: more than 262144 examples over all clusters "
                     "(the fixed scratch holds 262144)");
    return GCPSL_E_INVAL;
  }
  gcpsl_status st;
  unsigned char* sc = scratch_for_current_device(&st);
  if (!sc) {
    set_global_error("gcpsl_sample_round_noalloc: cudaGetSymbolAddress of the scratch failed");
    return st;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint64_t* keys = reinterpret_cast<uint64_t*>(sc + kKeysOff);
  int32_t* perm = reinterpret_cast<int32_t*>(sc + kPermOff);
  int64_t* off = reinterpret_cast<int64_t*>(sc + kOffOff);
  int32_t* rounds = reinterpret_cast<int32_t*>(sc + kRoundsOff);
  int64_t* t = reinterpret_cast<int64_t*>(sc + kTOff);
  // every word the kernels read is rewritten here: nothing carries over from
  // the previous call
  cudaError_t e = cudaMemcpyAsync(off, cluster_offsets, sizeof(int64_t) * (C + 1),
                                  cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(rounds, r.data(), sizeof(int32_t) * C, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(t, &round, sizeof(int64_t), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) {
    const dim3 grid((unsigned)((max_nc + 255) / 256), (unsigned)C);
    k_keys_any_round<<<grid, 256, 0, s>>>(ids, off, rounds, t, cluster_id_base, (uint32_t)seed,
                                          (uint32_t)(seed >> 32), keys);
    k_rank_any_round<<<grid, 256, 0, s>>>(ids, off, keys, perm);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess)
    e = launch_sample(s, perm, off, rounds, rounds, t, owner, labels, K, B, C, idx, counts,
                      active, batch_labels, nullptr);
  // the host copies above read pageable memory; finish them before the
  // vectors go out of scope
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    set_global_error(cudaGetErrorString(e));
    return GCPSL_E_CUDA;
  }
  return GCPSL_OK;
}
