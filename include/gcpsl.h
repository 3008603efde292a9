/*
 * gcpsl.h -- C ABI of the GB300 GCPSL training-step library (libgcpsl.so).
 *
 * GCPSL ("Concurrent Split Learning Through Stable Client Clustering",
 * Kohankhaki, Rentschler, Schmeink) assigns K clients to N fixed clusters,
 * runs one GPSL workload with a fixed batch B per cluster, and fuses the
 * split-model replicas every F local rounds (Algorithm 2).  This library
 * keeps the C cluster replicas (the paper's N) resident on one GPU and runs
 * one local round of all of them per call, as grouped CUDA kernels with the
 * replica index in the grid.
 *
 * Conventions shared by every entry point
 *  - Every call returns a gcpsl_status and never aborts the process.
 *  - Host pointers passed in are owned by the caller.  gcpsl_init copies
 *    what it needs (except the images with data_on_host = 1, see below), so
 *    the caller may free its arrays after init returns.
 *  - The context owns all device memory it allocates; gcpsl_destroy frees it.
 *  - gcpsl_step and gcpsl_fuse are asynchronous on the context's stream;
 *    every getter synchronises that stream first.
 *  - After a CUDA error or a device-side timeout the context is "sticky":
 *    later calls return GCPSL_E_STATE.  gcpsl_last_error describes the cause.
 *  - One host thread at a time per context.
 */
#ifndef GCPSL_H
#define GCPSL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  GCPSL_OK = 0,
  GCPSL_E_INVAL = 1,        /* bad argument (value, size, NULL) */
  GCPSL_E_NOMEM = 2,        /* host or device allocation failed */
  GCPSL_E_CUDA = 3,         /* a CUDA runtime call failed */
  GCPSL_E_STATE = 4,        /* call on a context in the error state */
  GCPSL_E_TIMEOUT = 5,      /* a device-side wait gave up */
  GCPSL_E_UNSUPPORTED = 6   /* architecture / dtype combination not built */
} gcpsl_status;

/* Split-model architectures.  Conv layers are 3x3, stride 1, padding 1, with
 * bias, each followed by ReLU; "pool" is a 2x2 stride-2 max-pool.
 *  TINY_CNN : client conv 3->16 pool | server conv 16->32 pool, FC 2048->10
 *  SPLIT_CNN: client conv 3->32, conv 32->64 pool (cut 64x16x16) |
 *             server conv 64->128 pool, conv 128->128 pool, FC 2048->10
 *  RESNET18 : the CIFAR ResNet-18 split after stage 1 (Section V-A): client
 *             conv3x3 3->64 stem + GroupNorm(32) + ReLU, stage 1 (two basic
 *             blocks of 64 channels, GroupNorm) (cut 64x32x32) | server
 *             stages 2-4 (128/256/512 channels, stride 2, train-mode
 *             BatchNorm), global average pool, FC 512->10; no conv bias
 *  RESNET18_C100: the same split with FC 512->100 (the CIFAR-100 shape)   */
enum { GCPSL_TINY_CNN = 0, GCPSL_SPLIT_CNN = 1, GCPSL_RESNET18 = 2, GCPSL_RESNET18_C100 = 3 };
enum { GCPSL_F32 = 0, GCPSL_BF16 = 1 };
enum { GCPSL_CLIENT = 0, GCPSL_SERVER = 1, GCPSL_BN_STATE = 2 };
enum { GCPSL_CUT_ACT = 0, GCPSL_CUT_GRAD = 1 };

/* Model and optimiser description.
 *  operand_dtype: GCPSL_F32 computes in fp32 throughout; GCPSL_BF16 stores
 *    weights (as a shadow of the fp32 master), activations and gradients of
 *    activations in bf16 and accumulates in fp32.
 *  SGD follows PyTorch: g += weight_decay*theta; v = momentum*v + g (v starts
 *    at 0, so the first round takes v = g); theta -= lr*(nesterov ? g +
 *    momentum*v : v); with momentum 0, theta -= lr*g.
 *  label_smoothing e: cross-entropy target (1-e)*onehot + e/classes.
 *  cluster_id_base: cluster n draws its sampler keys with cluster id
 *    cluster_id_base + n (lets C one-cluster contexts reproduce one
 *    C-cluster context exactly).
 *  data_on_host: 0 = images copied to device memory at init; 1 = images stay
 *    in pinned, device-mapped host memory owned by the context and each round
 *    gathers its B sampled images per cluster from there.
 *  augment: 0 = the sampled images as stored; 1 = the training augmentation
 *    of Section V-A (random crop from the 4-pixel zero-padded image, then a
 *    random horizontal flip), drawn per round, cluster and batch position
 *    from Philox4x32-10 with counter (b, t, cluster_id_base + n, 1) and key
 *    `seed`: dy = (o0 * 9) >> 32, dx = (o1 * 9) >> 32, flip = o2 & 1, and
 *    out[ch][y][x] = img[ch][y + dy - 4][x' + dx - 4], x' = flip ? 31 - x : x,
 *    0 outside the image.  (The synthetic images are N(0,1) already, so the
 *    dataset normalisation of Section V-A is the identity.)
 *  gn_groups, bn_momentum, norm_eps (ResNet-18 split; Section IV-B keeps
 *    BatchNorm in the server and puts GroupNorm in the client without fixing
 *    these): GroupNorm's group count, one of 1, 2, 4, 8, 16, 32 (0 selects
 *    32); the BatchNorm running-statistics momentum in (0, 1] (0 selects
 *    PyTorch's 0.1); the eps of both norms, > 0 (0 selects 1e-5).
 *  client_average: how a cluster's client gradient averages the round's
 *    active clients (Sec. IV-B).  0 (default): the gradient of the
 *    batch-mean loss, i.e. each client weighted by its b_{k,t} examples.
 *    1: the unweighted mean over the active clients A of each client's
 *    mean-loss gradient: the gradient at the cut is multiplied, example by
 *    example, by B / (|A| b_{k,t}) before the client segment's backward
 *    (the server segment keeps the batch mean; gcpsl_get_cut's gradient is
 *    the scaled one).                                                     */
typedef struct {
  int arch;
  int operand_dtype;
  float lr, momentum, weight_decay;
  int nesterov;
  float label_smoothing;
  int cluster_id_base;
  int data_on_host;
  int augment;
  int gn_groups;
  float bn_momentum, norm_eps;
  int client_average;
} gcpsl_model_desc;

/* Training data of all K clients (Section III-A: client k owns D_k).
 *  images: n x 3 x 32 x 32 fp32, NCHW;  labels: n values in [0, classes);
 *  owner: client id of each example, in [0, K).                          */
typedef struct {
  const float* images;
  const int32_t* labels;
  const int32_t* owner;
  int64_t n;
  int num_classes;        /* the architecture's: 100 for RESNET18_C100, else 10 */
} gcpsl_dataset;

/* Per-round statistics, written by gcpsl_step when non-NULL (forces a sync).
 *  loss[n]: mean softmax cross-entropy of cluster n's batch;
 *  active[n]: |A_{n,t}|, clients that supplied >= 1 example (Eq. 3).     */
typedef struct {
  float* loss;            /* caller-owned, C entries */
  int32_t* active;        /* caller-owned, C entries */
} gcpsl_step_stats;

typedef struct gcpsl_ctx gcpsl_ctx;

/* gcpsl_init -- set up C cluster workloads (Algorithm 2, "initialize all
 * split-model replicas equally").
 *  desc: model/optimiser; K clients; C clusters;
 *  assignment[K]: cluster of each client (Algorithm 1's fixed map), in
 *    [0, C), or -1 for a client this context does not serve;
 *  B: per-cluster batch (Eq. 1, sum_k b_{k,t} = B); F: fuse after every F-th
 *    round (0 = never; gcpsl_fuse can still be called), every cluster taking
 *    a local round every round (lockstep); or F = -1: the epoch schedule of
 *    Section IV-C -- a system epoch is R = max_n r_n rounds (r_n = n_c / B),
 *    cluster n takes local rounds 0 .. r_n - 1 of it and then waits at the
 *    fusion barrier (no padded optimizer step, no BatchNorm-state update;
 *    its batch in a waiting round is its last one, computed but not
 *    applied, reported with loss 0 and |A| = 0), and the replicas are fused
 *    after every system epoch;
 *  seed: sampler seed (Philox4x32-10 key);
 *  data: the dataset (see gcpsl_dataset);
 *  init_params: NULL or the initial parameters of one replica as fp32, client
 *    segment then server segment, each in PyTorch state_dict order (conv
 *    weights OIHW, linear weight [out][in]); NULL draws them from a fixed
 *    Philox stream as U(-1/sqrt(fan_in), 1/sqrt(fan_in));
 *  out: receives the context.
 * Rejects (GCPSL_E_INVAL): NULL pointers, K/C/B <= 0, F < -1, norm
 * hyper-parameters outside the ranges above, augment or client_average
 * other than 0 / 1, assignment
 * outside [-1, C), owner outside [0, K), num_classes other than the
 * architecture's, labels outside [0, num_classes), a cluster with fewer
 * than B examples.  Fusion weights are
 * q_n = n_c / sum_m n_m over this context's clusters (Eq. 5).            */
gcpsl_status gcpsl_init(const gcpsl_model_desc* desc, int K, int C, const int32_t* assignment,
                        int B, int F, uint64_t seed, const gcpsl_dataset* data,
                        const float* init_params, gcpsl_ctx** out);

/* gcpsl_step -- one local round of every cluster (Algorithm 2's inner loop
 * body): GPSL sampling of B examples (Eq. 1; epoch = one pass over a random
 * permutation of the cluster's examples, the n_c mod B remainder left out),
 * client-segment forward to the cut, server forward, softmax cross-entropy
 * (mean over the batch), backward to the cut gradient and through the client
 * segment, and an SGD update of every replica; then, when the number of
 * rounds taken is a multiple of F, fusion (Eq. 5).  stats may be NULL.   */
gcpsl_status gcpsl_step(gcpsl_ctx* ctx, gcpsl_step_stats* stats);

/* gcpsl_fuse -- Eq. 5: theta_bar = sum_n q_n theta_n for all parameters,
 * written back to every replica (Section IV-C broadcast).  Momentum buffers
 * stay per replica.                                                      */
gcpsl_status gcpsl_fuse(gcpsl_ctx* ctx);

/* gcpsl_get_params -- copy replica `cluster`'s parameters of `segment`
 * (GCPSL_CLIENT / GCPSL_SERVER) as fp32 in the init_params order into dst.
 * With the ResNet-18 split, segment GCPSL_BN_STATE gives the BatchNorm
 * running statistics (per BatchNorm layer in module order: running_mean
 * then running_var; fused with q like the parameters, Eq. 5).
 * dst == NULL (or len too small) only reports the needed count in *needed
 * (and returns GCPSL_E_INVAL if dst is non-NULL but too small).          */
gcpsl_status gcpsl_get_params(gcpsl_ctx* ctx, int cluster, int segment, float* dst, size_t len,
                              size_t* needed);

/* gcpsl_set_params -- overwrite replica `cluster`'s parameters (both
 * segments, init_params order and length).  Momentum is left unchanged.  */
gcpsl_status gcpsl_set_params(gcpsl_ctx* ctx, int cluster, const float* src, size_t len);

/* gcpsl_set_bn_state -- overwrite replica `cluster`'s BatchNorm running
 * statistics (ResNet-18 split only; len = gcpsl_num_params(arch,
 * GCPSL_BN_STATE)).                                                       */
gcpsl_status gcpsl_set_bn_state(gcpsl_ctx* ctx, int cluster, const float* src, size_t len);

/* gcpsl_get_momentum / gcpsl_set_momentum -- replica `cluster`'s SGD
 * momentum buffer (Section IV-C: optimiser state stays per replica), both
 * segments in the init_params order; len must equal the parameter count.
 * With set_params this checkpoints and restores a replica exactly.       */
gcpsl_status gcpsl_get_momentum(gcpsl_ctx* ctx, int cluster, float* dst, size_t len);
gcpsl_status gcpsl_set_momentum(gcpsl_ctx* ctx, int cluster, const float* src, size_t len);

/* gcpsl_get_pool_codes -- the last round's max-pool decisions of conv layer
 * `layer` (0-based over client then server layers; it must be pooled), one
 * byte per pooled output, laid out [C][B][channels][h/2][w/2]: bits 0-1 are
 * the window position of the first maximum in row-major order, bit 2 is set
 * when that maximum is positive (the output then carries a gradient).     */
gcpsl_status gcpsl_get_pool_codes(gcpsl_ctx* ctx, int layer, uint8_t* dst, size_t len);

/* gcpsl_get_relu_masks -- ResNet-18 split only: the last round's ReLU
 * decisions, one byte per activation (1: the ReLU output is positive),
 * laid out [C][B][E] with, per example, the stem's decisions, then for
 * each of the 8 blocks those of its inner ReLU (a1) and of its output, each
 * in [channels][h][w] order (E = 64*32*32 + sum over blocks of 2*ch*h*w).
 * A test's record of which branch of every ReLU the round took.
 * dst == NULL only reports the count in *needed.                          */
gcpsl_status gcpsl_get_relu_masks(gcpsl_ctx* ctx, uint8_t* dst, size_t len, size_t* needed);

/* gcpsl_get_cut -- the last round's cut activation z (GCPSL_CUT_ACT) or cut
 * gradient dL/dz (GCPSL_CUT_GRAD) of every cluster as fp32, laid out
 * [C][B][channels][h][w].  len is in floats; dst NULL reports nothing but
 * returns GCPSL_E_INVAL (use gcpsl_cut_elems).                           */
gcpsl_status gcpsl_get_cut(gcpsl_ctx* ctx, int which, float* dst, size_t len);
size_t gcpsl_cut_elems(const gcpsl_ctx* ctx);

/* gcpsl_get_sample -- the last round's batches: idx[C][B] global example
 * ids ordered by (owner, id) within each cluster, and counts[C][K] with
 * counts[n][k] = b_{k,t} of Eq. 1 (0 for clients outside cluster n).
 * Either pointer may be NULL.                                            */
gcpsl_status gcpsl_get_sample(gcpsl_ctx* ctx, int32_t* idx, int32_t* counts);

/* gcpsl_num_params -- parameters per replica of a segment (-1: bad arch). */
int64_t gcpsl_num_params(int arch, int segment);

/* gcpsl_rounds -- local rounds taken so far.                             */
int64_t gcpsl_rounds(const gcpsl_ctx* ctx);

/* gcpsl_set_stream -- run on the caller's cudaStream_t (passed as void*);
 * NULL returns to the context's own stream.  Synchronises the old stream. */
gcpsl_status gcpsl_set_stream(gcpsl_ctx* ctx, void* cuda_stream);

/* gcpsl_set_graph -- rounds after the first are replayed from CUDA graphs
 * (default on): each round variant (epoch boundary or not, timed or not) is
 * captured from the stream on first use and relaunched with one
 * cudaGraphLaunch.  A replay enqueues exactly the kernels and arguments of
 * the eager path, so results are identical bit for bit; 0 switches to eager
 * launches.  Synchronises the stream.  Not part of the paper: a launch-cost
 * measure for small rounds.                                              */
gcpsl_status gcpsl_set_graph(gcpsl_ctx* ctx, int enable);

/* Kernel timing: when enabled, every kernel the context launches is
 * bracketed by CUDA events on its stream (event-record nodes in a graph).  gcpsl_kernel_times fills, for up
 * to `cap` kernel kinds, the name (static string), the number of launches
 * and the summed device milliseconds since the last reset, and returns the
 * number of kinds (synchronises).                                        */
gcpsl_status gcpsl_set_timing(gcpsl_ctx* ctx, int enable);
/* gcpsl_kernels_launched -- kernels the context has launched so far
 * (eager launches and the kernel nodes of replayed graphs); -1 for NULL.  */
int64_t gcpsl_kernels_launched(const gcpsl_ctx* ctx);

/* gcpsl_set_timing_filter -- time only the kernels whose name starts with
 * `prefix` (NULL or "" = all), so that a timed round carries few event
 * records.  Synchronises the stream.                                     */
gcpsl_status gcpsl_set_timing_filter(gcpsl_ctx* ctx, const char* prefix);
int gcpsl_kernel_times(gcpsl_ctx* ctx, const char** names, int64_t* launches, double* ms,
                       int cap);
void gcpsl_reset_kernel_times(gcpsl_ctx* ctx);

/* gcpsl_sample_round_noalloc -- the GPSL round sampler of gcpsl_step for
 * callers that cannot allocate device memory.  The paper has no counterpart:
 * this is a deployment variant.  It is for code that may not call cudaMalloc
 * while it runs, e.g. a plug-in inside a host framework whose allocator owns
 * the whole device, or a process that reserves all of its device memory up
 * front and forbids later allocations.  The caller passes every input and
 * output; the entry point calls no cudaMalloc, cudaFree or other allocating
 * routine.  Its working storage is a fixed file-scope device array of about
 * 3.2 MB, which every GPU that loads the library holds until the process
 * exits.
 *
 * It returns, for round `round` (0-based) of C clusters, the batches that a
 * context with the same clusters, B, seed and cluster_id_base draws in that
 * round (gcpsl_get_sample), including the epoch permutation rebuild.
 *  ids:             device, the clusters' example ids concatenated, each
 *                   cluster's ids in ascending order (cluster n owns
 *                   ids[cluster_offsets[n] .. cluster_offsets[n+1]));
 *  cluster_offsets: host, C+1 entries, cluster_offsets[0] = 0;
 *  owner, labels:   device, indexed by example id;
 *  idx:             device out [C][B], ids ordered by (owner, id);
 *  counts:          device out [C][K], b_{k,t} (Eq. 1);
 *  active:          device out [C], |A_{n,t}|;
 *  batch_labels:    device out [C][B], labels of idx;
 *  stream:          cudaStream_t (NULL = legacy default stream).
 * Limits: 1 <= C <= 1024, 1 <= B <= 1024, every cluster >= B examples, at most
 * 262144 examples over all clusters; violations return GCPSL_E_INVAL with a
 * message in gcpsl_last_error(NULL).  The first call on a device looks up the
 * array's device address with that device current; make that first call
 * before any stream capture.  Every call shares the one array and rewrites
 * all of it that it reads, so calls do not depend on earlier ones, but calls
 * that overlap on the GPU (other streams, other host threads) race on it.
 * The call returns after the stream has finished the batch.               */
gcpsl_status gcpsl_sample_round_noalloc(const int32_t* ids, const int64_t* cluster_offsets,
                                        const int32_t* owner, const int32_t* labels, int K, int C,
                                        int B, int64_t round, int cluster_id_base, uint64_t seed,
                                        int32_t* idx, int32_t* counts, int32_t* active,
                                        int32_t* batch_labels, void* stream);

/* gcpsl_check_wait_timeout -- exercises the failure path of the library's
 * bounded device-side waits: one block waits on a shared-memory mbarrier
 * that nothing arrives on, gives up after limit_ns nanoseconds of device
 * time (1 <= limit_ns <= 1e9), sets the context's device error word and
 * exits, as every kernel of the library does when a TMA, MMA or bulk-copy
 * completion never comes.  Returns GCPSL_E_TIMEOUT (after which the context
 * is in the error state: later calls return GCPSL_E_STATE); GCPSL_E_INVAL
 * for a bad limit; GCPSL_E_STATE on a context already in the error state.
 * No fault, trap or unbounded wait is involved: the GPU stays usable for
 * other contexts.                                                         */
gcpsl_status gcpsl_check_wait_timeout(gcpsl_ctx* ctx, uint64_t limit_ns);

/* gcpsl_last_error -- static description of the context's last failure
 * (or of the last failed gcpsl_init when ctx is NULL).                   */
const char* gcpsl_last_error(const gcpsl_ctx* ctx);

/* gcpsl_destroy -- free the context (NULL is a no-op).                   */
void gcpsl_destroy(gcpsl_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* GCPSL_H */
