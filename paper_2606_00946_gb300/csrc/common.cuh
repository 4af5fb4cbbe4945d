// Internal declarations of the Lodestar GB300 library: context layout, device
// helpers shared by the kernels, and the launchers each .cu file provides.
#pragma once

#include <utility>

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <algorithm>
#include <cstdint>
#include <mutex>
#include <vector>

#include "lodestar.h"

namespace ls {

constexpr uint64_t kG = 0x9E3779B97F4A7C15ull;  // floor(2^64 / golden ratio)
constexpr int kBlockTok = LS_BLOCK_TOKENS;
constexpr int kPair = LS_PAIR_FEATURES;

// ---------------------------------------------------------------------------
// predictor layout
// ---------------------------------------------------------------------------
struct MlpDesc {
  int n_layers;
  int w[LS_MAX_LAYERS + 1];
  int64_t woff[LS_MAX_LAYERS];   // W_l offset in the flat parameter vector
  int64_t boff[LS_MAX_LAYERS];   // b_l offset
  int64_t wtoff[LS_MAX_LAYERS];  // offset of the transposed copy W_l^T [in, out]
  int bf16;                      // 1: bf16 operands (weights, layer input, hidden activations)
  int max_width;
};

// Layout of the tensor-core scorer (k_score_tc.cu), planned once per context.
struct TcPlan {
  int n_tc = 0;                    // tensor-core layers (all but the width-1 output layer)
  int in_pad[LS_MAX_LAYERS] = {};  // K of layer l rounded up to 64
  int out[LS_MAX_LAYERS] = {};     // N of layer l
  int nc[LS_MAX_LAYERS] = {};      // N columns per MMA chunk (<= 256)
  int64_t img_off[LS_MAX_LAYERS] = {};
  int64_t chunk_off[64] = {};      // byte offset of weight chunk q (per-tile order)
  int32_t chunk_len[64] = {};
  int chunks = 0;
  int64_t img_bytes = 0;
  int chunk_bytes = 0;
  int a_bytes = 0;
  int stages = 0;
  int resident = 0;
  int smem = 0;
  uint32_t tmem_cols = 0;
  int d_pad = 0;
  int64_t w_last_off = 0;
  int64_t b_last_off = 0;
  int pipe = 0;                    // pipelined kernel applies (two hidden layers, resident weights)
  int pipe_smem = 0;
  int wide = 0;                    // wide kernel applies (two hidden layers of multiples of 128, streamed weights)
  int wide_smem = 0;
  int wide_stages = 0;
  int wide_q = 1;                  // weight slices per stage of the wide kernel
  int pair = 0;                    // pair kernel applies (two hidden layers of multiples of 256, 2-SM products)
  int pair_smem = 0;
  int pair_stages = 0;
  int pair_q = 1;                  // 16 KB half-slices per stage of the pair kernel
  int pair_slices = 0;             // half-slices per CTA per tile (the per-rank stream of the image)
  int pair_clusters = 0;           // co-resident CTA pairs (0: not queried)
};

// One published weight version (Sec. 4.3.1 P2: the routing side reads a
// version that training never writes).
struct Published {
  float* params = nullptr;  // flat, same layout as the master; weights rounded in bf16 mode
  float* wt = nullptr;      // per-layer transposed weights [in, out]
  uint8_t* img = nullptr;   // pre-swizzled bf16 hidden-layer weights (tensor-core scorer)
  float* bounds = nullptr;  // feature bounds published with the weights: lo [d], then hi [d]
  uint64_t version = 0;
};

// Counters that change with every step live in device memory so that a whole
// step (snapshot, route, log, train, publish) can be captured once in a CUDA
// graph and replayed: kernels read and advance them at execution time.
struct DevState {
  int64_t ring_count;       // records appended to the sample ring so far
  int64_t step;             // optimiser steps taken
  int32_t cur;              // published buffer routes read (-1: none yet)
  int32_t route_b;          // buffer chosen by the route in flight (set by its prefix kernel)
  uint64_t version;         // publishes completed
  uint64_t pub_version[2];  // version held by each buffer
  uint32_t done[6];         // per-kernel block arrival counters (last-block updates)
  float adam_bc[2];         // 1 - beta1^t, 1 - beta2^t of the step in flight, t = step + 1
  double beta_pow[2];       // beta1^step, beta2^step (fp64 running products)
  int64_t replay_count;     // records in the replay pool
  int64_t admitted;         // evicted stream positions below this were considered for the replay pool
  int32_t train_abort;      // set by a training step's gather (empty buffer, bad slot): the step's
                            // optimiser changes nothing and clears it
  uint32_t walk_next;       // next request of the prefix walk in flight (0 between walks)
};

// Row of training-buffer index u (Sec. 4.3.2: a round trains on F u R): ring
// slot u for u < nF, else replay record u - nF at row replay_base + u - nF.
__host__ __device__ __forceinline__ int64_t union_row(int64_t u, int64_t nF, int64_t replay_base) {
  return u < nF ? u : replay_base + (u - nF);
}

// Adam bias corrections of the coming step, 1 - beta^(step+1), from the fp64
// running powers (one multiply each, by one thread of the step's first kernel).
__device__ __forceinline__ void set_adam_bc(DevState* st) {
  st->adam_bc[0] = (float)(1.0 - st->beta_pow[0] * 0.9);
  st->adam_bc[1] = (float)(1.0 - st->beta_pow[1] * 0.999);
}

// The optimiser's last block, after a step: advance the counter and the powers.
__device__ __forceinline__ void advance_step(DevState* st, int64_t t) {
  st->step = t;
  st->beta_pow[0] *= 0.9;
  st->beta_pow[1] *= 0.999;
}
enum { DONE_RING = 0, DONE_OPT = 1, DONE_PUB = 2, DONE_BOUNDS = 3 };
enum { DONE_REPLAY = 4, DONE_WALK = 5 };  // DevState::done has 6 entries

// Kernel-level tracing: when enabled, every launch is bracketed by CUDA events
// recorded on the launching stream; ls_trace_read() sums the elapsed times.
enum TraceId {
  TR_HASH, TR_INSERT, TR_PREFIX, TR_SCORE, TR_ARGMIN, TR_ASSEMBLE, TR_RING, TR_PUBLISH,
  TR_GATHER, TR_GEMM_FWD, TR_LOSS, TR_GEMM_DW, TR_REDUCE, TR_COLSUM, TR_GEMM_DX, TR_OPT,
  TR_MEMSET, TR_SCORE_TC, TR_NORM_ROWS, TR_PUBLISH_TC, TR_HASH_BATCH, TR_SCREEN, TR_WALK,
  TR_GEMM_TC_FWD, TR_GEMM_TC_DW, TR_GEMM_TC_DX, TR_PREFIX_INDEX, TR_INDEX_INSERT,
  TR_GUARDS, TR_BOUNDS, TR_REPLAY, TR_TRAIN_STEP, TR_ROUTE_SEQ, TR_COUNT
};
extern const char* const kTraceNames[TR_COUNT];

struct Tracer {
  static constexpr int kPool = 8192;
  bool on = false;
  bool ready = false;
  cudaEvent_t ev[kPool];
  int used = 0;
  struct Pending { int id, a, launches; };
  std::vector<Pending> pend;
  int64_t launches[TR_COUNT] = {};
  int64_t timed[TR_COUNT] = {};   // launches whose time is in ms[] (the rest found the event pool full)
  double ms[TR_COUNT] = {};
  int64_t dropped = 0;
  std::mutex mu;

  int begin(cudaStream_t s) {
    if (!on) return -1;
    std::lock_guard<std::mutex> g(mu);
    if (used + 2 > kPool) return -2;
    const int t = used;
    used += 2;
    cudaEventRecord(ev[t], s);
    return t;
  }
  void end(int t, int id, int n, cudaStream_t s) {
    if (t == -1) return;
    std::lock_guard<std::mutex> g(mu);
    launches[id] += n;
    if (t < 0) { ++dropped; return; }
    cudaEventRecord(ev[t + 1], s);
    pend.push_back({id, t, n});
  }
};

// Buffers of the tensor-core training step (k_train_fast.cu): bf16 operand
// images of activations, gradients and weights, ReLU mask bits, and the
// fp32 partials the optimiser sums.
struct TrainFast {
  bool on = false;
  int rows_max = 0;                        // max_train_batch rounded up to 128
  int in_pad[LS_MAX_LAYERS] = {};          // K of layer l (input width padded to 64)
  uint8_t* imgA[LS_MAX_LAYERS] = {};       // A_l  [rows, in_pad[l]]
  uint8_t* imgAT[LS_MAX_LAYERS] = {};      // A_l^T [in_pad[l], rows]
  uint8_t* imgDZ[2] = {};                  // dz of a hidden layer [rows, width], by layer parity
  uint8_t* imgDZT[2] = {};                 // its transpose [width padded to 128, rows]
  uint16_t* mask[LS_MAX_LAYERS + 1] = {};  // bits of [A_l > 0] as [width/16][rows]
  uint8_t* imgW[LS_MAX_LAYERS] = {};       // bf16 W_l  [out, in_pad]
  uint8_t* imgWT[LS_MAX_LAYERS] = {};      // bf16 W_l^T [in_pad, out]
  float* partW[LS_MAX_LAYERS] = {};        // dW split partials [splits][out][in_pad]
  float* partB[LS_MAX_LAYERS] = {};        // db tile partials [tiles][out]
  float* partWL = nullptr;                 // output-layer dW tile partials [tiles][in]
  float* partBL = nullptr;                 // output-layer db tile partials [tiles]
  float* partLoss = nullptr;               // squared-error tile partials [tiles]
  int splits[LS_MAX_LAYERS] = {};
  uint8_t* base = nullptr;                 // allocations
  float* parts = nullptr;
};

struct Ctx {
  ls_config cfg{};
  MlpDesc mlp{};
  int d = 0;
  int64_t n_params = 0;
  int64_t wt_total = 0;

  // snapshot (Sec. 4.2): instance state rows and per-instance key tables
  int n_inst = 0;
  int64_t slots = 0;       // per-instance table slots (power of two)
  uint32_t mask = 0;
  uint64_t* tables = nullptr;
  int32_t* table_count = nullptr;
  float* inst_state = nullptr;
  float* mean = nullptr;
  float* stdv = nullptr;
  bool have_norm = false;

  // parameters and optimiser state
  float* master = nullptr;
  float* adam_m = nullptr;
  float* adam_v = nullptr;
  bool have_params = false;

  // publish / swap: two buffers, the device-side index st->cur says which
  // one routes read; a publish writes the other and flips it
  Published pub[2];
  bool have_published = false;   // a publish has been enqueued (host order)
  uint64_t version = 0;          // publishes enqueued (host order)
  cudaEvent_t ev_pub = nullptr;    // after the last publish enqueued
  cudaEvent_t ev_route = nullptr;  // after the last route enqueued
  bool pub_recorded = false, route_recorded = false;
  DevState* st = nullptr;

  // sample ring (Sec. 4.3.2): rows [0, C) the FIFO pool, [C, C + P) the
  // pending ring of evicted records, [C + P, C + P + Rc) the replay pool
  float* ring_x = nullptr;
  float* ring_y = nullptr;
  int64_t replay_base = 0;        // C + P
  // replay admission scratch
  float* remb = nullptr;          // embeddings [P + Rc, H] fp32 (candidates, then kept)
  float* rnorm = nullptr;         // |bf16(g)|^2 [P + Rc] (+inf for rows not in use)
  float* rpart = nullptr;         // row-min partials [max(P, Rc), kRowMinParts]
  float* rd = nullptr;            // d per candidate [P]
  float* rn = nullptr;            // n per kept record [Rc]
  int32_t* rinv = nullptr;        // rank -> candidate [P], then rank -> kept slot [Rc]
  int32_t* rrank = nullptr;       // rank of each candidate [P], then of each kept record [Rc]
  int64_t* rcount = nullptr;      // candidates and kept records of the round in flight [2]
  uint8_t* rimg = nullptr;        // bf16 embedding image (128-row tiles, MMA layout) for bf16 predictors
  int64_t ring_enqueued = 0;     // records appended (host order); the device count is st->ring_count
  // feature bounds of the ring (Algorithm 4 [l, u]): staged by ls_refresh_bounds,
  // published by ls_publish into pub[b].bounds
  float* bounds_stage = nullptr;  // lo [d], hi [d]
  uint32_t* benc = nullptr;       // bounds being reduced, order-preserving codes [2][d]
  ls_guards guards{};             // Algorithm 4 guard parameters of guarded routes

  // route scratch
  int32_t* hits = nullptr;    // [max_requests, max_instances]
  float* scores = nullptr;    // [max_requests, max_instances]
  // prefix index over all instances (LS_PREFIX_INDEX): key -> instance bitmask
  bool use_index = false;
  int gW = 0;                 // 64-bit mask words per slot
  int64_t gslots = 0;
  uint64_t* gkeys = nullptr;  // [gslots]
  uint64_t* gmask = nullptr;  // [gslots, gW]
  uint64_t* bkeys = nullptr;  // block keys of the batch, slot tok_off[r]/16 + b
  int64_t bkeys_cap = 0;
  uint32_t* work = nullptr;   // (request, instance) pairs that hit block 0
  int* work_n = nullptr;
  uint16_t* xin = nullptr;    // bf16 instance template rows [max_instances, d_pad]
  uint16_t* xrq = nullptr;    // bf16 request template rows [max_requests, d_pad]
  uint4* pairx = nullptr;     // bf16 pair features of each (request, instance), 16 bytes: chunk 0 of its row
  uint8_t* ximg = nullptr;    // pipelined scorer: bf16 feature rows of the batch as MMA-layout tiles
  bool use_tc = false;
  TcPlan tc;

  // train scratch
  float* tx = nullptr;        // activations a_0..a_{L-1}, [B, sum w[0..L-1]]
  float* tz = nullptr;        // pre-activations z_1..z_L, [B, sum w[1..L]]
  float* ty = nullptr;        // targets [B]
  float* dz0 = nullptr;       // [B, max_width]
  float* dz1 = nullptr;
  float* grad = nullptr;      // [n_params]
  float* gpart = nullptr;     // split-K partials (also column-sum partials)
  int64_t gpart_floats = 0;
  float* loss_tmp = nullptr;  // [1]
  TrainFast tf;               // tensor-core training buffers (when tf.on)
  int train_ctas = 0;         // > 0: persistent training step of that many CTAs
  uint32_t* tr_bar = nullptr; // [2]: its grid-barrier arrivals and abort flag

  int* d_err = nullptr;       // first device-side error (0 = none)
  int sms = 148;              // SM count of the context's device
  std::mutex mu;
  Tracer tracer;
};

inline bool capturing(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  return cudaStreamIsCapturing(s, &st) == cudaSuccess && st != cudaStreamCaptureStatusNone;
}

// Launch bracketed by trace events (skipped while the stream is being captured).
template <class F>
cudaError_t traced(Ctx& c, int id, int n_launch, cudaStream_t s, F&& f) {
  const int t = c.tracer.on && !capturing(s) ? c.tracer.begin(s) : -1;
  const cudaError_t e = f();
  c.tracer.end(t, id, n_launch, s);
  return e;
}

// ---------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float round_bf16(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

__device__ __forceinline__ void latch_error(int* err, int code) {
  atomicCAS(err, 0, code);
}

// The route's choice of published buffer, taken once per route (by thread 0
// of block 0 of its prefix kernel) so that every scorer CTA reads one version.
__device__ __forceinline__ void route_snapshot(DevState* st) {
  if (st && blockIdx.x == 0 && threadIdx.x == 0)
    st->route_b = *reinterpret_cast<volatile int32_t*>(&st->cur);
}

// True in exactly one block of the grid: the last to arrive at `done`, after
// every block has passed this point (so every block's earlier reads of the
// state it will update are done).  The counter is reset for the next launch.
__device__ __forceinline__ bool last_block(uint32_t* done) {
  __shared__ bool is_last;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t nb = gridDim.x * gridDim.y * gridDim.z;
    const uint32_t t = atomicAdd(done, 1u);
    is_last = (t == nb - 1);
    if (is_last) *done = 0u;
  }
  __syncthreads();
  return is_last;
}

// Order-preserving 32-bit code of a float: unsigned comparison of codes is
// the float comparison, -0 below +0.
__device__ __forceinline__ uint32_t ord_code(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// (a, i) precedes (b, j) in the order (score, index): NaN after every number,
// -0 == +0, ties to the lower index (the greedy selection of Algorithm 4).
__device__ __forceinline__ bool score_precedes(float a, int i, float b, int j) {
  const bool an = isnan(a), bn = isnan(b);
  if (an != bn) return bn;
  if (!an && a != b) return a < b;
  return i < j;
}

// Raw feature k of pair (request with prompt length L and hit length h,
// instance row inst, request extras req):  [L, h, 16h, 16h/L, L-16h,
// ceil(L/16)-h || inst[0..d_inst) || req[0..d_req)]  (Sec. 4.1 Features).
__device__ __forceinline__ float raw_feature(int k, int64_t L, int h, const float* inst,
                                            int d_inst, const float* req) {
  switch (k) {
    case 0: return (float)L;
    case 1: return (float)h;
    case 2: return (float)((int64_t)kBlockTok * h);
    case 3: return L > 0 ? (float)((int64_t)kBlockTok * h) / (float)L : 0.0f;
    case 4: return (float)(L - (int64_t)kBlockTok * h);
    case 5: return (float)((L + kBlockTok - 1) / kBlockTok - h);
    default: break;
  }
  k -= kPair;
  return k < d_inst ? inst[k] : req[k - d_inst];
}

// Per-feature z-score (Algorithm 4, Normalize); std below 1e-12 -> 1.
__device__ __forceinline__ float zscore(float x, float mu, float sd) {
  float s = sd < 1e-12f ? 1.0f : sd;
  return (x - mu) / s;
}

// Launch of a kernel of the route or training chain with programmatic
// dependent launch: it may start (and run what precedes its pdl_wait()) while
// the previous kernel of the stream finishes.  `cluster` > 1 adds a cluster
// dimension.
template <typename... KArgs, typename... Args>
cudaError_t launch_chained(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                           int cluster, Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int n = 1;
  if (cluster > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    n = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------------------
// launchers (each returns the launch status)
// ---------------------------------------------------------------------------
cudaError_t launch_hash_blocks(int n_seq, const int32_t* tok, const int64_t* tok_off,
                               uint64_t* keys_out, const int64_t* key_off, int64_t cap, int* err,
                               cudaStream_t s);
cudaError_t launch_hash_screen(int n_req, const int32_t* tok, const int64_t* tok_off, uint64_t* keys,
                               int64_t cap, int* err, const uint64_t* tables, uint32_t mask, int64_t slots,
                               int n_inst, int32_t* hits, uint32_t* work, int* work_n, int sms,
                               DevState* st, cudaStream_t s);
cudaError_t launch_probe_walk(int n_inst, const int64_t* tok_off, const uint64_t* keys, int64_t cap,
                              const uint64_t* tables, uint32_t mask, int64_t slots, int32_t* hits,
                              const uint32_t* work, const int* work_n, int sms, cudaStream_t s);
cudaError_t launch_table_insert(const uint64_t* keys, const int64_t* key_off, int n_inst,
                                int64_t n_keys, uint64_t* tables, uint32_t mask, int64_t slots,
                                int32_t* counts, int64_t max_keys, int* err, cudaStream_t s);
cudaError_t launch_prefix_match(int n_req, const int32_t* tok, const int64_t* tok_off,
                                const uint64_t* tables, uint32_t mask, int64_t slots, int n_inst,
                                int32_t* hits, DevState* st, cudaStream_t s);

cudaError_t launch_assemble_features(int n_req, int n_inst, const int64_t* tok_off,
                                     const int32_t* hits, const float* inst_state, int d_inst,
                                     const float* req_feats, int d_req, const float* mean,
                                     const float* stdv, float* x_out, cudaStream_t s);
cudaError_t launch_score_simt(const MlpDesc& mlp, const Published* pub, const int32_t* sel, int n_req, int n_inst,
                              const int64_t* tok_off, const int32_t* hits, const float* inst_state,
                              int d_inst, const float* req_feats, int d_req, const float* mean,
                              const float* stdv, float* scores, cudaStream_t s);
cudaError_t launch_argmin(int n_req, int n_inst, const float* scores, int32_t* choice,
                          float* best, cudaStream_t s);
// Algorithm 4 guards.  benc must hold the identity codes (0xff800000 in
// [0, d), 0x007fffff in [d, 2d)) before a bounds launch; each launch leaves
// them so.
cudaError_t launch_ring_bounds(int d, const float* ring_x, int64_t capacity, int64_t replay_base,
                               int64_t replay_capacity, uint32_t* benc, float* stage, DevState* st, int sms,
                               cudaStream_t s);
cudaError_t launch_guards(const ls_guards& g, int n_req, int n_inst, const int32_t* tok, const int64_t* tok_off,
                          const int32_t* hits, const float* scores, const float* inst, int d_inst,
                          const float* req, int d_req, const Published* pub, const DevState* st,
                          int32_t* choice, float* best, int32_t* status, int32_t* fallback, int sms,
                          cudaStream_t s);
constexpr int kGuardHeurMaxInst = 1024;  // instances the heuristic keeps in shared memory

// Plan the tensor-core scorer; `allow_pair` false leaves the pair kernel out
// (and its image layout), `allow_pipe` false the pipelined one.
bool plan_tc(const MlpDesc& m, TcPlan& p, bool allow_pair = true, bool allow_pipe = true);
// CTA pairs of the pair kernel that can be resident at once (0: none).
int pair_max_clusters(const TcPlan& p);
// Publish the master weights into buffer 1 - st->cur (fp32 params, the
// transposed copy when `want_wt`, the tensor-core image when `tc`, the staged
// feature bounds), then flip st->cur and bump the version; one launch.
cudaError_t launch_publish(const MlpDesc& m, const TcPlan* tc, const float* master, const Published* pub,
                           int want_wt, const float* bounds_stage, DevState* st, int sms, cudaStream_t s);
cudaError_t launch_norm_rows(const int64_t* tok_off, const int32_t* hits, uint4* pairx, int n_inst, int d_inst,
                             const float* inst, int n_req, int d_req,
                             const float* req, const float* mean, const float* stdv, int d_pad,
                             uint16_t* xin, uint16_t* xrq, int sms, cudaStream_t s);
size_t route_seq_smem(int n_inst, int d_inst, int wmax, int W);
cudaError_t launch_read_features(int64_t row0, int64_t n_rows, int d, const TcPlan& p, int n_inst,
                                 const uint8_t* ximg, const uint4* pairx, const uint16_t* xin, const uint16_t* xrq,
                                 uint16_t* out, cudaStream_t s);
cudaError_t launch_route_seq(int n_req, int n_inst, int d_inst, int d_req, int q_col, const int64_t* tok_off,
                             const uint64_t* bkeys, int64_t bcap, const float* req, float* inst, const float* mean,
                             const float* stdv, const Published* pub, const DevState* st, const MlpDesc& m,
                             uint64_t* gkeys, uint64_t* gmask, int W, uint64_t gslots_mask, int32_t* counts,
                             int64_t max_keys, int32_t* choice, float* best, float* scores, int32_t* hits, int* err,
                             cudaStream_t s);
cudaError_t launch_inst_templates(int n_inst, int d_inst, const float* inst, const float* mean, const float* stdv,
                                  int d_pad, uint16_t* xin, int sms, cudaStream_t s);
cudaError_t launch_feature_image(const int64_t* tok_off, const int32_t* hits, int n_inst, const uint16_t* xin,
                                 int d_inst, int n_req, int d_req, const float* req, const float* mean,
                                 const float* stdv, int d_pad, uint8_t* ximg, int sms, cudaStream_t s);
// With the pipelined kernel and n_inst dividing 32 the selector runs inside the
// scorer (choice/best written, scores only when non-NULL); see scorer_selects().
inline bool scorer_selects(const TcPlan& p, int n_inst) { return p.pipe && n_inst <= 32 && 32 % n_inst == 0; }
cudaError_t launch_score_tc(const MlpDesc& m, const TcPlan& p, const Published* pub, const int32_t* sel,
                            int n_req, int n_inst, const uint4* pairx, const uint8_t* ximg, int32_t* choice,
                            float* best,
                            const uint16_t* xin, const uint16_t* xrq, int d_inst, int d_req,
                            const float* mean, const float* stdv, float* scores, int* err, int sms,
                            cudaStream_t s);
cudaError_t launch_ring_append(int n, int d, const float* x, const float* y, float* ring_x,
                               float* ring_y, DevState* st, int64_t capacity, int64_t pending, cudaStream_t s);
// forward of B rows already in c.tx (layer inputs), keeping z_l in c.tz and a_l in c.tx;
// rows_dev (device, nullable): rows in use, the tensor-core products skip tiles past it
cudaError_t forward_rows(Ctx& c, int B, cudaStream_t s, const int64_t* rows_dev = nullptr);
cudaError_t run_replay_admit(Ctx& c, float* d_out, float* n_out, cudaStream_t s);
// row-min distance GEMM: out[row * ldp + part] = min over this CTA's columns n of
// na[row] + nb[n] - 2 sum_k A(row, k) B(n, k), skipping n == row + self_off
// rows_dev / cols_dev (device, nullable): rows / columns in use; CTAs whose
// tile starts past them write +inf partials and stop.
cudaError_t launch_rowmin_tc(int M, int N, int K, const float* A, int64_t lda, const float* B, int64_t ldb,
                             const float* na, const float* nb, int64_t self_off, float* part, int64_t ldp,
                             const int64_t* rows_dev, const int64_t* cols_dev, int* parts_used, int* err, int sms,
                             cudaStream_t s);
constexpr int kRowMinParts = 256;  // partial columns per row of rpart
cudaError_t run_train_step(Ctx& c, int batch, const int32_t* idx, int opt, float lr,
                           float* loss_out, cudaStream_t s);
cudaError_t launch_gemm_tc(int M, int N, int K, const float* A, int64_t sam, int64_t sak, const float* B,
                           int64_t sbn, int64_t sbk, int splits, int epi, float* C, int64_t ldc,
                           int64_t split_stride, const float* bias, float* act, int64_t ld_act, int hidden,
                           const float* zprev, int64_t ld_zprev, int* err, int sms, cudaStream_t s,
                           const int64_t* rows_dev = nullptr);  // rows in use (device): later tiles skip
int gemm_tc_splits_used(int K, int splits);
int index_words(int max_instances);
bool plan_train_fast(const MlpDesc& m, int max_batch, TrainFast& f);
int64_t train_fast_bytes(const MlpDesc& m, const TrainFast& f, int64_t* parts_floats);
void train_fast_bind(const MlpDesc& m, TrainFast& f, uint8_t* base, float* parts);
cudaError_t train_fast_images(Ctx& c, cudaStream_t s);
cudaError_t run_train_fast(Ctx& c, int batch, const int32_t* idx, int opt, float lr, float* loss_out,
                           cudaStream_t s);
void set_last_error(const char* msg);  // sets the text ls_last_error() returns
cudaError_t launch_prefix_index(int n_req, const int32_t* tok, const int64_t* tok_off, const uint64_t* gkeys,
                                const uint64_t* gmask, int W, uint64_t gmask_slots, int n_inst, int32_t* hits,
                                int sms, DevState* st, cudaStream_t s);
cudaError_t launch_index_insert(const uint64_t* keys, const int64_t* key_off, int n_inst, int64_t n_keys,
                                uint64_t* gkeys, uint64_t* gmask, int W, uint64_t gmask_slots, int32_t* counts,
                                int64_t max_keys, int* err, int sms, cudaStream_t s);

}  // namespace ls
