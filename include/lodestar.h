/*
 * lodestar.h -- C ABI of the GB300 routing hot path of Lodestar, an
 * online-learned LLM inference router.
 *
 * Per routing batch the library computes, for every (request, instance) pair,
 * the prefix-cache hit length of the request's prompt on the instance, the
 * pair's feature vector, the predicted TTFT of the shared reward model, and
 * per request the instance with the lowest prediction.  It also logs
 * (features, observed TTFT) records and runs minibatch training steps of the
 * predictor, publishing new weights atomically to the routing side.
 *
 * Conventions (all entry points):
 *  - Every array argument is a DEVICE pointer owned by the caller unless the
 *    comment says otherwise; it is read or written only by work enqueued on
 *    the given stream, so it must stay valid until that work completes.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Calls are asynchronous with respect to the host.
 *  - Return value: LS_OK (0) or a negative ls_status.  Argument errors are
 *    detected on the host before anything is enqueued.  Errors found on the
 *    device (table overflow, an out-of-range ring slot) are latched in the
 *    context and reported by ls_sync_status().  ls_last_error() gives a
 *    message for the last failing call on the calling thread.
 *  - No call aborts, traps or throws across the ABI.
 *  - A context is used from one host thread at a time, except that
 *    ls_route_batch (on one stream) may run concurrently with
 *    ls_log_samples / ls_train_step / ls_publish (on another stream).
 *  - Block size is 16 tokens; prompts are int32 token ids.
 *  - The counters that advance every step (records in the sample ring,
 *    optimiser steps, which published buffer routing reads, the weight
 *    version) live in device memory and are read and advanced by the kernels
 *    when they run.  So the calls of one step -- ls_snapshot_update,
 *    ls_route_batch, ls_log_samples, ls_train_step, ls_publish -- can be
 *    recorded once into a CUDA graph by stream capture and replayed; each
 *    replay behaves like issuing the calls again.  While a stream is being
 *    captured these calls skip their cross-stream ordering (the events that
 *    make a publish wait for earlier routes and a route wait for the last
 *    publish), so a replayed graph must be the context's only user while it
 *    runs, on one stream.  Host-side argument checks and the version written
 *    to *weight_version_out happen at capture time.
 */
#ifndef LODESTAR_H
#define LODESTAR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LS_MAX_LAYERS 8
#define LS_BLOCK_TOKENS 16
#define LS_PAIR_FEATURES 6

typedef struct ls_ctx ls_ctx;

typedef enum {
    LS_OK = 0,
    LS_ERR_ARG = -1,        /* invalid argument (null pointer, bad size, ...) */
    LS_ERR_CUDA = -2,       /* a CUDA runtime call failed */
    LS_ERR_OOM = -3,        /* device allocation failed */
    LS_ERR_TABLE_FULL = -4, /* an instance holds more keys than configured */
    LS_ERR_TIMEOUT = -5,    /* a bounded device-side wait gave up */
    LS_ERR_STATE = -6       /* call not valid in the current state */
} ls_status;

enum { LS_F32 = 0, LS_BF16 = 1 };      /* predictor arithmetic */
enum { LS_REPLACE = 0, LS_INSERT = 1 };/* ls_snapshot_update key modes */
enum { LS_SGD = 0, LS_ADAM = 1 };      /* ls_train_step optimisers */
enum { LS_SCORER_AUTO = 0, LS_SCORER_CUDA_CORES = 1, LS_SCORER_TENSOR_CORES = 2 };
enum { LS_PREFIX_AUTO = 0, LS_PREFIX_TWO_PHASE = 1, LS_PREFIX_FUSED = 2, LS_PREFIX_INDEX = 3 };

/* Predictor and capacity configuration, fixed at ls_create.
 * widths[0] = d = 6 + d_inst + d_req (pair features, instance state, request
 * extras), widths[1..n_layers-1] = hidden widths, widths[n_layers] = 1. */
typedef struct {
    int32_t n_layers;                    /* Linear layers, 1..LS_MAX_LAYERS */
    int32_t widths[LS_MAX_LAYERS + 1];
    int32_t d_inst;                      /* instance-state features per instance */
    int32_t d_req;                       /* request extras per request */
    int32_t dtype;                       /* LS_F32 or LS_BF16 */
    int32_t max_instances;
    int32_t max_requests;                /* per ls_route_batch call */
    int64_t max_keys_per_instance;       /* cached blocks tracked per instance */
    float max_load;                      /* hash-table load bound in (0, 1) */
    int64_t ring_capacity;               /* logged samples kept (oldest evicted) */
    int32_t max_train_batch;
    int64_t max_batch_tokens;            /* prompt tokens per ls_route_batch call (sizes the
                                            block-key scratch; more latches LS_ERR_ARG) */
    int32_t prefix_mode;                 /* LS_PREFIX_*: INDEX keeps one table over all
                                            instances (key -> instance bitmask; needs
                                            max_instances <= 512) and looks each block up once
                                            per request, stopping once no instance matches;
                                            TWO_PHASE hashes every block, then screens block 0
                                            per pair and walks the survivors in per-instance
                                            tables; FUSED probes per-instance tables per request
                                            with early exit.  AUTO = INDEX when possible, else
                                            TWO_PHASE.  All modes give identical hits. */
    int32_t scorer;                      /* LS_SCORER_*: AUTO picks the tensor-core scorer
                                            for bf16 predictors whose hidden widths are
                                            multiples of 64 (<= 512), CUDA cores otherwise;
                                            TENSOR_CORES on an unsupported shape -> LS_ERR_ARG */
    /* Two-pool training data (Sec. 4.3.2): the sample ring is the FIFO pool;
     * replay_capacity > 0 adds a replay pool of that many records, fed by
     * ls_replay_admit from the records the FIFO evicted, which wait in a
     * pending ring of pending_capacity records (>= 1 with a replay pool, 0
     * without).  0 / 0: FIFO only. */
    int64_t replay_capacity;
    int64_t pending_capacity;
    /* Dropout between hidden layers during training (Sec. 4.1 Model
     * architecture: 0.1), 0 <= dropout < 1; 0 = none.  Unit o of hidden
     * activation h (one that feeds another hidden layer) in minibatch row j
     * at optimiser step t is kept when (u >> 11) >= ceil(dropout 2^53), u =
     * mix64(mix64(dropout_seed ^ ((t << 16) | h)) ^ ((j << 20) | o)), and
     * kept units are scaled by fp32(1 / (1 - dropout)).  Needs the
     * tensor-core training path (bf16, hidden widths <= 256): LS_ERR_ARG
     * otherwise. */
    float dropout;
    uint64_t dropout_seed;
    /* Launch shape of a tensor-core training step (bf16, hidden widths <=
     * 256): <= 0 uses one launch per phase (gather, each product, optimiser;
     * the default and the faster one measured), > 0 runs the whole step as
     * one persistent launch of that many CTAs (at most the SM count) that
     * meet at a grid barrier between phases.  Results are the same bits
     * either way. */
    int32_t train_ctas;
} ls_config;

typedef struct {
    int32_t n_inst;              /* instances in the current snapshot */
    int32_t d;                   /* feature width */
    int64_t n_params;            /* predictor parameter count */
    int64_t table_slots;         /* slots per instance table */
    int64_t ring_count;          /* samples ever logged */
    int64_t train_steps;         /* training steps taken */
    uint64_t weight_version;     /* version of the last published weights, 0 = none */
    int32_t scorer;              /* LS_SCORER_CUDA_CORES or LS_SCORER_TENSOR_CORES in use */
    int64_t replay_count;        /* records in the replay pool */
    int64_t pending_count;       /* evicted records waiting for ls_replay_admit */
    int32_t tc_kernel;           /* tensor-core scorer variant routes run (ls_tc_kernel) */
} ls_info;

/* Tensor-core scorer variants (all compute the same forward; which one runs is
 * fixed by the predictor widths when the context is created):
 *   GENERIC    any bf16 predictor with hidden widths multiples of 64, <= 512;
 *   PIPELINED  two hidden layers <= 256 wide, weights resident in shared memory;
 *   PAIR       otherwise two hidden layers of multiples of 256, or three of
 *              exactly 256, and a feature width <= 128: CTA pairs running 2-SM
 *              products, weights streamed;
 *   WIDE       two hidden layers of multiples of 128 and a feature width
 *              <= 128 on one CTA per tile, where PAIR does not apply or CTA
 *              pairs cannot be resident together.
 * The environment variables LS_TC_PAIR and LS_TC_PIPE set to "0" at context
 * creation plan without the PAIR and the PIPELINED variant respectively. */
typedef enum {
    LS_TC_NONE = 0,
    LS_TC_GENERIC = 1,
    LS_TC_PIPELINED = 2,
    LS_TC_WIDE = 3,
    LS_TC_PAIR = 4
} ls_tc_kernel;

/* Number of predictor parameters: sum over layers of out*in + out. */
int64_t ls_param_count(const ls_config *cfg);

/* Create a context on the current CUDA device.  Allocates all device memory
 * the context will ever use (tables, weights, optimiser state, sample ring,
 * scratch).  *out receives the context.  LS_ERR_ARG on an invalid config,
 * LS_ERR_OOM if an allocation fails. */
int ls_create(const ls_config *cfg, ls_ctx **out);

/* Release the context and its device memory (synchronises the device). */
void ls_destroy(ls_ctx *ctx);

/* Message for the last failing call on this thread ("" if none). */
const char *ls_last_error(void);

/* Blocks until all work of the device has completed, then returns and clears
 * the first error latched by device code (LS_OK if none). */
int ls_sync_status(ls_ctx *ctx);

/* Context facts; ring_count, train_steps and weight_version are read from the
 * device after synchronising it. */
int ls_get_info(ls_ctx *ctx, ls_info *out /* host */);

/* Set the fp32 master parameters (device, ls_param_count floats: W1 [w1,w0]
 * row-major, b1 [w1], W2, b2, ...), reset optimiser state and step count
 * (synchronises `stream`).  Routing keeps using the previously published
 * weights until ls_publish. */
int ls_set_params(ls_ctx *ctx, const float *params, void *stream);
int ls_get_params(ls_ctx *ctx, float *params_out, void *stream);

/* Optimiser state for checkpointing: Adam first and second moments (device,
 * n_params floats each) and the step count (host value; both calls
 * synchronise `stream` to move it). */
int ls_get_opt_state(ls_ctx *ctx, float *m_out, float *v_out, int64_t *step_out, void *stream);
int ls_set_opt_state(ls_ctx *ctx, const float *m, const float *v, int64_t step, void *stream);

/* Per-feature normalisation statistics (Algorithm 4, Normalize): mean[d],
 * std[d] (device floats).  Features are z-scored as (x - mean) / std, with a
 * std below 1e-12 replaced by 1. */
int ls_set_normalizer(ls_ctx *ctx, const float *mean, const float *std, void *stream);

/* Cluster snapshot (Sec. 4.2 cluster snapshot manager, prefix KV-cache tracker).
 * n_inst instances; inst_state [n_inst, d_inst] row-major floats (queued and
 * running requests, inflight prefill / decode tokens, KV utilisation, ...).
 * keys: cached-block keys of each instance as CSR, keys[key_off[i] ..
 * key_off[i+1]) for instance i, key_off [n_inst+1] int64 on the device,
 * n_keys = key_off[n_inst] given on the host.  keys == NULL updates the state
 * rows only.  mode LS_REPLACE empties the tables of instances 0..n_inst-1
 * first; LS_INSERT adds to them.  A key value 0 is stored as 1 (0 marks an
 * empty slot).  More than max_keys_per_instance distinct keys in one table
 * latches LS_ERR_TABLE_FULL. */
int ls_snapshot_update(ls_ctx *ctx, int32_t n_inst, const float *inst_state,
                       const uint64_t *keys, const int64_t *key_off, int64_t n_keys,
                       int32_t mode, void *stream);

/* Block keys of token sequences (the keys the prefix tracker stores).
 * Sequence s is tok[tok_off[s] .. tok_off[s+1]) (tok_off int64 [n_seq+1]);
 * its floor(L_s/16) full blocks get keys keys_out[key_off[s] + b].
 * Definition (this library's reading; the paper says only that the prefix
 * index may be a hash table, Sec. 2):
 *   mix64 = SplitMix64 output finaliser, G = 0x9E3779B97F4A7C15;
 *   c_b = mix64( XOR_{j<8} mix64(w_{b,j} + (j+1) G) ), w_{b,j} the 64-bit word
 *         of tokens 16b+2j (low half) and 16b+2j+1 (high half);
 *   s_{-1} = G, s_b = s_{b-1} G + c_b (mod 2^64); key_b = mix64(s_b), 0 -> 1.
 * key_b depends on every token of blocks 0..b (prefix reuse is strictly
 * sequential, Sec. 2). */
int ls_hash_blocks(ls_ctx *ctx, int32_t n_seq, const int32_t *tok, const int64_t *tok_off,
                   uint64_t *keys_out, const int64_t *key_off, void *stream);

/* Normalised feature rows of all (request, instance) pairs for given hit
 * lengths (hits [n_req, n_inst] int32): row r*n_inst + i of x_out [n_req*n_inst, d]
 * is the z-scored [L, h, 16h, 16h/L, L-16h, ceil(L/16)-h || inst_state[i] ||
 * req_feats[r]] (Sec. 4.1 Features; Algorithm 4 Normalize), L = prompt length
 * from tok_off.  Parity hook; ls_route_batch computes the same rows on chip. */
int ls_assemble_features(ls_ctx *ctx, int32_t n_req, const int64_t *tok_off, const int32_t *hits,
                         const float *req_feats, float *x_out, void *stream);

/* Route a batch (Sec. 4.1 reward model, Algorithm 4): for each request r
 * (prompt tok[tok_off[r] .. tok_off[r+1]), request extras req_feats [n_req,
 * d_req]) and each snapshot instance i: hit length h[r,i] (leading full blocks
 * whose keys are all in instance i's table, stopping at the first miss),
 * features, predicted TTFT yhat[r,i] from the last published weights, and
 * choice[r] = argmin_i yhat[r,i] (ties -> lowest index, NaN last),
 * best[r] = yhat[r, choice[r]].  Optional outputs (NULL to skip):
 * scores_opt [n_req, n_inst] floats, hits_opt [n_req, n_inst] int32.
 * *weight_version_out (HOST pointer, nullable) receives the version used.
 * All requests of a batch see the same snapshot.  LS_ERR_STATE if no
 * weights were published or the snapshot is empty. */
int ls_route_batch(ls_ctx *ctx, int32_t n_req, const int32_t *tok, const int64_t *tok_off,
                   const float *req_feats, int32_t *choice, float *best, float *scores_opt,
                   int32_t *hits_opt, uint64_t *weight_version_out, void *stream);

/* Append n logged records (raw feature rows feats [n, d], observed TTFT in
 * seconds ttft [n]) to the sample ring: record j goes to slot
 * (count + j) mod ring_capacity, evicting the oldest (Sec. 4.3.2); count is
 * the number of records appended before, kept on the device.  With a replay
 * pool, every record the call evicts is first copied to the pending ring
 * (the record at stream position p to pending slot p mod pending_capacity,
 * overwriting the oldest pending record when full), and n must not exceed
 * ring_capacity (LS_ERR_ARG). */
int ls_log_samples(ls_ctx *ctx, int32_t n, const float *feats, const float *ttft, void *stream);

/* One minibatch step of the predictor on the training buffer F u R (Sec.
 * 4.3.2): index u < nF is ring slot u, nF <= u < nF + nR is replay record
 * u - nF (nF = min(count, ring_capacity), nR = records in the replay pool,
 * 0 without one).  idx [batch] int32 on the device; NULL = indices
 * (k*batch + j) mod (nF + nR) at step k; k, count and nR are the device
 * counters when the step runs.  A step before any ls_log_samples call is
 * refused with LS_ERR_STATE.  A step that still finds the buffer empty on the
 * device (records logged on another stream it is not ordered after) latches
 * LS_ERR_STATE, and a step with an idx entry outside the filled buffer
 * latches LS_ERR_ARG; such a step reads no record past the buffer and changes
 * nothing: master weights, Adam moments and the step count stay as they
 * were, and *loss_out receives NaN.
 * Loss = mean squared error of the predicted TTFT (seconds).  opt LS_SGD:
 * theta -= lr g; LS_ADAM: beta1 0.9, beta2 0.999, eps 1e-8, bias-corrected.
 * Updates the master weights only; routing sees them after ls_publish.
 * loss_out: device float (nullable) receives the minibatch loss before the
 * update. */
int ls_train_step(ls_ctx *ctx, int32_t batch, const int32_t *idx, int32_t opt, float lr,
                  float *loss_out, void *stream);

/* Atomically publish the master weights to routing (Sec. 4.3.1 P2: swap of the
 * model pointer).  One kernel writes the buffer routing is not reading and,
 * when all of it is written, switches the device-side buffer index.  Route
 * calls enqueued after this call (in host order) use the new version once
 * this stream reaches the publish point; earlier routes keep the version they
 * started with (each route takes the index once, before it scores). */
int ls_publish(ls_ctx *ctx, void *stream);

/* The bf16 feature rows the tensor-core scorer read for the last routed batch
 * (Sec. 4.1 Features; Algorithm 4 Normalize), rows row0 .. row0 + n_rows - 1
 * of the batch (row r * n_inst + i), d bf16 values each (raw bit patterns),
 * written to DEVICE out [n_rows, d].  Decoded from the buffers the scorer
 * consumes -- the feature image's operand tiles (pipelined scorer) or the pair
 * chunks and instance / request template rows the other tensor-core scorers
 * combine on chip -- so this is a parity hook on the production features, not
 * a recomputation.  Rows of the batch only (beyond it the contents are stale).
 * LS_ERR_STATE with the CUDA-core scorer (its rows never leave registers). */
int ls_read_features(ls_ctx *ctx, int64_t row0, int64_t n_rows, uint16_t *out, void *stream);

/* Sequential-commit routing (Sec. 4.2 cluster snapshot manager and prefix
 * KV-cache tracker; Sec. 4.3.1 P1: the gateway routes one request at a time):
 * the requests are routed in order, r = 0, 1, ..., and each decision is
 * committed before request r + 1 is scored:
 *   - inst_state[choice[r], queue_col] += 1 (fp32; skipped for queue_col -1):
 *     the chosen instance queues one more request;
 *   - every full-block key of prompt r joins the chosen instance's cache (the
 *     prefix index gains the instance's bit; distinct keys count against
 *     max_keys_per_instance, more latch LS_ERR_TABLE_FULL).
 * Request r is scored exactly as ls_route_batch scores it (hits, features,
 * predictor, argmin, ties to the lowest index, NaN last) against the snapshot
 * as the decisions for requests 0..r-1 left it.  The updates stay in the
 * context's snapshot after the call (until the next ls_snapshot_update).
 * scores_opt / hits_opt (DEVICE [n_req, n_inst], nullable): each request's
 * predictions and hit lengths as seen when it was decided.  Needs the prefix
 * index mode and n_inst x (widest layer) small enough for one CTA's shared
 * memory (LS_ERR_ARG otherwise; the large cluster is beyond it).  One CTA walks
 * the requests, so the call's time grows with n_req.  Other arguments, the
 * stream rules and errors are those of ls_route_batch. */
int ls_route_sequential(ls_ctx *ctx, int32_t n_req, const int32_t *tok, const int64_t *tok_off,
                        const float *req_feats, int32_t queue_col, int32_t *choice, float *best, float *scores_opt,
                        int32_t *hits_opt, uint64_t *weight_version_out, void *stream);

/* ---- Algorithm 4 guards (Sec. 4.3.1 fallback; Sec. 4.1 consistent hashing) ----
 * Per-request status of a guarded route.  The low bits say whether the
 * router decided (OK) or hands the request back to the gateway's fallback
 * heuristic (Algorithm 3) with choice -1 and best NaN:
 *   LS_ROUTE_COLD_START  fewer than n_min records were ever logged;
 *   LS_ROUTE_OOD         some raw feature of some (request, instance) pair
 *                        lies outside the published bounds [lo_j, hi_j]
 *                        (a NaN feature is outside).
 * LS_ROUTE_KFILTER is added to OK when the K-filter applied to the request. */
enum { LS_ROUTE_OK = 0, LS_ROUTE_COLD_START = 1, LS_ROUTE_OOD = 2, LS_ROUTE_KFILTER = 4 };

typedef struct {
    int64_t n_min;     /* cold start while records logged < n_min (<= 0: off) */
    int32_t ood;       /* nonzero: out-of-range check against the published bounds */
    int32_t k;         /* K-filter candidates (0: filter off) */
    int32_t kv_col;    /* instance-state column holding KV-cache utilisation */
    float tau_sat;     /* filter when mean_i inst[i, kv_col] > tau_sat ... */
    float tau_ben;     /* ... and max_i 16 h[r,i] (kappa_i |r|, hit tokens) > tau_ben */
    /* Fallback heuristic written to fallback_opt (Algorithm 3 pre-computes it
     * so that a cold-start / out-of-range status costs the gateway nothing):
     * LS_HEUR_NONE, LS_HEUR_PREFIX_LOAD (Algorithm 1) or LS_HEUR_PREFIX
     * (Algorithm 2). */
    int32_t heuristic;
    int32_t count_col[2];  /* request count c_i = inst[i, count_col[0]] (+ inst[i, count_col[1]]
                              when count_col[1] >= 0), summed in fp64 */
    float theta_imbal;     /* Algorithm 1: c_max - c_min > theta_imbal -> least loaded */
    float k_overload;      /* Algorithm 1: eligible when c_i <= mean + k_overload * std */
    float tau_prefix;      /* Algorithm 2: best prefix match kept when m > tau_prefix */
} ls_guards;

enum { LS_HEUR_NONE = 0, LS_HEUR_PREFIX_LOAD = 1, LS_HEUR_PREFIX = 2 };

/* Set the guard parameters used by later ls_route_batch_guarded calls (host
 * state, read when a route is enqueued or captured).  All off after
 * ls_create.  LS_ERR_ARG for k < 0, k > max_instances, k > 0 with kv_col
 * outside [0, d_inst), an unknown heuristic, a heuristic with count_col[0]
 * outside [0, d_inst) or count_col[1] outside [-1, d_inst), or a heuristic
 * with max_instances > 1024. */
int ls_set_guards(ls_ctx *ctx, const ls_guards *g /* host */);

/* Feature bounds of the training buffer (Algorithm 4 input [l, u]): one kernel
 * takes, for every feature column j, the smallest and largest value over the
 * records the training buffer holds when it runs (the sample ring's first
 * min(count, ring_capacity) slots and the replay pool's records; NaN values
 * skipped; a column without a number gets the empty range lo = +inf,
 * hi = -inf) into a staging copy.  The next
 * ls_publish publishes the staged bounds together with the weights, so a
 * route sees the bounds of the data its weights were trained beside.  Before
 * the first refresh the staging copy holds the empty range in every column. */
int ls_refresh_bounds(ls_ctx *ctx, void *stream);

/* One admission round of the replay pool (Sec. 4.3.2: evicted samples are
 * admitted only if their last-hidden-layer activations weighted by the
 * prediction residual are the most diverse with respect to those kept).
 * Candidates: the pending records not yet considered (stream order), m of
 * them.  With the current master weights every candidate and kept record
 * gets the embedding g = (yhat - y) a (a = last hidden activation); then
 *   d_e = min over kept j of |g_e - g_j|^2        (+inf with nothing kept),
 *   n_j = min over kept k != j of |g_j - g_k|^2   (+inf without another),
 * candidates ranked by (d desc, stream order), kept records by (n asc, slot);
 * the first free = replay_capacity - nR candidates fill the free slots, then
 * the candidate of rank free + q replaces the kept record of rank q while
 * d > n (NaN counts as -inf).  All candidates count as considered.
 * Distances are formed as |g_e|^2 + |g_j|^2 - 2 g_e.g_j with bf16 products
 * and fp32 sums on tensor cores (shapes of at least 64 x 32), else fp32.
 * d_out [pending_capacity] / n_out [replay_capacity] (DEVICE, nullable):
 * d of candidate t (t < m) and n of replay slot j (j < nR, before the round).
 * LS_ERR_STATE without a replay pool or without parameters / normaliser. */
int ls_replay_admit(ls_ctx *ctx, float *d_out, float *n_out, void *stream);

/* Copy the replay pool: DEVICE x_out [replay_capacity, d], y_out
 * [replay_capacity] (slots >= *n_out are left as they are), HOST *n_out
 * (synchronises the device). */
int ls_get_replay(ls_ctx *ctx, float *x_out, float *y_out, int64_t *n_out, void *stream);

/* Copy bounds to DEVICE lo_out [d], hi_out [d]: which = 0 the staging copy,
 * 1 the bounds routing reads now (synchronises the device). */
int ls_get_bounds(ls_ctx *ctx, int32_t which, float *lo_out, float *hi_out, void *stream);

/* ls_route_batch with the guards of Algorithm 4 and a status per request
 * (DEVICE int32 status [n_req]).  Per request, in order:
 *   1. cold start: records logged (device count when the route runs) < n_min;
 *   2. out of range (when ood): any raw feature [L, h, 16h, 16h/L, L-16h,
 *      ceil(L/16)-h || inst_state[i] || req_feats[r]] of any instance i
 *      outside [lo, hi] of the bounds published with the weights this route
 *      reads;
 *   3. choice = argmin_i yhat[r,i] as in ls_route_batch, then the K-filter
 *      (when k >= 1 and the prompt has a full block): if the mean of
 *      inst_state[:, kv_col] exceeds tau_sat (the fp64 mean: sum in instance
 *      order, divided by N) and
 *      16 max_i h[r,i] exceeds tau_ben, the candidates are the k instances
 *      with the largest rendezvous weights mix64(g ^ mix64((i+1) G)) (ties
 *      to the lower index), g = key of the prompt's first block (the prefix
 *      group, as ls_hash_blocks defines keys); a choice outside them is
 *      replaced by the argmin over them (same order).
 * Exploration and the random tiebreak of Algorithm 4 are not taken
 * (epsilon = 0, equal scores go to the lowest index).
 * fallback_opt (DEVICE int32 [n_req], nullable; written when a heuristic is
 * set): the heuristic's instance for every request, whatever its status.
 * With m_i = 16 h[r,i] / L (fp32) and c_i the request counts:
 *   Algorithm 1: if c_max - c_min > theta_imbal the least-loaded instance;
 *     else, with mu and sigma the mean and population standard deviation of
 *     c (sums in instance order, two passes, sqrt correctly rounded), the
 *     first instance with c_i <= mu + k_overload sigma in the order (m desc,
 *     c asc, index asc); none: the least loaded.  Counts, spread, mean,
 *     deviation and every comparison of counts are fp64.
 *   Algorithm 2: the largest m (lowest index) if it exceeds tau_prefix, else
 *     the least loaded.
 * Least loaded = smallest c_i, lowest index among equals, NaN last.
 * Other arguments, the stream rules and errors are those of ls_route_batch. */
int ls_route_batch_guarded(ls_ctx *ctx, int32_t n_req, const int32_t *tok, const int64_t *tok_off,
                           const float *req_feats, int32_t *choice, float *best, int32_t *status,
                           int32_t *fallback_opt, float *scores_opt, int32_t *hits_opt,
                           uint64_t *weight_version_out, void *stream);

/* Kernel tracing.  While enabled, each kernel launch of this context is
 * bracketed by CUDA events on its launching stream (a few microseconds of host
 * time per launch; launches recorded into a CUDA graph are not traced).
 * ls_trace_read synchronises the device, writes up to max_entries per-kernel
 * totals to the HOST array out, sets *n_out, and resets the totals: launches
 * counted, total_ms summed over the timed_launches of them that got events
 * (8192 events are pooled between reads; later launches are counted only). */
typedef struct {
    char name[32];
    int64_t launches;
    double total_ms;
    int64_t timed_launches;
} ls_trace_entry;

int ls_trace_enable(ls_ctx *ctx, int32_t on);
int ls_trace_read(ls_ctx *ctx, ls_trace_entry *out, int32_t max_entries, int32_t *n_out);

/* Prefix hit lengths without any device allocation (no counterpart in the
 * paper).  Computes the same h[r, i] as the prefix stage of ls_route_batch --
 * the number of leading full blocks of prompt r whose keys are all in
 * instance i's table -- using the two-phase kernels (hash + block-0 screen,
 * then a walk of the pairs that hit block 0), but needs no context and takes
 * its scratch from one statically sized device array compiled into the
 * library.
 *
 * Who needs it: callers that must not allocate device memory while routing --
 * a routing thread that is latency-critical (cudaMalloc/cudaFree can
 * synchronise the device), code inside stream capture (allocation calls are
 * not capturable), and plugins inside a host process whose memory pool owns
 * all device memory.  The cost: LS_STATIC_SCRATCH_BYTES of device memory is
 * reserved on every GPU the library is loaded on, for the life of the process.
 *
 *   n_req       requests (>= 0; 0 returns LS_OK with nothing enqueued)
 *   tok         DEVICE int32 tokens of the batch (CSR values)
 *   tok_off     DEVICE int64 [n_req + 1] CSR offsets (non-decreasing)
 *   n_tokens    HOST copy of tok_off[n_req] - tok_off[0]; the call checks the
 *               batch's block count against LS_STATIC_MAX_BLOCKS with it, and
 *               that check is only as good as this value: if it understates
 *               the span, blocks past the static capacity count as misses
 *               (hits come out short, nothing is written out of bounds) and
 *               no status reports it.
 *   tables      DEVICE uint64 [n_inst * slots_per_instance]: per-instance
 *               open-addressing tables of block keys (key 0 = empty slot,
 *               linear probing from key & (slots - 1)), 16-byte aligned
 *   slots_per_instance  power of two in [16, 2^31]
 *   n_inst      instances (>= 1)
 *   hits_out    DEVICE int32 [n_req, n_inst] row-major, fully overwritten
 *   stream      cudaStream_t (NULL = legacy default stream)
 *
 * Scratch: keys [LS_STATIC_MAX_BLOCKS] uint64, a work list of
 * [LS_STATIC_MAX_PAIRS] uint32, and two int32 counters that must start at
 * zero for every call; the call zeroes them itself with cudaMemsetAsync on
 * `stream`, before its kernels.  The scratch is shared by every caller on a
 * device, so two calls whose kernels overlap in time (different streams,
 * different host threads) race and may return wrong hit lengths: serialise
 * them on one stream or with events.
 * The first call on a device (with that device current) looks up the
 * scratch address with cudaGetSymbolAddress and keeps it for the life of the
 * process; make that first call outside any stream capture.  After a
 * cudaDeviceReset (or any teardown of the device's primary context) the kept
 * address is stale and calls on that device are undefined.  Returns LS_ERR_ARG for bad arguments or a batch
 * beyond the static limits (with a message in ls_last_error), LS_ERR_CUDA if
 * the lookup or a launch fails, else LS_OK once the work is enqueued. */
#define LS_STATIC_MAX_BLOCKS 262144 /* full 16-token blocks per batch */
#define LS_STATIC_MAX_PAIRS 262144  /* n_req * n_inst per batch */
#define LS_STATIC_SCRATCH_BYTES (LS_STATIC_MAX_BLOCKS * 8 + LS_STATIC_MAX_PAIRS * 4 + 256)
int ls_prefix_hits_static(int32_t n_req, const int32_t *tok, const int64_t *tok_off, int64_t n_tokens,
                          const uint64_t *tables, int64_t slots_per_instance, int32_t n_inst,
                          int32_t *hits_out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* LODESTAR_H */
