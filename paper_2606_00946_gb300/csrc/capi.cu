// C ABI entry points (include/lodestar.h): argument checks, the context's
// device memory, stream ordering of publish / route, and error reporting.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "common.cuh"

using namespace ls;

namespace ls {
const char* const kTraceNames[TR_COUNT] = {
    "hash_blocks", "table_insert", "prefix_match", "score_simt", "argmin", "assemble_features",
    "ring_append", "publish", "train_gather", "gemm_fwd", "loss_grad", "gemm_dw", "reduce_dw",
    "colsum_db", "gemm_dx", "optimizer", "memset", "score_tc", "features", "publish_tc",
    "hash_screen", "probe_screen", "probe_walk", "gemm_tc_fwd", "gemm_tc_dw", "gemm_tc_dx", "prefix_index",
    "index_insert", "guards", "ring_bounds", "replay_admit", "train_step", "route_seq"};
}

struct ls_ctx {
  Ctx c;
};

namespace {

thread_local std::string g_err;

int fail(int code, const std::string& msg) {
  g_err = msg;
  return code;
}

int cuda_fail(cudaError_t e, const char* where) {
  g_err = std::string(where) + ": " + cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? LS_ERR_OOM : LS_ERR_CUDA;
}

}  // namespace

namespace ls {
// Message for ls_last_error() from entry points defined in other files.
void set_last_error(const char* msg) { g_err = msg; }
}  // namespace ls

namespace {

#define LS_CK(call)                                   \
  do {                                                \
    cudaError_t e_ = (call);                          \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
  } while (0)

inline cudaStream_t S(void* p) { return reinterpret_cast<cudaStream_t>(p); }

int64_t count_params(const ls_config& c) {
  int64_t n = 0;
  for (int l = 0; l < c.n_layers; ++l) n += (int64_t)c.widths[l + 1] * c.widths[l] + c.widths[l + 1];
  return n;
}

bool check_config(const ls_config* c, std::string& why) {
  if (!c) { why = "config is NULL"; return false; }
  if (c->n_layers < 1 || c->n_layers > LS_MAX_LAYERS) { why = "n_layers must be 1..8"; return false; }
  if (c->d_inst < 0 || c->d_req < 0) { why = "d_inst and d_req must be >= 0"; return false; }
  if (c->widths[0] != LS_PAIR_FEATURES + c->d_inst + c->d_req) {
    why = "widths[0] must equal 6 + d_inst + d_req";
    return false;
  }
  for (int l = 0; l <= c->n_layers; ++l)
    if (c->widths[l] < 1 || c->widths[l] > 1024) { why = "widths must be 1..1024"; return false; }
  if (c->widths[c->n_layers] != 1) { why = "the output width must be 1"; return false; }
  if (c->dtype != LS_F32 && c->dtype != LS_BF16) { why = "dtype must be LS_F32 or LS_BF16"; return false; }
  if (c->max_instances < 1 || c->max_instances > 8192) { why = "max_instances must be 1..8192"; return false; }
  if (c->max_requests < 1) { why = "max_requests must be >= 1"; return false; }
  if (c->max_keys_per_instance < 1) { why = "max_keys_per_instance must be >= 1"; return false; }
  if (!(c->max_load > 0.0f && c->max_load < 1.0f)) { why = "max_load must be in (0, 1)"; return false; }
  if (c->ring_capacity < 1) { why = "ring_capacity must be >= 1"; return false; }
  if (c->max_train_batch < 1) { why = "max_train_batch must be >= 1"; return false; }
  if (c->scorer < LS_SCORER_AUTO || c->scorer > LS_SCORER_TENSOR_CORES) { why = "bad scorer"; return false; }
  if (c->prefix_mode < LS_PREFIX_AUTO || c->prefix_mode > LS_PREFIX_INDEX) { why = "bad prefix_mode"; return false; }
  if (c->prefix_mode == LS_PREFIX_INDEX && c->max_instances > 512) {
    why = "prefix_mode INDEX needs max_instances <= 512";
    return false;
  }
  if (c->max_batch_tokens < 1) { why = "max_batch_tokens must be >= 1"; return false; }
  if (!(c->dropout >= 0.0f && c->dropout < 1.0f)) { why = "dropout must be in [0, 1)"; return false; }
  if (c->replay_capacity < 0 || c->pending_capacity < 0 || ((c->replay_capacity > 0) != (c->pending_capacity > 0))) {
    why = "replay_capacity and pending_capacity must both be 0 or both be >= 1";
    return false;
  }
  const double need = std::ceil((double)c->max_keys_per_instance / (double)c->max_load);
  if (need > (double)(1ull << 31)) { why = "table would exceed 2^31 slots"; return false; }
  return true;
}

int64_t table_slots(const ls_config& c) {
  const double need = std::ceil((double)c.max_keys_per_instance / (double)c.max_load);
  int64_t s = 16;
  while ((double)s < need) s <<= 1;
  return s;
}

template <class T>
cudaError_t dalloc(T** p, int64_t n) {
  *p = nullptr;
  if (n <= 0) n = 1;
  return cudaMalloc(reinterpret_cast<void**>(p), (size_t)n * sizeof(T));
}

void free_all(Ctx& c) {
  void* ptrs[] = {c.tables, c.table_count, c.inst_state, c.mean, c.stdv, c.master, c.adam_m,
                  c.adam_v, c.pub[0].params, c.pub[0].wt, c.pub[1].params, c.pub[1].wt,
                  c.ring_x, c.ring_y, c.hits, c.scores, c.tx, c.tz, c.ty, c.dz0, c.dz1, c.grad,
                  c.gpart, c.loss_tmp, c.d_err, c.pub[0].img, c.pub[1].img, c.xin, c.xrq, c.pairx, c.ximg,
                  c.bkeys, c.work, c.work_n, c.gkeys, c.gmask, c.st, c.tf.base, c.tf.parts,
                  c.pub[0].bounds, c.pub[1].bounds, c.bounds_stage, c.benc, c.remb, c.rnorm, c.rpart, c.rd,
                  c.rn, c.rinv, c.rcount, c.rimg, c.rrank, c.tr_bar};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  if (c.ev_pub) cudaEventDestroy(c.ev_pub);
  if (c.ev_route) cudaEventDestroy(c.ev_route);
  if (c.tracer.ready)
    for (int i = 0; i < Tracer::kPool; ++i) cudaEventDestroy(c.tracer.ev[i]);
}

}  // namespace

extern "C" {

int64_t ls_param_count(const ls_config* cfg) {
  std::string why;
  if (!check_config(cfg, why)) return fail(LS_ERR_ARG, why);
  return count_params(*cfg);
}

const char* ls_last_error(void) { return g_err.c_str(); }

int ls_create(const ls_config* cfg, ls_ctx** out) {
  std::string why;
  if (!out) return fail(LS_ERR_ARG, "out is NULL");
  *out = nullptr;
  if (!check_config(cfg, why)) return fail(LS_ERR_ARG, why);
  ls_ctx* h = new ls_ctx();
  Ctx& c = h->c;
  c.cfg = *cfg;
  MlpDesc& m = c.mlp;
  m.n_layers = cfg->n_layers;
  m.bf16 = cfg->dtype == LS_BF16;
  int64_t off = 0, wt = 0;
  m.max_width = 1;
  for (int l = 0; l <= cfg->n_layers; ++l) {
    m.w[l] = cfg->widths[l];
    m.max_width = std::max(m.max_width, cfg->widths[l]);
  }
  for (int l = 0; l < cfg->n_layers; ++l) {
    m.woff[l] = off;
    off += (int64_t)m.w[l + 1] * m.w[l];
    m.boff[l] = off;
    off += m.w[l + 1];
    m.wtoff[l] = wt;
    wt += (int64_t)m.w[l + 1] * m.w[l];
  }
  c.d = m.w[0];
  c.n_params = off;
  {
    // LS_TC_PAIR=0 in the environment plans without the pair kernel (the
    // one-CTA wide kernel takes its shapes), LS_TC_PIPE=0 without the
    // pipelined one, so that each kernel stays exercised on shapes another
    // one would take
    const char* pair_env = std::getenv("LS_TC_PAIR");
    const char* pipe_env = std::getenv("LS_TC_PIPE");
    const bool allow_pair = !(pair_env && pair_env[0] == '0');
    const bool allow_pipe = !(pipe_env && pipe_env[0] == '0');
    const bool can_tc = plan_tc(m, c.tc, allow_pair, allow_pipe);
    if (cfg->scorer == LS_SCORER_TENSOR_CORES && !can_tc) {
      delete h;
      return fail(LS_ERR_ARG, "tensor-core scorer needs a bf16 predictor with hidden widths that are "
                              "multiples of 64 and at most 512");
    }
    c.use_tc = can_tc && cfg->scorer != LS_SCORER_CUDA_CORES;
    if (c.use_tc && c.tc.pair) {  // the pair kernel needs CTA pairs that fit together on the device
      const int k = pair_max_clusters(c.tc);
      if (k < 1)
        plan_tc(m, c.tc, false, allow_pipe);
      else
        c.tc.pair_clusters = k;
    }
  }
  c.wt_total = wt;
  {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&c.sms, cudaDevAttrMultiProcessorCount, dev);
  }
  c.slots = table_slots(*cfg);
  c.mask = (uint32_t)(c.slots - 1);

  const int64_t NI = cfg->max_instances, R = cfg->max_requests, B = cfg->max_train_batch;
  int64_t sum_in = 0, sum_out = 0, max_wl = 1;
  for (int l = 0; l < cfg->n_layers; ++l) {
    sum_in += m.w[l];
    sum_out += m.w[l + 1];
    max_wl = std::max<int64_t>(max_wl, (int64_t)m.w[l] * m.w[l + 1]);
  }
  cudaError_t e = cudaSuccess;
  auto A = [&](cudaError_t r) { if (e == cudaSuccess) e = r; };
  c.use_index = cfg->prefix_mode == LS_PREFIX_INDEX ||
                (cfg->prefix_mode == LS_PREFIX_AUTO && cfg->max_instances <= 512);
  if (c.use_index) {
    c.gW = index_words(cfg->max_instances);
    const double need = std::ceil((double)cfg->max_instances * (double)cfg->max_keys_per_instance /
                                  (double)cfg->max_load);
    c.gslots = 16;
    while ((double)c.gslots < need) c.gslots <<= 1;
    // one mask word: (key, mask) entries interleaved in gkeys; else separate arrays
    A(dalloc(&c.gkeys, c.gW == 1 ? 2 * c.gslots : c.gslots));
    if (c.gW > 1) A(dalloc(&c.gmask, c.gslots * c.gW));
  } else {
    A(dalloc(&c.tables, NI * c.slots));
  }
  A(dalloc(&c.table_count, NI));
  A(dalloc(&c.inst_state, NI * std::max(1, cfg->d_inst)));
  A(dalloc(&c.mean, c.d));
  A(dalloc(&c.stdv, c.d));
  A(dalloc(&c.master, c.n_params));
  A(dalloc(&c.adam_m, c.n_params));
  A(dalloc(&c.adam_v, c.n_params));
  for (int b = 0; b < 2; ++b) {
    A(dalloc(&c.pub[b].params, c.n_params));
    A(dalloc(&c.pub[b].wt, c.wt_total));
    if (c.use_tc) A(dalloc(&c.pub[b].img, c.tc.img_bytes));
    A(dalloc(&c.pub[b].bounds, 2 * (int64_t)c.d));
  }
  A(dalloc(&c.bounds_stage, 2 * (int64_t)c.d));
  A(dalloc(&c.benc, 2 * (int64_t)c.d));
  c.bkeys_cap = cfg->max_batch_tokens / kBlockTok + 1;
  if (!c.use_index && cfg->prefix_mode != LS_PREFIX_FUSED) {
    A(dalloc(&c.bkeys, c.bkeys_cap));
    A(dalloc(&c.work, R * NI));
  } else if (c.use_index) {
    A(dalloc(&c.bkeys, c.bkeys_cap));  // block keys of a sequential-commit batch
  }
  A(dalloc(&c.work_n, 1));
  A(dalloc(&c.xin, NI * std::max(1, c.tc.d_pad)));
  A(dalloc(&c.xrq, R * std::max(1, c.tc.d_pad)));
  if (c.use_tc && !c.tc.pipe) A(dalloc(&c.pairx, R * NI));
  if (c.use_tc && c.tc.pipe)
    A(dalloc(&c.ximg, (R * NI + 127) / 128 * ((int64_t)c.tc.d_pad / 64) * 16384));
  // FIFO, pending ring, replay pool (Sec. 4.3.2 two-pool training data)
  const int64_t ring_rows = cfg->ring_capacity + cfg->pending_capacity + cfg->replay_capacity;
  c.replay_base = cfg->ring_capacity + cfg->pending_capacity;
  A(dalloc(&c.ring_x, ring_rows * c.d));
  A(dalloc(&c.ring_y, ring_rows));
  if (cfg->replay_capacity > 0) {
    const int64_t er = cfg->pending_capacity + cfg->replay_capacity;
    A(dalloc(&c.remb, er * m.w[m.n_layers - 1]));
    A(dalloc(&c.rnorm, er));
    A(dalloc(&c.rpart, er * kRowMinParts));
    const int H = m.w[m.n_layers - 1];
    if (m.bf16 && H % 64 == 0 && H <= 256)  // tensor-core distances from a bf16 image
      A(dalloc(&c.rimg, ((cfg->pending_capacity + 127) / 128 + (cfg->replay_capacity + 127) / 128) * 128 * H * 2));
    A(dalloc(&c.rd, cfg->pending_capacity));
    A(dalloc(&c.rn, cfg->replay_capacity));
    A(dalloc(&c.rinv, er));
    A(dalloc(&c.rrank, er));
    A(dalloc(&c.rcount, 2 + (er + cfg->max_train_batch - 1) / cfg->max_train_batch));
  }
  A(dalloc(&c.hits, R * NI));
  A(dalloc(&c.scores, R * NI));
  A(dalloc(&c.tx, B * sum_in));
  A(dalloc(&c.tz, B * sum_out));
  A(dalloc(&c.ty, B));
  A(dalloc(&c.dz0, B * m.max_width));
  A(dalloc(&c.dz1, B * m.max_width));
  A(dalloc(&c.grad, c.n_params));
  c.gpart_floats = 64 * max_wl + 64 * (int64_t)m.max_width;  // dW partials, then column-sum partials
  A(dalloc(&c.gpart, c.gpart_floats));
  A(dalloc(&c.loss_tmp, 1));
  A(dalloc(&c.d_err, 1));
  A(dalloc(&c.st, 1));
  int64_t tf_bytes = 0;
  const bool fast_train = plan_train_fast(m, cfg->max_train_batch, c.tf);
  if (cfg->dropout > 0.0f && !fast_train) {
    free_all(c);
    delete h;
    return fail(LS_ERR_ARG, "dropout needs the tensor-core training path (bf16, hidden widths <= 256)");
  }
  if (fast_train) {
    int64_t pf = 0;
    tf_bytes = train_fast_bytes(m, c.tf, &pf);
    A(dalloc(&c.tf.base, tf_bytes));
    A(dalloc(&c.tf.parts, pf));
    A(dalloc(&c.tr_bar, 2));
    if (e == cudaSuccess) train_fast_bind(m, c.tf, c.tf.base, c.tf.parts);
    c.train_ctas = cfg->train_ctas > 0 ? std::min(cfg->train_ctas, c.sms) : 0;
  }
  if (e == cudaSuccess) {
    A(cudaEventCreateWithFlags(&c.ev_pub, cudaEventDisableTiming));
    A(cudaEventCreateWithFlags(&c.ev_route, cudaEventDisableTiming));
  }
  if (e == cudaSuccess) {
    if (c.tables) A(cudaMemset(c.tables, 0, (size_t)NI * c.slots * sizeof(uint64_t)));
    if (c.gkeys) A(cudaMemset(c.gkeys, 0, (size_t)c.gslots * (c.gW == 1 ? 2 : 1) * sizeof(uint64_t)));
    if (c.gmask) A(cudaMemset(c.gmask, 0, (size_t)c.gslots * c.gW * sizeof(uint64_t)));
    A(cudaMemset(c.table_count, 0, (size_t)NI * sizeof(int32_t)));
    A(cudaMemset(c.adam_m, 0, (size_t)c.n_params * sizeof(float)));
    A(cudaMemset(c.adam_v, 0, (size_t)c.n_params * sizeof(float)));
    A(cudaMemset(c.d_err, 0, sizeof(int)));
    if (c.tf.base) A(cudaMemset(c.tf.base, 0, (size_t)tf_bytes));
    {  // no record seen yet: the empty range in every column
      std::vector<float> empty(2 * (size_t)c.d);
      std::fill(empty.begin(), empty.begin() + c.d, INFINITY);
      std::fill(empty.begin() + c.d, empty.end(), -INFINITY);
      const size_t nb = empty.size() * sizeof(float);
      A(cudaMemcpy(c.bounds_stage, empty.data(), nb, cudaMemcpyHostToDevice));
      A(cudaMemcpy(c.pub[0].bounds, empty.data(), nb, cudaMemcpyHostToDevice));
      A(cudaMemcpy(c.pub[1].bounds, empty.data(), nb, cudaMemcpyHostToDevice));
      std::vector<uint32_t> ident(2 * (size_t)c.d, 0xff800000u);  // codes of +inf, then -inf
      std::fill(ident.begin() + c.d, ident.end(), 0x007fffffu);
      A(cudaMemcpy(c.benc, ident.data(), ident.size() * sizeof(uint32_t), cudaMemcpyHostToDevice));
    }
    DevState init{};
    init.cur = -1;
    init.route_b = 0;
    init.beta_pow[0] = init.beta_pow[1] = 1.0;
    A(cudaMemcpy(c.st, &init, sizeof(DevState), cudaMemcpyHostToDevice));
    A(cudaDeviceSynchronize());
  }
  if (e != cudaSuccess) {
    int rc = cuda_fail(e, "ls_create");
    free_all(c);
    delete h;
    return rc;
  }
  *out = h;
  return LS_OK;
}

void ls_destroy(ls_ctx* h) {
  if (!h) return;
  cudaDeviceSynchronize();
  free_all(h->c);
  delete h;
}

int ls_sync_status(ls_ctx* h) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  LS_CK(cudaDeviceSynchronize());
  int code = 0;
  LS_CK(cudaMemcpy(&code, h->c.d_err, sizeof(int), cudaMemcpyDeviceToHost));
  LS_CK(cudaMemset(h->c.d_err, 0, sizeof(int)));
  LS_CK(cudaDeviceSynchronize());
  if (code) return fail(code, "error latched by device code");
  return LS_OK;
}

int ls_get_info(ls_ctx* h, ls_info* out) {
  if (!h || !out) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  DevState ds{};
  LS_CK(cudaDeviceSynchronize());
  LS_CK(cudaMemcpy(&ds, c.st, sizeof(DevState), cudaMemcpyDeviceToHost));
  std::lock_guard<std::mutex> g(c.mu);
  out->n_inst = c.n_inst;
  out->d = c.d;
  out->n_params = c.n_params;
  out->table_slots = c.use_index ? c.gslots : c.slots;
  out->ring_count = ds.ring_count;
  out->train_steps = ds.step;
  out->weight_version = ds.version;
  out->scorer = c.use_tc ? LS_SCORER_TENSOR_CORES : LS_SCORER_CUDA_CORES;
  out->tc_kernel = !c.use_tc ? LS_TC_NONE
                   : c.tc.pipe ? LS_TC_PIPELINED
                   : c.tc.pair ? LS_TC_PAIR
                   : c.tc.wide ? LS_TC_WIDE
                               : LS_TC_GENERIC;
  out->replay_count = ds.replay_count;
  out->pending_count = 0;
  if (c.cfg.replay_capacity > 0) {  // evicted positions [lo, hi) not yet considered
    const int64_t hi = std::max<int64_t>(0, ds.ring_count - c.cfg.ring_capacity);
    const int64_t lo = std::min(hi, std::max(ds.admitted, hi - c.cfg.pending_capacity));
    out->pending_count = hi - lo;
  }
  return LS_OK;
}

int ls_set_params(ls_ctx* h, const float* params, void* stream) {
  if (!h || !params) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  const size_t n = (size_t)c.n_params * sizeof(float);
  LS_CK(cudaMemcpyAsync(c.master, params, n, cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaMemsetAsync(c.adam_m, 0, n, S(stream)));
  LS_CK(cudaMemsetAsync(c.adam_v, 0, n, S(stream)));
  {
    const int64_t zero = 0;
    const double ones[2] = {1.0, 1.0};
    LS_CK(cudaMemcpyAsync(&c.st->step, &zero, sizeof(zero), cudaMemcpyHostToDevice, S(stream)));
    LS_CK(cudaMemcpyAsync(c.st->beta_pow, ones, sizeof(ones), cudaMemcpyHostToDevice, S(stream)));
    LS_CK(cudaStreamSynchronize(S(stream)));  // the host values above are locals
  }
  if (c.tf.on) LS_CK(train_fast_images(c, S(stream)));
  c.have_params = true;
  return LS_OK;
}

int ls_get_params(ls_ctx* h, float* params_out, void* stream) {
  if (!h || !params_out) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  LS_CK(cudaMemcpyAsync(params_out, c.master, (size_t)c.n_params * sizeof(float),
                        cudaMemcpyDeviceToDevice, S(stream)));
  return LS_OK;
}

int ls_get_opt_state(ls_ctx* h, float* m_out, float* v_out, int64_t* step_out, void* stream) {
  if (!h || !m_out || !v_out || !step_out) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  const size_t n = (size_t)c.n_params * sizeof(float);
  LS_CK(cudaMemcpyAsync(m_out, c.adam_m, n, cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaMemcpyAsync(v_out, c.adam_v, n, cudaMemcpyDeviceToDevice, S(stream)));
  int64_t step = 0;
  LS_CK(cudaMemcpyAsync(&step, &c.st->step, sizeof(int64_t), cudaMemcpyDeviceToHost, S(stream)));
  LS_CK(cudaStreamSynchronize(S(stream)));
  *step_out = step;
  return LS_OK;
}

int ls_set_opt_state(ls_ctx* h, const float* m, const float* v, int64_t step, void* stream) {
  if (!h || !m || !v || step < 0) return fail(LS_ERR_ARG, "bad argument");
  Ctx& c = h->c;
  const size_t n = (size_t)c.n_params * sizeof(float);
  LS_CK(cudaMemcpyAsync(c.adam_m, m, n, cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaMemcpyAsync(c.adam_v, v, n, cudaMemcpyDeviceToDevice, S(stream)));
  const int64_t st_step = step;
  // the running powers exactly as the device forms them, one multiply per step
  double pw[2] = {1.0, 1.0};
  for (int64_t t = 0; t < step; ++t) {
    pw[0] *= 0.9;
    pw[1] *= 0.999;
  }
  LS_CK(cudaMemcpyAsync(&c.st->step, &st_step, sizeof(int64_t), cudaMemcpyHostToDevice, S(stream)));
  LS_CK(cudaMemcpyAsync(c.st->beta_pow, pw, sizeof(pw), cudaMemcpyHostToDevice, S(stream)));
  LS_CK(cudaStreamSynchronize(S(stream)));
  return LS_OK;
}

int ls_set_normalizer(ls_ctx* h, const float* mean, const float* stdv, void* stream) {
  if (!h || !mean || !stdv) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  LS_CK(cudaMemcpyAsync(c.mean, mean, (size_t)c.d * sizeof(float), cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaMemcpyAsync(c.stdv, stdv, (size_t)c.d * sizeof(float), cudaMemcpyDeviceToDevice, S(stream)));
  c.have_norm = true;
  if (c.use_tc && c.tc.pipe && c.n_inst > 0)  // instance template rows follow the normaliser
    LS_CK(launch_inst_templates(c.n_inst, c.cfg.d_inst, c.inst_state, c.mean, c.stdv, c.tc.d_pad, c.xin, c.sms,
                                S(stream)));
  return LS_OK;
}

int ls_snapshot_update(ls_ctx* h, int32_t n_inst, const float* inst_state, const uint64_t* keys,
                       const int64_t* key_off, int64_t n_keys, int32_t mode, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (n_inst < 1 || n_inst > c.cfg.max_instances) return fail(LS_ERR_ARG, "n_inst out of range");
  if (c.cfg.d_inst > 0 && !inst_state) return fail(LS_ERR_ARG, "inst_state is NULL");
  if (mode != LS_REPLACE && mode != LS_INSERT) return fail(LS_ERR_ARG, "bad mode");
  if (keys && (!key_off || n_keys < 0)) return fail(LS_ERR_ARG, "keys need key_off and n_keys >= 0");
  if (!keys && n_keys != 0) return fail(LS_ERR_ARG, "n_keys given without keys");
  if (c.cfg.d_inst > 0)
    LS_CK(cudaMemcpyAsync(c.inst_state, inst_state, (size_t)n_inst * c.cfg.d_inst * sizeof(float),
                          cudaMemcpyDeviceToDevice, S(stream)));
  if (c.use_tc && c.tc.pipe && c.have_norm)  // instance template rows follow the snapshot
    LS_CK(traced(c, TR_NORM_ROWS, 1, S(stream), [&] {
      return launch_inst_templates(n_inst, c.cfg.d_inst, c.inst_state, c.mean, c.stdv, c.tc.d_pad, c.xin, c.sms,
                                   S(stream));
    }));
  if (keys && c.use_index) {
    if (mode == LS_REPLACE) {
      // the index holds every instance: replacing the listed instances
      // (all of the snapshot) rebuilds it
      LS_CK(cudaMemsetAsync(c.gkeys, 0, (size_t)c.gslots * (c.gW == 1 ? 2 : 1) * sizeof(uint64_t), S(stream)));
      if (c.gmask) LS_CK(cudaMemsetAsync(c.gmask, 0, (size_t)c.gslots * c.gW * sizeof(uint64_t), S(stream)));
      LS_CK(cudaMemsetAsync(c.table_count, 0, (size_t)c.cfg.max_instances * sizeof(int32_t), S(stream)));
    }
    LS_CK(traced(c, TR_INDEX_INSERT, 1, S(stream), [&] {
      return launch_index_insert(keys, key_off, n_inst, n_keys, c.gkeys, c.gmask, c.gW, (uint64_t)(c.gslots - 1),
                                 c.table_count, c.cfg.max_keys_per_instance, c.d_err, c.sms, S(stream));
    }));
  } else if (keys) {
    if (mode == LS_REPLACE) {
      LS_CK(cudaMemsetAsync(c.tables, 0, (size_t)n_inst * c.slots * sizeof(uint64_t), S(stream)));
      LS_CK(cudaMemsetAsync(c.table_count, 0, (size_t)n_inst * sizeof(int32_t), S(stream)));
    }
    LS_CK(traced(c, TR_INSERT, 1, S(stream), [&] {
      return launch_table_insert(keys, key_off, n_inst, n_keys, c.tables, c.mask, c.slots,
                                 c.table_count, c.cfg.max_keys_per_instance, c.d_err, S(stream));
    }));
  }
  c.n_inst = n_inst;
  return LS_OK;
}

int ls_hash_blocks(ls_ctx* h, int32_t n_seq, const int32_t* tok, const int64_t* tok_off,
                   uint64_t* keys_out, const int64_t* key_off, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  if (n_seq < 0) return fail(LS_ERR_ARG, "n_seq < 0");
  if (n_seq == 0) return LS_OK;
  if (!tok || !tok_off || !keys_out || !key_off) return fail(LS_ERR_ARG, "NULL argument");
  LS_CK(traced(h->c, TR_HASH, 1, S(stream), [&] {
    return launch_hash_blocks(n_seq, tok, tok_off, keys_out, key_off, 0, h->c.d_err, S(stream));
  }));
  return LS_OK;
}

int ls_assemble_features(ls_ctx* h, int32_t n_req, const int64_t* tok_off, const int32_t* hits,
                         const float* req_feats, float* x_out, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (n_req < 0) return fail(LS_ERR_ARG, "n_req < 0");
  if (n_req == 0) return LS_OK;
  if (!tok_off || !hits || !x_out || (c.cfg.d_req > 0 && !req_feats))
    return fail(LS_ERR_ARG, "NULL argument");
  if (c.n_inst < 1) return fail(LS_ERR_STATE, "no snapshot");
  if (!c.have_norm) return fail(LS_ERR_STATE, "normaliser not set");
  LS_CK(traced(c, TR_ASSEMBLE, 1, S(stream), [&] {
    return launch_assemble_features(n_req, c.n_inst, tok_off, hits, c.inst_state, c.cfg.d_inst,
                                    req_feats, c.cfg.d_req, c.mean, c.stdv, x_out, S(stream));
  }));
  return LS_OK;
}

}  // extern "C"

namespace {

// One route; `status` non-NULL selects the guarded selection of Algorithm 4
// (scores are then always materialised and the guard kernel replaces argmin).
int route_impl(ls_ctx* h, int32_t n_req, const int32_t* tok, const int64_t* tok_off, const float* req_feats,
               int32_t* choice, float* best, int32_t* status, int32_t* fallback, bool guarded, float* scores_opt,
               int32_t* hits_opt, uint64_t* weight_version_out, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (n_req < 0 || n_req > c.cfg.max_requests) return fail(LS_ERR_ARG, "n_req out of range");
  if (n_req > 0 && (!tok || !tok_off || !choice || !best || (c.cfg.d_req > 0 && !req_feats) ||
                    (guarded && !status)))
    return fail(LS_ERR_ARG, "NULL argument");
  if (c.n_inst < 1) return fail(LS_ERR_STATE, "no snapshot");
  if (!c.have_norm) return fail(LS_ERR_STATE, "normaliser not set");
  cudaStream_t s = S(stream);
  const bool cap = capturing(s);
  uint64_t v;
  {
    std::lock_guard<std::mutex> g(c.mu);
    if (!c.have_published) return fail(LS_ERR_STATE, "no weights published");
    v = c.version;
    // the route reads the latest publish enqueued before it (host order)
    if (!cap && c.pub_recorded) LS_CK(cudaStreamWaitEvent(s, c.ev_pub, 0));
  }
  if (weight_version_out) *weight_version_out = v;
  if (n_req == 0) return LS_OK;
  int32_t* hits = hits_opt ? hits_opt : c.hits;
  const bool fused_select = !guarded && c.use_tc && scorer_selects(c.tc, c.n_inst);
  float* scores = scores_opt ? scores_opt : (fused_select ? nullptr : c.scores);
  if (c.use_index) {
    LS_CK(traced(c, TR_PREFIX_INDEX, 1, s, [&] {
      return launch_prefix_index(n_req, tok, tok_off, c.gkeys, c.gmask, c.gW, (uint64_t)(c.gslots - 1), c.n_inst,
                                 hits, c.sms, c.st, s);
    }));
  } else if (c.cfg.prefix_mode == LS_PREFIX_FUSED) {
    LS_CK(traced(c, TR_PREFIX, 1, s, [&] {
      return launch_prefix_match(n_req, tok, tok_off, c.tables, c.mask, c.slots, c.n_inst, hits, c.st, s);
    }));
  } else {
    LS_CK(traced(c, TR_MEMSET, 1, s, [&] { return cudaMemsetAsync(c.work_n, 0, sizeof(int), s); }));
    LS_CK(traced(c, TR_HASH_BATCH, 1, s, [&] {
      return launch_hash_screen(n_req, tok, tok_off, c.bkeys, c.bkeys_cap, c.d_err, c.tables, c.mask, c.slots,
                                c.n_inst, hits, c.work, c.work_n, c.sms, c.st, s);
    }));
    LS_CK(traced(c, TR_WALK, 1, s, [&] {
      return launch_probe_walk(c.n_inst, tok_off, c.bkeys, c.bkeys_cap, c.tables, c.mask, c.slots, hits,
                               c.work, c.work_n, c.sms, s);
    }));
  }
  if (c.use_tc) {
    LS_CK(traced(c, TR_NORM_ROWS, 1, s, [&] {
      if (c.tc.pipe)
        return launch_feature_image(tok_off, hits, c.n_inst, c.xin, c.cfg.d_inst, n_req, c.cfg.d_req, req_feats,
                                    c.mean, c.stdv, c.tc.d_pad, c.ximg, c.sms, s);
      return launch_norm_rows(tok_off, hits, c.pairx, c.n_inst, c.cfg.d_inst, c.inst_state, n_req, c.cfg.d_req,
                              req_feats, c.mean,
                              c.stdv, c.tc.d_pad, c.xin, c.xrq, c.sms, s);
    }));
    LS_CK(traced(c, TR_SCORE_TC, 1, s, [&] {
      return launch_score_tc(c.mlp, c.tc, c.pub, &c.st->route_b, n_req, c.n_inst, c.pairx, c.ximg,
                             fused_select ? choice : nullptr, fused_select ? best : nullptr,
                             c.xin, c.xrq, c.cfg.d_inst, c.cfg.d_req, c.mean, c.stdv, scores, c.d_err, c.sms,
                             s);
    }));
  } else {
    LS_CK(traced(c, TR_SCORE, 1, s, [&] {
      return launch_score_simt(c.mlp, c.pub, &c.st->route_b, n_req, c.n_inst, tok_off, hits, c.inst_state,
                               c.cfg.d_inst, req_feats, c.cfg.d_req, c.mean, c.stdv, scores, s);
    }));
  }
  if (guarded)
    LS_CK(traced(c, TR_GUARDS, 1, s, [&] {
      return launch_guards(c.guards, n_req, c.n_inst, tok, tok_off, hits, scores, c.inst_state, c.cfg.d_inst,
                           req_feats, c.cfg.d_req, c.pub, c.st, choice, best, status, fallback, c.sms, s);
    }));
  else if (!fused_select)
    LS_CK(traced(c, TR_ARGMIN, 1, s, [&] { return launch_argmin(n_req, c.n_inst, scores, choice, best, s); }));
  if (!cap) {
    std::lock_guard<std::mutex> g(c.mu);
    LS_CK(cudaEventRecord(c.ev_route, s));
    c.route_recorded = true;
  }
  return LS_OK;
}

}  // namespace

extern "C" {

int ls_route_batch(ls_ctx* h, int32_t n_req, const int32_t* tok, const int64_t* tok_off,
                   const float* req_feats, int32_t* choice, float* best, float* scores_opt,
                   int32_t* hits_opt, uint64_t* weight_version_out, void* stream) {
  return route_impl(h, n_req, tok, tok_off, req_feats, choice, best, nullptr, nullptr, false, scores_opt, hits_opt,
                    weight_version_out, stream);
}

int ls_read_features(ls_ctx* h, int64_t row0, int64_t n_rows, uint16_t* out, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (!c.use_tc) return fail(LS_ERR_STATE, "the CUDA-core scorer assembles feature rows in registers only");
  if (row0 < 0 || n_rows < 0 || (n_rows > 0 && !out)) return fail(LS_ERR_ARG, "bad rows or NULL output");
  const int64_t cap = (int64_t)c.cfg.max_requests * c.cfg.max_instances;
  if (row0 + n_rows > cap) return fail(LS_ERR_ARG, "rows beyond the batch buffers");
  LS_CK(launch_read_features(row0, n_rows, c.d, c.tc, c.n_inst, c.ximg, c.pairx, c.xin, c.xrq, out, S(stream)));
  return LS_OK;
}

int ls_route_sequential(ls_ctx* h, int32_t n_req, const int32_t* tok, const int64_t* tok_off,
                        const float* req_feats, int32_t queue_col, int32_t* choice, float* best, float* scores_opt,
                        int32_t* hits_opt, uint64_t* weight_version_out, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (n_req < 0 || n_req > c.cfg.max_requests) return fail(LS_ERR_ARG, "n_req out of range");
  if (n_req > 0 && (!tok || !tok_off || !choice || !best || (c.cfg.d_req > 0 && !req_feats)))
    return fail(LS_ERR_ARG, "NULL argument");
  if (queue_col < -1 || queue_col >= c.cfg.d_inst) return fail(LS_ERR_ARG, "queue_col outside [-1, d_inst)");
  if (!c.use_index) return fail(LS_ERR_ARG, "sequential routing needs the prefix index mode");
  if (c.n_inst < 1) return fail(LS_ERR_STATE, "no snapshot");
  if (!c.have_norm) return fail(LS_ERR_STATE, "normaliser not set");
  int wmax = 1;
  for (int l = 0; l <= c.mlp.n_layers; ++l) wmax = std::max(wmax, c.mlp.w[l]);
  if (!route_seq_smem(c.n_inst, c.cfg.d_inst, wmax, c.gW))
    return fail(LS_ERR_ARG, "sequential routing: instances x widest layer beyond its shared-memory limit");
  cudaStream_t s = S(stream);
  const bool cap = capturing(s);
  uint64_t v;
  {
    std::lock_guard<std::mutex> g(c.mu);
    if (!c.have_published) return fail(LS_ERR_STATE, "no weights published");
    v = c.version;
    if (!cap && c.pub_recorded) LS_CK(cudaStreamWaitEvent(s, c.ev_pub, 0));
  }
  if (weight_version_out) *weight_version_out = v;
  if (n_req == 0) return LS_OK;
  LS_CK(traced(c, TR_HASH, 1, s, [&] {
    return launch_hash_blocks(n_req, tok, tok_off, c.bkeys, nullptr, c.bkeys_cap, c.d_err, s);
  }));
  LS_CK(traced(c, TR_ROUTE_SEQ, 1, s, [&] {
    return launch_route_seq(n_req, c.n_inst, c.cfg.d_inst, c.cfg.d_req, queue_col, tok_off, c.bkeys, c.bkeys_cap,
                            req_feats, c.inst_state, c.mean, c.stdv, c.pub, c.st, c.mlp, c.gkeys, c.gmask, c.gW,
                            (uint64_t)(c.gslots - 1), c.table_count, c.cfg.max_keys_per_instance, choice, best,
                            scores_opt, hits_opt, c.d_err, s);
  }));
  if (c.use_tc && c.tc.pipe)  // instance template rows follow the updated instance rows
    LS_CK(traced(c, TR_NORM_ROWS, 1, s, [&] {
      return launch_inst_templates(c.n_inst, c.cfg.d_inst, c.inst_state, c.mean, c.stdv, c.tc.d_pad, c.xin, c.sms,
                                   s);
    }));
  if (!cap) {
    std::lock_guard<std::mutex> g(c.mu);
    LS_CK(cudaEventRecord(c.ev_route, s));
    c.route_recorded = true;
  }
  return LS_OK;
}

int ls_route_batch_guarded(ls_ctx* h, int32_t n_req, const int32_t* tok, const int64_t* tok_off,
                           const float* req_feats, int32_t* choice, float* best, int32_t* status,
                           int32_t* fallback_opt, float* scores_opt, int32_t* hits_opt, uint64_t* weight_version_out,
                           void* stream) {
  return route_impl(h, n_req, tok, tok_off, req_feats, choice, best, status, fallback_opt, true, scores_opt,
                    hits_opt, weight_version_out, stream);
}

int ls_set_guards(ls_ctx* h, const ls_guards* g) {
  if (!h || !g) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  if (g->k < 0 || g->k > c.cfg.max_instances) return fail(LS_ERR_ARG, "k out of range");
  if (g->k > 0 && (g->kv_col < 0 || g->kv_col >= c.cfg.d_inst))
    return fail(LS_ERR_ARG, "kv_col outside the instance-state columns");
  if (g->heuristic < LS_HEUR_NONE || g->heuristic > LS_HEUR_PREFIX) return fail(LS_ERR_ARG, "unknown heuristic");
  if (g->heuristic != LS_HEUR_NONE) {
    if (g->count_col[0] < 0 || g->count_col[0] >= c.cfg.d_inst || g->count_col[1] < -1 ||
        g->count_col[1] >= c.cfg.d_inst)
      return fail(LS_ERR_ARG, "count_col outside the instance-state columns");
    if (c.cfg.max_instances > kGuardHeurMaxInst) return fail(LS_ERR_ARG, "heuristic needs max_instances <= 1024");
  }
  c.guards = *g;
  return LS_OK;
}

int ls_refresh_bounds(ls_ctx* h, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  LS_CK(traced(c, TR_BOUNDS, 1, S(stream), [&] {
    return launch_ring_bounds(c.d, c.ring_x, c.cfg.ring_capacity, c.replay_base, c.cfg.replay_capacity, c.benc,
                              c.bounds_stage, c.st, c.sms,
                              S(stream));
  }));
  return LS_OK;
}

int ls_replay_admit(ls_ctx* h, float* d_out, float* n_out, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (c.cfg.replay_capacity < 1) return fail(LS_ERR_STATE, "no replay pool configured");
  if (!c.have_params) return fail(LS_ERR_STATE, "parameters not set");
  if (!c.have_norm) return fail(LS_ERR_STATE, "normaliser not set");
  LS_CK(run_replay_admit(c, d_out, n_out, S(stream)));
  return LS_OK;
}

int ls_get_replay(ls_ctx* h, float* x_out, float* y_out, int64_t* n_out, void* stream) {
  if (!h || !x_out || !y_out || !n_out) return fail(LS_ERR_ARG, "NULL argument");
  Ctx& c = h->c;
  if (c.cfg.replay_capacity < 1) return fail(LS_ERR_STATE, "no replay pool configured");
  int64_t nr = 0;
  LS_CK(cudaDeviceSynchronize());
  LS_CK(cudaMemcpy(&nr, &c.st->replay_count, sizeof(nr), cudaMemcpyDeviceToHost));
  if (nr > 0) {
    LS_CK(cudaMemcpyAsync(x_out, c.ring_x + c.replay_base * c.d, (size_t)nr * c.d * sizeof(float),
                          cudaMemcpyDeviceToDevice, S(stream)));
    LS_CK(cudaMemcpyAsync(y_out, c.ring_y + c.replay_base, (size_t)nr * sizeof(float), cudaMemcpyDeviceToDevice,
                          S(stream)));
    LS_CK(cudaStreamSynchronize(S(stream)));
  }
  *n_out = nr;
  return LS_OK;
}

int ls_get_bounds(ls_ctx* h, int32_t which, float* lo_out, float* hi_out, void* stream) {
  if (!h || !lo_out || !hi_out) return fail(LS_ERR_ARG, "NULL argument");
  if (which != 0 && which != 1) return fail(LS_ERR_ARG, "which must be 0 or 1");
  Ctx& c = h->c;
  const float* src = c.bounds_stage;
  if (which == 1) {
    int32_t cur = -1;
    LS_CK(cudaDeviceSynchronize());
    LS_CK(cudaMemcpy(&cur, &c.st->cur, sizeof(cur), cudaMemcpyDeviceToHost));
    if (cur < 0) return fail(LS_ERR_STATE, "no weights published");
    src = c.pub[cur].bounds;
  }
  const size_t nb = (size_t)c.d * sizeof(float);
  LS_CK(cudaMemcpyAsync(lo_out, src, nb, cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaMemcpyAsync(hi_out, src + c.d, nb, cudaMemcpyDeviceToDevice, S(stream)));
  LS_CK(cudaStreamSynchronize(S(stream)));
  return LS_OK;
}

int ls_log_samples(ls_ctx* h, int32_t n, const float* feats, const float* ttft, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (n < 0) return fail(LS_ERR_ARG, "n < 0");
  if (n == 0) return LS_OK;
  if (!feats || !ttft) return fail(LS_ERR_ARG, "NULL argument");
  if (c.cfg.pending_capacity > 0 && n > c.cfg.ring_capacity)
    return fail(LS_ERR_ARG, "with a replay pool a log call holds at most ring_capacity records");
  LS_CK(traced(c, TR_RING, 1, S(stream), [&] {
    return launch_ring_append(n, c.d, feats, ttft, c.ring_x, c.ring_y, c.st, c.cfg.ring_capacity,
                              c.cfg.pending_capacity, S(stream));
  }));
  std::lock_guard<std::mutex> g(c.mu);
  c.ring_enqueued += n;
  return LS_OK;
}

int ls_train_step(ls_ctx* h, int32_t batch, const int32_t* idx, int32_t opt, float lr, float* loss_out,
                  void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (batch < 1 || batch > c.cfg.max_train_batch) return fail(LS_ERR_ARG, "batch out of range");
  if (opt != LS_SGD && opt != LS_ADAM) return fail(LS_ERR_ARG, "bad optimiser");
  if (!std::isfinite(lr)) return fail(LS_ERR_ARG, "lr is not finite");
  if (!c.have_params) return fail(LS_ERR_STATE, "parameters not set");
  if (!c.have_norm) return fail(LS_ERR_STATE, "normaliser not set");
  if (c.ring_enqueued < 1) return fail(LS_ERR_STATE, "sample ring is empty");
  LS_CK(c.tf.on ? run_train_fast(c, batch, idx, opt, lr, loss_out, S(stream))
                : run_train_step(c, batch, idx, opt, lr, loss_out, S(stream)));
  return LS_OK;
}

int ls_publish(ls_ctx* h, void* stream) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Ctx& c = h->c;
  if (!c.have_params) return fail(LS_ERR_STATE, "parameters not set");
  cudaStream_t s = S(stream);
  const bool cap = capturing(s);
  std::lock_guard<std::mutex> g(c.mu);
  // the buffer written (1 - cur) may still be read by routes enqueued
  // earlier, and publishes must not overlap one another
  if (!cap && c.route_recorded) LS_CK(cudaStreamWaitEvent(s, c.ev_route, 0));
  if (!cap && c.pub_recorded) LS_CK(cudaStreamWaitEvent(s, c.ev_pub, 0));
  LS_CK(traced(c, TR_PUBLISH, 1, s, [&] {
    return launch_publish(c.mlp, c.use_tc ? &c.tc : nullptr, c.master, c.pub, c.use_tc ? 0 : 1, c.bounds_stage,
                          c.st, c.sms, s);
  }));
  if (!cap) {
    LS_CK(cudaEventRecord(c.ev_pub, s));
    c.pub_recorded = true;
  }
  c.version += 1;
  c.have_published = true;
  return LS_OK;
}

int ls_trace_enable(ls_ctx* h, int32_t on) {
  if (!h) return fail(LS_ERR_ARG, "ctx is NULL");
  Tracer& t = h->c.tracer;
  std::lock_guard<std::mutex> g(t.mu);
  if (on && !t.ready) {
    for (int i = 0; i < Tracer::kPool; ++i) LS_CK(cudaEventCreate(&t.ev[i]));
    t.ready = true;
  }
  t.on = on != 0;
  return LS_OK;
}

int ls_trace_read(ls_ctx* h, ls_trace_entry* out, int32_t max_entries, int32_t* n_out) {
  if (!h || (!out && max_entries > 0) || max_entries < 0 || !n_out) return fail(LS_ERR_ARG, "bad argument");
  Tracer& t = h->c.tracer;
  LS_CK(cudaDeviceSynchronize());
  std::lock_guard<std::mutex> g(t.mu);
  for (const auto& p : t.pend) {
    float ms = 0.0f;
    LS_CK(cudaEventElapsedTime(&ms, t.ev[p.a], t.ev[p.a + 1]));
    t.ms[p.id] += ms;
    t.timed[p.id] += p.launches;
  }
  t.pend.clear();
  t.used = 0;
  int n = 0;
  for (int id = 0; id < TR_COUNT; ++id) {
    if (t.launches[id] == 0) continue;
    if (n < max_entries) {
      std::memset(out[n].name, 0, sizeof(out[n].name));
      std::strncpy(out[n].name, kTraceNames[id], sizeof(out[n].name) - 1);
      out[n].launches = t.launches[id];
      out[n].total_ms = t.ms[id];
      out[n].timed_launches = t.timed[id];
    }
    ++n;
    t.launches[id] = 0;
    t.timed[id] = 0;
    t.ms[id] = 0.0;
  }
  *n_out = n < max_entries ? n : max_entries;
  t.dropped = 0;
  return LS_OK;
}

}  // extern "C"
