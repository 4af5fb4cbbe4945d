// Guards of Algorithm 4 around the greedy selection (Sec. 4.3.1 "Fallback":
// cold start and out-of-range inputs hand the request back to the gateway's
// heuristic; Sec. 4.1 "Consistent hashing based filtering": under cluster
// memory saturation the choice is confined to K instances picked by
// consistent hashing of the request's prefix group).
//
//   k_ring_bounds  feature bounds [l, u] of the training buffer: column-wise
//                  minimum / maximum over the records the ring holds (NaN
//                  skipped), block results met by atomic min / max on
//                  order-preserving codes, decoded by the last block into the
//                  staging copy that the next publish makes visible.
//                  Bound: HBM, 4 d bytes per held record.
//   k_guards       one warp per request: cold-start test, out-of-range test of
//                  every raw feature of every pair, argmin, K-filter.  Reads
//                  the hits and scores of the request (8 bytes per pair), its
//                  first 64 prompt bytes and its extras; writes 12 bytes.
#include <climits>
#include <cmath>

#include "blockhash.cuh"
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
namespace {

constexpr unsigned kFull = 0xffffffffu;

// ---------------------------------------------------------------------------
// feature bounds of the sample ring
// ---------------------------------------------------------------------------

// The block minima / maxima meet in global memory through atomicMin /
// atomicMax on order-preserving codes (ord_code), so the result does not
// depend on which block finishes first.
__device__ __forceinline__ float ord_float(uint32_t e) {
  return __uint_as_float((e & 0x80000000u) ? (e & 0x7fffffffu) : ~e);
}
constexpr uint32_t kCodePosInf = 0xff800000u;  // ord_code(+inf): identity of the minimum
constexpr uint32_t kCodeNegInf = 0x007fffffu;  // ord_code(-inf): identity of the maximum

__device__ __forceinline__ void fold(float v, float& lo, float& hi) {  // NaN fails both tests: skipped
  lo = v < lo ? v : lo;
  hi = v > hi ? v : hi;
}

// Records of the training buffer F u R (union index u -> row union_row(u))
// split into gridDim.x contiguous ranges of u.
// d % 4 == 0: thread t reads 16-byte groups g = t % (d/4) of rows t / (d/4),
// t / (d/4) + P, ... (P = 256 / (d/4) rows per pass, so a pass is one
// contiguous run of P d floats), eight loads in flight.  Other d: the same
// with single floats (d <= 256), or columns t, t + 256, ... of every row.
// Block results go to the per-column codes in benc [2][d]; the last block
// decodes them into the staging copy and resets them for the next launch.
__global__ void __launch_bounds__(256) k_ring_bounds(int d, const float* __restrict__ ring_x, int64_t capacity,
                                                     int64_t replay_base, uint32_t* __restrict__ benc,
                                                     float* __restrict__ stage, DevState* st) {
  __shared__ float s_lo[1024], s_hi[1024];
  const int64_t count = *reinterpret_cast<volatile int64_t*>(&st->ring_count);
  const int64_t nF = count < capacity ? count : capacity;
  const int64_t rows = nF + *reinterpret_cast<volatile int64_t*>(&st->replay_count);
  const int64_t per = (rows + gridDim.x - 1) / gridDim.x;
  const int64_t r0 = (int64_t)blockIdx.x * per;
  const int64_t r1 = r0 + per < rows ? r0 + per : rows;
  const int t = threadIdx.x;
  if ((d & 3) == 0) {
    const int G = d >> 2, P = 256 / G, g = t % G, p = t / G;
    float lo[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
    float hi[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
    if (p < P) {
      const float4* base = reinterpret_cast<const float4*>(ring_x) + g;
      const float4 none = make_float4(NAN, NAN, NAN, NAN);  // rows past the range: folded as NaN, i.e. skipped
      for (int64_t r = r0 + p; r < r1; r += 8 * (int64_t)P) {
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          v[u] = r + (int64_t)u * P < r1 ? __ldcs(base + union_row(r + (int64_t)u * P, nF, replay_base) * G) : none;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          fold(v[u].x, lo[0], hi[0]);
          fold(v[u].y, lo[1], hi[1]);
          fold(v[u].z, lo[2], hi[2]);
          fold(v[u].w, lo[3], hi[3]);
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        s_lo[p * d + 4 * g + k] = lo[k];
        s_hi[p * d + 4 * g + k] = hi[k];
      }
    }
    __syncthreads();
    for (int c = t; c < d; c += 256) {
      float l = s_lo[c], h = s_hi[c];
      for (int q = 1; q < P; ++q) {
        l = fminf(l, s_lo[q * d + c]);  // +inf / -inf mark phases without a number
        h = fmaxf(h, s_hi[q * d + c]);
      }
      atomicMin(benc + c, ord_code(l));
      atomicMax(benc + d + c, ord_code(h));
    }
  } else {
    const bool narrow = d <= 256;
    const int P = narrow ? 256 / d : 1;
    const int p = narrow ? t / d : 0;
    for (int c = narrow ? t % d : t; c < d; c += narrow ? d : 256) {
      float lo = INFINITY, hi = -INFINITY;
      if (p < P)
        for (int64_t r = r0 + p; r < r1; r += 4 * (int64_t)P) {
          float v[4];
#pragma unroll
          for (int u = 0; u < 4; ++u)
            v[u] = r + (int64_t)u * P < r1 ? __ldcs(ring_x + union_row(r + (int64_t)u * P, nF, replay_base) * d + c)
                                           : NAN;
#pragma unroll
          for (int u = 0; u < 4; ++u) fold(v[u], lo, hi);
        }
      if (narrow) {
        if (p < P) {
          s_lo[t] = lo;
          s_hi[t] = hi;
        }
      } else {
        atomicMin(benc + c, ord_code(lo));
        atomicMax(benc + d + c, ord_code(hi));
      }
    }
    if (narrow) {
      __syncthreads();
      if (t < d) {
        float l = s_lo[t], h = s_hi[t];
        for (int q = 1; q < P; ++q) {
          l = fminf(l, s_lo[q * d + t]);
          h = fmaxf(h, s_hi[q * d + t]);
        }
        atomicMin(benc + t, ord_code(l));
        atomicMax(benc + d + t, ord_code(h));
      }
    }
  }
  if (last_block(&st->done[DONE_BOUNDS])) {
    for (int c = t; c < d; c += blockDim.x) {
      stage[c] = ord_float(atomicExch(benc + c, kCodePosInf));
      stage[d + c] = ord_float(atomicExch(benc + d + c, kCodeNegInf));
    }
  }
}

// ---------------------------------------------------------------------------
// guarded selection
// ---------------------------------------------------------------------------

struct GuardArgs {
  int n_req, n_inst, d_inst, d_req;
  const int32_t* tok;
  const int64_t* tok_off;
  const int32_t* hits;
  const float* scores;
  const float* inst;
  const float* req;
  const float* bounds[2];
  const DevState* st;
  int64_t n_min;
  int64_t h_ben;       // 16 h > tau_ben  <=>  h >= h_ben (h an integer; set on the host)
  int ood, K, kv_col;
  float tau_sat;
  // fallback heuristic (Algorithm 1: heur 1; Algorithm 2: heur 2; 0 = none)
  int heur, c_col0, c_col1;
  float theta_imbal, k_over, tau_prefix;
  int32_t* choice;
  float* best;
  int32_t* status;
  int32_t* fallback;
};

// (wa, a) ranks before (wb, b) in rendezvous order: larger weight, then lower index.
__device__ __forceinline__ bool hrw_before(uint64_t wa, int a, uint64_t wb, int b) {
  return wa != wb ? wa > wb : a < b;
}

__device__ __forceinline__ bool in_range(float x, float lo, float hi) { return x >= lo && x <= hi; }

constexpr int kHashedInst = kGuardHeurMaxInst;  // instance hashes kept in shared memory up to this count
constexpr int kGuardThreads = 256;  // warp 0: batch-wide terms; warps 1..7: requests

// Order-preserving 64-bit key of an fp64 value: keys compare as the values
// do, -0 and +0 get one key, NaN the largest key (after every number).
__device__ __forceinline__ uint64_t dkey(double v) {
  if (v != v) return ~0ull;
  const uint64_t b = (uint64_t)__double_as_longlong(__dadd_rn(v, 0.0));  // -0 + 0 = +0
  return (b >> 63) ? ~b : (b | 0x8000000000000000ull);
}
__device__ __forceinline__ double dkey_value(uint64_t k) {
  return __longlong_as_double((long long)((k >> 63) ? (k & 0x7fffffffffffffffull) : ~k));
}

constexpr float kU = 5.9604644775390625e-8f;  // 2^-24, unit roundoff of fp32

// The rare exact paths, out of line so that the common path keeps its
// registers: mu + k sigma of the counts (keys of fp64 values) and the mean of
// a strided fp32 column, each an fp64 chain in instance order, every
// operation rounded on its own.
__device__ __noinline__ double threshold64(const uint64_t* ck, int N, float k) {
  double m = 0.0;
  for (int i = 0; i < N; ++i) m = __dadd_rn(m, dkey_value(ck[i]));
  m = __ddiv_rn(m, (double)N);
  double v = 0.0;
  for (int i = 0; i < N; ++i) {
    const double dv = __dsub_rn(dkey_value(ck[i]), m);
    v = __dadd_rn(v, __dmul_rn(dv, dv));
  }
  v = __ddiv_rn(v, (double)N);
  return __dadd_rn(m, __dmul_rn((double)k, __dsqrt_rn(v)));
}

__device__ __noinline__ double mean64(const float* col, int stride, int N) {
  double s = 0.0;
  for (int i = 0; i < N; ++i) s = __dadd_rn(s, (double)__ldg(col + (int64_t)i * stride));
  return __ddiv_rn(s, (double)N);
}
constexpr int kBarBatch = 1, kBarInst = 2, kBarHeur = 3;

// Warp 0 of a block computes the terms shared by the whole batch and hands
// them over through named barriers, while warps 1..7 work on requests:
//   kBarBatch  instance hashes mix64((i + 1) G) and the gpu_kv decision;
//   kBarHeur   the heuristic's request counts, the least-loaded instance,
//              imbalance and which instances are within mu + k sigma;
//   kBarInst   whether some instance-state value lies outside its bounds.
// The heuristic (Algorithm 3 pre-computes it for the gateway's fallback) is
// formed for every request, cold or not.  Its prefix match ratio
// m_i = 16 h_i / L orders instances exactly as h_i does for a fixed L (fp32
// division is monotone, and distinct h < 2^24 give distinct ratios), so the
// kernel compares hit lengths.
// Requests: S lanes per request (a group; 32 / S requests per warp).  Lane j
// of a group takes instances j, j + S, ...; group results meet through
// log2(S) xor shuffles.  The out-of-range test of the pair features needs
// only the smallest and largest hit length of the request: every pair
// feature is a monotone function of h for a fixed L (L, h, 16h, 16h/L
// rounded, L - 16h, ceil(L/16) - h), so its extremes over the instances sit
// at those two.
template <int S>
__global__ void __launch_bounds__(kGuardThreads) k_guards(const __grid_constant__ GuardArgs a) {
  __shared__ uint64_t s_ih[kHashedInst];  // mix64((i + 1) G): the instance half of the rendezvous weight
  __shared__ uint64_t s_ck[kHashedInst];  // heuristic request counts (fp64) as order-preserving keys
  __shared__ float s_c[kHashedInst];      // the counts rounded to fp32 (fast statistics)
  __shared__ uint8_t s_elig[kHashedInst]; // c_i <= mu + k sigma
  __shared__ int s_kv, s_inst_bad, s_least, s_imb;
  const int N = a.n_inst, d = kPair + a.d_inst + a.d_req;
  const int b = *reinterpret_cast<const volatile int32_t*>(&a.st->route_b);
  const float* lo = a.bounds[b == 1 ? 1 : 0];
  const float* hi = lo + d;
  const bool cold = *reinterpret_cast<const volatile int64_t*>(&a.st->ring_count) < a.n_min;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool hashed = !cold && a.K >= 1 && a.K < N && N <= kHashedInst;
  const bool heur = a.heur != 0 && a.fallback != nullptr;  // the host keeps N <= kHashedInst then

  if (warp == 0) {
    if (heur) {
      // Algorithm 1's terms in fp64 (counts c_i = queued + running, their
      // mean and population standard deviation: sums in instance order, two
      // passes, each operation rounded on its own, sqrt correctly rounded).
      // Order statistics (least loaded, c_min, c_max, the c ordering of the
      // requests) are exact through order-preserving keys of the fp64 counts.
      // The threshold mu + k sigma is first formed in fp32 with a bound on its
      // distance from the fp64 value; only when some count lies within that
      // bound (or a count is not a finite fp32 number) does lane 0 form the
      // fp64 chain, so every eligibility is the fp64 decision.
      uint64_t kmin = dkey(INFINITY), kmax = dkey(-INFINITY), kl = ~0ull;
      int least = N;
      bool finite = true;
      for (int i = lane; i < N; i += 32) {
        double c = (double)__ldg(a.inst + (int64_t)i * a.d_inst + a.c_col0);
        if (a.c_col1 >= 0) c = __dadd_rn(c, (double)__ldg(a.inst + (int64_t)i * a.d_inst + a.c_col1));
        const uint64_t k = dkey(c);
        s_ck[i] = k;
        const float c32 = __double2float_rn(c);
        s_c[i] = c32;
        finite &= fabsf(c32) < 1e30f;  // NaN fails too
        if (k != ~0ull) {               // NaN counts are skipped by min / max
          kmin = k < kmin ? k : kmin;
          kmax = k > kmax ? k : kmax;
        }
        if (least == N || k < kl || (k == kl && i < least)) { kl = k; least = i; }  // NaN after numbers
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        const uint64_t omin = __shfl_xor_sync(kFull, kmin, o), omax = __shfl_xor_sync(kFull, kmax, o);
        kmin = omin < kmin ? omin : kmin;
        kmax = omax > kmax ? omax : kmax;
        const uint64_t ok = __shfl_xor_sync(kFull, kl, o);
        const int oi = __shfl_xor_sync(kFull, least, o);
        if (oi < N && (least == N || ok < kl || (ok == kl && oi < least))) { kl = ok; least = oi; }
      }
      finite = __all_sync(kFull, finite);
      __syncwarp();
      float mu = 0.0f, sa = 0.0f;
#pragma unroll 8
      for (int i = 0; i < N; ++i) {
        mu = __fadd_rn(mu, s_c[i]);
        sa = __fadd_rn(sa, fabsf(s_c[i]));
      }
      mu = __fdiv_rn(mu, (float)N);
      float var = 0.0f;
#pragma unroll 8
      for (int i = 0; i < N; ++i) {
        const float dv = __fsub_rn(s_c[i], mu);
        var = __fadd_rn(var, __fmul_rn(dv, dv));
      }
      var = __fdiv_rn(var, (float)N);
      const float sd = __fsqrt_rn(var);
      const float thr = __fadd_rn(mu, __fmul_rn(a.k_over, sd));
      // |thr - thr64| <= delta: the mean's error from recursive summation,
      // the variance's (second order in the mean's error, plus its own
      // summation), the square root's (|sqrt x - sqrt y| <= sqrt|x - y|, or
      // |x - y| / sqrt y), and the final roundings; doubled for margin
      const float fn = (float)N;
      const float dmu = 2.0f * (fn + 2.0f) * kU * (sa / fn);
      const float dvar = dmu * dmu + 2.0f * (fn + 4.0f) * kU * (var + dmu * dmu);
      float dsd = sqrtf(dvar);
      if (sd > 0.0f) dsd = fminf(dsd, dvar / sd);
      dsd += 2.0f * kU * sd;
      const float delta = 2.0f * (dmu + fabsf(a.k_over) * dsd + 4.0f * kU * (fabsf(mu) + fabsf(a.k_over) * sd));
      bool near = !finite || !(fabsf(thr) < 1e30f) || !(delta < 1e30f);
      for (int i = lane; i < N && !near; i += 32) {
        const float c = s_c[i];
        near = c == c && fabsf(__fsub_rn(c, thr)) <= delta + 2.0f * kU * fabsf(c);
      }
      near = __any_sync(kFull, near);
      if (near) {
        double thr64 = lane == 0 ? threshold64(s_ck, N, a.k_over) : 0.0;
        thr64 = __shfl_sync(kFull, thr64, 0);
        for (int i = lane; i < N; i += 32) s_elig[i] = dkey_value(s_ck[i]) <= thr64;
      } else {
        for (int i = lane; i < N; i += 32) s_elig[i] = s_c[i] <= thr;
      }
      if (lane == 0) {
        s_least = least;
        s_imb = __dsub_rn(dkey_value(kmax), dkey_value(kmin)) > (double)a.theta_imbal;
      }
      sm100::named_bar_arrive(kBarHeur, kGuardThreads);
    }
    if (cold) return;  // no request warp waits for the rest when the batch is cold
    if (hashed)
      for (int i = lane; i < N; i += 32) s_ih[i] = bh::mix64((uint64_t)(i + 1) * kG);
    // gpu_kv: the fp64 mean (sum in instance order, divided by N) against
    // tau_sat.  An fp32 sum in the same order (lanes load 32 values at a time,
    // the sum takes them one by one) decides unless its mean lies within the
    // recursive-summation bound of tau_sat; then lane 0 forms the fp64 sum.
    int kv = 0;
    if (a.K >= 1) {
      float sum = 0.0f, sa = 0.0f;
      for (int base = 0; base < N; base += 32) {
        const int i = base + lane;
        const float v = i < N ? __ldg(a.inst + (int64_t)i * a.d_inst + a.kv_col) : 0.0f;
        const int m = N - base < 32 ? N - base : 32;
#pragma unroll 8
        for (int q = 0; q < m; ++q) {
          const float x = __shfl_sync(kFull, v, q);
          sum = __fadd_rn(sum, x);
          sa = __fadd_rn(sa, fabsf(x));
        }
      }
      const float mean = __fdiv_rn(sum, (float)N);
      const float tol = 2.0f * ((float)(N + 2) * kU * (sa / (float)N) + 2.0f * kU * fabsf(a.tau_sat));
      if (fabsf(mean) < 1e30f && tol < 1e30f && fabsf(__fsub_rn(mean, a.tau_sat)) > tol) {
        kv = mean > a.tau_sat;
      } else {
        if (lane == 0) kv = mean64(a.inst + a.kv_col, a.d_inst, N) > (double)a.tau_sat;
        kv = __shfl_sync(kFull, kv, 0);
      }
    }
    if (lane == 0) s_kv = kv;
    sm100::named_bar_arrive(kBarBatch, kGuardThreads);
    // instance rows are the same for every request of the batch: lane t takes
    // elements t, t + 32, ... of the N x d_inst block, 16 loads in flight
    int bad = 0;
    if (a.ood && a.d_inst > 0) {
      const int total = N * a.d_inst;
      const int step_i = 32 / a.d_inst, step_k = 32 % a.d_inst;
      int ei = lane / a.d_inst, ek = lane % a.d_inst;
      for (int e0 = lane; e0 < total; e0 += 16 * 32) {
        float v[16], l[16], h[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const bool ok = e0 + u * 32 < total;
          v[u] = ok ? __ldg(a.inst + (int64_t)ei * a.d_inst + ek) : 0.0f;
          l[u] = ok ? __ldg(lo + kPair + ek) : 0.0f;
          h[u] = ok ? __ldg(hi + kPair + ek) : 0.0f;
          ei += step_i;
          ek += step_k;
          if (ek >= a.d_inst) { ek -= a.d_inst; ++ei; }
        }
#pragma unroll
        for (int u = 0; u < 16; ++u) bad |= !in_range(v[u], l[u], h[u]);
      }
    }
    bad = __any_sync(kFull, bad);
    if (lane == 0) s_inst_bad = bad;
    sm100::named_bar_arrive(kBarInst, kGuardThreads);
    return;
  }

  constexpr int kPerWarp = 32 / S;
  const int j = lane & (S - 1);  // lane within the group
  const int64_t groups = (int64_t)gridDim.x * (kGuardThreads / 32 - 1) * kPerWarp;
  // every lane of a warp runs the same number of iterations (shuffles stay converged)
  const int64_t iters = ((int64_t)a.n_req + groups - 1) / groups;
  float plo[kPair], phi[kPair];
  if (a.ood) {
#pragma unroll
    for (int k = 0; k < kPair; ++k) {
      plo[k] = __ldg(lo + k);
      phi[k] = __ldg(hi + k);
    }
  }
  bool kv_ok = false, inst_bad = false;
  for (int64_t it = 0; it < iters; ++it) {
    const int64_t r = it * groups + ((int64_t)blockIdx.x * (kGuardThreads / 32 - 1) + (warp - 1)) * kPerWarp +
                      lane / S;
    const bool live = r < a.n_req;
    if (cold && live && j == 0) {
      a.choice[r] = -1;
      a.best[r] = __int_as_float(0x7fc00000);
      a.status[r] = LS_ROUTE_COLD_START;
    }
    if (cold && !heur) continue;
    // --- loads: offsets, then the first block's tokens; hits, scores, extras
    int64_t off = 0, L = 0;
    if (live) {
      off = __ldg(a.tok_off + r);
      L = __ldg(a.tok_off + r + 1) - off;
    }
    uint64_t part = 0;  // the group's lanes mix the 8 words of block 0 between them
    if (live && L >= kBlockTok)
      for (int w = j; w < 8; w += S) {
        const int32_t* p = a.tok + off + 2 * w;
        part ^= bh::word_mix((uint32_t)__ldg(p), (uint32_t)__ldg(p + 1), w);
      }
    const int32_t* hr = a.hits + r * N;
    const float* sr = a.scores + r * N;
    float bv = 0.0f;
    int bi = -1, hmax = 0, hmin = INT_MAX, bad = 0;
    if (live)
#pragma unroll 4
      for (int i = j; i < N; i += S) {
        const int h = __ldg(hr + i);
        const float v = __ldg(sr + i);
        if (bi < 0 || score_precedes(v, i, bv, bi)) { bv = v; bi = i; }
        hmax = h > hmax ? h : hmax;
        hmin = h < hmin ? h : hmin;
      }
    if (live && a.ood)
      for (int k = j; k < a.d_req; k += S) {
        const int q = kPair + a.d_inst + k;
        bad |= !in_range(__ldg(a.req + r * a.d_req + k), __ldg(lo + q), __ldg(hi + q));
      }
#pragma unroll
    for (int o = 1; o < S; o <<= 1) {
      const float ov = __shfl_xor_sync(kFull, bv, o);
      const int oi = __shfl_xor_sync(kFull, bi, o);
      if (oi >= 0 && (bi < 0 || score_precedes(ov, oi, bv, bi))) { bv = ov; bi = oi; }
      const int oh = __shfl_xor_sync(kFull, hmax, o), ol = __shfl_xor_sync(kFull, hmin, o);
      hmax = oh > hmax ? oh : hmax;
      hmin = ol < hmin ? ol : hmin;
      part ^= __shfl_xor_sync(kFull, part, o);
    }
    if (live && a.ood && j < 2) {  // lane 0 tests the pair features at hmin, lane 1 at hmax
      const int h = j == 0 ? hmin : hmax;
#pragma unroll
      for (int k = 0; k < kPair; ++k) bad |= !in_range(raw_feature(k, L, h, nullptr, 0, nullptr), plo[k], phi[k]);
    }
#pragma unroll
    for (int o = 1; o < S; o <<= 1) bad |= __shfl_xor_sync(kFull, bad, o);
    if (it == 0 && !cold) {  // the batch-wide terms from warp 0
      sm100::named_bar_sync(kBarBatch, kGuardThreads);
      kv_ok = s_kv != 0;
    }
    const bool filter = live && !cold && !bad && a.K >= 1 && L >= kBlockTok && kv_ok && (int64_t)hmax >= a.h_ben;
    // (a group filters or not as a whole; groups of one warp may differ, so
    // the shuffles below run in every group and only filtering groups use them)
    if (__any_sync(kFull, filter && a.K < N)) {
      // prefix group g = key of block 0: s_0 = G * G + c_0 (s_{-1} = G)
      const uint64_t g = bh::key_of(kG * kG + bh::mix64(part));
      // K rounds: each takes the best-ranked instance after the one taken
      // last.  The lane's weights are computed once (kept in registers for up
      // to kCached instances per lane, recomputed per round beyond that).
      constexpr int kCached = 32 / S < 4 ? 4 : 32 / S;
      uint64_t wc[kCached];
#pragma unroll
      for (int m = 0; m < kCached; ++m) {
        const int i = j + m * S;
        wc[m] = filter && i < N ? bh::mix64(g ^ (hashed ? s_ih[i] : bh::mix64((uint64_t)(i + 1) * kG))) : 0;
      }
      uint64_t tw = 0;
      int ti = -1, ci = -1;
      float cv = 0.0f;
      bool in = false;
      const int rounds = filter && a.K < N ? a.K : 0;  // K < N: every round finds an instance
      const int all_rounds = __reduce_max_sync(kFull, rounds);
      for (int k = 0; k < all_rounds; ++k) {
        uint64_t lw = 0;
        int li = -1;
        if (k < rounds) {
#pragma unroll
          for (int m = 0; m < kCached; ++m) {
            const int i = j + m * S;
            if (i < N && (ti < 0 || hrw_before(tw, ti, wc[m], i)) && (li < 0 || hrw_before(wc[m], i, lw, li))) {
              lw = wc[m];
              li = i;
            }
          }
          for (int i = j + kCached * S; i < N; i += S) {
            const uint64_t w = bh::mix64(g ^ (hashed ? s_ih[i] : bh::mix64((uint64_t)(i + 1) * kG)));
            if ((ti < 0 || hrw_before(tw, ti, w, i)) && (li < 0 || hrw_before(w, i, lw, li))) { lw = w; li = i; }
          }
        }
#pragma unroll
        for (int o = 1; o < S; o <<= 1) {
          const uint64_t ow = __shfl_xor_sync(kFull, lw, o);
          const int oi = __shfl_xor_sync(kFull, li, o);
          if (oi >= 0 && (li < 0 || hrw_before(ow, oi, lw, li))) { lw = ow; li = oi; }
        }
        if (k < rounds) {
          tw = lw;
          ti = li;
          in |= ti == bi;
          const float v = __ldg(sr + ti);
          if (ci < 0 || score_precedes(v, ti, cv, ci)) { cv = v; ci = ti; }
        }
      }
      if (filter && a.K < N && !in) { bv = cv; bi = ci; }
    }
    if (heur) {
      if (it == 0) sm100::named_bar_sync(kBarHeur, kGuardThreads);
      // Algorithm 1: the first eligible instance in the order (m desc, c asc,
      // index asc); Algorithm 2: argmax m (lowest index), kept if m > tau
      int hh = -1, hx = -1;
      uint64_t hc = 0;  // count key (fp64 order)
      if (live)
        for (int i = j; i < N; i += S) {
          if (a.heur == 1 && !s_elig[i]) continue;
          const int h = __ldg(hr + i);
          const uint64_t c = s_ck[i];
          if (hx < 0 || h > hh || (h == hh && a.heur == 1 && (c < hc || (c == hc && i < hx))) ||
              (h == hh && a.heur == 2 && i < hx)) {
            hh = h;
            hc = c;
            hx = i;
          }
        }
#pragma unroll
      for (int o = 1; o < S; o <<= 1) {
        const int oh = __shfl_xor_sync(kFull, hh, o), oi = __shfl_xor_sync(kFull, hx, o);
        const uint64_t oc = __shfl_xor_sync(kFull, hc, o);
        if (oi >= 0 && (hx < 0 || oh > hh || (oh == hh && a.heur == 1 && (oc < hc || (oc == hc && oi < hx))) ||
                        (oh == hh && a.heur == 2 && oi < hx))) {
          hh = oh;
          hc = oc;
          hx = oi;
        }
      }
      if (live && j == 0) {
        int pick = s_least;
        if (a.heur == 1 && !s_imb && hx >= 0) pick = hx;
        if (a.heur == 2 && raw_feature(3, L, hh, nullptr, 0, nullptr) > a.tau_prefix) pick = hx;
        a.fallback[r] = pick;
      }
    }
    if (cold) continue;
    if (it == 0) {  // out-of-range instance state puts every request out of range
      sm100::named_bar_sync(kBarInst, kGuardThreads);
      inst_bad = s_inst_bad != 0;
    }
    if (live && j == 0) {
      if (bad || inst_bad) {
        a.choice[r] = -1;
        a.best[r] = __int_as_float(0x7fc00000);
        a.status[r] = LS_ROUTE_OOD;
      } else {
        a.choice[r] = bi;
        a.best[r] = bv;
        a.status[r] = filter ? LS_ROUTE_KFILTER : LS_ROUTE_OK;
      }
    }
  }
}

}  // namespace

cudaError_t launch_ring_bounds(int d, const float* ring_x, int64_t capacity, int64_t replay_base,
                               int64_t replay_capacity, uint32_t* benc, float* stage, DevState* st, int sms,
                               cudaStream_t s) {
  // at least 64 rows per block, at most four blocks per SM
  int64_t grid = std::min<int64_t>((capacity + replay_capacity + 63) / 64, 4 * (int64_t)sms);
  grid = std::max<int64_t>(grid, 1);
  k_ring_bounds<<<(int)grid, 256, 0, s>>>(d, ring_x, capacity, replay_base, benc, stage, st);
  return cudaGetLastError();
}

cudaError_t launch_guards(const ls_guards& g, int n_req, int n_inst, const int32_t* tok, const int64_t* tok_off,
                          const int32_t* hits, const float* scores, const float* inst, int d_inst,
                          const float* req, int d_req, const Published* pub, const DevState* st,
                          int32_t* choice, float* best, int32_t* status, int32_t* fallback, int sms,
                          cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  GuardArgs a{};
  a.n_req = n_req;
  a.n_inst = n_inst;
  a.d_inst = d_inst;
  a.d_req = d_req;
  a.tok = tok;
  a.tok_off = tok_off;
  a.hits = hits;
  a.scores = scores;
  a.inst = inst;
  a.req = req;
  a.bounds[0] = pub[0].bounds;
  a.bounds[1] = pub[1].bounds;
  a.st = st;
  a.n_min = g.n_min;
  a.ood = g.ood != 0;
  a.K = g.k;
  a.kv_col = g.kv_col;
  a.tau_sat = g.tau_sat;
  {  // 16 h > tau_ben for an integer h  <=>  h >= floor(tau_ben / 16) + 1 (exact: a power-of-two divide)
    const double t = (double)g.tau_ben / 16.0;
    if (std::isnan(t) || t >= 9.0e18) a.h_ben = INT64_MAX;  // never
    else if (t < 0.0) a.h_ben = 0;                            // every h >= 0
    else a.h_ben = (int64_t)std::floor(t) + 1;
  }
  a.choice = choice;
  a.best = best;
  a.status = status;
  a.fallback = fallback;
  a.heur = g.heuristic;
  a.c_col0 = g.count_col[0];
  a.c_col1 = g.count_col[1];
  a.theta_imbal = g.theta_imbal;
  a.k_over = g.k_overload;
  a.tau_prefix = g.tau_prefix;
  constexpr int S = 8;
  const int64_t per_block = (kGuardThreads / 32 - 1) * (32 / S);
  const int grid = (int)std::min<int64_t>(((int64_t)n_req + per_block - 1) / per_block, (int64_t)sms * 8);
  k_guards<S><<<grid, kGuardThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace ls
