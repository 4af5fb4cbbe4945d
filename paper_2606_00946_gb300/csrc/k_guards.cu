// Guards of Algorithm 4 around the greedy selection (Sec. 4.3.1 "Fallback":
// cold start and out-of-range inputs hand the request back to the gateway's
// heuristic; Sec. 4.1 "Consistent hashing based filtering": under cluster
// memory saturation the choice is confined to K instances picked by
// consistent hashing of the request's prefix group).
//
//   k_ring_bounds  feature bounds [l, u] of the training buffer: column-wise
//                  minimum / maximum over the records the ring holds (NaN
//                  skipped), block partials combined by the last block into
//                  the staging copy that the next publish makes visible.
//                  Bound: HBM, 4 d bytes per held record.
//   k_guards       one warp per request: cold-start test, out-of-range test of
//                  every raw feature of every pair, argmin, K-filter.  Reads
//                  the hits and scores of the request (8 bytes per pair), its
//                  first 64 prompt bytes and its extras; writes 12 bytes.
#include "blockhash.cuh"
#include "common.cuh"

namespace ls {
namespace {

constexpr unsigned kFull = 0xffffffffu;

// ---------------------------------------------------------------------------
// feature bounds of the sample ring
// ---------------------------------------------------------------------------

// Rows [0, min(count, capacity)) split into gridDim.x contiguous ranges.  For
// d <= 256 the block reads P = 256 / d rows per pass (thread t: column t % d,
// row phase t / d), so one pass reads a contiguous run of P d floats; wider
// rows take columns t, t + 256, ... of every row.
__global__ void __launch_bounds__(256) k_ring_bounds(int d, const float* __restrict__ ring_x, int64_t capacity,
                                                     float* __restrict__ bpart, float* __restrict__ stage,
                                                     DevState* st) {
  __shared__ float s_lo[256], s_hi[256];
  const int64_t count = *reinterpret_cast<volatile int64_t*>(&st->ring_count);
  const int64_t rows = count < capacity ? count : capacity;
  const int64_t per = (rows + gridDim.x - 1) / gridDim.x;
  const int64_t r0 = (int64_t)blockIdx.x * per;
  const int64_t r1 = r0 + per < rows ? r0 + per : rows;
  const bool narrow = d <= 256;
  const int P = narrow ? 256 / d : 1;
  const int p = narrow ? (int)threadIdx.x / d : 0;
  float* part = bpart + (int64_t)blockIdx.x * 2 * d;
  for (int c = narrow ? (int)threadIdx.x % d : (int)threadIdx.x; c < d; c += narrow ? d : 256) {
    float lo = INFINITY, hi = -INFINITY;
    if (p < P) {
      const float* col = ring_x + c;
      int64_t r = r0 + p;
      // four rows in flight per thread
      for (; r + 3 * (int64_t)P < r1; r += 4 * (int64_t)P) {
        float v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = __ldcs(col + (r + (int64_t)u * P) * d);
#pragma unroll
        for (int u = 0; u < 4; ++u) {  // NaN fails both comparisons: skipped
          lo = v[u] < lo ? v[u] : lo;
          hi = v[u] > hi ? v[u] : hi;
        }
      }
      for (; r < r1; r += P) {
        const float v = __ldcs(col + r * d);
        lo = v < lo ? v : lo;
        hi = v > hi ? v : hi;
      }
    }
    if (narrow) {
      if (p < P) {
        s_lo[threadIdx.x] = lo;
        s_hi[threadIdx.x] = hi;
      }
    } else {
      part[c] = lo;
      part[d + c] = hi;
    }
  }
  if (narrow) {
    __syncthreads();
    if ((int)threadIdx.x < d) {
      float lo = s_lo[threadIdx.x], hi = s_hi[threadIdx.x];
      for (int q = 1; q < P; ++q) {
        const float l2 = s_lo[q * d + threadIdx.x], h2 = s_hi[q * d + threadIdx.x];
        lo = l2 < lo ? l2 : lo;
        hi = h2 > hi ? h2 : hi;
      }
      part[threadIdx.x] = lo;
      part[d + threadIdx.x] = hi;
    }
  }
  if (last_block(&st->done[DONE_BOUNDS])) {
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      float lo = INFINITY, hi = -INFINITY;
      for (int b = 0; b < (int)gridDim.x; ++b) {
        const float l2 = __ldcg(bpart + (int64_t)b * 2 * d + c);
        const float h2 = __ldcg(bpart + (int64_t)b * 2 * d + d + c);
        lo = l2 < lo ? l2 : lo;
        hi = h2 > hi ? h2 : hi;
      }
      stage[c] = lo;
      stage[d + c] = hi;
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
  int ood, K, kv_col;
  float tau_sat, tau_ben;
  int32_t* choice;
  float* best;
  int32_t* status;
};

// (wa, a) ranks before (wb, b) in rendezvous order: larger weight, then lower index.
__device__ __forceinline__ bool hrw_before(uint64_t wa, int a, uint64_t wb, int b) {
  return wa != wb ? wa > wb : a < b;
}

__device__ __forceinline__ bool in_range(float x, float lo, float hi) { return x >= lo && x <= hi; }

__global__ void __launch_bounds__(256) k_guards(const __grid_constant__ GuardArgs a) {
  __shared__ float s_lo[kPair], s_hi[kPair];
  __shared__ int s_kv;
  const int N = a.n_inst, d = kPair + a.d_inst + a.d_req;
  const int b = *reinterpret_cast<const volatile int32_t*>(&a.st->route_b);
  const float* lo = a.bounds[b == 1 ? 1 : 0];
  const float* hi = lo + d;
  const bool cold = *reinterpret_cast<const volatile int64_t*>(&a.st->ring_count) < a.n_min;
  int inst_bad = 0;
  if (!cold && a.ood) {
    // instance rows are the same for every request of the batch
    for (int e = threadIdx.x; e < N * a.d_inst; e += blockDim.x) {
      const int k = kPair + e % a.d_inst;
      inst_bad |= !in_range(__ldg(a.inst + e), __ldg(lo + k), __ldg(hi + k));
    }
    if (threadIdx.x < kPair) {
      s_lo[threadIdx.x] = __ldg(lo + threadIdx.x);
      s_hi[threadIdx.x] = __ldg(hi + threadIdx.x);
    }
  }
  if (threadIdx.x == 0) {
    int kv = 0;
    if (!cold && a.K >= 1) {  // gpu_kv mean: fp64, instance order
      double sum = 0.0;
      for (int i = 0; i < N; ++i) sum += (double)__ldg(a.inst + (int64_t)i * a.d_inst + a.kv_col);
      kv = sum / (double)N > (double)a.tau_sat;
    }
    s_kv = kv;
  }
  inst_bad = __syncthreads_or(inst_bad);
  const bool kv_ok = s_kv != 0;

  const int lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  for (int64_t r = (int64_t)blockIdx.x * warps + (threadIdx.x >> 5); r < a.n_req;
       r += (int64_t)gridDim.x * warps) {
    if (cold) {
      if (lane == 0) {
        a.choice[r] = -1;
        a.best[r] = __int_as_float(0x7fc00000);
        a.status[r] = LS_ROUTE_COLD_START;
      }
      continue;
    }
    const int64_t off = __ldg(a.tok_off + r);
    const int64_t L = __ldg(a.tok_off + r + 1) - off;
    const int32_t* hr = a.hits + r * N;
    const float* sr = a.scores + r * N;
    float bv = 0.0f;
    int bi = -1, hmax = 0, bad = inst_bad;
    for (int i = lane; i < N; i += 32) {
      const int h = __ldg(hr + i);
      const float v = __ldg(sr + i);
      if (bi < 0 || score_precedes(v, i, bv, bi)) { bv = v; bi = i; }
      hmax = h > hmax ? h : hmax;
      if (a.ood) {
#pragma unroll
        for (int k = 0; k < kPair; ++k)
          bad |= !in_range(raw_feature(k, L, h, nullptr, 0, nullptr), s_lo[k], s_hi[k]);
      }
    }
    if (a.ood)
      for (int k = lane; k < a.d_req; k += 32) {
        const int j = kPair + a.d_inst + k;
        bad |= !in_range(__ldg(a.req + r * a.d_req + k), __ldg(lo + j), __ldg(hi + j));
      }
    if (__any_sync(kFull, bad)) {
      if (lane == 0) {
        a.choice[r] = -1;
        a.best[r] = __int_as_float(0x7fc00000);
        a.status[r] = LS_ROUTE_OOD;
      }
      continue;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float ov = __shfl_xor_sync(kFull, bv, o);
      const int oi = __shfl_xor_sync(kFull, bi, o);
      if (oi >= 0 && (bi < 0 || score_precedes(ov, oi, bv, bi))) { bv = ov; bi = oi; }
    }
    hmax = __reduce_max_sync(kFull, hmax);
    int code = LS_ROUTE_OK;
    if (a.K >= 1 && L >= kBlockTok && kv_ok && 16.0 * (double)hmax > (double)a.tau_ben) {
      code = LS_ROUTE_KFILTER;
      if (a.K < N) {
        // prefix group g = key of block 0: s_0 = G * G + c_0 (s_{-1} = G)
        uint64_t part = 0;
        if (lane < 8) {
          const int32_t* p = a.tok + off + 2 * lane;
          part = bh::word_mix((uint32_t)__ldg(p), (uint32_t)__ldg(p + 1), lane);
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) part ^= __shfl_xor_sync(kFull, part, o);
        const uint64_t g = bh::key_of(kG * kG + bh::mix64(__shfl_sync(kFull, part, 0)));
        // K rounds: each takes the best-ranked instance after the one taken last
        uint64_t tw = 0;
        int ti = -1, ci = -1;
        float cv = 0.0f;
        bool in = false;
        for (int k = 0; k < a.K; ++k) {
          uint64_t lw = 0;
          int li = -1;
          for (int i = lane; i < N; i += 32) {
            const uint64_t w = bh::mix64(g ^ bh::mix64((uint64_t)(i + 1) * kG));
            if ((ti < 0 || hrw_before(tw, ti, w, i)) && (li < 0 || hrw_before(w, i, lw, li))) { lw = w; li = i; }
          }
#pragma unroll
          for (int o = 16; o; o >>= 1) {
            const uint64_t ow = __shfl_xor_sync(kFull, lw, o);
            const int oi = __shfl_xor_sync(kFull, li, o);
            if (oi >= 0 && (li < 0 || hrw_before(ow, oi, lw, li))) { lw = ow; li = oi; }
          }
          tw = lw;
          ti = li;
          in |= ti == bi;
          const float v = __ldg(sr + ti);
          if (ci < 0 || score_precedes(v, ti, cv, ci)) { cv = v; ci = ti; }
        }
        if (!in) { bv = cv; bi = ci; }
      }
    }
    if (lane == 0) {
      a.choice[r] = bi;
      a.best[r] = bv;
      a.status[r] = code;
    }
  }
}

}  // namespace

cudaError_t launch_ring_bounds(int d, const float* ring_x, int64_t capacity, float* bpart, float* stage,
                               DevState* st, int sms, cudaStream_t s) {
  // about 64 rows per block at least; never more blocks than partial slots
  int64_t grid = (capacity + 63) / 64;
  grid = std::min<int64_t>(grid, std::min<int64_t>(kBoundsBlocks, 2 * (int64_t)sms));
  grid = std::max<int64_t>(grid, 1);
  k_ring_bounds<<<(int)grid, 256, 0, s>>>(d, ring_x, capacity, bpart, stage, st);
  return cudaGetLastError();
}

cudaError_t launch_guards(const ls_guards& g, int n_req, int n_inst, const int32_t* tok, const int64_t* tok_off,
                          const int32_t* hits, const float* scores, const float* inst, int d_inst,
                          const float* req, int d_req, const Published* pub, const DevState* st,
                          int32_t* choice, float* best, int32_t* status, int sms, cudaStream_t s) {
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
  a.tau_ben = g.tau_ben;
  a.choice = choice;
  a.best = best;
  a.status = status;
  const int64_t blocks = ((int64_t)n_req + 7) / 8;
  const int grid = (int)std::min<int64_t>(blocks, (int64_t)sms * 8);
  k_guards<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace ls
