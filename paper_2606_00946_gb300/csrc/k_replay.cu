// Two-pool training data (Sec. 4.3.2 Training-data selection): a FIFO pool of
// recent records and a replay pool that admits evicted records when their
// gradient embeddings are the most diverse with respect to those kept.
//
// Rows of ring_x / ring_y: [0, C) FIFO, [C, C + P) pending ring (records the
// FIFO evicted, stream position p at row C + p mod P), [C + P, C + P + Rc)
// replay pool.  One admission round (run_replay_admit):
//   1. embedding rows: candidates t < P (pending positions not yet
//      considered, in stream order) then kept records k < Rc; chunks of the
//      training batch size go through k_replay_gather (z-score, bf16 rounding
//      in bf16 mode), the training forward, and k_replay_embed
//      (g = (yhat - y) a_last, |bf16(g)|^2, +inf for rows not in use);
//   2. nearest-neighbour distances on tensor cores (launch_rowmin_tc: bf16
//      products, fp32 sums, row minima per CTA) or on CUDA cores for small
//      shapes (k_rowmin_simt), minima combined by k_rowmin_reduce;
//   3. ranks (candidates by d desc, kept by n asc): k_replay_sort (bitonic,
//      one block per pool) when a pool fits 16384 keys, else k_replay_rank
//      (counting);
//   4. k_replay_apply: free slots filled, then pairs replaced while d > n;
//      the last block advances the pool size and the considered position.
#include "common.cuh"

namespace ls {
namespace {

constexpr unsigned kFull = 0xffffffffu;

struct ReplayGeom {
  int64_t C, P, Rc, base;  // FIFO capacity, pending capacity, replay capacity, replay row base
};

// Evicted stream positions waiting: [lo, hi), hi = count - C (>= 0), lo =
// max(admitted, hi - P): older evictions were overwritten in the pending ring.
__device__ __forceinline__ void pending_range(const DevState* st, const ReplayGeom& g, int64_t& lo, int64_t& hi) {
  const int64_t count = *reinterpret_cast<const volatile int64_t*>(&st->ring_count);
  const int64_t adm = *reinterpret_cast<const volatile int64_t*>(&st->admitted);
  hi = count > g.C ? count - g.C : 0;
  lo = hi - g.P > adm ? hi - g.P : adm;
  if (lo > hi) lo = hi;
}

// Ring row of embedding row r (candidates, then kept records), -1 if unused.
__device__ __forceinline__ int64_t embed_row_slot(int64_t r, const DevState* st, const ReplayGeom& g) {
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  if (r < g.P) return lo + r < hi ? g.C + (lo + r) % g.P : -1;
  const int64_t k = r - g.P;
  const int64_t nr = *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  return k < nr ? g.base + k : -1;
}

__global__ void k_replay_gather(int B, int64_t row0, int d, ReplayGeom g, const DevState* st,
                                const float* __restrict__ ring_x, const float* __restrict__ ring_y,
                                const float* __restrict__ mean, const float* __restrict__ stdv, int bf16,
                                float* __restrict__ x0, float* __restrict__ y, int64_t* __restrict__ counts) {
  if (row0 == 0 && blockIdx.x == 0 && threadIdx.x == 0) {  // the round's candidates and kept records
    int64_t lo, hi;
    pending_range(st, g, lo, hi);
    counts[0] = hi - lo;
    counts[1] = *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  }
  const int64_t total = (int64_t)B * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(e / d), k = (int)(e - (int64_t)j * d);
    const int64_t slot = embed_row_slot(row0 + j, st, g);
    float v = 0.0f;
    if (slot >= 0) {
      v = zscore(__ldg(ring_x + slot * d + k), __ldg(mean + k), __ldg(stdv + k));
      if (bf16) v = round_bf16(v);
    }
    x0[e] = v;
    if (k == 0) y[j] = slot >= 0 ? __ldg(ring_y + slot) : 0.0f;
  }
}

// One warp per row: g = (yhat - y) a_last (fp32), |bf16(g)|^2 summed in a
// fixed shuffle order; rows not in use get norm +inf (never nearest).
__global__ void k_replay_embed(int B, int64_t row0, int H, ReplayGeom g, const DevState* st,
                               const float* __restrict__ a_last, const float* __restrict__ yhat,
                               const float* __restrict__ y, float* __restrict__ emb, float* __restrict__ norm) {
  const int lane = threadIdx.x & 31;
  for (int64_t j = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; j < B;
       j += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t r = row0 + j;
    const bool used = embed_row_slot(r, st, g) >= 0;
    const float res = used ? yhat[j] - y[j] : 0.0f;
    float s = 0.0f;
    for (int k = lane; k < H; k += 32) {
      const float v = res * a_last[j * H + k];
      emb[r * H + k] = v;
      const float b = round_bf16(v);
      s = fmaf(b, b, s);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
    if (lane == 0) norm[r] = used ? s : INFINITY;
  }
}

// CUDA-core distances for shapes below a tensor-core tile: one warp per row,
// fp32 sums of squared differences, columns with norm +inf (unused) and the
// row's own column skipped.
__global__ void k_rowmin_simt(int M, int N, int K, const float* __restrict__ A, const float* __restrict__ Bm,
                              const float* __restrict__ na, const float* __restrict__ nb, int64_t self_off,
                              float* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  for (int64_t row = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; row < M;
       row += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    float best = INFINITY;
    for (int n = 0; n < N; ++n) {
      if (isinf(nb[n]) || (int64_t)n == row + self_off) continue;
      float s = 0.0f;
      for (int k = lane; k < K; k += 32) {
        const float t = A[row * K + k] - Bm[(int64_t)n * K + k];
        s = fmaf(t, t, s);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
      best = fminf(best, s);
    }
    if (lane == 0) out[row] = isinf(na[row]) ? INFINITY : best;
  }
}

__global__ void k_rowmin_reduce(int M, int parts, const float* __restrict__ part, int64_t ldp,
                                float* __restrict__ out) {
  for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < M; r += (int64_t)gridDim.x * blockDim.x) {
    float best = INFINITY;
    for (int q = 0; q < parts; ++q) best = fminf(best, part[r * ldp + q]);
    out[r] = best;
  }
}

__device__ __forceinline__ float div_key(float v) { return isnan(v) ? -INFINITY : v; }

// Ranks by counting.  Candidate t < m: #{f < m : (d_f, f) before (d_t, t)}
// with larger d first; kept j < nR: #{q < nR : (n_q, q) before (n_j, j)} with
// smaller n first.  inv[rank] = t (candidates), inv[P + rank] = j (kept).
__global__ void __launch_bounds__(256) k_replay_rank(ReplayGeom g, const DevState* st, const float* __restrict__ dc,
                                                     const float* __restrict__ nk, int32_t* __restrict__ inv) {
  __shared__ float tile[1024];
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  const int64_t m = hi - lo;
  const int64_t nr = *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  // blocks [0, cb) rank candidates, the rest rank kept records
  const int64_t cb = (g.P + blockDim.x - 1) / blockDim.x;
  const bool cand = blockIdx.x < cb;
  const int64_t i = (cand ? blockIdx.x : blockIdx.x - cb) * (int64_t)blockDim.x + threadIdx.x;
  const int64_t cnt = cand ? m : nr;
  const float* keys = cand ? dc : nk;
  const float mine = i < cnt ? div_key(keys[i]) : 0.0f;
  int64_t rank = 0;
  for (int64_t base = 0; base < cnt; base += 1024) {
    __syncthreads();
    for (int q = threadIdx.x; q < 1024; q += blockDim.x)
      tile[q] = base + q < cnt ? div_key(keys[base + q]) : 0.0f;
    __syncthreads();
    const int lim = cnt - base < 1024 ? (int)(cnt - base) : 1024;
    if (i < cnt)
      for (int q = 0; q < lim; ++q) {
        const float o = tile[q];
        const int64_t f = base + q;
        rank += cand ? (o > mine || (o == mine && f < i)) : (o < mine || (o == mine && f < i));
      }
  }
  if (i < cnt) inv[(cand ? 0 : g.P) + rank] = (int32_t)i;
}

// The same ranks by sorting, one block per pool (block 0 candidates, block 1
// kept records): 64-bit keys (order code << 32 | index; the candidates' code
// complemented for the descending order) sorted ascending in shared memory
// by a bitonic network over n2 (a power of two) keys, padding keys all ones.
__global__ void __launch_bounds__(1024) k_replay_sort(ReplayGeom g, const DevState* st, const float* __restrict__ dc,
                                                      const float* __restrict__ nk, int32_t* __restrict__ inv,
                                                      int n2c, int n2k) {
  extern __shared__ uint64_t key[];
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  const bool cand = blockIdx.x == 0;
  const int64_t cnt = cand ? hi - lo : *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  const int n2 = cand ? n2c : n2k;
  const float* v = cand ? dc : nk;
  for (int i = threadIdx.x; i < n2; i += blockDim.x) {
    uint64_t k = ~0ull;
    if (i < cnt) {
      const uint32_t code = ord_code(div_key(v[i]));
      k = ((uint64_t)(cand ? ~code : code) << 32) | (uint32_t)i;
    }
    key[i] = k;
  }
  __syncthreads();
  for (int k = 2; k <= n2; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += blockDim.x) {
        const int p = i ^ j;
        if (p > i) {
          const uint64_t a = key[i], b = key[p];
          if ((a > b) == ((i & k) == 0)) {
            key[i] = b;
            key[p] = a;
          }
        }
      }
      __syncthreads();
    }
  for (int r = threadIdx.x; r < cnt; r += blockDim.x) inv[(cand ? 0 : g.P) + r] = (int32_t)(key[r] & 0xffffffffu);
}

// One warp per candidate rank t: free slots first, then pairs while d > n.
__global__ void __launch_bounds__(256) k_replay_apply(int d, ReplayGeom g, DevState* st, const float* __restrict__ dc,
                                                      const float* __restrict__ nk, const int32_t* __restrict__ inv,
                                                      float* ring_x, float* ring_y) {
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  const int64_t m = hi - lo;
  const int64_t nr = *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  const int64_t free_slots = g.Rc - nr;
  const int lane = threadIdx.x & 31;
  for (int64_t t = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; t < m;
       t += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t c = inv[t];
    int64_t dest = -1;
    if (t < free_slots) {
      dest = nr + t;
    } else if (t - free_slots < nr) {
      const int64_t j = inv[g.P + (t - free_slots)];
      if (div_key(dc[c]) > div_key(nk[j])) dest = j;
    }
    if (dest < 0) continue;
    const int64_t src = g.C + (lo + c) % g.P, dst = g.base + dest;
    for (int k = lane; k < d; k += 32) ring_x[dst * d + k] = ring_x[src * d + k];
    if (lane == 0) ring_y[dst] = ring_y[src];
  }
  if (last_block(&st->done[DONE_REPLAY]) && threadIdx.x == 0) {
    st->replay_count = nr + (m < free_slots ? m : free_slots);
    st->admitted = hi;
  }
}

constexpr int kSortMax = 16384;  // keys a block sorts in shared memory (128 KB)

int grid_for(int64_t threads, int sms) {
  const int64_t b = (threads + 255) / 256;
  return (int)std::max<int64_t>(1, std::min<int64_t>(b, (int64_t)sms * 8));
}

}  // namespace

cudaError_t run_replay_admit(Ctx& c, float* d_out, float* n_out, cudaStream_t s) {
  const MlpDesc& m = c.mlp;
  const int L = m.n_layers;
  const int H = m.w[L - 1];
  ReplayGeom g{c.cfg.ring_capacity, c.cfg.pending_capacity, c.cfg.replay_capacity, c.replay_base};
  const int64_t rows = g.P + g.Rc;
  const int Bc = c.cfg.max_train_batch;
  cudaError_t e = cudaSuccess;
  // 1. embeddings, in chunks of the training batch size
  for (int64_t row0 = 0; row0 < rows; row0 += Bc) {
    const int B = (int)std::min<int64_t>(Bc, rows - row0);
    e = traced(c, TR_REPLAY, 1, s, [&] {
      k_replay_gather<<<grid_for((int64_t)B * m.w[0], c.sms), 256, 0, s>>>(
          B, row0, m.w[0], g, c.st, c.ring_x, c.ring_y, c.mean, c.stdv, m.bf16, c.tx, c.ty, c.rcount);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
    e = forward_rows(c, B, s);
    if (e != cudaSuccess) return e;
    int64_t xoff = 0, zoff = 0;
    for (int l = 0; l < L - 1; ++l) {
      xoff += (int64_t)B * m.w[l];
      zoff += (int64_t)B * m.w[l + 1];
    }
    e = traced(c, TR_REPLAY, 1, s, [&] {
      k_replay_embed<<<grid_for((int64_t)B * 32, c.sms), 256, 0, s>>>(B, row0, H, g, c.st, c.tx + xoff, c.tz + zoff,
                                                                        c.ty, c.remb, c.rnorm);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
  }
  // 2. nearest kept embedding of every candidate, nearest other kept of every kept record
  const float* Ec = c.remb;
  const float* Ek = c.remb + g.P * H;
  const float* nc = c.rnorm;
  const float* nkp = c.rnorm + g.P;
  const int64_t kNoSelf = -(int64_t(1) << 62);
  auto rowmin = [&](int M, const float* A, const float* na, int64_t self_off, const int64_t* rows_in_use,
                    float* out) -> cudaError_t {
    int parts = 0;
    cudaError_t r = traced(c, TR_REPLAY, 1, s, [&] {
      return launch_rowmin_tc(M, (int)g.Rc, H, A, H, Ek, H, na, nkp, self_off, c.rpart, kRowMinParts, rows_in_use,
                              c.rcount + 1, &parts, c.d_err, c.sms, s);
    });
    if (r == cudaSuccess) {
      return traced(c, TR_REPLAY, 1, s, [&] {
        k_rowmin_reduce<<<grid_for(M, c.sms), 256, 0, s>>>(M, parts, c.rpart, kRowMinParts, out);
        return cudaGetLastError();
      });
    }
    if (r != cudaErrorInvalidValue) return r;
    (void)cudaGetLastError();
    return traced(c, TR_REPLAY, 1, s, [&] {
      k_rowmin_simt<<<grid_for((int64_t)M * 32, c.sms), 256, 0, s>>>(M, (int)g.Rc, H, A, Ek, na, nkp, self_off, out);
      return cudaGetLastError();
    });
  };
  e = rowmin((int)g.P, Ec, nc, kNoSelf, c.rcount, c.rd);
  if (e != cudaSuccess) return e;
  e = rowmin((int)g.Rc, Ek, nkp, 0, c.rcount + 1, c.rn);
  if (e != cudaSuccess) return e;
  if (d_out) {
    e = cudaMemcpyAsync(d_out, c.rd, (size_t)g.P * sizeof(float), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
  }
  if (n_out) {
    e = cudaMemcpyAsync(n_out, c.rn, (size_t)g.Rc * sizeof(float), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
  }
  // 3. ranks, 4. admission
  e = traced(c, TR_REPLAY, 1, s, [&] {
    int n2c = 1, n2k = 1;
    while (n2c < g.P) n2c <<= 1;
    while (n2k < g.Rc) n2k <<= 1;
    const int n2 = std::max(n2c, n2k);
    if (n2 <= kSortMax) {
      const int smem = n2 * (int)sizeof(uint64_t);
      cudaError_t a = cudaFuncSetAttribute(k_replay_sort, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (a != cudaSuccess) return a;
      k_replay_sort<<<2, 1024, smem, s>>>(g, c.st, c.rd, c.rn, c.rinv, n2c, n2k);
    } else {
      const int blocks = (int)((g.P + 255) / 256 + (g.Rc + 255) / 256);
      k_replay_rank<<<blocks, 256, 0, s>>>(g, c.st, c.rd, c.rn, c.rinv);
    }
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  return traced(c, TR_REPLAY, 1, s, [&] {
    k_replay_apply<<<grid_for(g.P * 32, c.sms), 256, 0, s>>>(m.w[0], g, c.st, c.rd, c.rn, c.rinv, c.ring_x,
                                                             c.ring_y);
    return cudaGetLastError();
  });
}

}  // namespace ls
