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
//   3. ranks (candidates by d desc, kept by n asc) by counting over
//      (element tile, key tile) blocks (k_replay_rank), inverted by
//      k_replay_inv;
//   4. k_replay_apply: free slots filled, then pairs replaced while d > n;
//      the last block advances the pool size and the considered position.
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
namespace {
using namespace sm100;

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

// The forward runs over compact rows u: candidates t = u < m, then kept
// records k = u - m < nR.  Embedding row (the image's and the norms' index):
// candidate t -> t, kept record k -> P + k.
__device__ __forceinline__ int64_t compact_slot(int64_t u, const int64_t* counts, const ReplayGeom& g,
                                                int64_t lo) {
  const int64_t m = counts[0], nr = counts[1];
  if (u < m) return g.C + (lo + u) % g.P;
  return u < m + nr ? g.base + (u - m) : -1;
}

// The round's counts (candidates, kept records, rows in use per forward
// chunk of B) and every norm reset to +inf (rows the round does not use).
__global__ void k_replay_prep(ReplayGeom g, const DevState* st, int B, int nchunks, int64_t* __restrict__ counts,
                              float* __restrict__ norm, int32_t* __restrict__ rank) {
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  const int64_t m = hi - lo, nr = *reinterpret_cast<const volatile int64_t*>(&st->replay_count);
  if (threadIdx.x == 0) {
    counts[0] = m;
    counts[1] = nr;
    for (int c = 0; c < nchunks; ++c) {
      const int64_t v = m + nr - (int64_t)c * B;
      counts[2 + c] = v < 0 ? 0 : (v > B ? B : v);
    }
  }
  for (int64_t r = threadIdx.x; r < g.P + g.Rc; r += blockDim.x) {
    norm[r] = INFINITY;
    rank[r] = 0;
  }
}

__global__ void k_replay_gather(int B, int64_t row0, int d, ReplayGeom g, const DevState* st,
                                const float* __restrict__ ring_x, const float* __restrict__ ring_y,
                                const float* __restrict__ mean, const float* __restrict__ stdv, int bf16,
                                float* __restrict__ x0, float* __restrict__ y, const int64_t* __restrict__ counts) {
  int64_t lo, hi;
  pending_range(st, g, lo, hi);
  const int64_t total = (int64_t)B * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(e / d), k = (int)(e - (int64_t)j * d);
    const int64_t slot = compact_slot(row0 + j, counts, g, lo);
    float v = 0.0f;
    if (slot >= 0) {
      v = zscore(__ldg(ring_x + slot * d + k), __ldg(mean + k), __ldg(stdv + k));
      if (bf16) v = round_bf16(v);
    }
    x0[e] = v;
    if (k == 0) y[j] = slot >= 0 ? __ldg(ring_y + slot) : 0.0f;
  }
}

// One warp per compact row: g = (yhat - y) a_last (fp32) and |bf16(g)|^2
// (summed in a fixed shuffle order) at its embedding row; rows the round does
// not use keep the +inf norm k_replay_prep gave them (never nearest).  With an
// image (bf16 distances on tensor cores) the bf16 row also goes to its
// 128-row tile: candidate tiles first, then kept tiles.
__global__ void k_replay_embed(int B, int64_t row0, int H, ReplayGeom g, const int64_t* __restrict__ counts,
                               const float* __restrict__ a_last, const float* __restrict__ yhat,
                               const float* __restrict__ y, float* __restrict__ emb, float* __restrict__ norm,
                               uint8_t* __restrict__ img, int tilesC) {
  const int lane = threadIdx.x & 31;
  const int64_t m = counts[0], nr = counts[1];
  for (int64_t j = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; j < B;
       j += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t u = row0 + j;
    if (u >= m + nr) break;                 // rows past the round's records (warp-uniform)
    const int64_t r = u < m ? u : g.P + (u - m);
    const float res = yhat[j] - y[j];
    float s = 0.0f;
    uint8_t* trow = nullptr;
    int rr = 0;
    if (img) {
      const int64_t tl = r < g.P ? r / 128 : tilesC + (r - g.P) / 128;
      rr = (int)(r < g.P ? r % 128 : (r - g.P) % 128);
      trow = img + tl * (int64_t)128 * H * 2;
    }
    for (int k = lane; k < H; k += 32) {
      const float v = res * a_last[j * H + k];
      emb[r * H + k] = v;
      const float b = round_bf16(v);
      s = fmaf(b, b, s);
      if (trow) *reinterpret_cast<__nv_bfloat16*>(trow + sm100::sw128_offset(rr, k, 128)) = __float2bfloat16_rn(v);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
    if (lane == 0) norm[r] = s;
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

// Both pools' partial minima (rows [0, P) candidates, [P, P + Rc) kept).
__global__ void k_rowmin_reduce2(int P, int rows, int parts, const float* __restrict__ part, int64_t ldp,
                                 float* __restrict__ dc, float* __restrict__ nk) {
  for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x) {
    float best = INFINITY;
    for (int q = 0; q < parts; ++q) best = fminf(best, part[r * ldp + q]);
    if (r < P) dc[r] = best;
    else nk[r - P] = best;
  }
}

__device__ __forceinline__ float div_key(float v) { return isnan(v) ? -INFINITY : v; }

// ---------------------------------------------------------------------------
// nearest-neighbour distances on tensor cores from a bf16 embedding image
// ---------------------------------------------------------------------------
// The image holds the embeddings as 128-row tiles (candidate tiles, then kept
// tiles) of H/64 K-major 128-byte-swizzled slabs of 16 KB, so one bulk copy
// per slab lands a tile in the MMA layout.  CTA (row tile, column split):
// its 128 rows against a range of kept 128-row column tiles; warp 0 issues
// the MMAs into two TMEM accumulators, warp 1 bulk-copies the row tile once
// and the column tiles through two buffers, warps 2..5 (one TMEM lane
// quadrant each) turn each accumulator into the row minima of
// |g_r|^2 + |g_c|^2 - 2 g_r.g_c (the row's own kept column skipped).
constexpr int kDistThreads = 192;
constexpr int kSlab = 16384;       // 128 rows x 64 bf16

struct DistArgs {
  const uint8_t* img;
  const float* norm;               // [P + Rc] (+inf for rows not in use)
  float* part;                     // [(P + Rc), ldp]
  int64_t ldp;
  const int64_t* counts;           // [candidates, kept] of the round
  int P, Rc, H;
  int tilesC, tilesK, splits, per_split;  // column tiles per split
  int* err;
};

__global__ void __launch_bounds__(kDistThreads, 1) k_dist_rowmin(const __grid_constant__ DistArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int kb = a.H / 64;
  uint8_t* sA = smem;
  uint8_t* sB[2] = {smem + kb * kSlab, smem + 2 * kb * kSlab};
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 3 * kb * kSlab);
  uint64_t *a_full = bar, *b_full = bar + 1, *b_empty = bar + 3, *acc_full = bar + 5, *acc_empty = bar + 7;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bar + 9);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x / a.splits, split = blockIdx.x - tile * a.splits;
  const bool kept_rows = tile >= a.tilesC;
  const int rtile = kept_rows ? tile - a.tilesC : tile;       // row tile inside its region
  const int64_t rows_used = kept_rows ? a.counts[1] : a.counts[0];
  const int64_t ktiles_used = (a.counts[1] + 127) / 128;
  const int t0 = split * a.per_split;
  int T = (int)(ktiles_used - t0);
  T = T < 0 ? 0 : (T > a.per_split ? a.per_split : T);
  const int base_row = kept_rows ? a.P : 0;                   // first norm / partial row of the region
  // epilogue thread -> row: warps 2..5 own TMEM lane quadrants warp & 3
  const int q = warp & 3;
  const int row = rtile * 128 + 32 * q + lane;                // row inside the region
  const int region_rows = kept_rows ? a.Rc : a.P;
  if ((int64_t)rtile * 128 >= rows_used || T == 0) {          // nothing of this CTA is in use
    if (warp >= 2 && row < region_rows) a.part[(int64_t)(base_row + row) * a.ldp + split] = INFINITY;
    return;
  }
  if (tid == 0) {
    mbar_init(a_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_full + i, 1);
      mbar_init(b_empty + i, 1);
      mbar_init(acc_full + i, 1);
      mbar_init(acc_empty + i, 4);
    }
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t tile_bytes = (uint32_t)kb * kSlab;
  const uint8_t* imgA = a.img + (int64_t)tile * tile_bytes;
  const uint8_t* imgB = a.img + (int64_t)(a.tilesC + t0) * tile_bytes;
  bool ok = true;

  if (warp == 1) {
    if (lane == 0) {
      mbar_arrive_expect_tx(a_full, tile_bytes);
      for (int k = 0; k < kb; ++k) bulk_g2s(sA + k * kSlab, imgA + k * kSlab, kSlab, a_full);
      for (int t = 0; t < T && ok; ++t) {
        const int b = t & 1;
        if (t >= 2 && !mbar_wait(b_empty + b, (uint32_t)(((t - 2) >> 1) & 1))) ok = false;
        if (!ok) break;
        mbar_arrive_expect_tx(b_full + b, tile_bytes);
        for (int k = 0; k < kb; ++k)
          bulk_g2s(sB[b] + k * kSlab, imgB + (int64_t)t * tile_bytes + k * kSlab, kSlab, b_full + b);
      }
      if (!ok) latch_error(a.err, LS_ERR_TIMEOUT);
    }
  } else if (warp == 0) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, 128);
      if (!mbar_wait(a_full, 0)) ok = false;
      for (int t = 0; t < T && ok; ++t) {
        const int b = t & 1;
        if (!mbar_wait(b_full + b, (uint32_t)((t >> 1) & 1))) { ok = false; break; }
        if (t >= 2 && !mbar_wait(acc_empty + b, (uint32_t)(((t - 2) >> 1) & 1))) { ok = false; break; }
        tc_fence_after();
        const uint32_t ab = smem_u32(sA), bb = smem_u32(sB[b]);
        for (int k = 0; k < kb; ++k)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            umma_bf16(tmem + (uint32_t)(128 * b), sdesc_sw128(ab + k * kSlab + 32u * j),
                      sdesc_sw128(bb + k * kSlab + 32u * j), idesc, (k | j) ? 1u : 0u);
        umma_commit(b_empty + b);
        umma_commit(acc_full + b);
      }
      if (!ok) latch_error(a.err, LS_ERR_TIMEOUT);
    }
  } else {
    const float na = row < region_rows ? __ldg(a.norm + base_row + row) : INFINITY;
    const int self = kept_rows ? row : -1;                    // the row's own kept column
    const uint32_t lane_addr = (uint32_t)(32 * q) << 16;
    float rmin = INFINITY;
    for (int t = 0; t < T; ++t) {
      const int b = t & 1;
      const int col0 = (t0 + t) * 128;
      if (!mbar_wait(acc_full + b, (uint32_t)((t >> 1) & 1))) {
        if (lane == 0) latch_error(a.err, LS_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      for (int c = 0; c < 128; c += 32) {
        float nb[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) nb[u] = col0 + c + u < a.Rc ? __ldg(a.norm + a.P + col0 + c + u) : INFINITY;
        uint32_t v[32];
        tmem_ld32(tmem + lane_addr + (uint32_t)(128 * b + c), v);
        tmem_wait_ld();
#pragma unroll
        for (int u = 0; u < 32; ++u) {
          const float dist = na + nb[u] - 2.0f * __uint_as_float(v[u]);
          if (col0 + c + u != self) rmin = fminf(rmin, dist);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty + b);
    }
    if (row < region_rows) a.part[(int64_t)(base_row + row) * a.ldp + split] = rmin;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

// Ranks by counting, tiled over (element tile, key tile): each block counts,
// for its 256 elements, the keys of one 1024-key tile that come before them
// (candidates: larger d first; kept records: smaller n first; equal keys by
// index) and adds the count to rank[] (integer sums: the order of the
// additions does not matter).  rank[] was zeroed by k_replay_prep.
__global__ void __launch_bounds__(256) k_replay_rank(ReplayGeom g, const int64_t* __restrict__ counts,
                                                     const float* __restrict__ dc, const float* __restrict__ nk,
                                                     int32_t* __restrict__ rank) {
  __shared__ float tile[1024];
  const int64_t cb = (g.P + 255) / 256;               // element tiles of the candidates
  const bool cand = blockIdx.x < cb;
  const int64_t i = (cand ? blockIdx.x : blockIdx.x - cb) * 256 + threadIdx.x;
  const int64_t cnt = cand ? counts[0] : counts[1];
  const int64_t base = (int64_t)blockIdx.y * 1024;
  if ((cand ? blockIdx.x : blockIdx.x - cb) * 256 >= cnt || base >= cnt) return;   // block-uniform
  const float* keys = cand ? dc : nk;
  for (int q = threadIdx.x; q < 1024; q += 256) tile[q] = base + q < cnt ? div_key(keys[base + q]) : 0.0f;
  __syncthreads();
  if (i >= cnt) return;
  const float mine = div_key(keys[i]);
  const int lim = cnt - base < 1024 ? (int)(cnt - base) : 1024;
  int r = 0;
  for (int q = 0; q < lim; ++q) {
    const float o = tile[q];
    const int64_t f = base + q;
    r += cand ? (o > mine || (o == mine && f < i)) : (o < mine || (o == mine && f < i));
  }
  if (r) atomicAdd(rank + (cand ? 0 : g.P) + i, r);
}

// inv[rank] = element (candidates at [0, P), kept records at [P, P + Rc)).
__global__ void k_replay_inv(ReplayGeom g, const int64_t* __restrict__ counts, const int32_t* __restrict__ rank,
                             int32_t* __restrict__ inv) {
  const int64_t m = counts[0], nr = counts[1];
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < g.P + g.Rc;
       e += (int64_t)gridDim.x * blockDim.x) {
    const bool cand = e < g.P;
    const int64_t i = cand ? e : e - g.P;
    if (i < (cand ? m : nr)) inv[(cand ? 0 : g.P) + rank[e]] = (int32_t)i;
  }
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
  const int tilesC = (int)((g.P + 127) / 128), tilesK = (int)((g.Rc + 127) / 128);
  cudaError_t e = cudaSuccess;
  // 1. embeddings of the round's records (compact rows), in chunks of the training batch size
  const int nchunks = (int)((rows + Bc - 1) / Bc);
  e = traced(c, TR_REPLAY, 1, s, [&] {
    k_replay_prep<<<1, 1024, 0, s>>>(g, c.st, Bc, nchunks, c.rcount, c.rnorm, c.rrank);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  for (int64_t row0 = 0; row0 < rows; row0 += Bc) {
    const int B = (int)std::min<int64_t>(Bc, rows - row0);
    const int64_t* chunk_rows = c.rcount + 2 + row0 / Bc;
    e = traced(c, TR_REPLAY, 1, s, [&] {
      k_replay_gather<<<grid_for((int64_t)B * m.w[0], c.sms), 256, 0, s>>>(
          B, row0, m.w[0], g, c.st, c.ring_x, c.ring_y, c.mean, c.stdv, m.bf16, c.tx, c.ty, c.rcount);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
    e = forward_rows(c, B, s, chunk_rows);
    if (e != cudaSuccess) return e;
    int64_t xoff = 0, zoff = 0;
    for (int l = 0; l < L - 1; ++l) {
      xoff += (int64_t)B * m.w[l];
      zoff += (int64_t)B * m.w[l + 1];
    }
    e = traced(c, TR_REPLAY, 1, s, [&] {
      k_replay_embed<<<grid_for((int64_t)B * 32, c.sms), 256, 0, s>>>(B, row0, H, g, c.rcount, c.tx + xoff,
                                                                        c.tz + zoff, c.ty, c.remb, c.rnorm, c.rimg,
                                                                        tilesC);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
  }
  // 2. nearest kept embedding of every candidate, nearest other kept of every kept record
  if (c.rimg) {  // bf16 image: one launch for both, then one reduction
    DistArgs da{};
    da.img = c.rimg;
    da.norm = c.rnorm;
    da.part = c.rpart;
    da.ldp = kRowMinParts;
    da.counts = c.rcount;
    da.P = (int)g.P;
    da.Rc = (int)g.Rc;
    da.H = H;
    da.tilesC = tilesC;
    da.tilesK = tilesK;
    da.splits = std::max(1, std::min(std::min(tilesK, kRowMinParts), 2 * c.sms / (tilesC + tilesK)));
    da.per_split = (tilesK + da.splits - 1) / da.splits;
    da.err = c.d_err;
    const int smem = 1024 + 3 * (H / 64) * kSlab + 128;
    e = traced(c, TR_REPLAY, 1, s, [&] {
      cudaError_t a = cudaFuncSetAttribute(k_dist_rowmin, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (a != cudaSuccess) return a;
      k_dist_rowmin<<<(tilesC + tilesK) * da.splits, kDistThreads, smem, s>>>(da);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
    e = traced(c, TR_REPLAY, 1, s, [&] {
      k_rowmin_reduce2<<<grid_for(rows, c.sms), 256, 0, s>>>((int)g.P, (int)rows, da.splits, c.rpart, kRowMinParts,
                                                             c.rd, c.rn);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
  }
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
  if (!c.rimg) {
    e = rowmin((int)g.P, Ec, nc, kNoSelf, c.rcount, c.rd);
    if (e != cudaSuccess) return e;
    e = rowmin((int)g.Rc, Ek, nkp, 0, c.rcount + 1, c.rn);
    if (e != cudaSuccess) return e;
  }
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
    const dim3 grid((unsigned)((g.P + 255) / 256 + (g.Rc + 255) / 256),
                    (unsigned)((std::max(g.P, g.Rc) + 1023) / 1024));
    k_replay_rank<<<grid, 256, 0, s>>>(g, c.rcount, c.rd, c.rn, c.rrank);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  e = traced(c, TR_REPLAY, 1, s, [&] {
    k_replay_inv<<<grid_for(g.P + g.Rc, c.sms), 256, 0, s>>>(g, c.rcount, c.rrank, c.rinv);
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
