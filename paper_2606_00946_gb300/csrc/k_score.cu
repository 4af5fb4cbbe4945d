// Scoring kernels on CUDA cores: feature assembly (Sec. 4.1 Features,
// Algorithm 4 Normalize), the reward-model forward pass for small or fp32
// predictors (Sec. 4.1 Model architecture), the greedy argmin selector
// (Algorithm 4, argmax reward = argmin predicted TTFT) and the sample ring.
#include "common.cuh"

namespace ls {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float norm_feature(int k, int64_t L, int h, const float* inst,
                                             int d_inst, const float* req, const float* mean,
                                             const float* stdv) {
  return zscore(raw_feature(k, L, h, inst, d_inst, req), mean[k], stdv[k]);
}

__global__ void k_assemble(int n_req, int n_inst, const int64_t* __restrict__ tok_off,
                           const int32_t* __restrict__ hits, const float* __restrict__ inst_state,
                           int d_inst, const float* __restrict__ req_feats, int d_req,
                           const float* __restrict__ mean, const float* __restrict__ stdv,
                           float* __restrict__ x_out) {
  const int d = kPair + d_inst + d_req;
  const int64_t total = (int64_t)n_req * n_inst * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = e / d;
    const int k = (int)(e - row * d);
    const int r = (int)(row / n_inst), i = (int)(row - (int64_t)r * n_inst);
    const int64_t L = tok_off[r + 1] - tok_off[r];
    x_out[e] = norm_feature(k, L, hits[row], inst_state + (int64_t)i * d_inst, d_inst,
                            req_feats + (int64_t)r * d_req, mean, stdv);
  }
}

// Forward pass of a tile of TR pair rows (row = r * n_inst + i) held in shared
// memory.  Hidden layer: thread o computes output column o for all TR rows
// from the transposed weights W^T [in, out] (coalesced across threads);
// output layer (width 1): one warp per row, lanes split the dot product.
template <int TR>
__global__ void __launch_bounds__(256) k_score_simt(MlpDesc mlp, const float* __restrict__ pp0,
                                                    const float* __restrict__ wt0,
                                                    const float* __restrict__ pp1,
                                                    const float* __restrict__ wt1,
                                                    const int32_t* __restrict__ sel, int n_req,
                                                    int n_inst, const int64_t* __restrict__ tok_off,
                                                    const int32_t* __restrict__ hits,
                                                    const float* __restrict__ inst_state, int d_inst,
                                                    const float* __restrict__ req_feats, int d_req,
                                                    const float* __restrict__ mean,
                                                    const float* __restrict__ stdv,
                                                    float* __restrict__ scores) {
  extern __shared__ float smem[];
  const bool b1 = sel && *sel == 1;  // published buffer of this route
  const float* __restrict__ pp = b1 ? pp1 : pp0;
  const float* __restrict__ wt = b1 ? wt1 : wt0;
  const int H = mlp.max_width;
  float* a = smem;
  float* b = smem + TR * H;
  const int d = mlp.w[0];
  const int64_t rows = (int64_t)n_req * n_inst;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  for (int64_t row0 = (int64_t)blockIdx.x * TR; row0 < rows; row0 += (int64_t)gridDim.x * TR) {
    for (int e = threadIdx.x; e < TR * d; e += blockDim.x) {
      const int rr = e / d, k = e - rr * d;
      const int64_t g = row0 + rr;
      float v = 0.0f;
      if (g < rows) {
        const int r = (int)(g / n_inst), i = (int)(g - (int64_t)r * n_inst);
        const int64_t L = tok_off[r + 1] - tok_off[r];
        v = norm_feature(k, L, hits[g], inst_state + (int64_t)i * d_inst, d_inst,
                         req_feats + (int64_t)r * d_req, mean, stdv);
        if (mlp.bf16) v = round_bf16(v);
      }
      a[rr * d + k] = v;
    }
    __syncthreads();
    for (int l = 0; l < mlp.n_layers; ++l) {
      const int in = mlp.w[l], out = mlp.w[l + 1];
      const float* W = wt + mlp.wtoff[l];
      const float* bias = pp + mlp.boff[l];
      if (l == mlp.n_layers - 1) {  // output layer, width 1
        for (int rr = warp; rr < TR; rr += blockDim.x / 32) {
          float s = 0.0f;
          for (int k = lane; k < in; k += 32) s = fmaf(a[rr * in + k], W[k], s);
#pragma unroll
          for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
          const int64_t g = row0 + rr;
          if (lane == 0 && g < rows) scores[g] = s + bias[0];
        }
      } else {
        for (int o = threadIdx.x; o < out; o += blockDim.x) {
          float acc[TR];
#pragma unroll
          for (int rr = 0; rr < TR; ++rr) acc[rr] = 0.0f;
          for (int k = 0; k < in; ++k) {
            const float wv = W[(int64_t)k * out + o];
#pragma unroll
            for (int rr = 0; rr < TR; ++rr) acc[rr] = fmaf(a[rr * in + k], wv, acc[rr]);
          }
          const float bo = bias[o];
#pragma unroll
          for (int rr = 0; rr < TR; ++rr) {
            float z = acc[rr] + bo;
            z = z > 0.0f ? z : 0.0f;
            b[rr * out + o] = mlp.bf16 ? round_bf16(z) : z;
          }
        }
      }
      __syncthreads();
      float* t = a; a = b; b = t;
    }
  }
}

// One warp per request: lexicographic (score, index) minimum over instances.
__global__ void k_argmin(int n_req, int n_inst, const float* __restrict__ scores,
                         int32_t* __restrict__ choice, float* __restrict__ best) {
  const int lane = threadIdx.x & 31;
  const int64_t r = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  if (r >= n_req) return;
  const float* s = scores + r * n_inst;
  float bv = 0.0f;
  int bi = -1;
  for (int i = lane; i < n_inst; i += 32) {
    const float v = s[i];
    if (bi < 0 || score_precedes(v, i, bv, bi)) { bv = v; bi = i; }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float ov = __shfl_xor_sync(kFull, bv, o);
    const int oi = __shfl_xor_sync(kFull, bi, o);
    if (oi >= 0 && (bi < 0 || score_precedes(ov, oi, bv, bi))) { bv = ov; bi = oi; }
  }
  if (lane == 0) { choice[r] = bi; best[r] = bv; }
}

// Record j of the batch -> slot (count + j) mod capacity, count = records
// appended before this batch (device state); the last block advances the
// count by n.  When a batch is longer than the ring only its last `capacity`
// records are kept.  With a pending ring (pending > 0; then n <= capacity)
// the record a slot held, stream position p - capacity, is first copied to
// pending row capacity + (p - capacity) mod pending by the thread that then
// overwrites the same piece; of the records one call evicts only the newest
// `pending` are copied, so no two copies share a row.
__global__ void k_ring_append(int n, int d, const float* __restrict__ x, const float* __restrict__ y,
                              float* ring_x, float* ring_y, DevState* st, int64_t capacity, int64_t pending) {
  const int64_t count = *reinterpret_cast<volatile int64_t*>(&st->ring_count);
  const int64_t first = n > capacity ? n - capacity : 0;
  // piece = 4 consecutive columns of one record (the last piece of a record
  // may be short); pieces of a record share its slot
  const int per = (d + 3) / 4;
  const int64_t total = (int64_t)(n - first) * per;
  const bool vec = (d & 3) == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0 &&
                   (reinterpret_cast<uintptr_t>(ring_x) & 15) == 0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t jj = e / per;
    const int k = (int)(e - jj * per) * 4;
    const int64_t j = first + jj;
    const int64_t slot = (count + j) % capacity;
    const float* src = x + j * d + k;
    float* dst = ring_x + slot * d + k;
    // only the newest `pending` records this call evicts are kept (older ones
    // would land on the same pending rows)
    if (pending > 0 && count + j >= capacity && count + j - capacity >= count + n - capacity - pending) {
      const int64_t prow = capacity + (count + j - capacity) % pending;
      float* pdst = ring_x + prow * d + k;
      if (vec) {
        *reinterpret_cast<float4*>(pdst) = *reinterpret_cast<const float4*>(dst);
      } else {
        for (int u = 0; u < 4 && k + u < d; ++u) pdst[u] = dst[u];
      }
      if (k == 0) ring_y[prow] = ring_y[slot];
    }
    if (vec) {
      *reinterpret_cast<float4*>(dst) = __ldg(reinterpret_cast<const float4*>(src));
    } else {
      for (int u = 0; u < 4 && k + u < d; ++u) dst[u] = __ldg(src + u);
    }
    if (k == 0) ring_y[slot] = y[j];
  }
  if (last_block(&st->done[DONE_RING]) && threadIdx.x == 0) st->ring_count = count + n;
}

int sm_count() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;
}

int grid_1d(int64_t n, int threads, int per_sm = 8) {
  int64_t g = (n + threads - 1) / threads;
  const int64_t cap = (int64_t)sm_count() * per_sm;
  return (int)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

cudaError_t launch_assemble_features(int n_req, int n_inst, const int64_t* tok_off,
                                     const int32_t* hits, const float* inst_state, int d_inst,
                                     const float* req_feats, int d_req, const float* mean,
                                     const float* stdv, float* x_out, cudaStream_t s) {
  const int64_t total = (int64_t)n_req * n_inst * (kPair + d_inst + d_req);
  if (total <= 0) return cudaSuccess;
  k_assemble<<<grid_1d(total, 256), 256, 0, s>>>(n_req, n_inst, tok_off, hits, inst_state, d_inst,
                                                req_feats, d_req, mean, stdv, x_out);
  return cudaGetLastError();
}

cudaError_t launch_score_simt(const MlpDesc& mlp, const Published* pub, const int32_t* sel, int n_req, int n_inst,
                              const int64_t* tok_off, const int32_t* hits, const float* inst_state,
                              int d_inst, const float* req_feats, int d_req, const float* mean,
                              const float* stdv, float* scores, cudaStream_t s) {
  constexpr int TR = 16;
  const int64_t rows = (int64_t)n_req * n_inst;
  if (rows <= 0) return cudaSuccess;
  const size_t smem = (size_t)2 * TR * mlp.max_width * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(k_score_simt<TR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  int64_t tiles = (rows + TR - 1) / TR;
  const int64_t cap = (int64_t)sm_count() * 8;
  const int grid = (int)(tiles > cap ? cap : tiles);
  k_score_simt<TR><<<grid, 256, smem, s>>>(mlp, pub[0].params, pub[0].wt, pub[1].params, pub[1].wt, sel, n_req,
                                           n_inst, tok_off, hits,
                                           inst_state, d_inst, req_feats, d_req, mean, stdv, scores);
  return cudaGetLastError();
}

cudaError_t launch_argmin(int n_req, int n_inst, const float* scores, int32_t* choice, float* best,
                          cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  const int64_t threads = (int64_t)n_req * 32;
  k_argmin<<<(int)((threads + 255) / 256), 256, 0, s>>>(n_req, n_inst, scores, choice, best);
  return cudaGetLastError();
}

cudaError_t launch_ring_append(int n, int d, const float* x, const float* y, float* ring_x,
                               float* ring_y, DevState* st, int64_t capacity, int64_t pending, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int64_t keep = n > capacity ? capacity : n;
  const int64_t total = keep * ((d + 3) / 4);
  k_ring_append<<<grid_1d(total, 256), 256, 0, s>>>(n, d, x, y, ring_x, ring_y, st, capacity, pending);
  return cudaGetLastError();
}

}  // namespace ls
