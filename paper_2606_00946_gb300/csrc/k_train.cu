// Online training step of the reward predictor (Sec. 4.3.2 online learning;
// Sec. 4.3.1 P2 keeps it off the routing path).  The paper does not state the
// loss or optimiser; this library uses mean squared error on TTFT (seconds)
// and SGD or Adam (beta1 0.9, beta2 0.999, eps 1e-8, bias-corrected).
//
// bf16 mode: the operands of every product (layer input, weights, hidden
// activations, back-propagated dZ) are rounded to bf16; sums, biases, the
// master weights and optimiser state stay fp32.
#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace ls {
namespace {

constexpr int EPI_STORE = 0;  // C = acc (split-K partial when gridDim.z > 1)
constexpr int EPI_FWD = 1;    // Z = acc + bias; A_next = round(relu(Z)) for hidden layers
constexpr int EPI_MASK = 2;   // dZ_prev = acc * [Z_prev > 0]

struct GemmArgs {
  int M, N, K;
  const float* A; int lda;   // TA: A[k*lda + m], else A[m*lda + k]
  const float* B; int ldb;   // TB: B[n*ldb + k], else B[k*ldb + n]
  float* C; int ldc;
  int round_a, round_b;
  int kchunk;
  const float* bias;
  float* act; int ld_act; int hidden; int bf16;
  const float* zprev; int ld_zprev;
};

// 64x64 output tile, K steps of 16, 256 threads with 4x4 outputs each.
template <bool TA, bool TB, int EPI>
__global__ void __launch_bounds__(256) k_gemm(GemmArgs g) {
  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  const int kb = blockIdx.z * g.kchunk;
  const int ke = min(g.K, kb + g.kchunk);
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;

  for (int kk = kb; kk < ke; kk += 16) {
    for (int e = threadIdx.x; e < 1024; e += 256) {
      int mm, kx;
      if (TA) { kx = e >> 6; mm = e & 63; } else { mm = e >> 4; kx = e & 15; }
      const int m = m0 + mm, k = kk + kx;
      float v = 0.0f;
      if (m < g.M && k < ke) v = TA ? g.A[(int64_t)k * g.lda + m] : g.A[(int64_t)m * g.lda + k];
      As[kx][mm] = g.round_a ? round_bf16(v) : v;
    }
    for (int e = threadIdx.x; e < 1024; e += 256) {
      int nn, kx;
      if (TB) { nn = e >> 4; kx = e & 15; } else { kx = e >> 6; nn = e & 63; }
      const int n = n0 + nn, k = kk + kx;
      float v = 0.0f;
      if (n < g.N && k < ke) v = TB ? g.B[(int64_t)n * g.ldb + k] : g.B[(int64_t)k * g.ldb + n];
      Bs[kx][nn] = g.round_b ? round_bf16(v) : v;
    }
    __syncthreads();
#pragma unroll
    for (int kx = 0; kx < 16; ++kx) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kx][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kx][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* C = g.C + (int64_t)blockIdx.z * g.M * g.ldc;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= g.N) continue;
      if (EPI == EPI_STORE) {
        C[(int64_t)m * g.ldc + n] = acc[i][j];
      } else if (EPI == EPI_FWD) {
        const float z = acc[i][j] + g.bias[n];
        C[(int64_t)m * g.ldc + n] = z;
        if (g.hidden) {
          const float r = z > 0.0f ? z : 0.0f;
          g.act[(int64_t)m * g.ld_act + n] = g.bf16 ? round_bf16(r) : r;
        }
      } else {
        C[(int64_t)m * g.ldc + n] = g.zprev[(int64_t)m * g.ld_zprev + n] > 0.0f ? acc[i][j] : 0.0f;
      }
    }
  }
}

// Minibatch rows: slot = idx[j] (checked against the filled part of the ring)
// or (step*B + j) mod valid, with step and the ring's fill read from the device
// state; z-score in fp32, bf16-rounded in bf16 mode.  An empty buffer latches
// LS_ERR_STATE and reads nothing (the rows are zero).
__global__ void k_train_gather(int B, int d, const int32_t* __restrict__ idx, DevState* st,
                               int64_t capacity, int64_t replay_base, const float* __restrict__ ring_x,
                               const float* __restrict__ ring_y, const float* __restrict__ mean,
                               const float* __restrict__ stdv, int bf16, float* __restrict__ x0,
                               float* __restrict__ y, int* err) {
  const int64_t step = st->step;
  const int64_t count = st->ring_count;
  const int64_t nF = count < capacity ? count : capacity;
  const int64_t valid = nF + st->replay_count;  // F u R
  if (valid < 1 && blockIdx.x == 0 && threadIdx.x == 0) {
    latch_error(err, LS_ERR_STATE);
    st->train_abort = 1;  // the optimiser of this step leaves every parameter as it is
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) set_adam_bc(st);
  const int64_t total = (int64_t)B * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(e / d), k = (int)(e - (int64_t)j * d);
    int64_t slot;
    if (idx) {
      slot = idx[j];
      if (slot < 0 || slot >= valid) {
        if (k == 0) {
          latch_error(err, LS_ERR_ARG);
          st->train_abort = 1;
        }
        slot = 0;
      }
    } else {
      slot = valid > 0 ? (step * (int64_t)B + j) % valid : 0;
    }
    if (valid < 1) {  // nothing logged yet: no row to read
      x0[e] = 0.0f;
      if (k == 0) y[j] = 0.0f;
      continue;
    }
    slot = union_row(slot, nF, replay_base);
    const float v = zscore(ring_x[slot * d + k], mean[k], stdv[k]);
    x0[e] = bf16 ? round_bf16(v) : v;
    if (k == 0) y[j] = ring_y[slot];
  }
}

// dZ_L = 2 (yhat - y) / B and loss = mean (yhat - y)^2, one CTA (fixed order).
__global__ void __launch_bounds__(1024) k_loss_grad(int B, const float* __restrict__ yhat,
                                                    const float* __restrict__ y,
                                                    float* __restrict__ dz, float* loss_out,
                                                    const DevState* st) {
  __shared__ float part[32];
  float s = 0.0f;
  for (int j = threadIdx.x; j < B; j += blockDim.x) {
    const float e = yhat[j] - y[j];
    dz[j] = 2.0f * e / (float)B;
    s = fmaf(e, e, s);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    float t = threadIdx.x < (blockDim.x >> 5) ? part[threadIdx.x] : 0.0f;
#pragma unroll
    for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0 && loss_out) *loss_out = st->train_abort ? __int_as_float(0x7fc00000) : t / (float)B;
  }
}

// db[o] = sum_j dz[j, o] (unrounded dZ), first stage: CTA (x, y) sums rows
// y*rows_per .. of 32 columns into part[y][o]; k_reduce_partials adds the
// partials in order.
__global__ void __launch_bounds__(256) k_colsum(int B, int out, int rows_per, const float* __restrict__ dz,
                                                float* __restrict__ part) {
  __shared__ float red[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int o = blockIdx.x * 32 + tx;
  const int j0 = blockIdx.y * rows_per, j1 = min(B, j0 + rows_per);
  float s = 0.0f;
  if (o < out)
    for (int j = j0 + ty; j < j1; j += 8) s += dz[(int64_t)j * out + o];
  red[ty][tx] = s;
  __syncthreads();
  if (ty == 0 && o < out) {
    float t = 0.0f;
#pragma unroll
    for (int k = 0; k < 8; ++k) t += red[k][tx];
    part[(int64_t)blockIdx.y * out + o] = t;
  }
}

// Output layer (width 1) forward: z[j] = sum_k round(w[k]) a[j, k] + b, one
// warp per row (a is already bf16-valued in bf16 mode).
__global__ void k_out_fwd(int B, int K, const float* __restrict__ a, const float* __restrict__ w,
                          const float* __restrict__ b, int bf16, float* __restrict__ z) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t j = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; j < B; j += warps) {
    float s = 0.0f;
    for (int k = lane; k < K; k += 32) {
      const float wk = bf16 ? round_bf16(w[k]) : w[k];
      s = fmaf(a[j * (int64_t)K + k], wk, s);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) z[j] = s + b[0];
  }
}

// Output layer weight gradient, first stage: part[y][k] = sum over rows of
// block y of round(dz[j]) a[j, k]; k_reduce_partials adds the partials.
__global__ void __launch_bounds__(256) k_out_dw(int B, int K, int rows_per, const float* __restrict__ dz,
                                                const float* __restrict__ a, int bf16,
                                                float* __restrict__ part) {
  __shared__ float red[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int k = blockIdx.x * 32 + tx;
  const int j0 = blockIdx.y * rows_per, j1 = min(B, j0 + rows_per);
  float s = 0.0f;
  if (k < K)
    for (int j = j0 + ty; j < j1; j += 8) {
      const float g = bf16 ? round_bf16(dz[j]) : dz[j];
      s = fmaf(g, a[(int64_t)j * K + k], s);
    }
  red[ty][tx] = s;
  __syncthreads();
  if (ty == 0 && k < K) {
    float t = 0.0f;
#pragma unroll
    for (int q = 0; q < 8; ++q) t += red[q][tx];
    part[(int64_t)blockIdx.y * K + k] = t;
  }
}

// Output layer input gradient: dz_prev[j, k] = round(dz[j]) round(w[k]) [z[j, k] > 0].
__global__ void k_out_dx(int B, int K, const float* __restrict__ dz, const float* __restrict__ w,
                         const float* __restrict__ zprev, int bf16, float* __restrict__ out) {
  const int64_t n = (int64_t)B * K;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t j = e / K;
    const int k = (int)(e - j * K);
    const float g = bf16 ? round_bf16(dz[j]) : dz[j];
    const float wk = bf16 ? round_bf16(w[k]) : w[k];
    out[e] = zprev[e] > 0.0f ? g * wk : 0.0f;
  }
}

// dst[e] = sum over z of part[z * n + e], z in order (up to 16 loads in flight).
__global__ void k_reduce_partials(int S, int64_t n, const float* __restrict__ part,
                                  float* __restrict__ dst) {
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.0f;
    for (int z0 = 0; z0 < S; z0 += 16) {
      float v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] = z0 + u < S ? __ldg(part + (int64_t)(z0 + u) * n + e) : 0.0f;
#pragma unroll
      for (int u = 0; u < 16; ++u) s += v[u];
    }
    dst[e] = s;
  }
}

// The optimiser's last block, once every block has read the step counter and
// the abort flag: advance the step unless the gather aborted it, then clear
// the flag for the next step.
__device__ __forceinline__ void finish_step(DevState* st, int64_t t, bool aborted) {
  if (!aborted) advance_step(st, t);
  st->train_abort = 0;
}

// Optimiser updates.  Each advances the device step counter once (last block),
// after every block has read it.  A step whose gather found no record or a bad
// slot changes nothing.
__global__ void k_sgd(int64_t n, float lr, const float* __restrict__ g, float* __restrict__ p, DevState* st) {
  const int64_t t = st->step + 1;
  const bool aborted = st->train_abort != 0;
  if (!aborted)
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x)
      p[e] = p[e] - lr * g[e];
  if (last_block(&st->done[DONE_OPT]) && threadIdx.x == 0) finish_step(st, t, aborted);
}

// Adam, t = steps taken + 1: bias corrections 1 - beta^t formed in fp64 by
// the gather kernel of this step.
__global__ void k_adam(int64_t n, float lr, const float* __restrict__ g, float* __restrict__ p,
                       float* __restrict__ m, float* __restrict__ v, DevState* st) {
  const int64_t t = st->step + 1;
  const float bc1 = st->adam_bc[0], bc2 = st->adam_bc[1];
  const bool aborted = st->train_abort != 0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; !aborted && e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    const float ge = g[e];
    const float me = 0.9f * m[e] + 0.1f * ge;
    const float ve = 0.999f * v[e] + 0.001f * ge * ge;
    m[e] = me;
    v[e] = ve;
    const float mh = me / bc1, vh = ve / bc2;
    p[e] = p[e] - lr * mh / (sqrtf(vh) + 1e-8f);
  }
  if (last_block(&st->done[DONE_OPT]) && threadIdx.x == 0) finish_step(st, t, aborted);
}

template <bool TA, bool TB, int EPI>
cudaError_t gemm(const GemmArgs& a, int splits, cudaStream_t s) {
  dim3 grid((a.N + 63) / 64, (a.M + 63) / 64, splits);
  k_gemm<TA, TB, EPI><<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

int train_splits(int out, int in, int B, int n_sm) {
  const int tiles = ((out + 63) / 64) * ((in + 63) / 64);
  int S = (2 * n_sm + tiles - 1) / tiles;
  S = std::min(S, std::max(1, B / 64));
  return std::max(1, std::min(S, 64));
}

// Forward of B rows whose layer-0 inputs are in c.tx (z-scored, rounded in
// bf16 mode): z_l into c.tz, hidden activations a_l into c.tx (the training
// step's layout: layer l's input at c.tx + B * sum_{k<l} w_k).
cudaError_t forward_rows(Ctx& c, int B, cudaStream_t s, const int64_t* rows_dev) {
  const MlpDesc& m = c.mlp;
  const int L = m.n_layers;
  int64_t xoff[LS_MAX_LAYERS + 1], zoff[LS_MAX_LAYERS + 1];
  xoff[0] = zoff[0] = 0;
  for (int l = 0; l < L; ++l) {
    xoff[l + 1] = xoff[l] + (int64_t)B * m.w[l];
    zoff[l + 1] = zoff[l] + (int64_t)B * m.w[l + 1];
  }
  cudaError_t e = cudaSuccess;
  for (int l = 0; l < L; ++l) {
    GemmArgs a{};
    a.M = B; a.N = m.w[l + 1]; a.K = m.w[l];
    a.A = c.tx + xoff[l]; a.lda = m.w[l];
    a.B = c.master + m.woff[l]; a.ldb = m.w[l];
    a.C = c.tz + zoff[l]; a.ldc = m.w[l + 1];
    a.round_a = 0;  // activations were rounded when stored
    a.round_b = m.bf16;
    a.kchunk = ((a.K + 15) / 16) * 16;
    a.bias = c.master + m.boff[l];
    a.hidden = (l + 1 < L);
    a.act = a.hidden ? c.tx + xoff[l + 1] : nullptr;
    a.ld_act = m.w[l + 1];
    a.bf16 = m.bf16;
    bool done_tc = false;
    if (m.w[l + 1] == 1) {
      e = traced(c, TR_GEMM_FWD, 1, s, [&] {
        const int grid = (int)std::min<int64_t>(((int64_t)B * 32 + 255) / 256, (int64_t)c.sms * 8);
        k_out_fwd<<<grid, 256, 0, s>>>(B, m.w[l], a.A, a.B, a.bias, m.bf16, a.C);
        return cudaGetLastError();
      });
      if (e != cudaSuccess) return e;
      done_tc = true;
    } else if (m.bf16) {
      e = traced(c, TR_GEMM_TC_FWD, 1, s, [&] {
        return launch_gemm_tc(a.M, a.N, a.K, a.A, a.lda, 1, a.B, a.ldb, 1, 1, 1, a.C, a.ldc, 0, a.bias, a.act,
                              a.ld_act, a.hidden, nullptr, 0, c.d_err, c.sms, s, rows_dev);
      });
      if (e == cudaSuccess) done_tc = true;
      else if (e != cudaErrorInvalidValue) return e;
    }
    if (!done_tc) {
      e = traced(c, TR_GEMM_FWD, 1, s, [&] { return gemm<false, true, EPI_FWD>(a, 1, s); });
      if (e != cudaSuccess) return e;
    }
  }
  return cudaSuccess;
}

cudaError_t run_train_step(Ctx& c, int B, const int32_t* idx, int opt, float lr, float* loss_out,
                           cudaStream_t s) {
  const MlpDesc& m = c.mlp;
  const int L = m.n_layers;
  int64_t xoff[LS_MAX_LAYERS + 1], zoff[LS_MAX_LAYERS + 1];
  xoff[0] = zoff[0] = 0;
  for (int l = 0; l < L; ++l) {
    xoff[l + 1] = xoff[l] + (int64_t)B * m.w[l];
    zoff[l + 1] = zoff[l] + (int64_t)B * m.w[l + 1];
  }
  cudaError_t e;
  {
    const int64_t total = (int64_t)B * m.w[0];
    int grid = (int)std::min<int64_t>((total + 255) / 256, (int64_t)c.sms * 8);
    e = traced(c, TR_GATHER, 1, s, [&] {
      k_train_gather<<<std::max(grid, 1), 256, 0, s>>>(B, m.w[0], idx, c.st, c.cfg.ring_capacity, c.replay_base,
                                                       c.ring_x,
                                                       c.ring_y, c.mean, c.stdv, m.bf16, c.tx, c.ty,
                                                       c.d_err);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
  }
  // forward, keeping z_l and a_l
  e = forward_rows(c, B, s);
  if (e != cudaSuccess) return e;
  e = traced(c, TR_LOSS, 1, s, [&] {
    k_loss_grad<<<1, 1024, 0, s>>>(B, c.tz + zoff[L - 1], c.ty, c.dz0,
                                   loss_out ? loss_out : c.loss_tmp, c.st);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;

  float* dz = c.dz0;
  float* dzn = c.dz1;
  for (int l = L - 1; l >= 0; --l) {
    const int out = m.w[l + 1], in = m.w[l];
    // dW_l = round(dZ)^T A_l   (split over the batch, partials reduced in order)
    const int S = train_splits(out, in, B, c.sms);
    GemmArgs a{};
    a.M = out; a.N = in; a.K = B;
    a.A = dz; a.lda = out;
    a.B = c.tx + xoff[l]; a.ldb = in;
    a.C = c.gpart; a.ldc = in;
    a.round_a = m.bf16; a.round_b = 0;
    a.kchunk = (((B + S - 1) / S + 15) / 16) * 16;
    const int Seff = (B + a.kchunk - 1) / a.kchunk;
    int nparts = Seff;
    bool dw_tc = false;
    if (out == 1) {
      const int S1 = std::max(1, std::min(64, B / 64));
      const int rows_per = (B + S1 - 1) / S1;
      e = traced(c, TR_GEMM_DW, 1, s, [&] {
        k_out_dw<<<dim3((in + 31) / 32, S1), 256, 0, s>>>(B, in, rows_per, dz, c.tx + xoff[l], m.bf16, c.gpart);
        return cudaGetLastError();
      });
      if (e != cudaSuccess) return e;
      dw_tc = true;
      nparts = S1;
    } else if (m.bf16) {
      const int tiles = ((out + 127) / 128) * ((in + 127) / 128);
      const int S_tc = std::max(1, std::min({16, B / 64, (2 * c.sms + tiles - 1) / tiles}));
      e = traced(c, TR_GEMM_TC_DW, 1, s, [&] {
        return launch_gemm_tc(out, in, B, dz, 1, out, c.tx + xoff[l], 1, in, S_tc, 0, c.gpart, in,
                              (int64_t)out * in, nullptr, nullptr, 0, 0, nullptr, 0, c.d_err, c.sms, s);
      });
      if (e == cudaSuccess) { dw_tc = true; nparts = gemm_tc_splits_used(B, S_tc); }
      else if (e != cudaErrorInvalidValue) return e;
    }
    if (!dw_tc) {
      e = traced(c, TR_GEMM_DW, 1, s, [&] { return gemm<true, false, EPI_STORE>(a, Seff, s); });
      if (e != cudaSuccess) return e;
    }
    const int64_t nw = (int64_t)out * in;
    e = traced(c, TR_REDUCE, 1, s, [&] {
      k_reduce_partials<<<(int)std::min<int64_t>((nw + 255) / 256, (int64_t)c.sms * 8), 256, 0, s>>>(
          nparts, nw, c.gpart, c.grad + m.woff[l]);
      return cudaGetLastError();
    });
    if (e != cudaSuccess) return e;
    {
      const int S2 = std::max(1, std::min(64, B / 64));
      const int rows_per = (B + S2 - 1) / S2;
      float* part = c.gpart + (int64_t)64 * out * in;  // after the dW partials
      e = traced(c, TR_COLSUM, 1, s, [&] {
        k_colsum<<<dim3((out + 31) / 32, S2), 256, 0, s>>>(B, out, rows_per, dz, part);
        return cudaGetLastError();
      });
      if (e != cudaSuccess) return e;
      e = traced(c, TR_REDUCE, 1, s, [&] {
        k_reduce_partials<<<(out + 255) / 256, 256, 0, s>>>(S2, out, part, c.grad + m.boff[l]);
        return cudaGetLastError();
      });
      if (e != cudaSuccess) return e;
    }
    if (l > 0) {
      // dZ_{l-1} = (round(dZ_l) round(W_l)) * [z_{l-1} > 0]
      GemmArgs b{};
      b.M = B; b.N = in; b.K = out;
      b.A = dz; b.lda = out;
      b.B = c.master + m.woff[l]; b.ldb = in;
      b.C = dzn; b.ldc = in;
      b.round_a = m.bf16; b.round_b = m.bf16;
      b.kchunk = ((out + 15) / 16) * 16;
      b.zprev = c.tz + zoff[l - 1]; b.ld_zprev = in;
      bool dx_tc = false;
      if (out == 1) {
        e = traced(c, TR_GEMM_DX, 1, s, [&] {
          const int64_t n = (int64_t)B * in;
          const int grid = (int)std::min<int64_t>((n + 255) / 256, (int64_t)c.sms * 8);
          k_out_dx<<<grid, 256, 0, s>>>(B, in, dz, c.master + m.woff[l], c.tz + zoff[l - 1], m.bf16, dzn);
          return cudaGetLastError();
        });
        if (e != cudaSuccess) return e;
        dx_tc = true;
      } else if (m.bf16) {
        e = traced(c, TR_GEMM_TC_DX, 1, s, [&] {
          return launch_gemm_tc(B, in, out, dz, out, 1, c.master + m.woff[l], 1, in, 1, 2, dzn, in, 0, nullptr,
                                nullptr, 0, 0, c.tz + zoff[l - 1], in, c.d_err, c.sms, s);
        });
        if (e == cudaSuccess) dx_tc = true;
        else if (e != cudaErrorInvalidValue) return e;
      }
      if (!dx_tc) {
        e = traced(c, TR_GEMM_DX, 1, s, [&] { return gemm<false, false, EPI_MASK>(b, 1, s); });
        if (e != cudaSuccess) return e;
      }
      float* t = dz; dz = dzn; dzn = t;
    }
  }
  const int grid = (int)std::min<int64_t>((c.n_params + 255) / 256, (int64_t)c.sms * 8);
  return traced(c, TR_OPT, 1, s, [&] {
    if (opt == LS_SGD) k_sgd<<<grid, 256, 0, s>>>(c.n_params, lr, c.grad, c.master, c.st);
    else k_adam<<<grid, 256, 0, s>>>(c.n_params, lr, c.grad, c.master, c.adam_m, c.adam_v, c.st);
    return cudaGetLastError();
  });
}

}  // namespace ls
