// Training step of a bf16 predictor on tensor cores (Sec. 4.3.2 online
// learning; loss and optimiser as in k_train.cu: mean squared error, SGD or
// Adam), built around bf16 operand images.
//
// An "image" of a matrix X [R, C] is X in bf16 laid out exactly as a K-major
// 128-byte-swizzled MMA operand: element (r, c) at byte sw128_offset(r, c, R),
// so the 128 x 64 (or N x 64) tile of rows r0.. and K-block kb is one
// contiguous run of bytes that a single bulk copy lands in shared memory
// ready for tcgen05.mma.  Each product's epilogue writes the images the next
// products read, both row-major (X) and transposed (X^T, for the weight
// gradients, whose reduction runs over the batch):
//
//   gather     A_0 = bf16(zscore(x)) -> img(A_0), img(A_0^T)
//   forward l  Z = A_l W_l^T + b_l (TMEM) -> A_{l+1} = bf16(relu(Z)), mask [Z > 0]
//   last l     ... plus the width-1 output layer: yhat, loss, dz_L = 2 (yhat - y) / B,
//              dW_L, db_L partials, dz_l = bf16(dz_L) bf16(w_L) [Z > 0] -> img(dz_l), img(dz_l^T)
//   backward   dW_l = bf16(dz_l)^T A_l   (split over the batch, fp32 partials)
//              dz_{l-1} = (bf16(dz_l) W_l) [Z_{l-1} > 0] -> images   (same launch)
//   optimiser  gradient = ordered sum of the partials; SGD / Adam on the fp32
//              master; rewrites img(W_l), img(W_l^T) for the next step.
// Bias gradients are column sums of the unrounded dz, formed per 128-row tile
// in the epilogues.  The rounding points are those of the reference path
// (k_train.cu): bf16 operands of every product, fp32 sums, biases and state.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "sm100.cuh"

namespace ls {
using namespace sm100;

namespace {

constexpr int kT = 256;        // threads: 8 warps, 2 per TMEM lane quadrant
constexpr int kM = 128;        // rows per tile
constexpr int kMaxChunks = 4;  // K-blocks of 64 per CTA (all resident)

enum { TE_STORE = 0, TE_FWD = 1, TE_FWD_OUT = 2, TE_DX = 3 };

struct TrJob {
  int epi;
  int m_tiles, splits, nchunks, NT;  // CTA (m_tile, split) computes rows m_tile*128.., K-blocks split*nchunks..
  const uint8_t* A;                  // image, rA rows
  int rA;
  const uint8_t* B;                  // image, NT rows
  int M;                             // valid rows of D
  // TE_STORE: fp32 partial D to C[split][row][col]
  float* C;
  int ldc;
  int64_t split_stride;
  // TE_FWD / TE_FWD_OUT / TE_DX
  const float* bias;                 // layer bias (TE_FWD, TE_FWD_OUT)
  uint8_t* out;                      // row-major image of the result, rows = rows_pad (nullable)
  uint8_t* outT;                     // transposed image, rows = rT (nullable)
  int rT;
  uint32_t* mask_out;                // TE_FWD: [NT/32][rows_pad] bits of [Z > 0]
  const uint32_t* mask_in;           // TE_FWD_OUT keeps its own; TE_DX: bits of the previous layer
  float* colpart;                    // [m_tiles][NT] column sums of dz (TE_FWD_OUT, TE_DX)
  int rows_pad;                      // padded batch (multiple of 128)
  // TE_FWD_OUT: width-1 output layer
  const float* wL;                   // [NT] fp32 master weights of the output layer
  const float* bL;                   // [1]
  const float* y;                    // [batch] targets
  int batch;
  float* partWL;                     // [m_tiles][NT]
  float* partBL;                     // [m_tiles]
  float* partLoss;                   // [m_tiles]
};

struct TrArgs {
  TrJob job[2];
  int n_cta0;                        // CTAs of job 0; the rest run job 1
  int* err;
};

__device__ __forceinline__ uint16_t bf16_bits(float x) {
  __nv_bfloat16 v = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t*>(&v);
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Sum over the warp's 32 lanes of each of 32 per-lane values: afterwards lane
// u holds the sum for column u.  Fixed order (butterfly), 31 shuffles.
__device__ __forceinline__ float col_reduce32(float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) {
    const bool up = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < s; ++i) {
      const float send = up ? v[i] : v[i + s];
      const float keep = up ? v[i + s] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0];
}

// Row-major image: 32 bf16 values of row j, columns c0..c0+31 (c0 % 32 == 0).
__device__ __forceinline__ void store_row32(uint8_t* img, int rows, int j, int c0, const float (&v)[32]) {
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    uint4 q;
    q.x = pack2(v[8 * g], v[8 * g + 1]);
    q.y = pack2(v[8 * g + 2], v[8 * g + 3]);
    q.z = pack2(v[8 * g + 4], v[8 * g + 5]);
    q.w = pack2(v[8 * g + 6], v[8 * g + 7]);
    *reinterpret_cast<uint4*>(img + sw128_offset(j, c0 + 8 * g, rows)) = q;
  }
}

// Transposed image: element (c0 + u, j) for u < 32; lanes hold consecutive j,
// so each column is written as 2-byte pieces of one 64-byte run per warp.
__device__ __forceinline__ void store_col32(uint8_t* imgT, int rowsT, int j, int c0, const float (&v)[32]) {
#pragma unroll
  for (int u = 0; u < 32; ++u)
    *reinterpret_cast<uint16_t*>(imgT + sw128_offset(c0 + u, j, rowsT)) = bf16_bits(v[u]);
}

__global__ void __launch_bounds__(kT, 1) k_tr_gemm(const __grid_constant__ TrArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const bool second = (int)blockIdx.x >= args.n_cta0;
  const TrJob& J = args.job[second ? 1 : 0];
  const int li = second ? (int)blockIdx.x - args.n_cta0 : (int)blockIdx.x;
  const int mt = li % J.m_tiles, split = li / J.m_tiles;
  const int m0 = mt * kM;
  const int NT = J.NT, nch = J.nchunks;
  const uint32_t a_bytes = kM * 128, b_bytes = (uint32_t)NT * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  uint8_t* tail = smem + (size_t)kMaxChunks * (kM * 128 + 256 * 128);
  uint64_t* full = reinterpret_cast<uint64_t*>(tail);           // [kMaxChunks]
  uint64_t* done = full + kMaxChunks;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  float* red = reinterpret_cast<float*>(tail + 128);            // [2][4][256]
  float* xch = red + 2 * 4 * 256;                               // [2][128] row exchange

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint32_t tcols = 32;
  while ((int)tcols < NT) tcols <<= 1;
  if (tid == 0) {
    for (int c = 0; c < kMaxChunks; ++c) mbar_init(&full[c], 1);
    mbar_init(done, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, tcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  bool ok = true;
  if (tid == 0) {
    for (int c = 0; c < nch; ++c) {
      const int kb = split * nch + c;
      uint8_t* sa = smem + (size_t)c * stage_bytes;
      mbar_arrive_expect_tx(&full[c], stage_bytes);
      bulk_g2s(sa, J.A + (size_t)kb * J.rA * 128 + (size_t)m0 * 128, a_bytes, &full[c]);
      bulk_g2s(sa + a_bytes, J.B + (size_t)kb * NT * 128, b_bytes, &full[c]);
    }
    const uint32_t idesc = idesc_bf16_f32(kM, NT);
    for (int c = 0; c < nch; ++c) {
      if (!mbar_wait(&full[c], 0)) { ok = false; break; }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + (size_t)c * stage_bytes), sb = sa + a_bytes;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        umma_bf16(tmem, sdesc_sw128(sa + 32u * k), sdesc_sw128(sb + 32u * k), idesc, (c | k) ? 1u : 0u);
    }
    umma_commit(done);  // arrives once everything issued so far has completed
  }
  __syncwarp();
  if (!mbar_wait(done, 0)) ok = false;
  ok = __syncthreads_and(ok) != 0;  // one decision for the whole CTA
  if (!ok) {
    latch_error(args.err, LS_ERR_TIMEOUT);
    // copies that may still be in flight land in this CTA's own shared memory;
    // wait (bounded) for them before the CTA exits
    if (tid == 0)
      for (int c = 0; c < nch; ++c) mbar_wait(&full[c], 0);
  }
  tc_fence_after();

  const int q = warp & 3, h = warp >> 2;
  const int r = 32 * q + lane, j = m0 + r;
  const int half = NT / 2;
  const uint32_t lane_addr = (uint32_t)(32 * q) << 16;
  float* redA = red;              // [4][256]
  float* redB = red + 4 * 256;    // [4][256]

  if (ok && J.epi == TE_STORE) {
    if (j < J.M) {
      float* crow = J.C + (int64_t)split * J.split_stride + (int64_t)j * J.ldc;
      for (int c0 = h * half; c0 < (h + 1) * half; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(tmem + lane_addr + (uint32_t)c0, v);
        tmem_wait_ld();
#pragma unroll
        for (int g = 0; g < 8; ++g)
          reinterpret_cast<float4*>(crow + c0)[g] =
              make_float4(__uint_as_float(v[4 * g]), __uint_as_float(v[4 * g + 1]), __uint_as_float(v[4 * g + 2]),
                          __uint_as_float(v[4 * g + 3]));
      }
    }
  } else if (ok && J.epi == TE_FWD) {
    for (int c0 = h * half; c0 < (h + 1) * half; c0 += 32) {
      uint32_t v[32];
      tmem_ld32(tmem + lane_addr + (uint32_t)c0, v);
      tmem_wait_ld();
      float a[32];
      uint32_t bits = 0;
#pragma unroll
      for (int u = 0; u < 32; ++u) {
        const float z = __uint_as_float(v[u]) + __ldg(J.bias + c0 + u);
        bits |= (z > 0.0f ? 1u : 0u) << u;
        a[u] = round_bf16(z > 0.0f ? z : 0.0f);
      }
      J.mask_out[(int64_t)(c0 >> 5) * J.rows_pad + j] = bits;
      store_row32(J.out, J.rows_pad, j, c0, a);
      store_col32(J.outT, J.rT, j, c0, a);
    }
  } else if (ok && J.epi == TE_FWD_OUT) {
    // pass 1: activations, mask bits, this half's part of the output dot product
    uint32_t mbits[4];
    float dot = 0.0f;
    int w = 0;
    for (int c0 = h * half; c0 < (h + 1) * half; c0 += 32, ++w) {
      uint32_t v[32];
      tmem_ld32(tmem + lane_addr + (uint32_t)c0, v);
      tmem_wait_ld();
      uint32_t bits = 0;
#pragma unroll
      for (int u = 0; u < 32; ++u) {
        const float z = __uint_as_float(v[u]) + __ldg(J.bias + c0 + u);
        bits |= (z > 0.0f ? 1u : 0u) << u;
        const float a = round_bf16(z > 0.0f ? z : 0.0f);
        dot = fmaf(a, round_bf16(__ldg(J.wL + c0 + u)), dot);
      }
      mbits[w] = bits;
    }
    xch[h * kM + r] = dot;
    __syncthreads();
    const float yhat = (xch[r] + xch[kM + r]) + __ldg(J.bL);
    const bool valid = j < J.batch;
    const float e = valid ? yhat - __ldg(J.y + j) : 0.0f;
    const float dzL = valid ? 2.0f * e / (float)J.batch : 0.0f;
    const float rd = round_bf16(dzL);
    // loss and db_L partials: warp sums, then quadrants in order (half 0 only)
    float e2 = e * e, dsum = dzL;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      e2 += __shfl_xor_sync(0xffffffffu, e2, o);
      dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
    }
    __syncthreads();  // xch reused below
    if (h == 0 && lane == 0) {
      xch[q] = e2;
      xch[4 + q] = dsum;
    }
    // pass 2: dW_L partial (sum_j bf16(dz_L[j]) a[j, c]) and dz_l = bf16(dz_L) bf16(w_L) [Z > 0]
    w = 0;
    for (int c0 = h * half; c0 < (h + 1) * half; c0 += 32, ++w) {
      uint32_t v[32];
      tmem_ld32(tmem + lane_addr + (uint32_t)c0, v);
      tmem_wait_ld();
      float pw[32], dz[32];
#pragma unroll
      for (int u = 0; u < 32; ++u) {
        const float z = __uint_as_float(v[u]) + __ldg(J.bias + c0 + u);
        const float a = round_bf16(z > 0.0f ? z : 0.0f);
        pw[u] = rd * a;
        dz[u] = ((mbits[w] >> u) & 1u) ? rd * round_bf16(__ldg(J.wL + c0 + u)) : 0.0f;
      }
      if (J.out) store_row32(J.out, J.rows_pad, j, c0, dz);
      store_col32(J.outT, J.rT, j, c0, dz);
      const float sw = col_reduce32(pw);
      redA[q * 256 + c0 + lane] = sw;
      const float sb = col_reduce32(dz);
      redB[q * 256 + c0 + lane] = sb;
    }
    __syncthreads();
    for (int c = tid; c < NT; c += kT) {
      J.partWL[(int64_t)mt * NT + c] = ((redA[c] + redA[256 + c]) + redA[512 + c]) + redA[768 + c];
      J.colpart[(int64_t)mt * NT + c] = ((redB[c] + redB[256 + c]) + redB[512 + c]) + redB[768 + c];
    }
    if (tid == 0) {
      J.partLoss[mt] = ((xch[0] + xch[1]) + xch[2]) + xch[3];
      J.partBL[mt] = ((xch[4] + xch[5]) + xch[6]) + xch[7];
    }
  } else if (ok && J.epi == TE_DX) {
    for (int c0 = h * half; c0 < (h + 1) * half; c0 += 32) {
      uint32_t v[32];
      tmem_ld32(tmem + lane_addr + (uint32_t)c0, v);
      tmem_wait_ld();
      const uint32_t bits = J.mask_in[(int64_t)(c0 >> 5) * J.rows_pad + j];
      float dz[32];
#pragma unroll
      for (int u = 0; u < 32; ++u) dz[u] = ((bits >> u) & 1u) ? __uint_as_float(v[u]) : 0.0f;
      if (J.out) store_row32(J.out, J.rows_pad, j, c0, dz);
      store_col32(J.outT, J.rT, j, c0, dz);
      const float sb = col_reduce32(dz);
      redB[q * 256 + c0 + lane] = sb;
    }
    __syncthreads();
    for (int c = tid; c < NT; c += kT)
      J.colpart[(int64_t)mt * NT + c] = ((redB[c] + redB[256 + c]) + redB[512 + c]) + redB[768 + c];
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, tcols);
}

// Minibatch gather: row j of the batch (slot idx[j], or (step*B + j) mod
// valid) z-scored and rounded to bf16 into img(A_0) and img(A_0^T); rows past
// the batch and columns past d are zero.  Thread = (row j, 8 columns).
__global__ void k_tr_gather(int B, int rows_pad, int d, int d_pad, const int32_t* __restrict__ idx,
                            const DevState* st, int64_t capacity, const float* __restrict__ ring_x,
                            const float* __restrict__ ring_y, const float* __restrict__ mean,
                            const float* __restrict__ stdv, uint8_t* __restrict__ a0, uint8_t* __restrict__ a0t,
                            float* __restrict__ y, int* err) {
  const int64_t step = st->step;
  const int64_t count = st->ring_count;
  const int64_t valid = count < capacity ? count : capacity;
  if (valid < 1 && blockIdx.x == 0 && threadIdx.x == 0) latch_error(err, LS_ERR_STATE);
  const int64_t total = (int64_t)rows_pad * (d_pad / 8);
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(e % rows_pad), c0 = (int)(e / rows_pad) * 8;
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = 0.0f;
    if (j < B) {
      int64_t slot;
      if (idx) {
        slot = idx[j];
        if (slot < 0 || slot >= valid) {
          if (c0 == 0) latch_error(err, LS_ERR_ARG);
          slot = 0;
        }
      } else {
        slot = valid > 0 ? (step * (int64_t)B + j) % valid : 0;
      }
      const float* row = ring_x + slot * d;
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (c0 + u < d) v[u] = round_bf16(zscore(__ldg(row + c0 + u), __ldg(mean + c0 + u), __ldg(stdv + c0 + u)));
      if (c0 == 0) y[j] = ring_y[slot];
    }
    uint4 qv;
    qv.x = pack2(v[0], v[1]);
    qv.y = pack2(v[2], v[3]);
    qv.z = pack2(v[4], v[5]);
    qv.w = pack2(v[6], v[7]);
    *reinterpret_cast<uint4*>(a0 + sw128_offset(j, c0, rows_pad)) = qv;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      *reinterpret_cast<uint16_t*>(a0t + sw128_offset(c0 + u, j, d_pad)) = bf16_bits(v[u]);
  }
}

// sum_{s < n} src[s * stride], added in order, eight loads in flight.
__device__ __forceinline__ float ordered_sum(const float* __restrict__ src, int n, int64_t stride) {
  float g = 0.0f;
  int s = 0;
  for (; s + 8 <= n; s += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = __ldg(src + (int64_t)(s + u) * stride);
#pragma unroll
    for (int u = 0; u < 8; ++u) g += v[u];
  }
  for (; s < n; ++s) g += __ldg(src + (int64_t)s * stride);
  return g;
}

struct OptLayer {
  const float* partW;  // [S][out][ld] split partials of dW (hidden) or [T][in] tile partials (output)
  int S;
  int ld;
  const float* partB;  // [T][out] (hidden) or [T] (output)
  uint8_t* imgW;       // [out rows, in_pad] image of bf16(W) (hidden layers)
  uint8_t* imgWT;      // [in_pad rows, out] image of bf16(W)^T
  int in_pad;
};

struct OptArgs {
  MlpDesc m;
  OptLayer L[LS_MAX_LAYERS];
  int T;               // row tiles of the batch
  int64_t n;           // parameters
  int mode;            // 0: images only, 1: SGD, 2: Adam
  float lr;
  float* p;
  float* mo;
  float* vo;
  DevState* st;
  const float* partLoss;
  int B;
  float* loss_out;
};

// Gradient of every parameter as an ordered sum of its partials, the
// optimiser update of the fp32 master, and the bf16 images of the updated
// hidden-layer weights.  Block 0 also forms the minibatch loss.
__global__ void __launch_bounds__(256) k_tr_opt(const __grid_constant__ OptArgs a) {
  __shared__ float bc[2];
  const int64_t t = a.st->step + 1;
  if (threadIdx.x == 0) {
    bc[0] = (float)(1.0 - pow(0.9, (double)t));
    bc[1] = (float)(1.0 - pow(0.999, (double)t));
  }
  __syncthreads();
  const MlpDesc& m = a.m;
  const int nl = m.n_layers;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < a.n;
       e += (int64_t)gridDim.x * blockDim.x) {
    int l = 0;
    while (l + 1 < nl && e >= m.woff[l + 1]) ++l;
    const int out = m.w[l + 1], in = m.w[l];
    const OptLayer& P = a.L[l];
    const bool is_w = e < m.boff[l];
    int o = 0, i = 0;
    float p = a.p[e];
    if (a.mode != 0) {
      float g = 0.0f;
      if (l + 1 < nl) {
        if (is_w) {
          const int64_t u = e - m.woff[l];
          o = (int)(u / in);
          i = (int)(u - (int64_t)o * in);
          g = ordered_sum(P.partW + (int64_t)o * P.ld + i, P.S, (int64_t)out * P.ld);
        } else {
          o = (int)(e - m.boff[l]);
          g = ordered_sum(P.partB + o, a.T, out);
        }
      } else {
        if (is_w) {
          i = (int)(e - m.woff[l]);
          g = ordered_sum(P.partW + i, a.T, P.ld);
        } else {
          g = ordered_sum(P.partB, a.T, 1);
        }
      }
      if (a.mode == 1) {
        p = p - a.lr * g;
      } else {
        const float me = 0.9f * a.mo[e] + 0.1f * g;
        const float ve = 0.999f * a.vo[e] + 0.001f * g * g;
        a.mo[e] = me;
        a.vo[e] = ve;
        const float mh = me / bc[0], vh = ve / bc[1];
        p = p - a.lr * mh / (sqrtf(vh) + 1e-8f);
      }
      a.p[e] = p;
    } else if (l + 1 < nl && is_w) {
      const int64_t u = e - m.woff[l];
      o = (int)(u / in);
      i = (int)(u - (int64_t)o * in);
    }
    if (l + 1 < nl && is_w) {
      const uint16_t b = bf16_bits(p);
      *reinterpret_cast<uint16_t*>(P.imgW + sw128_offset(o, i, out)) = b;
      *reinterpret_cast<uint16_t*>(P.imgWT + sw128_offset(i, o, P.in_pad)) = b;
    }
  }
  if (a.mode != 0 && blockIdx.x == 0 && threadIdx.x == 0 && a.loss_out) {
    float s = 0.0f;
    for (int tt = 0; tt < a.T; ++tt) s += a.partLoss[tt];
    *a.loss_out = s / (float)a.B;
  }
  if (a.mode != 0 && last_block(&a.st->done[DONE_OPT]) && threadIdx.x == 0) a.st->step = t;
}

int gemm_smem_bytes() { return 1024 + kMaxChunks * (kM * 128 + 256 * 128) + 128 + (2 * 4 * 256 + 2 * kM) * 4; }

cudaError_t launch_tr_gemm(const TrJob& j0, const TrJob* j1, int* err, cudaStream_t s) {
  TrArgs a{};
  a.job[0] = j0;
  a.n_cta0 = j0.m_tiles * j0.splits;
  int n = a.n_cta0;
  if (j1) {
    a.job[1] = *j1;
    n += j1->m_tiles * j1->splits;
  }
  a.err = err;
  const int smem = gemm_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(k_tr_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  k_tr_gemm<<<n, kT, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

// The fast path applies to bf16 predictors with at least one hidden layer,
// hidden widths that are multiples of 64 up to 256 and an input width of at
// most 256 (padded to 64).
bool plan_train_fast(const MlpDesc& m, int max_batch, TrainFast& f) {
  f = TrainFast{};
  if (!m.bf16 || m.n_layers < 2) return false;
  f.in_pad[0] = ((m.w[0] + 63) / 64) * 64;
  if (f.in_pad[0] > 256) return false;
  for (int l = 1; l < m.n_layers; ++l) {
    if (m.w[l] % 64 != 0 || m.w[l] > 256) return false;
    f.in_pad[l] = m.w[l];
  }
  f.rows_max = ((max_batch + kM - 1) / kM) * kM;
  f.on = true;
  return true;
}

int64_t train_fast_bytes(const MlpDesc& m, const TrainFast& f, int64_t* parts_floats) {
  const int nh = m.n_layers - 1;
  const int64_t R = f.rows_max;
  int64_t bytes = 0;
  for (int l = 0; l < nh; ++l) bytes += 2 * R * f.in_pad[l] * 2;  // A_l, A_l^T
  int hmax = 0;
  for (int l = 1; l <= nh; ++l) hmax = std::max(hmax, m.w[l]);
  const int64_t hpad = ((hmax + 127) / 128) * 128;
  bytes += 2 * (R * hmax * 2 + hpad * R * 2);                       // dz images, two parities
  for (int l = 1; l <= nh; ++l) bytes += (int64_t)(m.w[l] / 32) * R * 4;  // masks
  for (int l = 0; l < nh; ++l) bytes += 2 * (int64_t)m.w[l + 1] * f.in_pad[l] * 2;  // weight images
  const int64_t T = R / kM;
  int64_t pf = 0;
  for (int l = 0; l < nh; ++l) pf += (R / 128) * (int64_t)m.w[l + 1] * f.in_pad[l] + T * m.w[l + 1];
  pf += T * m.w[nh] + T + T;  // output layer weight / bias partials, loss partials
  *parts_floats = pf;
  return bytes;
}

// Carve the context's fast-path buffers out of one allocation.
void train_fast_bind(const MlpDesc& m, TrainFast& f, uint8_t* base, float* parts) {
  const int nh = m.n_layers - 1;
  const int64_t R = f.rows_max;
  uint8_t* p = base;
  for (int l = 0; l < nh; ++l) {
    f.imgA[l] = p;
    p += R * f.in_pad[l] * 2;
    f.imgAT[l] = p;
    p += R * f.in_pad[l] * 2;
  }
  int hmax = 0;
  for (int l = 1; l <= nh; ++l) hmax = std::max(hmax, m.w[l]);
  const int64_t hpad = ((hmax + 127) / 128) * 128;
  for (int b = 0; b < 2; ++b) {
    f.imgDZ[b] = p;
    p += R * hmax * 2;
    f.imgDZT[b] = p;
    p += hpad * R * 2;
  }
  for (int l = 1; l <= nh; ++l) {
    f.mask[l] = reinterpret_cast<uint32_t*>(p);
    p += (int64_t)(m.w[l] / 32) * R * 4;
  }
  for (int l = 0; l < nh; ++l) {
    f.imgW[l] = p;
    p += (int64_t)m.w[l + 1] * f.in_pad[l] * 2;
    f.imgWT[l] = p;
    p += (int64_t)m.w[l + 1] * f.in_pad[l] * 2;
  }
  const int64_t T = R / kM;
  float* q = parts;
  for (int l = 0; l < nh; ++l) {
    f.partW[l] = q;
    q += (R / 128) * (int64_t)m.w[l + 1] * f.in_pad[l];
    f.partB[l] = q;
    q += T * m.w[l + 1];
  }
  f.partWL = q;
  q += T * m.w[nh];
  f.partBL = q;
  q += T;
  f.partLoss = q;
}

// bf16 images of the master's hidden-layer weights (after ls_set_params).
cudaError_t train_fast_images(Ctx& c, cudaStream_t s) {
  const MlpDesc& m = c.mlp;
  TrainFast& f = c.tf;
  OptArgs a{};
  a.m = m;
  for (int l = 0; l + 1 < m.n_layers; ++l) {
    a.L[l].imgW = f.imgW[l];
    a.L[l].imgWT = f.imgWT[l];
    a.L[l].in_pad = f.in_pad[l];
  }
  a.n = c.n_params;
  a.mode = 0;
  a.p = c.master;
  a.st = c.st;
  const int grid = (int)std::min<int64_t>((c.n_params + 255) / 256, (int64_t)c.sms * 4);
  k_tr_opt<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t run_train_fast(Ctx& c, int B, const int32_t* idx, int opt, float lr, float* loss_out, cudaStream_t s) {
  const MlpDesc& m = c.mlp;
  TrainFast& f = c.tf;
  const int nh = m.n_layers - 1;  // hidden layers 0..nh-1, output layer nh
  const int R = ((B + kM - 1) / kM) * kM;
  const int T = R / kM;
  cudaError_t e;
  e = traced(c, TR_GATHER, 1, s, [&] {
    const int64_t total = (int64_t)R * (f.in_pad[0] / 8);
    const int grid = (int)std::min<int64_t>((total + 255) / 256, (int64_t)c.sms * 8);
    k_tr_gather<<<grid, 256, 0, s>>>(B, R, m.w[0], f.in_pad[0], idx, c.st, c.cfg.ring_capacity, c.ring_x, c.ring_y,
                                     c.mean, c.stdv, f.imgA[0], f.imgAT[0], c.ty, c.d_err);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  // forward: hidden layers; the last one also runs the output layer and the loss
  for (int l = 0; l < nh; ++l) {
    const bool last = l == nh - 1;
    TrJob J{};
    J.epi = last ? TE_FWD_OUT : TE_FWD;
    J.m_tiles = T;
    J.splits = 1;
    J.nchunks = f.in_pad[l] / 64;
    J.NT = m.w[l + 1];
    J.A = f.imgA[l];
    J.rA = R;
    J.B = f.imgW[l];
    J.M = R;
    J.bias = c.master + m.boff[l];
    J.rows_pad = R;
    if (!last) {
      J.out = f.imgA[l + 1];
      J.outT = f.imgAT[l + 1];
      J.rT = f.in_pad[l + 1];
      J.mask_out = f.mask[l + 1];
    } else {
      J.out = l > 0 ? f.imgDZ[l & 1] : nullptr;
      J.outT = f.imgDZT[l & 1];
      J.rT = ((m.w[l + 1] + 127) / 128) * 128;
      J.colpart = f.partB[l];
      J.wL = c.master + m.woff[nh];
      J.bL = c.master + m.boff[nh];
      J.y = c.ty;
      J.batch = B;
      J.partWL = f.partWL;
      J.partBL = f.partBL;
      J.partLoss = f.partLoss;
    }
    e = traced(c, TR_GEMM_TC_FWD, 1, s, [&] { return launch_tr_gemm(J, nullptr, c.d_err, s); });
    if (e != cudaSuccess) return e;
  }
  // backward: dW_l (split over the batch) and, for l > 0, dz_{l-1} in the same launch
  const int kpc = 2;  // K-blocks (of 64 rows) per dW CTA
  for (int l = nh - 1; l >= 0; --l) {
    const int out = m.w[l + 1];
    TrJob W{};
    W.epi = TE_STORE;
    W.m_tiles = (out + kM - 1) / kM;
    W.nchunks = std::min(kpc, R / 64);
    W.splits = (R / 64) / W.nchunks;
    W.NT = f.in_pad[l];
    W.A = f.imgDZT[l & 1];
    W.rA = ((out + 127) / 128) * 128;
    W.B = f.imgAT[l];
    W.M = out;
    W.C = f.partW[l];
    W.ldc = f.in_pad[l];
    W.split_stride = (int64_t)out * f.in_pad[l];
    f.splits[l] = W.splits;
    TrJob X{};
    if (l > 0) {
      X.epi = TE_DX;
      X.m_tiles = T;
      X.splits = 1;
      X.nchunks = out / 64;
      X.NT = m.w[l];
      X.A = f.imgDZ[l & 1];
      X.rA = R;
      X.B = f.imgWT[l];
      X.M = R;
      X.rows_pad = R;
      X.mask_in = f.mask[l];
      X.out = l > 1 ? f.imgDZ[(l - 1) & 1] : nullptr;
      X.outT = f.imgDZT[(l - 1) & 1];
      X.rT = ((m.w[l] + 127) / 128) * 128;
      X.colpart = f.partB[l - 1];
    }
    e = traced(c, l > 0 ? TR_GEMM_TC_DX : TR_GEMM_TC_DW, 1, s,
               [&] { return launch_tr_gemm(W, l > 0 ? &X : nullptr, c.d_err, s); });
    if (e != cudaSuccess) return e;
  }
  OptArgs a{};
  a.m = m;
  for (int l = 0; l < nh; ++l) {
    a.L[l].partW = f.partW[l];
    a.L[l].S = f.splits[l];
    a.L[l].ld = f.in_pad[l];
    a.L[l].partB = f.partB[l];
    a.L[l].imgW = f.imgW[l];
    a.L[l].imgWT = f.imgWT[l];
    a.L[l].in_pad = f.in_pad[l];
  }
  a.L[nh].partW = f.partWL;
  a.L[nh].ld = m.w[nh];
  a.L[nh].partB = f.partBL;
  a.T = T;
  a.n = c.n_params;
  a.mode = opt == LS_SGD ? 1 : 2;
  a.lr = lr;
  a.p = c.master;
  a.mo = c.adam_m;
  a.vo = c.adam_v;
  a.st = c.st;
  a.partLoss = f.partLoss;
  a.B = B;
  a.loss_out = loss_out ? loss_out : c.loss_tmp;
  return traced(c, TR_OPT, 1, s, [&] {
    const int grid = (int)std::min<int64_t>((c.n_params + 255) / 256, (int64_t)c.sms * 4);
    k_tr_opt<<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
  });
}

}  // namespace ls
