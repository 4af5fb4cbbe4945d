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

#include "blockhash.cuh"
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
using namespace sm100;

namespace {

constexpr int kT = 512;        // 16 warps: TMEM lane quadrant = warp % 4, column quarter = warp / 4
constexpr int kM = 128;        // rows per tile
constexpr int kMaxChunks = 4;  // K-blocks of 64 per CTA (all resident)

enum { TE_STORE = 0, TE_FWD = 1, TE_FWD_OUT = 2, TE_DX = 3 };

// One product D = A B^T over a K range, tiled as 128-row tiles x n_split
// column parts x splits of K; CTA li -> (column part li % n_split, row tile,
// split), so the column parts of a tile are adjacent (a cluster for TE_FWD_OUT).
struct TrJob {
  int epi;
  int m_tiles, n_split, splits, nchunks;
  int NT;                            // columns per CTA; the product's N = NT * n_split
  const uint8_t* A;                  // image, rA rows
  int rA;
  const uint8_t* B;                  // image, N rows
  int M;                             // valid rows of D
  // TE_STORE: fp32 partial D to C[split][row][col]
  float* C;
  int ldc;
  int64_t split_stride;
  // TE_FWD / TE_FWD_OUT / TE_DX
  const float* bias;                 // layer bias (TE_FWD, TE_FWD_OUT)
  uint8_t* out;                      // row-major image of the result, rows = rows_pad (nullable)
  uint8_t* outT;                     // transposed image, rows = rT
  int rT;
  uint16_t* mask_out;                // TE_FWD: bits of [Z > 0] as [N/16][rows_pad]
  const uint16_t* mask_in;           // TE_DX: bits of the layer input's ReLU
  float* colpart;                    // [m_tiles][N] column sums of dz (TE_FWD_OUT, TE_DX)
  int rows_pad;                      // padded batch (multiple of 128)
  // TE_FWD_OUT: width-1 output layer
  const float* wL;                   // [N] fp32 master weights of the output layer
  const float* bL;                   // [1]
  const float* y;                    // [batch] targets
  int batch;
  float* partWL;                     // [m_tiles][N]
  float* partBL;                     // [m_tiles]
  float* partLoss;                   // [m_tiles]
  // dropout between hidden layers (0 = none): TE_FWD drops units of hidden
  // activation drop_h and scales the kept ones; TE_DX scales the gradient of
  // the dropped activation drop_h (its keep bits are in mask_in)
  int drop_h;
};

struct TrArgs {
  TrJob job[2];
  int n_cta0;                        // CTAs of job 0; the rest run job 1
  int n_cta;                         // CTAs of both jobs
  int* err;
  const DevState* st;                // optimiser step counter (dropout stream)
  uint64_t drop_seed, drop_thr;      // keep <=> (u >> 11) >= drop_thr
  float drop_scale;                  // fp32 1 / (1 - p)
};

__device__ __forceinline__ uint16_t bf16_bits(float x) {
  __nv_bfloat16 v = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t*>(&v);
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Sum over the warp's 32 lanes of each of 16 per-lane values: afterwards
// lanes u and u + 16 hold the sum for column u.  Fixed order (butterfly).
__device__ __forceinline__ float col_reduce16(float (&v)[16]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 8; s >= 1; s >>= 1) {
    const bool up = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < s; ++i) {
      const float send = up ? v[i] : v[i + s];
      const float keep = up ? v[i + s] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0] + __shfl_xor_sync(0xffffffffu, v[0], 16);
}

// Row-major image from packed bf16 pairs: w[h] holds columns c + 2h (low
// half) and c + 2h + 1 (high half) of row j; c % 16 == 0.
__device__ __forceinline__ void store_row16p(uint8_t* img, int rows, int j, int c, const uint32_t (&w)[8]) {
  *reinterpret_cast<uint4*>(img + sw128_offset(j, c, rows)) = make_uint4(w[0], w[1], w[2], w[3]);
  *reinterpret_cast<uint4*>(img + sw128_offset(j, c + 8, rows)) = make_uint4(w[4], w[5], w[6], w[7]);
}

// Transposed image [rowsT x 128] from packed bf16 pairs: element (c + u, r)
// for u < 16, c % 16 == 0, r < 128 the tile row.  The same bytes as
// sw128_offset(c + u, r, rowsT), with the row's swizzle phase (c + u) & 7 =
// u & 7 folded into per-store constants.
__device__ __forceinline__ void store_col16p(uint8_t* imgT, int rowsT, int r, int c, const uint32_t (&w)[8]) {
  uint8_t* base = imgT + (size_t)(r >> 6) * rowsT * 128 + (size_t)c * 128 + (r & 7) * 2;
  const uint32_t cx = (uint32_t)((r & 63) >> 3) << 4;
#pragma unroll
  for (int u = 0; u < 16; ++u) {
    const uint16_t v = (u & 1) ? (uint16_t)(w[u >> 1] >> 16) : (uint16_t)(w[u >> 1] & 0xffffu);
    *reinterpret_cast<uint16_t*>(base + u * 128 + (cx ^ ((uint32_t)(u & 7) << 4))) = v;
  }
}

// Forward epilogue of one warp's columns [cbeg, cbeg + cw) of its 32 tile
// rows (r the thread's row): Z + b, ReLU and, with `drop`, dropout of unit
// n0 + c under the stream h1 (key rowkey + c, rowkey = (row << 20) | n0),
// each activation rounded to bf16 once as packed pairs that both images take
// their bytes from, and the 16-bit masks [Z > 0 and kept].
__device__ __forceinline__ void fwd_cols(uint32_t taddr, const float* s_bias, int cbeg, int cw, uint8_t* S1,
                                         uint8_t* S2, int NT, int r, uint16_t* mask_out, int64_t rows_pad,
                                         bool drop, uint64_t h1, uint64_t rowkey, uint64_t drop_thr,
                                         float drop_scale) {
  for (int c = cbeg; c < cbeg + cw; c += 16) {
    uint32_t v[16];
    tmem_ld16x(taddr + (uint32_t)c, v);
    tmem_wait_ld();
    uint32_t w[8];
    uint32_t bits = 0;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const float4 q4 = reinterpret_cast<const float4*>(s_bias + c)[g];
      const float bq[4] = {q4.x, q4.y, q4.z, q4.w};
      float a4[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int u = 4 * g + e;
        const float z = __uint_as_float(v[u]) + bq[e];
        float rv = z > 0.0f ? z : 0.0f;
        bool on = z > 0.0f;
        if (drop) {
          const uint64_t hu = bh::mix64(h1 ^ (rowkey + (uint64_t)(c + u)));
          const bool keep = (hu >> 11) >= drop_thr;
          on = on && keep;
          rv = keep ? rv * drop_scale : 0.0f;
        }
        bits |= (on ? 1u : 0u) << u;
        a4[e] = rv;
      }
      w[2 * g] = pack2(a4[0], a4[1]);
      w[2 * g + 1] = pack2(a4[2], a4[3]);
    }
    mask_out[(int64_t)(c >> 4) * rows_pad] = (uint16_t)bits;
    store_row16p(S1, kM, r, c, w);
    store_col16p(S2, NT, r, c, w);
  }
}

// Shared memory of a training-product CTA: kMaxChunks stages of one 128-row A
// tile and one (<= 256)-row B tile, then the barriers and epilogue scratch.
__device__ __forceinline__ uint8_t* tr_tail(uint8_t* smem) {
  return smem + (size_t)kMaxChunks * (kM * 128 + 256 * 128);
}

// The part of tile `bid` that reads nothing the step's earlier products
// write: arm every chunk barrier for the tile (the chunk barriers it does not
// use are arrived on with no bytes, so each advances one phase per tile),
// copy the weight operand (forward and input-gradient products read the
// weight images, which only the optimiser of the previous step writes) and
// stage the epilogue's bias and output weights (the fp32 master).  A
// per-launch product runs it before waiting for its predecessor.
__device__ __forceinline__ void tr_tile_pre(const TrArgs& args, int bid, uint8_t* smem) {
  const bool second = bid >= args.n_cta0;
  const TrJob& J = args.job[second ? 1 : 0];
  const int li = second ? bid - args.n_cta0 : bid;
  const int ns = li % J.n_split, rest = li / J.n_split;
  const int split = rest / J.m_tiles;
  const int NT = J.NT, N = NT * J.n_split, n0 = ns * NT, nch = J.nchunks;
  const uint32_t a_bytes = kM * 128, b_bytes = (uint32_t)NT * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  uint8_t* tail = tr_tail(smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(tail);
  float* s_bias = reinterpret_cast<float*>(tail + 128);
  float* s_w = s_bias + 256;
  const int tid = threadIdx.x;
  if (tid == 0) {
    const bool b_static = J.epi != TE_STORE;  // the weight-gradient products read activations
    for (int c = 0; c < nch; ++c) {
      const int kb = split * nch + c;
      mbar_arrive_expect_tx(&full[c], stage_bytes);
      if (b_static) bulk_g2s(smem + (size_t)c * stage_bytes + a_bytes, J.B + (size_t)kb * N * 128 + (size_t)n0 * 128,
                             b_bytes, &full[c]);
    }
    for (int c = nch; c < kMaxChunks; ++c) mbar_arrive(&full[c]);
  }
  for (int t = tid; t < NT; t += kT) {
    if (J.bias) s_bias[t] = __ldg(J.bias + n0 + t);
    if (J.epi == TE_FWD_OUT) s_w[t] = round_bf16(__ldg(J.wL + n0 + t));
  }
}

// The operand copies of tile `bid` that tr_tile_pre left (the activation or
// gradient operand; both operands of a weight-gradient product), by one
// thread, onto the barriers tr_tile_pre armed.
__device__ __forceinline__ void tr_tile_copies(const TrArgs& args, int bid, uint8_t* smem) {
  const bool second = bid >= args.n_cta0;
  const TrJob& J = args.job[second ? 1 : 0];
  const int li = second ? bid - args.n_cta0 : bid;
  const int ns = li % J.n_split, rest = li / J.n_split;
  const int mt = rest % J.m_tiles, split = rest / J.m_tiles;
  const int m0 = mt * kM;
  const int NT = J.NT, N = NT * J.n_split, n0 = ns * NT, nch = J.nchunks;
  const uint32_t a_bytes = kM * 128, b_bytes = (uint32_t)NT * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(tr_tail(smem));
  for (int c = 0; c < nch; ++c) {
    const int kb = split * nch + c;
    uint8_t* sa = smem + (size_t)c * stage_bytes;
    bulk_g2s(sa, J.A + (size_t)kb * J.rA * 128 + (size_t)m0 * 128, a_bytes, &full[c]);
    if (J.epi == TE_STORE) bulk_g2s(sa + a_bytes, J.B + (size_t)kb * N * 128 + (size_t)n0 * 128, b_bytes, &full[c]);
  }
}

// One output tile (part `bid` of the products in `args`) on this CTA's shared
// memory and TMEM accumulator, after tr_tile_pre of the same tile (and, when
// `copied`, tr_tile_copies).  Every
// mbarrier advances by one phase per tile (parity `par`).  `drain` waits for
// the tile's image stores to reach global memory (other CTAs of the grid read
// them); otherwise only until they have read shared memory.  Returns false
// after a timed-out wait (error latched, copies in flight waited for).
__device__ __forceinline__ bool tr_tile(const TrArgs& args, int bid, uint8_t* smem, uint32_t tmem, uint32_t par,
                                        bool drain, bool copied) {
  const bool second = bid >= args.n_cta0;
  const TrJob& J = args.job[second ? 1 : 0];
  const int li = second ? bid - args.n_cta0 : bid;
  const int ns = li % J.n_split, rest = li / J.n_split;
  const int mt = rest % J.m_tiles, split = rest / J.m_tiles;
  const int m0 = mt * kM;
  const int NT = J.NT, N = NT * J.n_split, n0 = ns * NT, nch = J.nchunks;
  const uint32_t a_bytes = kM * 128, b_bytes = (uint32_t)NT * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  uint8_t* tail = tr_tail(smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(tail);           // [kMaxChunks]
  uint64_t* done = full + kMaxChunks;
  float* s_bias = reinterpret_cast<float*>(tail + 128);         // [256]
  float* s_w = s_bias + 256;                                    // [256] bf16-rounded output weights
  float* red = s_w + 256;                                       // [4][256] column sums by lane quadrant
  float* red2 = red + 4 * 256;                                  // [4][256]
  float* rowq = red2 + 4 * 256;                                 // [8][128] row dots by column group
  float* rowdot = rowq + 8 * 128;                               // [128] this CTA's row dots
  float* yrow = rowdot + 128;                                   // [128] predictions
  float* wsum = yrow + 128;                                     // [8] warp partials

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  bool ok = true;
  if (tid == 0) {
    if (!copied) tr_tile_copies(args, bid, smem);
    const uint32_t idesc = idesc_bf16_f32(kM, NT);
    for (int c = 0; c < nch; ++c) {
      if (!mbar_wait(&full[c], par)) { ok = false; break; }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + (size_t)c * stage_bytes), sb = sa + a_bytes;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        umma_bf16(tmem, sdesc_sw128(sa + 32u * k), sdesc_sw128(sb + 32u * k), idesc, (c | k) ? 1u : 0u);
    }
    umma_commit(done);  // arrives once everything issued so far has completed
  }
  __syncwarp();
  if (!mbar_wait(done, par)) ok = false;
  ok = __syncthreads_and(ok) != 0;  // one decision for the whole CTA
  if (!ok) {
    latch_error(args.err, LS_ERR_TIMEOUT);
    // copies that may still be in flight land in this CTA's own shared memory;
    // wait (bounded) for them before the CTA exits
    if (tid == 0)
      for (int c = 0; c < nch; ++c) mbar_wait(&full[c], par);
  }
  tc_fence_after();

  const int q = warp & 3, cq = warp >> 2;
  const int r = 32 * q + lane, j = m0 + r;
  // the epilogues stage their image tiles in the (now free) operand stages,
  // in the images' own byte layout: the row-major tile [128 rows x NT] as
  // NT / 64 runs of 16 KB, the transposed tile [NT rows x 128] as two runs of
  // NT x 128 bytes; bulk copies then write each run with one instruction
  uint8_t* S1 = smem;
  uint8_t* S2 = smem + 65536;
  const int cw = NT / 4, cbeg = cq * cw;  // this warp's columns (CTA-local)
  const uint32_t lane_addr = (uint32_t)(32 * q) << 16;

  if (ok && J.epi == TE_STORE) {
    if (j < J.M) {
      float* crow = J.C + (int64_t)split * J.split_stride + (int64_t)j * J.ldc + n0;
      for (int c = cbeg; c < cbeg + cw; c += 16) {
        uint32_t v[16];
        tmem_ld16x(tmem + lane_addr + (uint32_t)c, v);
        tmem_wait_ld();
#pragma unroll
        for (int g = 0; g < 4; ++g)
          reinterpret_cast<float4*>(crow + c)[g] =
              make_float4(__uint_as_float(v[4 * g]), __uint_as_float(v[4 * g + 1]), __uint_as_float(v[4 * g + 2]),
                          __uint_as_float(v[4 * g + 3]));
      }
    }
  } else if (ok && J.epi == TE_FWD) {
    // dropout stream of this activation at step t = step + 1 (Sec. 4.1: dropout
    // between hidden layers): h1 = mix64(seed ^ ((t << 16) | h)),
    // u = mix64(h1 ^ ((row << 20) | unit)), kept when (u >> 11) >= thr
    uint64_t h1 = 0;
    if (J.drop_h > 0) {
      const uint64_t t = (uint64_t)(*reinterpret_cast<const volatile int64_t*>(&args.st->step) + 1);
      h1 = bh::mix64(args.drop_seed ^ ((t << 16) | (uint64_t)J.drop_h));
    }
    uint16_t* mask_out = J.mask_out + j + (int64_t)(n0 >> 4) * J.rows_pad;
    const bool drop = J.drop_h > 0;
    fwd_cols(tmem + lane_addr, s_bias, cbeg, cw, S1, S2, NT, r, mask_out, J.rows_pad, drop, h1,
             ((uint64_t)j << 20) | (uint64_t)n0, args.drop_thr, args.drop_scale);
  } else if (ok && J.epi == TE_DX) {
    for (int c = cbeg; c < cbeg + cw; c += 16) {
      uint32_t v[16];
      tmem_ld16x(tmem + lane_addr + (uint32_t)c, v);
      tmem_wait_ld();
      const uint32_t bits = J.mask_in[(int64_t)((n0 + c) >> 4) * J.rows_pad + j];
      float dz[16];
      const float sc = J.drop_h > 0 ? args.drop_scale : 1.0f;
#pragma unroll
      for (int u = 0; u < 16; ++u) dz[u] = ((bits >> u) & 1u) ? __uint_as_float(v[u]) * sc : 0.0f;
      uint32_t w[8];
#pragma unroll
      for (int h = 0; h < 8; ++h) w[h] = pack2(dz[2 * h], dz[2 * h + 1]);
      if (J.out) store_row16p(S1, kM, r, c, w);
      store_col16p(S2, NT, r, c, w);
      const float sb = col_reduce16(dz);
      if (lane < 16) red[q * 256 + c + lane] = sb;
    }
    __syncthreads();
    for (int c = tid; c < NT; c += kT)
      J.colpart[(int64_t)mt * N + n0 + c] = ((red[c] + red[256 + c]) + red[512 + c]) + red[768 + c];
  }
  if (J.epi == TE_FWD_OUT) {
    // pass 1: activations and this warp's part of the output dot product
    // With all 256 columns in one CTA (no cluster), each warp keeps its two
    // 32-column halves apart and the row dot is added as the two 128-column
    // CTAs of the cluster form add it: the same order, the same bits.
    const bool whole = NT == 256;
    if (ok) {
      float dot[2] = {0.0f, 0.0f};
      for (int c = cbeg; c < cbeg + cw; c += 16) {
        uint32_t v[16];
        tmem_ld16x(tmem + lane_addr + (uint32_t)c, v);
        tmem_wait_ld();
        const int hh = whole && c >= cbeg + 32 ? 1 : 0;
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const float z = __uint_as_float(v[u]) + s_bias[c + u];
          dot[hh] = fmaf(round_bf16(z > 0.0f ? z : 0.0f), s_w[c + u], dot[hh]);
        }
      }
      if (whole) {
        rowq[(2 * cq) * 128 + r] = dot[0];
        rowq[(2 * cq + 1) * 128 + r] = dot[1];
      } else {
        rowq[cq * 128 + r] = dot[0];
      }
    }
    __syncthreads();
    if (ok && tid < kM) {
      const float lo = ((rowq[tid] + rowq[128 + tid]) + rowq[256 + tid]) + rowq[384 + tid];
      rowdot[tid] = whole ? lo + (((rowq[512 + tid] + rowq[640 + tid]) + rowq[768 + tid]) + rowq[896 + tid]) : lo;
    }
    if (J.n_split > 1) cluster_sync();
    else __syncthreads();
    if (ok && tid < kM) {
      float tot = rowdot[tid];
      if (J.n_split > 1) {
        const uint32_t me = cluster_ctarank();
        const float other = ld_dsmem_f32(rowdot + tid, me ^ 1u);
        tot = me == 0 ? tot + other : other + tot;  // rank 0's part first on both
      }
      yrow[tid] = tot + __ldg(J.bL);
    }
    if (J.n_split > 1) cluster_sync();  // the partner has read this CTA's rowdot
    else __syncthreads();
    if (ok) {
      const bool valid = j < J.batch;
      const float yhat = yrow[r];
      const float e = valid ? yhat - __ldg(J.y + j) : 0.0f;
      const float dzL = valid ? 2.0f * e / (float)J.batch : 0.0f;
      const float rd = round_bf16(dzL);
      if (ns == 0 && cq == 0) {
        float e2 = e * e, dsum = dzL;
#pragma unroll
        for (int o = 16; o; o >>= 1) {
          e2 += __shfl_xor_sync(0xffffffffu, e2, o);
          dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
        }
        if (lane == 0) {
          wsum[q] = e2;
          wsum[4 + q] = dsum;
        }
      }
      // pass 2 (Z re-read from TMEM, so [Z > 0] is the same test as in pass 1):
      // dW_L partial (sum_j bf16(dz_L[j]) a[j, c]) and dz = bf16(dz_L) bf16(w_L) [Z > 0]
      for (int c = cbeg; c < cbeg + cw; c += 16) {
        uint32_t v[16];
        tmem_ld16x(tmem + lane_addr + (uint32_t)c, v);
        tmem_wait_ld();
        float pw[16], dz[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const float z = __uint_as_float(v[u]) + s_bias[c + u];
          const bool pos = z > 0.0f;
          pw[u] = rd * round_bf16(pos ? z : 0.0f);
          dz[u] = pos ? rd * s_w[c + u] : 0.0f;
        }
        uint32_t w[8];
#pragma unroll
        for (int h = 0; h < 8; ++h) w[h] = pack2(dz[2 * h], dz[2 * h + 1]);
        if (J.out) store_row16p(S1, kM, r, c, w);
        store_col16p(S2, NT, r, c, w);
        const float sw = col_reduce16(pw);
        if (lane < 16) red2[q * 256 + c + lane] = sw;
        const float sb = col_reduce16(dz);
        if (lane < 16) red[q * 256 + c + lane] = sb;
      }
    }
    __syncthreads();
    if (ok) {
      for (int c = tid; c < NT; c += kT) {
        J.partWL[(int64_t)mt * N + n0 + c] = ((red2[c] + red2[256 + c]) + red2[512 + c]) + red2[768 + c];
        J.colpart[(int64_t)mt * N + n0 + c] = ((red[c] + red[256 + c]) + red[512 + c]) + red[768 + c];
      }
      if (ns == 0 && tid == 0) {
        J.partLoss[mt] = ((wsum[0] + wsum[1]) + wsum[2]) + wsum[3];
        J.partBL[mt] = ((wsum[4] + wsum[5]) + wsum[6]) + wsum[7];
      }
    }
  }
  if (ok && (J.epi == TE_FWD || J.epi == TE_DX || J.epi == TE_FWD_OUT)) {
    fence_async_smem();  // staged tiles are read by the bulk copies (async proxy)
    __syncthreads();
    if (tid == 0) {
      if (J.out)
        for (int kb = 0; kb < NT / 64; ++kb)
          bulk_s2g(J.out + ((int64_t)(n0 / 64 + kb) * J.rows_pad + m0) * 128, S1 + (size_t)kb * kM * 128, kM * 128);
      for (int h = 0; h < kM / 64; ++h)
        bulk_s2g(J.outT + ((int64_t)(m0 / 64 + h) * J.rT + n0) * 128, S2 + (size_t)h * NT * 128,
                 (uint32_t)NT * 128);
      if (drain) bulk_commit_wait_all();
      else bulk_commit_wait_read();  // before the stages are reused or the CTA exits
    }
  }
  tc_fence_before();
  __syncthreads();
  return ok;
}

// One launch per product (or pair of products): CTA b runs tile b.
__global__ void __launch_bounds__(kT, 1) k_tr_gemm(const __grid_constant__ TrArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(tr_tail(smem));
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(full + kMaxChunks + 1);
  const int NT = args.job[(int)blockIdx.x >= args.n_cta0 ? 1 : 0].NT;
  uint32_t tcols = 32;
  while ((int)tcols < NT) tcols <<= 1;
  if (threadIdx.x == 0) {
    for (int c = 0; c <= kMaxChunks; ++c) mbar_init(&full[c], 1);  // chunk barriers, then `done`
    fence_mbar_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(tmem_holder, tcols);
    tmem_relinquish();
  }
  // The next product may start now: its CTAs take SMs this grid leaves idle
  // and run their own prologue while this one works.  Every kernel of the
  // step after the gather starts only after the gather has passed its wait
  // (it lets its successor in at its end), so after the previous step's
  // optimiser has completed: the weight images and the master read before
  // the wait below are final.
  pdl_trigger();
  tr_tile_pre(args, (int)blockIdx.x, smem);
  // the activation and gradient operands come from the previous kernels of the
  // stream: their copies start as soon as the wait returns
  pdl_wait();
  if (threadIdx.x == 0) tr_tile_copies(args, (int)blockIdx.x, smem);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  // image stores may still be in flight when the CTA exits: the grid's
  // completion makes them visible to the next kernel
  tr_tile(args, (int)blockIdx.x, smem, tmem, 0, false, true);
  if (threadIdx.x < 32) tmem_dealloc(tmem, tcols);
}

// Minibatch gather: row j of the batch (slot idx[j], or (step*B + j) mod
// valid) z-scored and rounded to bf16 into img(A_0) and img(A_0^T); rows past
// the batch and columns past d are zero.  Thread = (row j, 8 columns).
struct GatherArgs {
  int B, rows_pad, d, d_pad;
  const int32_t* idx;
  DevState* st;
  int64_t capacity, replay_base;
  const float* ring_x;
  const float* ring_y;
  const float* mean;
  const float* stdv;
  uint8_t* a0;
  uint8_t* a0t;
  float* y;
  int* err;
};

// Items [first, total) with stride `stride` of the minibatch gather; `lead`:
// this thread also checks the buffer and sets the Adam bias corrections.
__device__ __forceinline__ void tr_gather_items(const GatherArgs& g, int64_t first, int64_t stride, bool lead) {
  const int B = g.B, rows_pad = g.rows_pad, d = g.d, d_pad = g.d_pad;
  const int32_t* __restrict__ idx = g.idx;
  const float* __restrict__ ring_x = g.ring_x;
  const float* __restrict__ ring_y = g.ring_y;
  const float* __restrict__ mean = g.mean;
  const float* __restrict__ stdv = g.stdv;
  uint8_t* __restrict__ a0 = g.a0;
  uint8_t* __restrict__ a0t = g.a0t;
  float* __restrict__ y = g.y;
  int* err = g.err;
  DevState* st = g.st;
  const int64_t step = st->step;
  const int64_t count = st->ring_count;
  const int64_t nF = count < g.capacity ? count : g.capacity;
  const int64_t valid = nF + st->replay_count;  // F u R
  const int64_t replay_base = g.replay_base;
  if (valid < 1 && lead) {
    latch_error(err, LS_ERR_STATE);
    st->train_abort = 1;  // the optimiser of this step leaves every parameter as it is
  }
  if (lead) set_adam_bc(st);
  const int total = rows_pad * (d_pad / 8);  // at most 2^31 / 16 rows of 128 columns
  // rows of a multiple of four columns are read as 16-byte vectors
  const bool vec = (d & 3) == 0;
  for (int64_t e = first; e < total; e += stride) {
    const int ei = (int)e;
    const int j = ei % rows_pad, c0 = (ei / rows_pad) * 8;
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = 0.0f;
    if (j < B && valid > 0) {  // an empty buffer (error latched above) reads nothing: zero rows
      int64_t slot;
      if (idx) {
        slot = idx[j];
        if (slot < 0 || slot >= valid) {
          if (c0 == 0) {
            latch_error(err, LS_ERR_ARG);
            st->train_abort = 1;
          }
          slot = 0;
        }
      } else {
        slot = valid > 0 ? (step * (int64_t)B + j) % valid : 0;
      }
      slot = union_row(slot, nF, replay_base);
      const float* row = ring_x + slot * d;
      if (vec && c0 + 8 <= d) {
        float x[8], mu[8], sd[8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const float4 xv = __ldg(reinterpret_cast<const float4*>(row + c0) + h);
          const float4 mv = __ldg(reinterpret_cast<const float4*>(mean + c0) + h);
          const float4 sv = __ldg(reinterpret_cast<const float4*>(stdv + c0) + h);
          x[4 * h] = xv.x, x[4 * h + 1] = xv.y, x[4 * h + 2] = xv.z, x[4 * h + 3] = xv.w;
          mu[4 * h] = mv.x, mu[4 * h + 1] = mv.y, mu[4 * h + 2] = mv.z, mu[4 * h + 3] = mv.w;
          sd[4 * h] = sv.x, sd[4 * h + 1] = sv.y, sd[4 * h + 2] = sv.z, sd[4 * h + 3] = sv.w;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = round_bf16(zscore(x[u], mu[u], sd[u]));
      } else {
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (c0 + u < d) v[u] = round_bf16(zscore(__ldg(row + c0 + u), __ldg(mean + c0 + u), __ldg(stdv + c0 + u)));
      }
      if (c0 == 0) y[j] = ring_y[slot];
    } else if (j < B && c0 == 0) {
      y[j] = 0.0f;
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

__global__ void k_tr_gather(const __grid_constant__ GatherArgs g) {
  pdl_wait();  // the ring and the device counters from the previous kernels of the stream
  tr_gather_items(g, blockIdx.x * (int64_t)blockDim.x + threadIdx.x, (int64_t)gridDim.x * blockDim.x,
                  blockIdx.x == 0 && threadIdx.x == 0);
  pdl_trigger();
}

// sum_{s < n} src[s * stride], added in order, sixteen loads in flight.
__device__ __forceinline__ float ordered_sum(const float* __restrict__ src, int n, int64_t stride) {
  float g = 0.0f;
  int s = 0;
  for (; s + 16 <= n; s += 16) {
    float v[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) v[u] = __ldg(src + (int64_t)(s + u) * stride);
#pragma unroll
    for (int u = 0; u < 16; ++u) g += v[u];
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
  // one-pass launch: block b holds 256 parameters of layer l, blk0[l] <= b <
  // blk0[l + 1], from the layer's first parameter on (opt_blocks)
  int blk0[LS_MAX_LAYERS + 1];
};

// Gradient of every parameter as an ordered sum of its partials, the
// optimiser update of the fp32 master, and the bf16 images of the updated
// hidden-layer weights, for parameters [first, n) with stride `stride`.
// Gradient (ordered sum of its partials), optimiser update and bf16 image
// writes of parameter e of layer l.  A step whose gather found no record or a
// bad slot (`aborted`) changes nothing: the images already hold the unchanged
// weights.
__device__ __forceinline__ void tr_opt_one(const OptArgs& a, int l, int64_t e, bool aborted, float bc1, float bc2) {
  const MlpDesc& m = a.m;
  const int out = m.w[l + 1], in = m.w[l];
  const OptLayer& P = a.L[l];
  const bool hidden = l + 1 < m.n_layers, is_w = e < m.boff[l];
  int o = 0, i = 0;
  if (is_w) {
    const int u = (int)(e - m.woff[l]);  // index within one layer's weights
    if (hidden) {
      o = u / in;
      i = u - o * in;
    } else {
      i = u;
    }
  } else {
    o = (int)(e - m.boff[l]);
  }
  float p = a.p[e];
  if (a.mode != 0) {
    // the moments do not depend on the gradient: their loads overlap the partials'
    float mo = 0.0f, vo = 0.0f;
    if (a.mode == 2) {
      mo = a.mo[e];
      vo = a.vo[e];
    }
    float g;
    if (hidden)
      g = is_w ? ordered_sum(P.partW + (int64_t)o * P.ld + i, P.S, (int64_t)out * P.ld)
               : ordered_sum(P.partB + o, a.T, out);
    else
      g = is_w ? ordered_sum(P.partW + i, a.T, P.ld) : ordered_sum(P.partB, a.T, 1);
    if (aborted) return;
    if (a.mode == 1) {
      p = p - a.lr * g;
    } else {
      const float me = 0.9f * mo + 0.1f * g;
      const float ve = 0.999f * vo + 0.001f * g * g;
      a.mo[e] = me;
      a.vo[e] = ve;
      const float mh = me / bc1, vh = ve / bc2;
      p = p - a.lr * mh / (sqrtf(vh) + 1e-8f);
    }
    a.p[e] = p;
  }
  if (hidden && is_w) {
    const uint16_t b = bf16_bits(p);
    *reinterpret_cast<uint16_t*>(P.imgW + sw128_offset(o, i, out)) = b;
    *reinterpret_cast<uint16_t*>(P.imgWT + sw128_offset(i, o, P.in_pad)) = b;
  }
}

// Every parameter in [first, n) with stride `stride` (the persistent step).
__device__ __forceinline__ void tr_opt_items(const OptArgs& a, int64_t first, int64_t stride) {
  const MlpDesc& m = a.m;
  const int nl = m.n_layers;
  const bool aborted = a.mode != 0 && a.st->train_abort != 0;
  const float bc1 = a.st->adam_bc[0], bc2 = a.st->adam_bc[1];  // set by the gather kernel
  for (int64_t e = first; e < a.n; e += stride) {
    // the layer of parameter e: layer starts increase, so count those at or before e
    int l = 0;
#pragma unroll
    for (int k = 1; k < LS_MAX_LAYERS; ++k) l += (k < nl && e >= m.woff[k]) ? 1 : 0;
    tr_opt_one(a, l, e, aborted, bc1, bc2);
  }
}

// The minibatch loss (sum of the tile partials in order), by one warp: the
// lanes load 32 partials at once, every lane adds them in tile order, lane 0
// writes the result.
__device__ __forceinline__ void tr_loss_warp(const OptArgs& a) {
  if (a.mode != 0 && a.loss_out) {
    const int lane = threadIdx.x & 31;
    const bool abort = a.st->train_abort != 0;
    float s = 0.0f;
    for (int t0 = 0; t0 < a.T; t0 += 32) {
      const float v = t0 + lane < a.T ? a.partLoss[t0 + lane] : 0.0f;
      const int n = min(32, a.T - t0);
      for (int k = 0; k < n; ++k) s += __shfl_sync(0xffffffffu, v, k);
    }
    if (lane == 0) *a.loss_out = abort ? __int_as_float(0x7fc00000) : s / (float)a.B;
  }
}

__global__ void __launch_bounds__(256) k_tr_opt(const __grid_constant__ OptArgs a) {
  pdl_wait();  // gradient partials from the previous kernels of the stream
  pdl_trigger();
  const int64_t t = a.st->step + 1;
  const bool aborted = a.mode != 0 && a.st->train_abort != 0;
  const float bc1 = a.st->adam_bc[0], bc2 = a.st->adam_bc[1];  // set by the gather kernel
  {
    // this block's layer and parameters (one pass: a parameter per thread)
    const int nl = a.m.n_layers;
    int l = 0;
#pragma unroll
    for (int k = 1; k < LS_MAX_LAYERS; ++k) l += (k < nl && (int)blockIdx.x >= a.blk0[k]) ? 1 : 0;
    const int64_t e = a.m.woff[l] + (int64_t)((int)blockIdx.x - a.blk0[l]) * 256 + threadIdx.x;
    if (e < a.m.boff[l] + a.m.w[l + 1]) tr_opt_one(a, l, e, aborted, bc1, bc2);
  }
  if (blockIdx.x == 0 && threadIdx.x < 32) tr_loss_warp(a);
  // the last block, once every block has read the counter and the flag
  if (a.mode != 0 && last_block(&a.st->done[DONE_OPT]) && threadIdx.x == 0) {
    if (!aborted) advance_step(a.st, t);
    a.st->train_abort = 0;
  }
}

// ---------------------------------------------------------------------------
// The whole step as one persistent launch of a few CTAs (the rest of the GPU
// stays with routing): the gather, each product of the forward and backward
// passes (a phase: its tiles spread over the CTAs) and the optimiser, with a
// grid barrier between phases.  Same tiles, same epilogues and same order of
// every sum as the launch-per-phase path, so the same bits.
// ---------------------------------------------------------------------------
constexpr int kMaxPhases = 2 * (LS_MAX_LAYERS - 1);
constexpr uint32_t kGridSpin = 1u << 21;  // barrier polls before giving up (a second or so)

struct StepArgs {
  GatherArgs g;
  TrArgs ph[kMaxPhases];
  int n_ph;
  OptArgs opt;
  uint32_t* bar;  // [0] arrivals, [1] abort flag; zero at launch
};
static_assert(sizeof(StepArgs) <= 32000, "kernel parameters of the persistent step");

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// All CTAs meet (arrival `k` of each CTA: target k * gridDim.x).  Generic
// writes before it are visible to every read after it, bulk copies included.
// False for every CTA once one has given up (bounded wait) or failed a tile.
__device__ __forceinline__ bool tr_grid_sync(uint32_t* bar, uint32_t target, int* err) {
  __shared__ int s_go;
  asm volatile("fence.proxy.async.global;" ::: "memory");
  __syncthreads();
  if (threadIdx.x == 0) {
    volatile uint32_t* abort = bar + 1;
    __threadfence();
    atomicAdd(bar, 1u);
    int go = 1;
    for (uint32_t it = 0; ld_acquire_u32(bar) < target; ++it) {
      if (*abort || it >= kGridSpin) {
        if (!*abort) {
          atomicExch(bar + 1, 1u);
          latch_error(err, LS_ERR_TIMEOUT);
        }
        go = 0;
        break;
      }
      __nanosleep(64);
    }
    if (*abort) go = 0;
    s_go = go;
  }
  __syncthreads();
  asm volatile("fence.proxy.async.global;" ::: "memory");
  return s_go != 0;
}

__global__ void __launch_bounds__(kT, 1) k_tr_step(const __grid_constant__ StepArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(tr_tail(smem));
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(full + kMaxChunks + 1);
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int c = 0; c <= kMaxChunks; ++c) mbar_init(&full[c], 1);  // chunk barriers, then `done`
    fence_mbar_init();
  }
  if (tid < 32) {
    tmem_alloc(tmem_holder, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  int* err = a.g.err;
  const int64_t first = blockIdx.x * (int64_t)kT + tid, stride = (int64_t)gridDim.x * kT;
  uint32_t arrivals = 0;
  tr_gather_items(a.g, first, stride, blockIdx.x == 0 && tid == 0);
  bool go = tr_grid_sync(a.bar, ++arrivals * gridDim.x, err);
  uint32_t par = 0;
  for (int ph = 0; go && ph < a.n_ph; ++ph) {
    const TrArgs& P = a.ph[ph];
    for (int b = blockIdx.x; b < P.n_cta; b += gridDim.x) {
      tr_tile_pre(P, b, smem);
      if (!tr_tile(P, b, smem, tmem, par, true, false)) {
        if (tid == 0) atomicExch(a.bar + 1, 1u);
        go = false;
        break;
      }
      par ^= 1u;
    }
    if (go) go = tr_grid_sync(a.bar, ++arrivals * gridDim.x, err);
  }
  if (go) {
    tr_opt_items(a.opt, first, stride);
    if (tr_grid_sync(a.bar, ++arrivals * gridDim.x, err) && blockIdx.x == 0 && tid < 32) {
      tr_loss_warp(a.opt);
      __syncwarp();  // every lane has read the abort flag before lane 0 clears it
      if (tid == 0 && a.opt.mode != 0) {
        if (!a.opt.st->train_abort) advance_step(a.opt.st, a.opt.st->step + 1);
        a.opt.st->train_abort = 0;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid < 32) tmem_dealloc(tmem, 256);
}

int gemm_smem_bytes() {
  return 1024 + kMaxChunks * (kM * 128 + 256 * 128) + 128 + (256 + 256 + 8 * 256 + 8 * 128 + 128 + 128 + 8) * 4;
}

TrArgs tr_args(const Ctx& c, const TrJob& j0, const TrJob* j1, int* err) {
  TrArgs a{};
  a.st = c.st;
  a.drop_seed = c.cfg.dropout_seed;
  a.drop_thr = c.cfg.dropout > 0.0f ? (uint64_t)std::ceil((double)c.cfg.dropout * 9007199254740992.0) : 0;
  a.drop_scale = (float)(1.0 / (1.0 - (double)c.cfg.dropout));
  a.job[0] = j0;
  a.n_cta0 = j0.m_tiles * j0.n_split * j0.splits;
  int n = a.n_cta0;
  if (j1) {
    a.job[1] = *j1;
    n += j1->m_tiles * j1->n_split * j1->splits;
  }
  a.err = err;
  a.n_cta = n;
  return a;
}

cudaError_t launch_tr_gemm(const Ctx& c, const TrJob& j0, const TrJob* j1, int* err, cudaStream_t s) {
  const TrArgs a = tr_args(c, j0, j1, err);
  const int n = a.n_cta;
  const int smem = gemm_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(k_tr_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  // the column parts of a TE_FWD_OUT tile exchange row sums through
  // distributed shared memory: one cluster per tile
  const int cl = (j0.epi == TE_FWD_OUT && !j1) ? j0.n_split : 1;
  return launch_chained(k_tr_gemm, dim3(n), dim3(kT), (size_t)smem, s, cl, a);
}

// Column parts per tile: two when the columns split into halves that are
// multiples of 64 (each warp then owns a multiple of 16 columns).
int n_split_for(int N) { return N % 128 == 0 ? 2 : 1; }

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
    f.mask[l] = reinterpret_cast<uint16_t*>(p);
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

// Blocks of the one-pass optimiser launch: 256 parameters each, within one
// layer.  Returns the grid size.
int opt_blocks(const MlpDesc& m, OptArgs& a) {
  int b = 0;
  for (int l = 0; l < m.n_layers; ++l) {
    a.blk0[l] = b;
    const int64_t n_l = m.boff[l] + m.w[l + 1] - m.woff[l];
    b += (int)((n_l + 255) / 256);
  }
  for (int l = m.n_layers; l <= LS_MAX_LAYERS; ++l) a.blk0[l] = b;
  return b;
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
  const int grid = opt_blocks(m, a);
  k_tr_opt<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

namespace {
GatherArgs gather_args(const Ctx& c, int B, const int32_t* idx) {
  GatherArgs g{};
  g.B = B;
  g.rows_pad = ((B + kM - 1) / kM) * kM;
  g.d = c.mlp.w[0];
  g.d_pad = c.tf.in_pad[0];
  g.idx = idx;
  g.st = c.st;
  g.capacity = c.cfg.ring_capacity;
  g.replay_base = c.replay_base;
  g.ring_x = c.ring_x;
  g.ring_y = c.ring_y;
  g.mean = c.mean;
  g.stdv = c.stdv;
  g.a0 = c.tf.imgA[0];
  g.a0t = c.tf.imgAT[0];
  g.y = c.ty;
  g.err = c.d_err;
  return g;
}
}  // namespace

cudaError_t run_train_fast(Ctx& c, int B, const int32_t* idx, int opt, float lr, float* loss_out, cudaStream_t s) {
  const MlpDesc& m = c.mlp;
  TrainFast& f = c.tf;
  const int nh = m.n_layers - 1;  // hidden layers 0..nh-1, output layer nh
  const int R = ((B + kM - 1) / kM) * kM;
  const int T = R / kM;
  // one persistent launch (the products become its phases) or one launch each
  const bool one = c.train_ctas > 0;
  static thread_local StepArgs step;
  step = StepArgs{};
  cudaError_t e = cudaSuccess;
  if (!one) {
    e = traced(c, TR_GATHER, 1, s, [&] {
      const int64_t total = (int64_t)R * (f.in_pad[0] / 8);
      const int grid = (int)std::min<int64_t>((total + 255) / 256, (int64_t)c.sms * 8);
      return launch_chained(k_tr_gather, dim3(grid), dim3(256), 0, s, 1, gather_args(c, B, idx));
    });
    if (e != cudaSuccess) return e;
  }
  // forward: hidden layers; the last one also runs the output layer and the loss
  for (int l = 0; l < nh; ++l) {
    const bool last = l == nh - 1;
    TrJob J{};
    J.epi = last ? TE_FWD_OUT : TE_FWD;
    J.m_tiles = T;
    // the persistent launch has no clusters: the output layer's row dot
    // products stay within one CTA (all columns of the tile).  A hidden
    // layer of 256 columns runs as four 64-column parts (128 CTAs for a
    // batch of 4096: half the epilogue and image stores per SM)
    J.n_split = (last && one) ? 1 : (!last && !one && m.w[l + 1] % 256 == 0) ? 4 : n_split_for(m.w[l + 1]);
    J.splits = 1;
    J.nchunks = f.in_pad[l] / 64;
    J.NT = m.w[l + 1] / J.n_split;
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
    // dropout on hidden activation l + 1 when it feeds another hidden layer
    J.drop_h = (c.cfg.dropout > 0.0f && l + 2 < m.n_layers) ? l + 1 : 0;
    if (one) {
      step.ph[step.n_ph++] = tr_args(c, J, nullptr, c.d_err);
      continue;
    }
    e = traced(c, TR_GEMM_TC_FWD, 1, s, [&] { return launch_tr_gemm(c, J, nullptr, c.d_err, s); });
    if (e != cudaSuccess) return e;
  }
  // backward: dW_l (split over the batch) and, for l > 0, dz_{l-1} in the same launch
  for (int l = nh - 1; l >= 0; --l) {
    const int out = m.w[l + 1];
    TrJob W{};
    W.epi = TE_STORE;
    W.m_tiles = (out + kM - 1) / kM;
    W.n_split = n_split_for(f.in_pad[l]);
    // K-blocks (of 64 batch rows) per CTA: 4 when that still gives 48 CTAs,
    // else 2 (more CTAs, more partials for the optimiser to add)
    const int kpc = W.m_tiles * W.n_split * (R / 256) >= 48 ? 4 : 2;
    W.nchunks = std::min(kpc, R / 64);
    W.splits = (R / 64) / W.nchunks;
    W.NT = f.in_pad[l] / W.n_split;
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
      X.n_split = n_split_for(m.w[l]);
      X.splits = 1;
      X.nchunks = out / 64;
      X.NT = m.w[l] / X.n_split;
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
      X.drop_h = (c.cfg.dropout > 0.0f && l < m.n_layers - 1) ? l : 0;  // input a_l was dropped
    }
    if (one) {
      step.ph[step.n_ph++] = tr_args(c, W, l > 0 ? &X : nullptr, c.d_err);
      continue;
    }
    e = traced(c, l > 0 ? TR_GEMM_TC_DX : TR_GEMM_TC_DW, 1, s,
               [&] { return launch_tr_gemm(c, W, l > 0 ? &X : nullptr, c.d_err, s); });
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
  if (one) {
    step.g = gather_args(c, B, idx);
    step.opt = a;
    step.bar = c.tr_bar;
    return traced(c, TR_TRAIN_STEP, 1, s, [&] {
      cudaError_t e2 = cudaMemsetAsync(c.tr_bar, 0, 2 * sizeof(uint32_t), s);
      if (e2 != cudaSuccess) return e2;
      const int smem = gemm_smem_bytes();
      e2 = cudaFuncSetAttribute(k_tr_step, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e2 != cudaSuccess) return e2;
      cudaLaunchConfig_t cfg{};
      cfg.gridDim = dim3(c.train_ctas);
      cfg.blockDim = dim3(kT);
      cfg.dynamicSmemBytes = smem;
      cfg.stream = s;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident: the grid barrier needs it
      attr[0].val.cooperative = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      return cudaLaunchKernelEx(&cfg, k_tr_step, step);
    });
  }
  return traced(c, TR_OPT, 1, s, [&] {
    const int grid = opt_blocks(m, a);
    return launch_chained(k_tr_opt, dim3(grid), dim3(256), 0, s, 1, a);
  });
}

}  // namespace ls
