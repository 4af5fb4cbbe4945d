// Sequential-commit routing (Sec. 4.2 cluster snapshot manager and prefix
// KV-cache tracker; Sec. 4.3.1 P1: the gateway routes one request at a time):
// the requests of a batch are routed in order, and each decision is committed
// before the next request is scored -- the chosen instance's queue count grows
// by one and the prompt's full blocks join its cache (the prefix index gains
// the instance's bit for each block key), so a later request with the same
// prefix sees the hit and the longer queue.
//
// One persistent CTA walks the requests (the chain is inherently serial); per
// request:
//   1. hit lengths for every instance from the prefix index: the CTA's
//      threads look up a chunk of the prompt's block keys at once, a block-wide
//      prefix AND of their instance masks gives the instances matching every
//      block so far, and each instance finds where its bit dies by bisection;
//   2. feature rows (pair block, the instance rows as updated by earlier
//      decisions, request extras), z-scored, bf16-rounded in bf16 mode;
//   3. the predictor on CUDA cores: warp per output column, lanes across K,
//      rows in turn, published weights (bf16-rounded in bf16 mode, fp32 sums);
//   4. the argmin (lowest (score, index), NaN last);
//   5. the commit: queue count + 1, index insertion of the prompt's keys with
//      the chosen instance's bit (distinct keys counted against the table
//      capacity).
// Index reads bypass L1 (the CTA's own insertions must be visible to it).
#include "blockhash.cuh"
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
namespace {
using namespace bh;

constexpr int kSeqThreads = 512;
constexpr int kSeqWarps = kSeqThreads / 32;
constexpr int kSeqMaxW = 8;  // instance-mask words (512 instances)

struct SeqArgs {
  int n_req, n_inst, d_inst, d_req, q_col;
  const int64_t* tok_off;
  const uint64_t* bkeys;  // block keys of the batch at (tok_off[r] - tok_off[0]) / 16 + b
  const float* req;
  float* inst;            // [n_inst, d_inst] instance rows (updated in place at the end)
  const float* mean;
  const float* stdv;
  const float* params0;
  const float* params1;
  const DevState* st;
  MlpDesc m;
  int wmax;               // widest layer input / output
  int wsm;                // 1: the weights are copied into shared memory once per call
  int64_t wbytes;         // size of that weight region
  int64_t woff_s[LS_MAX_LAYERS];  // byte offset of layer l's transposed weights in the weight region
  uint64_t* gkeys;
  uint64_t* gmask;
  int W;
  uint64_t gslots_mask;
  int32_t* counts;
  int64_t max_keys;
  int32_t* choice;
  float* best;
  float* scores;          // [n_req, n_inst] or NULL
  int32_t* hits;          // [n_req, n_inst] or NULL
  int* err;
};

// Index lookups through L2 (ld.global.cg), so that keys this CTA inserted are seen.
__device__ __forceinline__ void seq_lookup(const SeqArgs& a, uint64_t key, uint64_t (&mw)[kSeqMaxW]) {
#pragma unroll
  for (int w = 0; w < kSeqMaxW; ++w) mw[w] = 0;
  const uint64_t mslots = a.gslots_mask;
  uint64_t s = key & mslots;
  for (uint64_t n = 0; n <= mslots; ++n) {
    const uint64_t k = a.W == 1 ? __ldcg(a.gkeys + 2 * s) : __ldcg(a.gkeys + s);
    if (k == key) {
      if (a.W == 1) mw[0] = __ldcg(a.gkeys + 2 * s + 1);
      else
        for (int w = 0; w < a.W; ++w) mw[w] = __ldcg(a.gmask + s * a.W + w);
      return;
    }
    if (k == 0) return;
    s = (s + 1) & mslots;
  }
}

// Insertion of `key` for instance `inst` (the protocol of the snapshot's index
// insert: CAS on an empty slot, OR of the instance's bit, a newly set bit
// counts one distinct key of the instance).
__device__ __forceinline__ void seq_insert(const SeqArgs& a, uint64_t key, int inst) {
  unsigned long long* tab = reinterpret_cast<unsigned long long*>(a.gkeys);
  const int kstride = a.W == 1 ? 2 : 1;
  uint64_t s = key & a.gslots_mask;
  int64_t slot = -1;
  for (uint64_t n = 0; n <= a.gslots_mask; ++n) {
    const unsigned long long prev = atomicCAS(tab + s * kstride, 0ull, (unsigned long long)key);
    if (prev == 0ull || prev == key) { slot = (int64_t)s; break; }
    s = (s + 1) & a.gslots_mask;
  }
  if (slot < 0) { latch_error(a.err, LS_ERR_TABLE_FULL); return; }
  const unsigned long long bit = 1ull << (inst & 63);
  unsigned long long* mword = a.W == 1 ? tab + 2 * slot + 1
                                       : reinterpret_cast<unsigned long long*>(a.gmask + slot * a.W + (inst >> 6));
  const unsigned long long old = atomicOr(mword, bit);
  if (!(old & bit)) {
    const int cnt = atomicAdd(a.counts + inst, 1);
    if (cnt >= a.max_keys) latch_error(a.err, LS_ERR_TABLE_FULL);
  }
}

__device__ __forceinline__ bool seq_precedes(float a, int i, float b, int j) {
  const bool an = a != a, bn = b != b;
  if (an != bn) return bn;
  if (!an && a != b) return a < b;
  return i < j;
}

// Byte offsets of the shared-memory arrays (each 16-byte aligned).  Layer
// inputs and activations take `xe` bytes each: 2 in bf16 mode (their values
// are bf16-rounded, so bf16 holds them exactly), 4 in fp32 mode.  The weight
// region (`wbytes`, 0 when the weights stay in global memory) holds every
// layer's W^T [in][out] in the predictor's element type.
struct SeqSmem {
  size_t inst, x0, x1, sc, hh, pa, wtot, carry, rv, ri, w, total;
};
__host__ __device__ __forceinline__ size_t seq_al(size_t b) { return (b + 15) & ~(size_t)15; }
__host__ __device__ __forceinline__ SeqSmem seq_smem(int N, int DI, int wmax, int W, int xe, size_t wbytes) {
  SeqSmem o;
  o.inst = 0;                                                   // [N][d_inst] fp32
  o.x0 = seq_al(o.inst + (size_t)N * (DI > 0 ? DI : 1) * 4);    // [N][wmax] activations
  o.x1 = seq_al(o.x0 + (size_t)N * wmax * xe);                  // [N][wmax] activations
  o.sc = seq_al(o.x1 + (size_t)N * wmax * xe);                  // [N] scores
  o.hh = seq_al(o.sc + (size_t)N * 4);                          // [N] hit lengths
  o.pa = seq_al(o.hh + (size_t)N * 4);                          // [kSeqThreads][W] prefix AND
  o.wtot = seq_al(o.pa + (size_t)kSeqThreads * W * 8);          // [kSeqWarps][W]
  o.carry = seq_al(o.wtot + (size_t)kSeqWarps * W * 8);         // [W]
  o.rv = seq_al(o.carry + (size_t)W * 8);                       // [kSeqWarps] argmin values
  o.ri = seq_al(o.rv + (size_t)kSeqWarps * 4);                  // [kSeqWarps] argmin indices
  o.w = seq_al(o.ri + (size_t)kSeqWarps * 4);                   // transposed weights (optional)
  o.total = seq_al(o.w + wbytes);
  return o;
}

// Activation element i of an array of `xe`-byte elements, as fp32 / stored.
__device__ __forceinline__ float seq_xget(const uint8_t* X, int64_t i, bool bf) {
  return bf ? __uint_as_float((uint32_t)reinterpret_cast<const uint16_t*>(X)[i] << 16)
            : reinterpret_cast<const float*>(X)[i];
}
__device__ __forceinline__ void seq_xset(uint8_t* X, int64_t i, float v, bool bf) {
  if (bf) reinterpret_cast<uint16_t*>(X)[i] = (uint16_t)(__float_as_uint(round_bf16(v)) >> 16);
  else reinterpret_cast<float*>(X)[i] = v;
}

// One hidden or output layer of the predictor in bf16, weights W^T [in][out]
// in shared memory: thread per (four rows, CT outputs).  Per pair of K steps
// one weight load of CT values per step and one 4-byte load per row (x[k],
// x[k+1]) feed 8·CT fp32 fused multiply-adds of bf16 inputs: the same
// products, each sum in K order, as the plain fp32 loop.  ReLU and bf16
// rounding of hidden outputs; the output layer's values go to sc.
template <int CT>
__device__ __forceinline__ void seq_layer_bf16(const uint8_t* Wt, const uint8_t* xin, uint8_t* xout,
                                               const float* __restrict__ bl, int N, int in, int out, int wmax,
                                               bool last_layer, float* sc) {
  const int n4 = (N + 3) >> 2, oc = out / CT;
  for (int e = threadIdx.x; e < n4 * oc; e += kSeqThreads) {
    const int o0 = CT * (e % oc), i0 = 4 * (e / oc);
    const uint8_t* xr[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) xr[q] = xin + (size_t)min(i0 + q, N - 1) * wmax * 2;
    float acc[4][CT];
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int j = 0; j < CT; ++j) acc[q][j] = 0.0f;
    const uint8_t* wp = Wt + (size_t)o0 * 2;
    const size_t wrow = (size_t)out * 2;
    uint32_t w0[CT / 2], w1[CT / 2];
    int k = 0;
    for (; k + 2 <= in; k += 2, wp += 2 * wrow) {
#pragma unroll
      for (int h = 0; h < CT / 2; ++h) {
        w0[h] = reinterpret_cast<const uint32_t*>(wp)[h];
        w1[h] = reinterpret_cast<const uint32_t*>(wp + wrow)[h];
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t xv = *reinterpret_cast<const uint32_t*>(xr[q] + (size_t)k * 2);
        const uint32_t x0 = __byte_perm(xv, 0u, 0x1010), x1 = __byte_perm(xv, 0u, 0x3232);
#pragma unroll
        for (int h = 0; h < CT / 2; ++h) sm100::fma2_bf16_f32(x0, w0[h], acc[q][2 * h], acc[q][2 * h + 1]);
#pragma unroll
        for (int h = 0; h < CT / 2; ++h) sm100::fma2_bf16_f32(x1, w1[h], acc[q][2 * h], acc[q][2 * h + 1]);
      }
    }
    if (k < in) {  // an odd K: the last step alone
#pragma unroll
      for (int h = 0; h < CT / 2; ++h) w0[h] = reinterpret_cast<const uint32_t*>(wp)[h];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t xs = reinterpret_cast<const uint16_t*>(xr[q])[k];
        const uint32_t x0 = xs | (xs << 16);
#pragma unroll
        for (int h = 0; h < CT / 2; ++h) sm100::fma2_bf16_f32(x0, w0[h], acc[q][2 * h], acc[q][2 * h + 1]);
      }
    }
#pragma unroll
    for (int j = 0; j < CT; ++j) {
      const float bo = __ldg(bl + o0 + j);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (i0 + q >= N) break;
        const float z = acc[q][j] + bo;
        if (last_layer) sc[i0 + q] = z;
        else seq_xset(xout, (int64_t)(i0 + q) * wmax + o0 + j, fmaxf(z, 0.0f), true);
      }
    }
  }
}

__global__ void __launch_bounds__(kSeqThreads, 1) k_route_seq(const __grid_constant__ SeqArgs a, int64_t bcap) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  const int N = a.n_inst, DI = a.d_inst, W = a.W;
  const MlpDesc& m = a.m;
  const int d = m.w[0];
  const bool bf = m.bf16 != 0;
  const SeqSmem o = seq_smem(N, DI, a.wmax, W, bf ? 2 : 4, a.wsm ? (size_t)a.wbytes : 0);
  float* sinst = reinterpret_cast<float*>(smem_raw + o.inst);
  uint8_t* X0 = smem_raw + o.x0;
  uint8_t* X1 = smem_raw + o.x1;
  uint8_t* Wsm = smem_raw + o.w;
  float* sc = reinterpret_cast<float*>(smem_raw + o.sc);
  int32_t* hh = reinterpret_cast<int32_t*>(smem_raw + o.hh);
  uint64_t* PA = reinterpret_cast<uint64_t*>(smem_raw + o.pa);
  uint64_t* wtot = reinterpret_cast<uint64_t*>(smem_raw + o.wtot);
  uint64_t* carry = reinterpret_cast<uint64_t*>(smem_raw + o.carry);
  float* rv = reinterpret_cast<float*>(smem_raw + o.rv);
  int* ri = reinterpret_cast<int*>(smem_raw + o.ri);
  __shared__ int s_buf, s_go, s_choice;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) s_buf = *reinterpret_cast<const volatile int32_t*>(&a.st->cur) == 1 ? 1 : 0;
  for (int e = tid; e < N * DI; e += kSeqThreads) sinst[e] = a.inst[e];
  __syncthreads();
  const float* __restrict__ params = s_buf ? a.params1 : a.params0;
  if (a.wsm) {
    // every layer's W^T [in][out] in shared memory for the whole call (the
    // published weights, bf16-valued in bf16 mode, so bf16 holds them exactly);
    // read along W's rows (coalesced), written transposed
    for (int l = 0; l < m.n_layers; ++l) {
      const int in = m.w[l], out = m.w[l + 1];
      const float* __restrict__ Wl = params + m.woff[l];
      uint8_t* Wt = Wsm + a.woff_s[l];
      for (int e = tid; e < in * out; e += kSeqThreads) {
        const int oo = e / in, k = e - oo * in;
        seq_xset(Wt, (int64_t)k * out + oo, __ldg(Wl + e), bf);
      }
    }
    __syncthreads();
  }
  const int64_t base = a.tok_off[0];
  for (int r = 0; r < a.n_req; ++r) {
    const int64_t t0 = a.tok_off[r];
    const int64_t L = a.tok_off[r + 1] - t0;
    const int64_t nb = L / kBlockTok;
    const int64_t k0 = (t0 - base) / kBlockTok;
    // ---- 1. hit lengths
    for (int i = tid; i < N; i += kSeqThreads) hh[i] = -1;
    if (tid < W) {
      const int lo = 64 * tid;
      carry[tid] = N >= lo + 64 ? ~0ull : (N > lo ? ((1ull << (N - lo)) - 1ull) : 0ull);
    }
    __syncthreads();
    for (int64_t p = 0; p < nb; p += kSeqThreads) {
      const int64_t b = p + tid;
      uint64_t mw[kSeqMaxW];
      if (b < nb) {
        const uint64_t key = k0 + b < bcap ? a.bkeys[k0 + b] : 0ull;  // past the key scratch: a miss
        if (key) seq_lookup(a, key, mw);
        else
#pragma unroll
          for (int w = 0; w < kSeqMaxW; ++w) mw[w] = 0;
      } else {
#pragma unroll
        for (int w = 0; w < kSeqMaxW; ++w) mw[w] = ~0ull;  // past the prompt: changes nothing
      }
#pragma unroll
      for (int w = 0; w < kSeqMaxW; ++w) {
        if (w >= W) break;
        uint64_t x = mw[w];
#pragma unroll
        for (int k = 0; k < 5; ++k) {
          const uint64_t y = __shfl_up_sync(kFull, x, 1 << k);
          if (lane >= (1 << k)) x &= y;
        }
        mw[w] = x;
        if (lane == 31) wtot[warp * W + w] = x;
      }
      __syncthreads();
#pragma unroll
      for (int w = 0; w < kSeqMaxW; ++w) {
        if (w >= W) break;
        uint64_t e = carry[w];
        for (int v = 0; v < warp; ++v) e &= wtot[v * W + w];
        PA[tid * W + w] = e & mw[w];
      }
      __syncthreads();
      const int last = (int)(nb - p < kSeqThreads ? nb - p : kSeqThreads) - 1;
      for (int i = tid; i < N; i += kSeqThreads) {
        if (hh[i] >= 0) continue;
        const int wi = i >> 6;
        const uint64_t bit = 1ull << (i & 63);
        if (PA[last * W + wi] & bit) continue;  // still matching after this chunk
        int lo = 0, hi = last;                   // first t whose prefix AND lost the bit
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (PA[mid * W + wi] & bit) lo = mid + 1; else hi = mid;
        }
        hh[i] = (int32_t)(p + lo);
      }
      __syncthreads();
      if (tid == 0) {
        int any = 0;
        for (int w = 0; w < W; ++w) {
          carry[w] = PA[last * W + w];
          any |= carry[w] != 0;
        }
        s_go = any;
      }
      __syncthreads();
      if (!s_go) break;
    }
    for (int i = tid; i < N; i += kSeqThreads)
      if (hh[i] < 0) hh[i] = (int32_t)nb;  // matching every full block
    __syncthreads();
    // ---- 2. feature rows
    for (int e = tid; e < N * d; e += kSeqThreads) {
      const int i = e / d, k = e - i * d;
      float raw;
      if (k < kPair) raw = raw_feature(k, L, hh[i], nullptr, 0, nullptr);
      else if (k < kPair + DI) raw = sinst[i * DI + (k - kPair)];
      else raw = a.req[(int64_t)r * a.d_req + (k - kPair - DI)];
      const float x = zscore(raw, a.mean[k], a.stdv[k]);
      seq_xset(X0, (int64_t)i * a.wmax + k, x, bf);
    }
    __syncthreads();
    // ---- 3. the predictor
    uint8_t* xin = X0;
    uint8_t* xout = X1;
    for (int l = 0; l < m.n_layers; ++l) {
      const int in = m.w[l], out = m.w[l + 1];
      const bool last_layer = l + 1 == m.n_layers;
      const float* __restrict__ bl = params + m.boff[l];
      if (a.wsm && out < 32) {
        // a narrow layer (the output layer): warp per row, lanes across K
        const uint8_t* Wt = Wsm + a.woff_s[l];
        for (int e = warp; e < N * out; e += kSeqWarps) {
          const int i = e / out, oo = e - i * out;
          float part = 0.0f;
          for (int k = lane; k < in; k += 32)
            part = fmaf(seq_xget(Wt, (int64_t)k * out + oo, bf), seq_xget(xin, (int64_t)i * a.wmax + k, bf), part);
#pragma unroll
          for (int sft = 16; sft; sft >>= 1) part += __shfl_xor_sync(kFull, part, sft);
          if (lane == 0) {
            const float z = part + __ldg(bl + oo);
            if (last_layer) sc[i] = z;
            else seq_xset(xout, (int64_t)i * a.wmax + oo, fmaxf(z, 0.0f), bf);
          }
        }
      } else if (a.wsm && bf && (out & 3) == 0 && (a.wmax & 1) == 0) {
        // bf16: thread per (four rows, four outputs) (two outputs a thread,
        // for more threads when the rows are few, measured no faster)
        seq_layer_bf16<4>(Wsm + a.woff_s[l], xin, xout, bl, N, in, out, a.wmax, last_layer, sc);
      } else if (a.wsm) {
        // thread per (output, four rows): one weight and four broadcast
        // inputs per K step, fp32 sums, the bias added after the sum
        const uint8_t* Wt = Wsm + a.woff_s[l];
        const int nb4 = (N + 3) >> 2;
        const int xe = bf ? 2 : 4;
        for (int e = tid; e < nb4 * out; e += kSeqThreads) {
          const int oo = e % out, i0 = (e / out) * 4;
          const uint8_t* xr[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) xr[q] = xin + (size_t)min(i0 + q, N - 1) * a.wmax * xe;
          const uint8_t* wp = Wt + (size_t)oo * xe;
          const int wstep = out * xe;
          float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll 4
          for (int k = 0; k < in; ++k, wp += wstep) {
            const float wv = seq_xget(wp, 0, bf);
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[q] = fmaf(wv, seq_xget(xr[q], k, bf), acc[q]);
          }
          const float bo = __ldg(bl + oo);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (i0 + q >= N) break;
            const float z = acc[q] + bo;
            if (last_layer) sc[i0 + q] = z;
            else seq_xset(xout, (int64_t)(i0 + q) * a.wmax + oo, fmaxf(z, 0.0f), bf);
          }
        }
      } else {
        // weights too large for shared memory: warp per output column, lanes
        // across K, the column's weights in registers
        const float* __restrict__ Wl = params + m.woff[l];
        for (int oo = warp; oo < out; oo += kSeqWarps) {
          float wr[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int k = lane + 32 * j;
            wr[j] = k < in ? __ldg(Wl + (int64_t)oo * in + k) : 0.0f;
          }
          const float bo = __ldg(bl + oo);
          for (int i = 0; i < N; ++i) {
            float part = 0.0f;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int k = lane + 32 * j;
              if (k < in) part = fmaf(wr[j], seq_xget(xin, (int64_t)i * a.wmax + k, bf), part);
            }
#pragma unroll
            for (int sft = 16; sft; sft >>= 1) part += __shfl_xor_sync(kFull, part, sft);
            if (lane == 0) {
              const float z = part + bo;
              if (last_layer) sc[i] = z;
              else seq_xset(xout, (int64_t)i * a.wmax + oo, fmaxf(z, 0.0f), bf);
            }
          }
        }
      }
      __syncthreads();
      uint8_t* t = xin;
      xin = xout;
      xout = t;
    }
    // ---- 4. selection
    {
      float bv = 0.0f;
      int bi = -1;
      for (int i = tid; i < N; i += kSeqThreads)
        if (bi < 0 || seq_precedes(sc[i], i, bv, bi)) { bv = sc[i]; bi = i; }
#pragma unroll
      for (int s = 16; s; s >>= 1) {
        const float ov = __shfl_xor_sync(kFull, bv, s);
        const int oi = __shfl_xor_sync(kFull, bi, s);
        if (oi >= 0 && (bi < 0 || seq_precedes(ov, oi, bv, bi))) { bv = ov; bi = oi; }
      }
      if (lane == 0) { rv[warp] = bv; ri[warp] = bi; }
      __syncthreads();
      if (tid == 0) {
        float v = rv[0];
        int c = ri[0];
        for (int w = 1; w < kSeqWarps; ++w)
          if (ri[w] >= 0 && (c < 0 || seq_precedes(rv[w], ri[w], v, c))) { v = rv[w]; c = ri[w]; }
        s_choice = c;
        a.choice[r] = c;
        a.best[r] = v;
        if (a.q_col >= 0 && c >= 0) sinst[c * DI + a.q_col] += 1.0f;  // ---- 5a. the queue grows
      }
    }
    if (a.scores)
      for (int i = tid; i < N; i += kSeqThreads) a.scores[(int64_t)r * N + i] = sc[i];
    if (a.hits)
      for (int i = tid; i < N; i += kSeqThreads) a.hits[(int64_t)r * N + i] = hh[i];
    __syncthreads();
    // ---- 5b. the chosen instance caches the prompt's blocks
    const int c = s_choice;
    if (c >= 0)
      for (int64_t b = tid; b < nb; b += kSeqThreads)
        if (k0 + b < bcap) seq_insert(a, a.bkeys[k0 + b], c);
    __syncthreads();
  }
  for (int e = tid; e < N * DI; e += kSeqThreads) a.inst[e] = sinst[e];
}

}  // namespace

// Shared memory of the sequential route without the weight region, 0 if the
// shape does not fit (bf16 activations: the smaller of the two layouts).
size_t route_seq_smem(int n_inst, int d_inst, int wmax, int W) {
  if (W < 1 || W > kSeqMaxW || wmax > 512 || n_inst < 1) return 0;
  const size_t b = seq_smem(n_inst, d_inst, wmax, W, 4, 0).total;
  return b <= 200 * 1024 ? b : 0;
}

cudaError_t launch_route_seq(int n_req, int n_inst, int d_inst, int d_req, int q_col, const int64_t* tok_off,
                             const uint64_t* bkeys, int64_t bcap, const float* req, float* inst, const float* mean,
                             const float* stdv, const Published* pub, const DevState* st, const MlpDesc& m,
                             uint64_t* gkeys, uint64_t* gmask, int W, uint64_t gslots_mask, int32_t* counts,
                             int64_t max_keys, int32_t* choice, float* best, float* scores, int32_t* hits, int* err,
                             cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  SeqArgs a{};
  a.n_req = n_req;
  a.n_inst = n_inst;
  a.d_inst = d_inst;
  a.d_req = d_req;
  a.q_col = q_col;
  a.tok_off = tok_off;
  a.bkeys = bkeys;
  a.req = req;
  a.inst = inst;
  a.mean = mean;
  a.stdv = stdv;
  a.params0 = pub[0].params;
  a.params1 = pub[1].params;
  a.st = st;
  a.m = m;
  int wmax = 1;
  for (int l = 0; l <= m.n_layers; ++l) wmax = std::max(wmax, m.w[l]);
  a.wmax = wmax;
  a.gkeys = gkeys;
  a.gmask = gmask;
  a.W = W;
  a.gslots_mask = gslots_mask;
  a.counts = counts;
  a.max_keys = max_keys;
  a.choice = choice;
  a.best = best;
  a.scores = scores;
  a.hits = hits;
  a.err = err;
  if (!route_seq_smem(n_inst, d_inst, wmax, W)) return cudaErrorInvalidValue;
  const int xe = m.bf16 ? 2 : 4;
  int64_t wb = 0;
  for (int l = 0; l < m.n_layers; ++l) {
    a.woff_s[l] = wb;
    wb += (((int64_t)m.w[l] * m.w[l + 1] * xe) + 15) & ~(int64_t)15;
  }
  // the weights go to shared memory when they fit beside the rest
  const size_t with_w = seq_smem(n_inst, d_inst, wmax, W, xe, (size_t)wb).total;
  a.wsm = with_w <= 224 * 1024 ? 1 : 0;
  a.wbytes = a.wsm ? wb : 0;
  const size_t smem = a.wsm ? with_w : seq_smem(n_inst, d_inst, wmax, W, xe, 0).total;
  cudaError_t e = cudaFuncSetAttribute(k_route_seq, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_route_seq<<<1, kSeqThreads, smem, s>>>(a, bcap);
  return cudaGetLastError();
}

}  // namespace ls
