// Tensor-core scorer for bf16 predictors (Sec. 4.1 reward model; Algorithm 4
// batched forward): every hidden Linear layer is a tcgen05 MMA with the fp32
// accumulator in tensor memory; feature tiles and hidden activations are
// built in shared memory in the 128-byte-swizzled K-major layout the MMA
// reads; weights arrive by bulk copy (TMA engine) from a pre-swizzled bf16
// image written at publish time; the width-1 output layer is a dot product in
// the last epilogue.
//
// One persistent CTA per SM (512 threads) walks 128-row tiles (row = r*N + i).
// Per tile: build the feature tile -> for each hidden layer: one thread issues
// the MMAs (K = 16 per instruction, N-chunks of <= 256 columns), all warps then
// read the accumulator (warp w: TMEM lanes 32*(w%4).., column quarter w/4), add
// the bias, apply ReLU, round to bf16 and write the next layer's operand tile.
// When every weight chunk fits in shared memory the weights are loaded once per
// CTA; otherwise they stream through a ring of stages, the next chunk's copy
// overlapping the current MMAs.
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
using namespace sm100;

namespace {

constexpr int kTileM = 128;
constexpr int kThreadsTc = 512;  // 16 warps: 4 per TMEM lane quadrant
constexpr int kMaxChunks = 64;
constexpr int kMaxSmem = 232448;  // 227 KB opt-in per CTA

struct TcArgs {
  TcPlan p;
  const uint8_t* img0;     // published buffer 0 / 1: tensor-core weight image
  const uint8_t* img1;
  const float* params0;    // published buffer 0 / 1: flat fp32 parameters
  const float* params1;
  const int32_t* sel;      // buffer this route reads (device), NULL: buffer 0
  int64_t boff[LS_MAX_LAYERS];
  int64_t w_last_off;
  int n_req, n_inst, d, d_inst, d_req;
  const uint4* pairx;    // [rows] bf16 pair features (chunk 0 of each feature row, zeros past column 5)
  const uint8_t* ximg;   // pipelined kernel: feature tiles, tile t = xbytes at t * xbytes, in the MMA layout
  int32_t* choice;       // pipelined kernel with n_inst dividing 32: the selector runs in the epilogue
  float* best;
  int fuse_argmin;
  const uint16_t* xin;   // [n_inst, d_pad] bf16 instance template rows (zero outside inst columns)
  const uint16_t* xrq;   // [n_req, d_pad]  bf16 request template rows (zero outside req columns)
  const float* mean;
  const float* stdv;
  float* scores;
  int* err;
  int64_t rows;
  int n_tiles;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint16_t bf16_bits(float x) {
  __nv_bfloat16 v = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t*>(&v);
}

// 16-byte global load that leaves L1 alone (streamed feature inputs must not
// evict the epilogue's bias and weight lines)
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void st_shared_v4(uint8_t* p, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(smem_u32(p)), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}

// Feature tile of rows row0..row0+127: [pair(6) || inst || req || 0-pad] as bf16.
// The instance and request blocks come from template rows that hold the
// normalised values at their feature positions and zeros elsewhere, and the
// pair features of each row come as one 16-byte chunk with zeros past column
// 5 (k_norm_rows), so a 16-byte chunk of a feature row is the OR of at most
// three loaded chunks.  `nthr` threads (index `tr`) share the tile; each
// issues the loads of its U chunks before combining any of them, so that 3 U
// loads are in flight per thread (the loads are ordered asm, and a combine
// between them would wait for each group in turn).  Rows past the batch are
// zeros.
template <int U>
__device__ __forceinline__ void build_tile(const TcArgs& a, uint8_t* X, int64_t row0, int tr, int nthr) {
  const int cpr = a.p.d_pad / 8;  // 16-byte chunks per row
  const int total = kTileM * cpr;
  const int csh = (cpr & (cpr - 1)) == 0 ? __ffs(cpr) - 1 : -1;  // shift when cpr is a power of two
  const int64_t r0 = row0 / a.n_inst;
  const int i0 = (int)(row0 - r0 * a.n_inst);
  for (int base = 0; base < total; base += U * nthr) {
    uint4 ti[U], tq[U], tp[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int e = base + u * nthr + tr;
      ti[u] = tq[u] = tp[u] = make_uint4(0u, 0u, 0u, 0u);
      if (e >= total) continue;
      const int m = csh >= 0 ? e >> csh : e / cpr, c = e - m * cpr;
      const int64_t g = row0 + m;
      if (g >= a.rows) continue;
      int i = i0 + m;
      int64_t r = r0;
      if (a.n_inst >= 16) {
        while (i >= a.n_inst) { i -= a.n_inst; ++r; }
      } else {
        r += i / a.n_inst;
        i -= (i / a.n_inst) * a.n_inst;
      }
      ti[u] = ldg_stream(reinterpret_cast<const uint4*>(a.xin + (int64_t)i * a.p.d_pad) + c);
      tq[u] = ldg_stream(reinterpret_cast<const uint4*>(a.xrq + r * a.p.d_pad) + c);
      if (c == 0) tp[u] = ldg_stream(a.pairx + g);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int e = base + u * nthr + tr;
      if (e >= total) continue;
      const int m = csh >= 0 ? e >> csh : e / cpr, c = e - m * cpr;
      st_shared_v4(X + sw128_offset(m, c * 8, kTileM), ti[u].x | tq[u].x | tp[u].x, ti[u].y | tq[u].y | tp[u].y,
                   ti[u].z | tq[u].z | tp[u].z, ti[u].w | tq[u].w | tp[u].w);
    }
  }
}

// 16 consecutive fp32 columns of the warp's 32 TMEM lanes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ float4 ldg4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }

__global__ void __launch_bounds__(kThreadsTc, 1) k_score_tc(const __grid_constant__ TcArgs a) {
  const bool pb = a.sel && *a.sel == 1;  // published buffer of this route
  const uint8_t* __restrict__ img = pb ? a.img1 : a.img0;
  const float* __restrict__ params = pb ? a.params1 : a.params0;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const TcPlan& p = a.p;
  uint8_t* A = smem;
  uint8_t* ring = smem + p.a_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)p.stages * p.chunk_bytes);
  uint64_t* empty = full + p.stages;
  uint64_t* done = empty + p.stages;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_holder + 1);
  // partial dot products of the output layer [4][128]; they reuse the operand
  // tile, whose last reader (the final layer's MMA) has completed by then
  float* part = reinterpret_cast<float*>(A);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  const int my_tiles = blockIdx.x < a.n_tiles ? (a.n_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int64_t total = (int64_t)my_tiles * p.chunks;
  int64_t g_load = 0;  // thread 0: next chunk (in consumption order) to copy

  auto issue_load = [&](int64_t gq) {  // thread 0, streaming mode
    const int s = (int)(gq % p.stages);
    const int64_t u = gq / p.stages;
    if (u >= 1 && !mbar_wait(&empty[s], (uint32_t)((u - 1) & 1))) return false;
    const int q = (int)(gq % p.chunks);
    mbar_arrive_expect_tx(&full[s], (uint32_t)p.chunk_len[q]);
    bulk_g2s(ring + (size_t)s * p.chunk_bytes, img + p.chunk_off[q], (uint32_t)p.chunk_len[q], &full[s]);
    return true;
  };

  if (tid == 0 && my_tiles > 0) {
    if (p.resident) {
      for (int q = 0; q < p.chunks; ++q) {
        mbar_arrive_expect_tx(&full[q], (uint32_t)p.chunk_len[q]);
        bulk_g2s(ring + (size_t)q * p.chunk_bytes, img + p.chunk_off[q], (uint32_t)p.chunk_len[q], &full[q]);
      }
    } else {
      while (g_load < total && g_load < p.stages - 1) {
        if (!issue_load(g_load)) { *abort_flag = 1; break; }
        ++g_load;
      }
    }
  }
  uint32_t done_phase = 0;
  const int q4 = warp & 3;   // TMEM lane quadrant: rows 32*q4 .. 32*q4+31
  const int cq = warp >> 2;  // column quarter handled by this warp
  const int row = 32 * q4 + lane;
  const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;

  for (int it = 0; it < my_tiles; ++it) {
    const int64_t row0 = (int64_t)(blockIdx.x + (int64_t)it * gridDim.x) * kTileM;
    build_tile<4>(a, A, row0, threadIdx.x, kThreadsTc);
    fence_async_smem();
    __syncthreads();
    if (*abort_flag) break;
    int q = 0;
    for (int l = 0; l < p.n_tc; ++l) {
      if (tid == 0) {
        tc_fence_after();
        bool ok = true;
        const int nk = p.in_pad[l] / 64, nn = p.out[l] / p.nc[l];
        const uint32_t idesc = idesc_bf16_f32(kTileM, p.nc[l]);
        for (int nci = 0; nci < nn && ok; ++nci) {
          for (int kb = 0; kb < nk && ok; ++kb, ++q) {
            const int64_t gq = (int64_t)it * p.chunks + q;
            int s;
            uint32_t par;
            if (p.resident) { s = q; par = 0; }
            else { s = (int)(gq % p.stages); par = (uint32_t)((gq / p.stages) & 1); }
            if (!mbar_wait(&full[s], par)) { ok = false; break; }
            tc_fence_after();
            const uint32_t a_base = smem_u32(A) + (uint32_t)kb * kTileM * 128u;
            const uint32_t b_base = smem_u32(ring + (size_t)s * p.chunk_bytes);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              umma_bf16(tmem + (uint32_t)(nci * p.nc[l]), sdesc_sw128(a_base + 32u * j),
                        sdesc_sw128(b_base + 32u * j), idesc, (kb | j) ? 1u : 0u);
            if (!p.resident) {
              umma_commit(&empty[s]);
              while (ok && g_load < total && g_load < gq + p.stages) {
                ok = issue_load(g_load);
                ++g_load;
              }
            }
          }
        }
        umma_commit(done);
        if (!ok) {
          *abort_flag = 1;
          latch_error(a.err, LS_ERR_TIMEOUT);
        }
      }
      __syncwarp();
      if (!mbar_wait(done, done_phase)) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
      }
      done_phase ^= 1u;
      tc_fence_after();
      const int qw = p.out[l] / 4;  // columns per warp
      const int cbeg = cq * qw;
      const float* bias = params + a.boff[l];
      if (l + 1 < p.n_tc) {
        // hidden epilogue: bias, ReLU, bf16 -> next layer's operand tile
        for (int c0 = cbeg; c0 < cbeg + qw; c0 += 16) {
          uint32_t v[16];
          tmem_ld16(tmem + lane_addr + (uint32_t)c0, v);
          tmem_wait_ld();
          uint32_t pk[8];
#pragma unroll
          for (int j4 = 0; j4 < 4; ++j4) {
            const float4 b = ldg4(bias + c0 + 4 * j4);
            pk[2 * j4] = pack_bf16(fmaxf(__uint_as_float(v[4 * j4]) + b.x, 0.0f),
                                   fmaxf(__uint_as_float(v[4 * j4 + 1]) + b.y, 0.0f));
            pk[2 * j4 + 1] = pack_bf16(fmaxf(__uint_as_float(v[4 * j4 + 2]) + b.z, 0.0f),
                                       fmaxf(__uint_as_float(v[4 * j4 + 3]) + b.w, 0.0f));
          }
          st_shared_v4(A + sw128_offset(row, c0, kTileM), pk[0], pk[1], pk[2], pk[3]);
          st_shared_v4(A + sw128_offset(row, c0 + 8, kTileM), pk[4], pk[5], pk[6], pk[7]);
        }
        tc_fence_before();
        fence_async_smem();
        __syncthreads();
      } else {
        // last hidden layer: bias, ReLU, bf16 rounding, then the width-1 output layer
        const float* wl = params + a.w_last_off;
        float sacc = 0.0f;
        for (int c0 = cbeg; c0 < cbeg + qw; c0 += 16) {
          uint32_t v[16];
          tmem_ld16(tmem + lane_addr + (uint32_t)c0, v);
          tmem_wait_ld();
#pragma unroll
          for (int j4 = 0; j4 < 4; ++j4) {
            const float4 b = ldg4(bias + c0 + 4 * j4);
            const float4 w = ldg4(wl + c0 + 4 * j4);
            const __nv_bfloat162 lo = __floats2bfloat162_rn(fmaxf(__uint_as_float(v[4 * j4]) + b.x, 0.0f),
                                                            fmaxf(__uint_as_float(v[4 * j4 + 1]) + b.y, 0.0f));
            const __nv_bfloat162 hi = __floats2bfloat162_rn(fmaxf(__uint_as_float(v[4 * j4 + 2]) + b.z, 0.0f),
                                                            fmaxf(__uint_as_float(v[4 * j4 + 3]) + b.w, 0.0f));
            sacc = fmaf(__low2float(lo), w.x, sacc);
            sacc = fmaf(__high2float(lo), w.y, sacc);
            sacc = fmaf(__low2float(hi), w.z, sacc);
            sacc = fmaf(__high2float(hi), w.w, sacc);
          }
        }
        part[cq * kTileM + row] = sacc;
        tc_fence_before();
        __syncthreads();
        if (tid < kTileM) {
          const int64_t g = row0 + tid;
          if (g < a.rows)
            a.scores[g] = ((part[tid] + part[kTileM + tid]) + (part[2 * kTileM + tid] + part[3 * kTileM + tid])) +
                          __ldg(params + a.p.b_last_off);
        }
        __syncthreads();
      }
      if (*abort_flag) break;
    }
    if (*abort_flag) break;
  }
  __syncthreads();
  // streaming copies still in flight (only after an abort): wait for them, bounded
  if (tid == 0 && !p.resident) {
    for (int64_t gq = g_load - 1; gq >= 0 && gq >= g_load - p.stages; --gq)
      mbar_wait(&full[gq % p.stages], (uint32_t)((gq / p.stages) & 1));
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, p.tmem_cols);
}

// ---------------------------------------------------------------------------
// Output-layer partial of 16 columns: the fp32 pair accumulator gains
// bf16(relu(z_c)) * w_c for the even and odd columns (w_c bf16, 8 per uint4).
__device__ __forceinline__ uint64_t out_dot16(const uint32_t (&v)[16], uint4 w0, uint4 w1, uint64_t acc) {
  const uint32_t wp[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
  float lo = __uint_as_float((uint32_t)acc), hi = __uint_as_float((uint32_t)(acc >> 32));
#pragma unroll
  for (int j = 0; j < 8; ++j)
    fma2_bf16_f32(cvt_relu_bf16x2(((uint64_t)v[2 * j + 1] << 32) | v[2 * j]), wp[j], lo, hi);
  return f2pack(lo, hi);
}

// Shared-memory loads as ordered asm: they stay below the tensor-memory
// loads and waits that precede them in the source, so the compiler does not
// hoist a whole epilogue's weights and biases into registers at once.
__device__ __forceinline__ uint4 lds_u4(const void* p) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(smem_u32(p)));
  return v;
}

// Pipelined variant for predictors with two hidden layers whose weights stay
// resident (widths <= 256), one persistent CTA per SM over 128-row tiles of
// the feature image.  Layer-1 activations go to the layer-2 MMA through a
// two-slot ring of 64-column K-blocks, so the layer-2 MMA of a tile runs while
// its layer-1 epilogue is still producing K-blocks; D1 and D2 sit in separate
// TMEM halves, so the output epilogue of tile t overlaps the layer-1 MMA and
// epilogue of tile t+1.  Each layer's accumulator starts from its bias (one
// K = 16 product), so the epilogues read no bias.
// ---------------------------------------------------------------------------
// Warp roles: 0 = MMA issuer (thread 0 also requests the weights and the
// first feature tile at the start), 1 = feature-tile loader (one bulk copy
// per later tile), 2..9 = layer-1 epilogue (E1), 10..17 = layer-2 + output
// epilogue (E2).  18 warps = at most 5 per SM sub-partition: 96 registers per
// thread at most.
constexpr int kEpiWarps = 8, kEpiThreads = kEpiWarps * 32;
constexpr int kE1Warp0 = 2, kE2Warp0 = kE1Warp0 + kEpiWarps;
constexpr int kThreadsPipe = (kE2Warp0 + kEpiWarps) * 32;  // 576
// Feature tiles in flight.  One suffices: the copy of tile t+1 starts when the
// layer-1 MMA of tile t completes and has the rest of tile t to land.
constexpr int kXB = 1;
// Barriers for the resident weight chunks (the last one takes every chunk past it).
constexpr int kWBars = 8;
__device__ __forceinline__ int wbar_of(int q) { return q < kWBars - 1 ? q : kWBars - 1; }

__global__ void __launch_bounds__(kThreadsPipe, 1) k_score_tc_pipe(const __grid_constant__ TcArgs a) {
  const bool pb = a.sel && *a.sel == 1;  // published buffer of this route
  const uint8_t* __restrict__ img = pb ? a.img1 : a.img0;
  const float* __restrict__ params = pb ? a.params1 : a.params0;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const TcPlan& p = a.p;
  const int H1 = p.out[0], H2 = p.out[1];
  const int nk0 = p.in_pad[0] / 64;       // K-blocks of layer 1 (feature tile)
  const int nk1 = H1 / 64;                // K-blocks of layer 2 (= 64-column blocks of D1)
  const int xbytes = nk0 * kTileM * 128;  // one feature tile
  uint8_t* W = smem;                                            // resident weight chunks
  uint8_t* X = W + (size_t)p.chunks * p.chunk_bytes;            // [kXB] feature tiles
  uint8_t* AR = X + kXB * (size_t)xbytes;                       // [2] activation K-blocks (16 KB)
  // biases as one K = 16 product per layer, D = ONE Bl^T ahead of the K-blocks:
  // ONE [128 x 16] has ones in columns 0..2 (all row groups read the same 8
  // rows: stride 0), Bl [256 x 16] holds the three bf16 terms hi + mid + lo
  // of each fp32 bias (their sum is the bias exactly)
  uint8_t* ONE = AR + 2 * kTileM * 128;                         // 256 B, no swizzle
  uint8_t* B1 = ONE + 8 * 32;                                   // 8 KB, no swizzle
  uint8_t* B2 = B1 + 256 * 32;                                  // 8 KB, no swizzle
  float* part = reinterpret_cast<float*>(B2 + 256 * 32);        // [2][128]
  uint16_t* sw3 = reinterpret_cast<uint16_t*>(part + 2 * kTileM);  // [256] bf16 output-layer weights
  uint64_t* bars = reinterpret_cast<uint64_t*>(sw3 + 256);
  uint64_t* x_full = bars;       // [2]
  uint64_t* x_empty = bars + 2;  // [2]
  uint64_t* a_full = bars + 4;   // [2]
  uint64_t* a_empty = bars + 6;  // [2]
  uint64_t* d1_full = bars + 8;
  uint64_t* d1_empty = bars + 9;
  uint64_t* d2_full = bars + 10;
  uint64_t* d2_empty = bars + 11;
  uint64_t* w_full = bars + 12;  // [kWBars]: weight chunk q lands on barrier min(q, kWBars - 1)
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 12 + kWBars);
  int* abort_flag = reinterpret_cast<int*>(tmem_holder + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int my_tiles = blockIdx.x < a.n_tiles ? (a.n_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  if (tid == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&x_full[b], 1);  // only the first kXB are used
      mbar_init(&x_empty[b], 1);
      mbar_init(&a_full[b], kEpiWarps);
      mbar_init(&a_empty[b], 1);
    }
    mbar_init(d1_full, 1);
    mbar_init(d1_empty, kEpiWarps);
    mbar_init(d2_full, 1);
    mbar_init(d2_empty, kEpiWarps);
    for (int b = 0; b < kWBars; ++b) mbar_init(&w_full[b], 1);
    *abort_flag = 0;
    fence_mbar_init();
    if (my_tiles > 0) {
      // the weight image is requested before anything else, so that it lands
      // during the prologue: the K-blocks of layer 1 (H1 x 128 B each), then
      // those of layer 2 (H2 x 128 B each), one resident chunk and barrier
      // each, so that tile 0's K-block kb waits only for its own chunk
      // (offsets from the widths, not from indexed tables)
      const int64_t l1_bytes = (int64_t)nk0 * H1 * 128;
      for (int q = 0; q < nk0 + nk1; ++q) {
        const uint32_t len = (uint32_t)(q < nk0 ? H1 : H2) * 128u;
        const int64_t off = q < nk0 ? (int64_t)q * H1 * 128 : l1_bytes + (int64_t)(q - nk0) * H2 * 128;
        mbar_expect_tx(&w_full[wbar_of(q)], len);
        bulk_g2s(W + (size_t)q * p.chunk_bytes, img + off, len, &w_full[wbar_of(q)]);
      }
      for (int b = 0; b < kWBars; ++b) mbar_arrive(&w_full[b]);  // a barrier without chunks completes here
    }
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, 512);
    tmem_relinquish();
  }
  for (int k = tid; k < H2; k += blockDim.x) sw3[k] = bf16_bits(__ldg(params + a.w_last_off + k));
  for (int e = tid; e < 8 * 2; e += blockDim.x) {  // 16-byte chunks: row e / 2, K half e % 2
    const uint4 q = (e & 1) ? make_uint4(0u, 0u, 0u, 0u) : make_uint4(0x3F803F80u, 0x3F80u, 0u, 0u);
    *reinterpret_cast<uint4*>(ONE + nosw16_offset(e >> 1, 8 * (e & 1))) = q;
  }
  for (int e = tid; e < 2 * 256 * 2; e += blockDim.x) {  // layer (e / 512), row n, K half
    const int l = e >> 9, n = (e >> 1) & 255;
    uint4 q = make_uint4(0u, 0u, 0u, 0u);
    if (!(e & 1) && n < (l ? H2 : H1)) {
      const float b = __ldg(params + a.boff[l] + n);
      const uint16_t hi = bf16_bits(b);
      uint16_t mid = 0, lo = 0;
      if (!isinf(b)) {  // b - hi and (b - hi) - mid are exact in fp32; lo holds the last 8 bits
        const float r1 = b - __uint_as_float((uint32_t)hi << 16);
        mid = bf16_bits(r1);
        lo = bf16_bits(r1 - __uint_as_float((uint32_t)mid << 16));
      }
      q.x = (uint32_t)hi | ((uint32_t)mid << 16);
      q.y = lo;
    }
    *reinterpret_cast<uint4*>((l ? B2 : B1) + nosw16_offset(n, 8 * (e & 1))) = q;
  }
  fence_async_smem();  // the bias operands are read by the tensor cores (async proxy)
  // everything above reads only the published weights; the feature tiles come
  // from the previous kernel of the stream
  pdl_wait();
  pdl_trigger();
  if (tid == 0 && my_tiles > 0) {
    mbar_arrive_expect_tx(&x_full[0], (uint32_t)xbytes);
    bulk_g2s(X, a.ximg + (int64_t)blockIdx.x * xbytes, (uint32_t)xbytes, &x_full[0]);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t D1 = tmem, D2 = tmem + 256;

  if (warp == 0) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && my_tiles > 0) {
      bool ok = true, x0_used = false;
      const uint32_t id1 = idesc_bf16_f32(kTileM, H1), id2 = idesc_bf16_f32(kTileM, H2);
      for (int t = 0; t < my_tiles && ok; ++t) {
        const int xb = t % kXB;
        ok = mbar_wait(&x_full[xb], (uint32_t)((t / kXB) & 1));
        x0_used = x0_used || ok;
        if (ok && t >= 1) ok = mbar_wait(d1_empty, (uint32_t)((t - 1) & 1));
        for (int kb = 0; ok && t == 0 && kb < nk0; ++kb) ok = mbar_wait(&w_full[wbar_of(kb)], 0);
        if (!ok) break;
        tc_fence_after();
        const uint32_t xa = smem_u32(X + (size_t)xb * xbytes);
        umma_bf16(D1, sdesc_nosw(smem_u32(ONE), 128, 0), sdesc_nosw(smem_u32(B1), 128, 256), id1, 0u);
        for (int kb = 0; kb < nk0; ++kb)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            umma_bf16(D1, sdesc_sw128(xa + (uint32_t)kb * kTileM * 128u + 32u * j),
                      sdesc_sw128(smem_u32(W + (size_t)kb * p.chunk_bytes) + 32u * j), id1, 1u);
        umma_commit(&x_empty[xb]);
        umma_commit(d1_full);
        if (t >= 1 && !mbar_wait(d2_empty, (uint32_t)((t - 1) & 1))) { ok = false; break; }
        tc_fence_after();
        umma_bf16(D2, sdesc_nosw(smem_u32(ONE), 128, 0), sdesc_nosw(smem_u32(B2), 128, 256), id2, 0u);
        for (int kb = 0; kb < nk1 && ok; ++kb) {
          const int64_t kq = (int64_t)t * nk1 + kb;
          const int slot = (int)(kq & 1);
          ok = mbar_wait(&a_full[slot], (uint32_t)((kq >> 1) & 1));
          if (ok && t == 0) ok = mbar_wait(&w_full[wbar_of(nk0 + kb)], 0);
          if (!ok) break;
          tc_fence_after();
          const uint32_t aa = smem_u32(AR + (size_t)slot * kTileM * 128);
          const uint32_t bb = smem_u32(W + (size_t)(nk0 + kb) * p.chunk_bytes);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            umma_bf16(D2, sdesc_sw128(aa + 32u * j), sdesc_sw128(bb + 32u * j), id2, 1u);
          umma_commit(&a_empty[slot]);
        }
        umma_commit(d2_full);
      }
      if (!ok) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
      }
      // copies issued at the start and still in flight land in this CTA's
      // shared memory: wait for them (bounded) before the CTA can exit
      for (int b = 0; b < kWBars; ++b) mbar_wait(&w_full[b], 0);
      if (!x0_used) mbar_wait(&x_full[0], 0);
    }
    __syncwarp();
  } else if (warp < kE1Warp0) {
    // ------------------------------------------------------------ feature-tile loader
    if (lane == 0) {
      int last[2] = {-1, -1};
      for (int t = 1; t < my_tiles; ++t) {  // tile 0 was requested by thread 0
        const int xb = t % kXB;
        if (t >= kXB && !mbar_wait(&x_empty[xb], (uint32_t)(((t - kXB) / kXB) & 1))) {
          *abort_flag = 1;
          latch_error(a.err, LS_ERR_TIMEOUT);
          break;
        }
        if (*reinterpret_cast<volatile int*>(abort_flag)) break;
        const int64_t tile = blockIdx.x + (int64_t)t * gridDim.x;
        mbar_arrive_expect_tx(&x_full[xb], (uint32_t)xbytes);
        bulk_g2s(X + (size_t)xb * xbytes, a.ximg + tile * xbytes, (uint32_t)xbytes, &x_full[xb]);
        last[xb] = t;
      }
      // copies still in flight land in this CTA's shared memory: wait for them
      // (bounded) before the CTA can exit
      for (int b = 0; b < kXB; ++b)
        if (last[b] >= 0) mbar_wait(&x_full[b], (uint32_t)((last[b] / kXB) & 1));
    }
    __syncwarp();
  } else if (warp < kE2Warp0) {
    // ------------------------------------------------------------ E1: layer-1 epilogue
    const int ew = warp - kE1Warp0;        // 0..7
    const int q4 = warp & 3;               // TMEM lane quadrant
    const int wk = ew >> 2;                // which 32 columns of each 64-column K-block
    const int row = 32 * q4 + lane;
    const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;
    for (int t = 0; t < my_tiles; ++t) {
      if (!mbar_wait(d1_full, (uint32_t)(t & 1))) { *abort_flag = 1; latch_error(a.err, LS_ERR_TIMEOUT); break; }
      tc_fence_after();
      bool ok = true;
      for (int kb = 0; kb < nk1; ++kb) {
        const int64_t kq = (int64_t)t * nk1 + kb;
        const int slot = (int)(kq & 1);
        const int colb = 64 * kb + 32 * wk;
        uint32_t v[2][16];  // D1 already holds z + b1
        tmem_ld16(D1 + lane_addr + (uint32_t)colb, v[0]);
        tmem_ld16(D1 + lane_addr + (uint32_t)(colb + 16), v[1]);
        tmem_wait_ld();
        if (kq >= 2 && !mbar_wait(&a_empty[slot], (uint32_t)(((kq - 2) >> 1) & 1))) { ok = false; break; }
        uint8_t* dst = AR + (size_t)slot * kTileM * 128;
#pragma unroll
        for (int g = 0; g < 2; ++g) {
          uint32_t pk[8];
#pragma unroll
          for (int j = 0; j < 8; ++j)
            pk[j] = cvt_relu_bf16x2(((uint64_t)v[g][2 * j + 1] << 32) | v[g][2 * j]);
          const int kcol = 32 * wk + 16 * g;  // column inside the K-block
          st_shared_v4(dst + sw128_offset(row, kcol, kTileM), pk[0], pk[1], pk[2], pk[3]);
          st_shared_v4(dst + sw128_offset(row, kcol + 8, kTileM), pk[4], pk[5], pk[6], pk[7]);
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&a_full[slot]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(d1_empty);
      if (!ok) { *abort_flag = 1; latch_error(a.err, LS_ERR_TIMEOUT); break; }
      if (*abort_flag) break;
    }
  } else {
    // ------------------------------------------------------------ E2: layer-2 epilogue + output layer
    const int ew = warp - kE2Warp0;        // 0..7
    const int q4 = warp & 3;
    const int wk = ew >> 2;                // column half of D2
    const int row = 32 * q4 + lane;
    const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;
    const float b3 = __ldg(params + p.b_last_off);
    const int half = H2 / 2;
    for (int t = 0; t < my_tiles; ++t) {
      const int64_t row0 = (int64_t)(blockIdx.x + (int64_t)t * gridDim.x) * kTileM;
      const bool ok2 = mbar_wait(d2_full, (uint32_t)(t & 1));
      tc_fence_after();
      uint64_t acc2 = 0;
      if (ok2) {
        // D2 already holds z + b2: two 16-column loads in flight, one consumed
        // while the next lands
        const uint32_t base = D2 + lane_addr;
        const int cb = wk * half, ce = cb + half;  // half is a multiple of 32
        uint32_t va[16], vb[16];
        tmem_ld16(base + (uint32_t)cb, va);
        for (int c0 = cb; c0 < ce; c0 += 32) {
          uint4 w0 = *reinterpret_cast<const uint4*>(sw3 + c0);
          uint4 w1 = *reinterpret_cast<const uint4*>(sw3 + c0 + 8);
          tmem_wait_ld_regs(va);
          tmem_ld16(base + (uint32_t)(c0 + 16), vb);
          acc2 = out_dot16(va, w0, w1, acc2);
          w0 = *reinterpret_cast<const uint4*>(sw3 + c0 + 16);
          w1 = *reinterpret_cast<const uint4*>(sw3 + c0 + 24);
          tmem_wait_ld_regs(vb);
          if (c0 + 32 < ce) tmem_ld16(base + (uint32_t)(c0 + 32), va);
          acc2 = out_dot16(vb, w0, w1, acc2);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(d2_empty);
      float* pt = part + (t & 1) * kTileM;  // double-buffered by tile parity
      if (wk == 1) pt[row] = __uint_as_float((uint32_t)acc2) + __uint_as_float((uint32_t)(acc2 >> 32));
      // all E2 warps continue, or all stop (a timeout here or elsewhere)
      if (!named_bar_and(1, kEpiThreads, ok2 && !*reinterpret_cast<volatile int*>(abort_flag))) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
        break;
      }
      if (wk == 0) {
        const int64_t g = row0 + row;
        const float mine = __uint_as_float((uint32_t)acc2) + __uint_as_float((uint32_t)(acc2 >> 32));
        const float yhat = (mine + pt[row]) + b3;
        if (g < a.rows && a.scores) a.scores[g] = yhat;
        if (a.fuse_argmin) {
          // n_inst divides 32 and tiles start at request boundaries: the
          // request's scores sit in n_inst consecutive lanes; lexicographic
          // (score, index) minimum, NaN last (Algorithm 4, greedy selection)
          const int n = a.n_inst;
          float bv = yhat;
          int bi = g < a.rows ? (lane & (n - 1)) : -1;
          for (int o = 1; o < n; o <<= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            const bool an = isnan(ov), bn = isnan(bv);
            const bool first = an != bn ? bn : (!an && ov != bv ? ov < bv : oi < bi);
            if (oi >= 0 && (bi < 0 || first)) { bv = ov; bi = oi; }
          }
          if ((lane & (n - 1)) == 0 && g < a.rows) {
            const int64_t r = g / n;
            a.choice[r] = bi;
            a.best[r] = bv;
          }
        }
      }
    }
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// Wide variant: two hidden layers whose widths are multiples of 128 (<= 512),
// weights streamed from L2 (they do not fit in shared memory), one persistent
// CTA per SM over 128-row tiles.  A job is one 128-column slice of a layer's
// output: its bias product (ones x three-term bias operand, as in the
// pipelined kernel), then its K-blocks, each a 16 KB [128 x 64] slice of the
// published weight image, whose 128-row N-chunks put the slices of a tile in
// the order they are consumed; a stage of the ring is Q consecutive slices
// brought by one bulk copy.  Layer-1 jobs read the feature tile from shared
// memory; their epilogue packs relu(z) to bf16 pairs and stores them in
// tensor memory, where the layer-2 jobs read them as the A operand -- so the
// 128 x H1 activation tile needs no shared memory and the layer-2 products
// read only their weights from it.  Accumulators alternate between two
// 128-column TMEM slots, so the epilogue of one job overlaps the next job's
// products.
// TMEM (512 columns): [0, 256) packed layer-1 activations, [256, 384) and
// [384, 512) the two slots.
// Warp roles (14 warps): 0 = MMA issuer (lane 0) and TMEM owner,
// 1 = weight producer (lane 0, one bulk copy per 16 KB slice into a ring of
// stages), 2..5 = feature-tile builders (template rows + pair chunk, as
// build_tile), 6..13 = epilogue: two warps per TMEM lane quadrant, each 64
// of a job's 128 columns.
// ---------------------------------------------------------------------------
constexpr int kWideBuild = 4, kWideEpi = 8;
constexpr int kWideBuild0 = 2, kWideEpi0 = kWideBuild0 + kWideBuild;
constexpr int kThreadsWide = (kWideEpi0 + kWideEpi) * 32;  // 448
constexpr int kWideChunk = kTileM * 128;                    // [128 N x 64 K] bf16 = 16 KB
constexpr uint32_t kSlot0 = 256;                             // TMEM column of accumulator slot 0

__global__ void __launch_bounds__(kThreadsWide, 1) k_score_wide(const __grid_constant__ TcArgs a) {
  const bool pb = a.sel && *a.sel == 1;  // published buffer of this route
  const uint8_t* __restrict__ img = pb ? a.img1 : a.img0;
  const float* __restrict__ params = pb ? a.params1 : a.params0;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const TcPlan& p = a.p;
  const int H1 = p.out[0], H2 = p.out[1];
  const int J1 = H1 / 128, J2 = H2 / 128;
  const int nk0 = p.in_pad[0] / 64, nk1 = H1 / 64;
  const int per_tile = J1 * nk0 + J2 * nk1;
  const int S = p.wide_stages, Q = p.wide_q;  // stages of Q slices each
  uint8_t* X = smem;                                              // [nk0] feature-tile K-blocks
  uint8_t* ring = X + (size_t)nk0 * kWideChunk;                   // [S][Q] weight slices
  uint8_t* ONE = ring + (size_t)S * Q * kWideChunk;               // 256 B, no swizzle
  uint8_t* BIAS = ONE + 256;                                      // [H1 + H2 rows x 16] no swizzle
  uint16_t* sw3 = reinterpret_cast<uint16_t*>(BIAS + (size_t)(H1 + H2) * 32);  // [H2] bf16
  float* part = reinterpret_cast<float*>(sw3 + H2);               // [2 tiles][2 halves][128]
  uint64_t* bars = reinterpret_cast<uint64_t*>(part + 4 * kTileM);
  uint64_t* full = bars;            // [S]
  uint64_t* empty = full + S;       // [S]
  uint64_t* x_full = empty + S;
  uint64_t* x_empty = x_full + 1;
  uint64_t* s_full = x_empty + 1;   // [2]
  uint64_t* s_empty = s_full + 2;   // [2]
  uint64_t* h1_ready = s_empty + 2;
  uint64_t* h1_free = h1_ready + 1;
  uint64_t* done = h1_free + 1;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int my_tiles = blockIdx.x < a.n_tiles ? (a.n_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  if (tid == 0) {
    for (int q = 0; q < S; ++q) {
      mbar_init(&full[q], 1);
      mbar_init(&empty[q], 1);
    }
    mbar_init(x_full, kWideBuild);
    mbar_init(x_empty, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_empty[b], kWideEpi);
    }
    mbar_init(h1_ready, kWideEpi * J1);
    mbar_init(h1_free, 1);
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, 512);
    tmem_relinquish();
  }
  // bias operands (three exact bf16 terms of each fp32 bias), the ones
  // operand and the bf16 output-layer weights, from the published parameters
  for (int k = tid; k < H2; k += blockDim.x) sw3[k] = bf16_bits(__ldg(params + a.w_last_off + k));
  for (int e = tid; e < 8 * 2; e += blockDim.x) {  // 16-byte chunks: row e / 2, K half e % 2
    const uint4 q = (e & 1) ? make_uint4(0u, 0u, 0u, 0u) : make_uint4(0x3F803F80u, 0x3F80u, 0u, 0u);
    *reinterpret_cast<uint4*>(ONE + nosw16_offset(e >> 1, 8 * (e & 1))) = q;
  }
  for (int e = tid; e < (H1 + H2) * 2; e += blockDim.x) {  // row n of [H1 | H2], K half e % 2
    const int n = e >> 1, l = n >= H1 ? 1 : 0, o = n - (l ? H1 : 0);
    uint4 q = make_uint4(0u, 0u, 0u, 0u);
    if (!(e & 1)) {
      const float b = __ldg(params + a.boff[l] + o);
      const uint16_t hi = bf16_bits(b);
      uint16_t mid = 0, lo = 0;
      if (!isinf(b)) {  // b - hi and (b - hi) - mid are exact in fp32; lo holds the last 8 bits
        const float r1 = b - __uint_as_float((uint32_t)hi << 16);
        mid = bf16_bits(r1);
        lo = bf16_bits(r1 - __uint_as_float((uint32_t)mid << 16));
      }
      q.x = (uint32_t)hi | ((uint32_t)mid << 16);
      q.y = lo;
    }
    *reinterpret_cast<uint4*>(BIAS + nosw16_offset(n, 8 * (e & 1))) = q;
  }
  fence_async_smem();  // the bias operands are read by the tensor cores (async proxy)
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t idesc = idesc_bf16_f32(kTileM, 128);

  if (warp == 0) {
    // ------------------------------------------------------------ MMA issuer
    // The tensor core's instruction queue is short: products must follow one
    // another with little scalar work between them, so this loop keeps plain
    // counters (stage, slice within the stage, slot), a parity bit per stage
    // and descriptors formed by addition (a shared-memory descriptor's address
    // field is the byte address / 16).
    if (lane == 0 && my_tiles > 0) {
      bool ok = true;
      int st = 0, part = 0;      // ring stage and slice within it
      uint32_t fpar = 0;         // bit s: parity of the next wait on full[s]
      uint32_t jslot = 0;        // jobs issued so far (slot = jslot & 1)
      const uint64_t ring_desc = sdesc_sw128(smem_u32(ring));
      const uint64_t one_desc = sdesc_nosw(smem_u32(ONE), 128, 0);
      const uint64_t bias_desc = sdesc_nosw(smem_u32(BIAS), 128, 256);
      const uint64_t x_desc = sdesc_sw128(smem_u32(X));
      for (int t = 0; t < my_tiles && ok; ++t) {
        ok = mbar_wait(x_full, (uint32_t)(t & 1));
        if (!ok) break;
        tc_fence_after();
        for (int j = 0; j < J1 + J2 && ok; ++j, ++jslot) {
          const bool l2 = j >= J1;
          if (j == J1) {
            umma_commit(x_empty);  // the feature tile is free once the layer-1 products are done
            ok = mbar_wait(h1_ready, (uint32_t)(t & 1));  // every layer-1 slice packed into TMEM
            if (!ok) break;
            tc_fence_after();
          }
          // the slot's previous epilogue has drained it
          const uint32_t slot = jslot & 1u;
          if (jslot >= 2 && !(ok = mbar_wait(&s_empty[slot], ((jslot >> 1) - 1) & 1u))) break;
          tc_fence_after();
          const uint32_t d = tmem + kSlot0 + 128u * slot;
          const int bias_row = l2 ? H1 + (j - J1) * 128 : j * 128;
          umma_bf16(d, one_desc, bias_desc + (uint64_t)(bias_row * 32 / 16), idesc, 0u);
          const int nk = l2 ? nk1 : nk0;
          for (int kb = 0; kb < nk; ++kb) {
            if (part == 0) {  // a new stage: wait for its copy
              if (!(ok = mbar_wait(&full[st], (fpar >> st) & 1u))) break;
              fpar ^= 1u << st;
              tc_fence_after();
            }
            const uint64_t bd = ring_desc + (uint64_t)((st * Q + part) * (kWideChunk / 16));
            if (l2) {
              const uint32_t a0 = tmem + (uint32_t)(32 * kb);
#pragma unroll
              for (int k = 0; k < 4; ++k) umma_bf16_ts(d, a0 + 8u * k, bd + 2u * k, idesc, 1u);
            } else {
              const uint64_t xd = x_desc + (uint64_t)(kb * (kWideChunk / 16));
#pragma unroll
              for (int k = 0; k < 4; ++k) umma_bf16(d, xd + 2u * k, bd + 2u * k, idesc, 1u);
            }
            if (++part == Q) {  // the stage is free once these products complete
              umma_commit(&empty[st]);
              part = 0;
              st = st + 1 == S ? 0 : st + 1;
            }
          }
          if (ok) umma_commit(&s_full[slot]);
        }
        if (ok) umma_commit(h1_free);  // the packed activations may be overwritten
      }
      if (!ok) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
      }
      umma_commit(done);  // every product issued has completed before TMEM is freed
      mbar_wait(done, 0);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ weight producer
    // The image holds the per-tile stream of slices contiguously (128-row
    // N-chunks, layer 1 then layer 2), so a stage of Q consecutive slices is
    // one bulk copy: large copies reach several times the rate of 16 KB ones.
    if (lane == 0 && my_tiles > 0) {
      const int64_t stages = (int64_t)my_tiles * per_tile / Q;
      const uint32_t bytes = (uint32_t)(Q * kWideChunk);
      int64_t G = 0;
      bool ok = true;
      for (; G < stages; ++G) {
        const int s = (int)(G % S);
        const int64_t u = G / S;
        if (u >= 1 && !(ok = mbar_wait(&empty[s], (uint32_t)((u - 1) & 1)))) break;
        if (*abort_flag) { ok = false; break; }
        const int q0 = (int)((G * Q) % per_tile);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_g2s(ring + (size_t)s * Q * kWideChunk, img + (int64_t)q0 * kWideChunk, bytes, &full[s]);
      }
      if (!ok) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
      }
      // stages issued and never consumed (only after an abort) land in this
      // CTA's shared memory: wait for them (bounded) before the CTA can exit
      for (int64_t h = G - 1; h >= 0 && h >= G - S; --h) mbar_wait(&full[h % S], (uint32_t)((h / S) & 1));
    }
    __syncwarp();
  } else if (warp < kWideEpi0) {
    // ------------------------------------------------------------ feature-tile builders
    const int bt = tid - kWideBuild0 * 32;
    pdl_wait();  // pair chunks and template rows from the previous kernel of the stream
    for (int t = 0; t < my_tiles; ++t) {
      if (t >= 1 && !mbar_wait(x_empty, (uint32_t)((t - 1) & 1))) {
        *abort_flag = 1;
        latch_error(a.err, LS_ERR_TIMEOUT);
        break;
      }
      if (*abort_flag) break;
      const int64_t row0 = (int64_t)(blockIdx.x + (int64_t)t * gridDim.x) * kTileM;
      build_tile<4>(a, X, row0, bt, kWideBuild * 32);
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(x_full);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kWideEpi0;       // 0..7
    const int q4 = warp & 3;               // TMEM lane quadrant
    const int h = ew >> 2;                 // which 64 of a job's 128 columns
    const int row = 32 * q4 + lane;
    const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;
    int64_t jg = 0;
    bool ok = true;
    for (int t = 0; t < my_tiles; ++t) {
      uint64_t acc = 0;  // output-layer partial, two fp32 lanes
      for (int c = 0; c < J1; ++c, ++jg) {
        const int slot = (int)(jg & 1);
        bool go = ok && !*abort_flag;
        if (go) go = mbar_wait(&s_full[slot], (uint32_t)((jg >> 1) & 1));
        if (go && c == 0 && t >= 1) go = mbar_wait(h1_free, (uint32_t)((t - 1) & 1));
        go = __all_sync(0xffffffffu, go);  // the tensor-memory accesses below are warp-wide
        if (!go) {
          ok = false;
          *abort_flag = 1;
        }
        if (go) {
          tc_fence_after();
          const uint32_t src = tmem + lane_addr + kSlot0 + 128u * (uint32_t)slot + 64u * (uint32_t)h;
          uint32_t v[4][16];
#pragma unroll
          for (int i = 0; i < 4; ++i) tmem_ld16(src + 16u * i, v[i]);
          tmem_wait_ld();
          uint32_t pk[32];
#pragma unroll
          for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j)
              pk[8 * i + j] = cvt_relu_bf16x2(((uint64_t)v[i][2 * j + 1] << 32) | v[i][2 * j]);
          tmem_st32(tmem + lane_addr + (uint32_t)(64 * c + 32 * h), pk);
          tmem_wait_st();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&s_empty[slot]);
          mbar_arrive(h1_ready);
        }
      }
      for (int n = 0; n < J2; ++n, ++jg) {
        const int slot = (int)(jg & 1);
        bool go = ok && !*abort_flag;
        if (go) go = mbar_wait(&s_full[slot], (uint32_t)((jg >> 1) & 1));
        go = __all_sync(0xffffffffu, go);
        if (!go) {
          ok = false;
          *abort_flag = 1;
        }
        if (go) {
          tc_fence_after();
          const uint32_t src = tmem + lane_addr + kSlot0 + 128u * (uint32_t)slot + 64u * (uint32_t)h;
          const uint4* w = reinterpret_cast<const uint4*>(sw3 + 128 * n + 64 * h);
          uint32_t va[16], vb[16];
          tmem_ld16(src, va);
#pragma unroll
          for (int i = 0; i < 4; i += 2) {
            tmem_wait_ld_regs(va);
            tmem_ld16(src + 16u * (i + 1), vb);
            acc = out_dot16(va, w[2 * i], w[2 * i + 1], acc);
            tmem_wait_ld_regs(vb);
            if (i + 2 < 4) tmem_ld16(src + 16u * (i + 2), va);
            acc = out_dot16(vb, w[2 * i + 2], w[2 * i + 3], acc);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_empty[slot]);
      }
      float* pt = part + (t & 1) * 2 * kTileM;
      pt[h * kTileM + row] = __uint_as_float((uint32_t)acc) + __uint_as_float((uint32_t)(acc >> 32));
      // the two halves of every row meet here; a stop is decided together
      if (!named_bar_and(1, kWideEpi * 32, ok)) break;
      if (h == 0) {
        const int64_t g = (int64_t)(blockIdx.x + (int64_t)t * gridDim.x) * kTileM + row;
        if (g < a.rows) a.scores[g] = (pt[row] + pt[kTileM + row]) + __ldg(params + p.b_last_off);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

// 16 loaded accumulator columns (the bias already in them) -> 8 packed bf16
// words relu(bf16(D)) at o[OFF..)
template <int OFF>
__device__ __forceinline__ void pack16_relu(const uint32_t (&v)[16], uint32_t (&o)[32]) {
#pragma unroll
  for (int j = 0; j < 8; ++j) o[OFF + j] = cvt_relu_bf16x2(((uint64_t)v[2 * j + 1] << 32) | v[2 * j]);
}
// 32 consecutive accumulator columns of the warp's lanes -> 16 packed words at
// o[OFF..OFF + 16).
template <int OFF>
__device__ __forceinline__ void pack32_relu(uint32_t taddr, uint32_t (&o)[32]) {
  uint32_t va[16], vb[16];
  tmem_ld16(taddr, va);
  tmem_ld16(taddr + 16u, vb);
  tmem_wait_ld_regs(va);
  pack16_relu<OFF>(va, o);
  tmem_wait_ld_regs(vb);
  pack16_relu<OFF + 8>(vb, o);
}
// 64 columns -> 32 packed words (o[0..32)); each 16-column load overlaps the
// packing of the one before.  Every column has been read when this returns.
__device__ __forceinline__ void pack64_relu(uint32_t taddr, uint32_t (&o)[32]) {
  uint32_t va[16], vb[16];
  tmem_ld16(taddr, va);
  tmem_wait_ld_regs(va);
  tmem_ld16(taddr + 16u, vb);
  pack16_relu<0>(va, o);
  tmem_wait_ld_regs(vb);
  tmem_ld16(taddr + 32u, va);
  pack16_relu<8>(vb, o);
  tmem_wait_ld_regs(va);
  tmem_ld16(taddr + 48u, vb);
  pack16_relu<16>(va, o);
  tmem_wait_ld_regs(vb);
  pack16_relu<24>(vb, o);
}
// Output-layer partial of 16 columns whose accumulators hold the bias: the
// fp32 pair accumulator (even columns low, odd columns high) gains
// bf16(relu(z_c)) * w_c, w the 16 bf16 output weights in shared memory.
__device__ __forceinline__ uint64_t out_dot16_wb(const uint32_t (&v)[16], const uint16_t* w, uint64_t acc) {
  float lo = __uint_as_float((uint32_t)acc), hi = __uint_as_float((uint32_t)(acc >> 32));
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const uint4 ww = lds_u4(w + 8 * q);
    const uint32_t wp[4] = {ww.x, ww.y, ww.z, ww.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = 4 * q + u;
      fma2_bf16_f32(cvt_relu_bf16x2(((uint64_t)v[2 * j + 1] << 32) | v[2 * j]), wp[u], lo, hi);
    }
  }
  return f2pack(lo, hi);
}

// ---------------------------------------------------------------------------
// Pair variant: the wide kernel's job for hidden widths that are multiples of
// 256, on a cluster of two CTAs (one TPC) whose tensor cores run 2-SM
// products (M = 256): CTA r builds and owns tile 2p + r of tile pair p, rows
// 0..127 of every product are CTA 0's tile and 128..255 CTA 1's.  Jobs are
// 256 output columns; the B operand of a job is split by rows, CTA r holding
// rows 128 r .. 128 r + 127 (its half-slices of 16 KB, streamed from its
// rank's part of the image).  Per SM this halves the weight bytes of the
// one-CTA wide kernel, whose per-SM copy rate bounded it.  256-column jobs
// keep the products long: each tcgen05 commit of a CTA pair stalls the
// product queue for a while, so a pair kernel wants few commits per product.
// TMEM, 512 columns in each CTA: the packed bf16 layer-1 activations H1 in
// columns [0, H1 / 2); the accumulator D0 = columns 0..255 for layer-1 job 0,
// compacted in place into H1 by its epilogue; D1 = columns 256..511 for
// layer-1 job 1 and every layer-2 job, released by the epilogue as soon as it
// has been read.  Each job's accumulator starts from its bias (one K = 16
// product), and the epilogues convert with one ReLU-and-round instruction per
// column pair: draining the single accumulator is the critical path.  With
// three hidden layers of 256 (kThree) the second layer is compaction job 1,
// its A operand H1 and its result packed into columns 128..255 (H2), which the
// output job reads.
// Warp roles in each CTA: 0 = MMA issuer (CTA 0) or stage relay (CTA 1), and
// the TMEM allocation; 1 = producer of this CTA's half-slices; 2..7 = feature
// tile builders; 8..15 = epilogue (lane quadrant warp % 4, column half
// (warp - 8) / 4 of a job's 256).  Barriers the issuer waits on count arrivals
// from both CTAs and live in CTA 0 (CTA 1 arrives remotely); barriers the
// issuer signals are committed to both CTAs.
// ---------------------------------------------------------------------------
constexpr int kPairBuild = 6, kPairEpi = 8;  // builder and epilogue warps of the pair kernel
constexpr int kPairBuild0 = 2, kPairEpi0 = kPairBuild0 + kPairBuild;
constexpr int kThreadsPair = (kPairEpi0 + kPairEpi) * 32;  // 512: 128 registers a thread at launch
constexpr int kHalfSlice = kTileM * 128;                   // [128 N x 64 K] bf16 = 16 KB

// A timeout anywhere in a CTA pair stops both CTAs.
__device__ __forceinline__ void pair_stop(volatile int* abort_flag, uint32_t rank, int* err) {
  *abort_flag = 1;
  st_cluster_u32((void*)abort_flag, rank ^ 1u, 1u);
  latch_error(err, LS_ERR_TIMEOUT);
}

template <bool kThree>  // three hidden layers of 256 (else two of multiples of 256)
__global__ void __launch_bounds__(kThreadsPair, 1) k_score_pair(const __grid_constant__ TcArgs a) {
  const bool pb = a.sel && *a.sel == 1;
  const uint8_t* __restrict__ img = pb ? a.img1 : a.img0;
  const float* __restrict__ params = pb ? a.params1 : a.params0;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const TcPlan& p = a.p;
  // Jobs of a tile: J1 "compaction" jobs, whose results are rounded into
  // packed bf16 TMEM columns 0..255 (H1), then J2 output jobs.  With three
  // hidden layers (all of 256) the second layer is compaction job 1: its A
  // operand is H1 (columns 0..127) and its result goes to columns 128..255
  // (H2), which the single output job (the third layer) reads.
  constexpr bool three = kThree;
  const int H2 = three ? 256 : p.out[1];  // the last hidden layer
  const int J1 = three ? 2 : p.out[0] / 256, J2 = three ? 1 : H2 / 256;
  const int nk0 = p.in_pad[0] / 64, nk1 = three ? 4 : p.in_pad[1] / 64;
  const uint32_t out_a = three ? 128u : 0u;  // TMEM column of the output jobs' A operand
  const int nk_c1 = three ? 4 : nk0;  // K-blocks of compaction job 1
  const int per_tile = p.pair_slices;
  const int S = p.pair_stages, Q = p.pair_q;
  uint8_t* X = smem;                                                  // [nk0] feature-tile K-blocks
  uint8_t* ring = X + (size_t)nk0 * kWideChunk;                       // [S][Q] half-slices
  // Each job's accumulator starts from its bias: one K = 16 product of ONE
  // [128 x 16] (ones in columns 0..2, every row group reading the same 8
  // rows: stride 0) and this CTA's 128 rows of the job's bias operand (the
  // three bf16 terms hi + mid + lo of each fp32 bias, whose sum is the bias
  // exactly), so the epilogues read no bias.
  uint8_t* ONE = ring + (size_t)S * Q * kHalfSlice;                   // 256 B, no swizzle
  uint8_t* BIAS = ONE + 8 * 32;                                       // [J1 + J2][128 x 16], no swizzle
  uint16_t* sw3 = reinterpret_cast<uint16_t*>(BIAS + (size_t)(J1 + J2) * kTileM * 32);  // [H2] bf16
  float* part = reinterpret_cast<float*>(sw3 + H2);                   // [2 tiles][2 halves][128]
  uint64_t* full = reinterpret_cast<uint64_t*>(part + 4 * kTileM);    // [S]
  uint64_t* empty = full + S;                                         // [S]
  uint64_t* x_full = empty + S;
  uint64_t* x_empty = x_full + 1;
  uint64_t* d0_full = x_empty + 1;
  uint64_t* d1_full = d0_full + 1;
  uint64_t* d1_empty = d1_full + 1;
  uint64_t* h1_ready = d1_empty + 1;  // [2]: layer-1 job j's activations are in H1
  uint64_t* done = h1_ready + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const uint32_t rank = cluster_ctarank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int pair_id = (int)(blockIdx.x >> 1), n_pairs = (int)(gridDim.x >> 1);
  const int tile_pairs = (a.n_tiles + 1) / 2;
  const int my_pairs = pair_id < tile_pairs ? (tile_pairs - 1 - pair_id) / n_pairs + 1 : 0;
  if (tid == 0) {
    for (int q = 0; q < S; ++q) {
      mbar_init(&full[q], rank == 0 ? 2 : 1);  // CTA 0: its own copy + the relayed arrival of CTA 1's
      mbar_init(&empty[q], 1);
    }
    mbar_init(x_full, 2 * kPairBuild);
    mbar_init(x_empty, 1);
    mbar_init(d0_full, 1);
    mbar_init(d1_full, 1);
    mbar_init(d1_empty, 2 * kPairEpi);
    mbar_init(&h1_ready[0], 2 * kPairEpi);
    mbar_init(&h1_ready[1], 2 * kPairEpi);
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc_pair(tmem_holder, 512);
    tmem_relinquish_pair();
  }
  for (int k = tid; k < H2; k += blockDim.x) sw3[k] = bf16_bits(__ldg(params + a.w_last_off + k));
  for (int e = tid; e < 8 * 2; e += blockDim.x) {  // 16-byte chunks: row e / 2, K half e % 2
    const uint4 q = (e & 1) ? make_uint4(0u, 0u, 0u, 0u) : make_uint4(0x3F803F80u, 0x3F80u, 0u, 0u);
    *reinterpret_cast<uint4*>(ONE + nosw16_offset(e >> 1, 8 * (e & 1))) = q;
  }
  // job jb's operand row i: output column 256 jb' + 128 rank + i of its layer
  // (this CTA supplies those 128 columns of the job's 256)
  for (int e = tid; e < (J1 + J2) * kTileM * 2; e += blockDim.x) {
    const int jb = e / (2 * kTileM), i = (e >> 1) % kTileM;
    const int l = three ? jb : (jb < J1 ? 0 : 1);
    const int col = (three ? 0 : (jb - (l ? J1 : 0)) * 256) + (int)rank * 128 + i;
    uint4 q = make_uint4(0u, 0u, 0u, 0u);
    if (!(e & 1)) {
      const float b = __ldg(params + a.boff[l] + col);
      const uint16_t hi = bf16_bits(b);
      uint16_t mid = 0, lo = 0;
      if (!isinf(b)) {  // b - hi and (b - hi) - mid are exact in fp32; lo holds the last 8 bits
        const float r1 = b - __uint_as_float((uint32_t)hi << 16);
        mid = bf16_bits(r1);
        lo = bf16_bits(r1 - __uint_as_float((uint32_t)mid << 16));
      }
      q.x = (uint32_t)hi | ((uint32_t)mid << 16);
      q.y = lo;
    }
    *reinterpret_cast<uint4*>(BIAS + (size_t)jb * kTileM * 32 + nosw16_offset(i, 8 * (e & 1))) = q;
  }
  fence_async_smem();  // both CTAs' bias operands are read by the tensor cores (async proxy)
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t idesc = idesc_bf16_f32(2 * kTileM, 256);
  // registers: warpgroups 0 and 1 (issuer, producer, builders) need few, the
  // two epilogue warpgroups read 64 accumulator columns per thread at once;
  // 256 x 88 + 256 x 168 = the 512 x 128 the CTA is launched with.  Each
  // warpgroup changes its budget at the head of its own branch.
  if (warp < kPairEpi0) {
    setmaxnreg_dec<88>();
  if (warp == 0) {
    if (rank == 0 && lane == 0) {
      // ---------------------------------------------------------- MMA issuer
      // As in the wide kernel: plain counters, a parity bit per stage and
      // descriptors formed by addition keep the products back to back.
      bool ok = true;
      int st = 0, part_i = 0;  // ring stage and half-slice within it
      uint32_t fpar = 0;       // bit s: parity of the next wait on full[s]
      uint32_t u1 = 0;         // D1 uses issued so far
      const uint64_t ring_desc = sdesc_sw128(smem_u32(ring));
      const uint64_t x_desc = sdesc_sw128(smem_u32(X));
      const uint64_t one_desc = sdesc_nosw(smem_u32(ONE), 128, 0);
      const uint64_t bias_desc = sdesc_nosw(smem_u32(BIAS), 128, 256);
      for (int t = 0; t < my_pairs && ok; ++t) {
        if (!(ok = mbar_wait_cl_short(x_full, (uint32_t)(t & 1)))) break;
        tc_fence_after();
        for (int j = 0; j < J1 + J2 && ok; ++j) {
          const bool l2 = j >= J1;
          // A operand in TMEM: the output jobs and, with three layers, job 1
          const bool a_tmem = l2 || (three && j == 1);
          // both feature tiles are free once the products reading them are done
          if (j == (three ? 1 : J1)) umma_pair_commit_both(x_empty);
          uint32_t d = tmem;  // D0: layer-1 job 0
          if (j > 0) {        // D1: its previous use has been read by both epilogues
            if (u1 >= 1 && !(ok = mbar_wait_cl_short(d1_empty, (u1 - 1) & 1u))) break;
            tc_fence_after();
            d = tmem + 256u;
          }
          const int nk = l2 ? nk1 : j == 1 ? nk_c1 : nk0;
          const uint32_t a_base = tmem + (l2 ? out_a : 0u);
          // the compaction job whose activations K-block 0 (three layers) or
          // each fourth K-block (two layers) of this job waits for, if any
          const bool wait_h = three ? j >= 1 : j == J1;
          umma_pair_bf16(d, one_desc, bias_desc + (uint64_t)(j * (kTileM * 32 / 16)), idesc, 0u);
          for (int kb = 0; kb < nk; ++kb) {
            // K-blocks 4 i.. of the output jobs read compaction job i's activations
            // (three layers: job 1 reads job 0's, the output job job 1's)
            if (wait_h && (three ? kb == 0 : (kb & 3) == 0)) {
              if (!(ok = mbar_wait_cl_short(&h1_ready[three ? j - 1 : kb >> 2], (uint32_t)(t & 1)))) break;
              tc_fence_after();
            }
            if (part_i == 0) {  // a new stage: both CTAs' copies have landed
              if (!(ok = mbar_wait_cl_short(&full[st], (fpar >> st) & 1u))) break;
              fpar ^= 1u << st;
              tc_fence_after();
            }
            const uint64_t bd = ring_desc + (uint64_t)((st * Q + part_i) * (kHalfSlice / 16));
            if (a_tmem) {
              const uint32_t a0 = a_base + (uint32_t)(32 * kb);
#pragma unroll
              for (int k = 0; k < 4; ++k) umma_pair_bf16_ts(d, a0 + 8u * k, bd + 2u * k, idesc, 1u);
            } else {
              const uint64_t xd = x_desc + (uint64_t)(kb * (kWideChunk / 16));
#pragma unroll
              for (int k = 0; k < 4; ++k) umma_pair_bf16(d, xd + 2u * k, bd + 2u * k, idesc, 1u);
            }
            if (++part_i == Q) {  // the stage is free in both CTAs once these products complete
              umma_pair_commit_both(&empty[st]);
              part_i = 0;
              st = st + 1 == S ? 0 : st + 1;
            }
          }
          if (!ok) break;
          if (j == 0) {
            umma_pair_commit_both(d0_full);
          } else {
            umma_pair_commit_both(d1_full);
            ++u1;
          }
        }
      }
      if (!ok) pair_stop(abort_flag, rank, a.err);
      umma_pair_commit_both(done);  // every product issued has completed before TMEM is freed
      mbar_wait(done, 0);
    } else if (rank == 1 && lane == 0) {
      // ---------------------------------------------------------- stage relay
      // this CTA's half of stage G has landed -> one arrival on CTA 0's full[s]
      const int64_t stages = (int64_t)my_pairs * per_tile / Q;
      for (int64_t G = 0; G < stages; ++G) {
        const int s = (int)(G % S);
        if (!mbar_wait(&full[s], (uint32_t)((G / S) & 1))) {
          pair_stop(abort_flag, rank, a.err);
          break;
        }
        if (*abort_flag) break;
        mbar_arrive_at(&full[s], 0);
      }
      mbar_wait(done, 0);  // the last commit has reached this CTA too
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ producer
    if (lane == 0 && my_pairs > 0) {
      const int64_t stages = (int64_t)my_pairs * per_tile / Q;
      const uint32_t bytes = (uint32_t)(Q * kHalfSlice);
      const uint8_t* src = img + (int64_t)rank * per_tile * kHalfSlice;
      int64_t G = 0;
      bool ok = true;
      for (; G < stages; ++G) {
        const int s = (int)(G % S);
        const int64_t u = G / S;
        if (u >= 1 && !(ok = mbar_wait_cl(&empty[s], (uint32_t)((u - 1) & 1)))) break;
        if (*abort_flag) {
          ok = false;
          break;
        }
        const int q0 = (int)((G * Q) % per_tile);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_g2s(ring + (size_t)s * Q * kHalfSlice, src + (int64_t)q0 * kHalfSlice, bytes, &full[s]);
      }
      if (!ok && !*abort_flag) pair_stop(abort_flag, rank, a.err);
      // stages issued and never consumed (only after an abort) land in this
      // CTA's shared memory: wait for them (bounded) before it can exit
      if (*abort_flag)
        for (int64_t h = G - 1; h >= 0 && h >= G - S; --h) mbar_wait(&full[h % S], (uint32_t)((h / S) & 1));
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ feature-tile builders
    const int bt = tid - kPairBuild0 * 32;
    pdl_wait();  // pair chunks and template rows from the previous kernel of the stream
    for (int t = 0; t < my_pairs; ++t) {
      if (t >= 1 && !mbar_wait_cl(x_empty, (uint32_t)((t - 1) & 1))) {
        pair_stop(abort_flag, rank, a.err);
        break;
      }
      if (*abort_flag) break;
      const int64_t tile = 2 * ((int64_t)pair_id + (int64_t)t * n_pairs) + rank;
      build_tile<4>(a, X, tile * kTileM, bt, kPairBuild * 32);  // rows past the batch: zeros
      fence_async_smem();  // the tile is read by the tensor cores (async proxy)
      __syncwarp();
      if (lane == 0) mbar_arrive_at(x_full, 0);
    }
  }
  } else {
    setmaxnreg_inc<168>();
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kPairEpi0;  // 0..7
    const int q4 = warp & 3;          // TMEM lane quadrant
    const int h = ew >> 2;            // which 128 of a job's 256 columns
    const int row = 32 * q4 + lane;
    const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;
    uint32_t u1 = 0;  // D1 uses read so far
    bool ok = true;
    for (int t = 0; t < my_pairs; ++t) {
      for (int j = 0; j < J1; ++j) {
        // layer-1 job j: relu(D + b1) -> bf16 -> H1 columns [128 j + 64 h, +64)
        bool go = ok && !*abort_flag;
        if (go) go = j == 0 ? mbar_wait_cl(d0_full, (uint32_t)(t & 1)) : mbar_wait_cl(d1_full, u1 & 1u);
        go = __all_sync(0xffffffffu, go);  // the tensor-memory accesses below are warp-wide
        if (!go && ok) {
          ok = false;
          // the issuer, whose waits need both CTAs' epilogues, runs out too and
          // latches the error for the pair
          if (lane == 0) *abort_flag = 1;
        }
        uint32_t pa[32], pb[32];
        if (j == 0) {
          // D0 is H1's own columns (packed column c holds features 2c, 2c + 1).
          // Half 1 overwrites columns 64..127, which half 0 of its quadrant
          // reads: half 0 reads them first and signals; each half then writes
          // a block of 32 packed columns once the columns under it are consumed.
          const uint32_t d0 = tmem + lane_addr;
          if (h == 0) {
            if (go) {
              tc_fence_after();
              pack64_relu(d0 + 64u, pb);  // features 64..127 -> columns 32..63
            }
            tc_fence_before();
            named_bar_arrive(2, kPairEpi * 32);
            if (go) {
              pack32_relu<16>(d0 + 32u, pa);  // features 32..63 -> columns 16..31
              tmem_st32(d0 + 32u, pb);                     // columns 32..63 are consumed now
              pack32_relu<0>(d0, pa);         // features 0..31 -> columns 0..15
              tmem_st32(d0, pa);
              tmem_wait_st();
            }
          } else {
            if (go) {
              tc_fence_after();
              pack64_relu(d0 + 128u, pa);  // features 128..191 -> columns 64..95
            }
            named_bar_sync(2, kPairEpi * 32);
            tc_fence_after();
            if (go) {
              tmem_st32(d0 + 64u, pa);
              pack64_relu(d0 + 192u, pb);  // features 192..255 -> columns 96..127
            }
            if (J1 > 1) {  // columns 128..255 read: layer-1 job 1 may write there
              tc_fence_before();
              named_bar_arrive(3, kPairEpi * 32);
            }
            if (go) {
              tmem_st32(d0 + 96u, pb);
              tmem_wait_st();
            }
          }
        } else {
          // D1 -> H1 columns [128 j + 64 h, +64), which job 0's columns 128..255
          // held: half 0 first waits until half 1 of its quadrant has read them
          const uint32_t src = tmem + lane_addr + 256u + 128u * (uint32_t)h;
          const uint32_t dst = tmem + lane_addr + (uint32_t)(128 * j + 64 * h);
          if (h == 0) {
            tc_fence_before();
            named_bar_sync(3, kPairEpi * 32);
          }
          if (go) {
            tc_fence_after();
            pack64_relu(src, pa);
            tmem_st32(dst, pa);
            pack64_relu(src + 64u, pb);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_at_relaxed(d1_empty, 0);  // D1 read: the next job may overwrite it
          ++u1;
          if (go) {
            tmem_st32(dst + 32u, pb);
            tmem_wait_st();
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_at_relaxed(&h1_ready[j], 0);
      }
      uint64_t acc = 0;  // output-layer partial, two fp32 lanes
      for (int n = 0; n < J2; ++n) {
        // layer-2 job n: acc += relu(bf16(D + b2)) . w3 over this warp's 128
        // columns; D1 is released once all are read
        bool go = ok && !*abort_flag;
        if (go) go = mbar_wait_cl(d1_full, u1 & 1u);
        go = __all_sync(0xffffffffu, go);
        if (!go && ok) {
          ok = false;
          if (lane == 0) *abort_flag = 1;
        }
        const uint32_t src = tmem + lane_addr + 256u + 128u * (uint32_t)h;
        const uint16_t* w = sw3 + 256 * n + 128 * h;
        uint32_t va[16], vb[16];
        if (go) {
          tc_fence_after();
          tmem_ld16(src, va);
#pragma unroll
          for (int i = 0; i < 6; i += 2) {
            tmem_wait_ld_regs(va);
            tmem_ld16(src + 16u * (i + 1), vb);
            acc = out_dot16_wb(va, w + 16 * i, acc);
            tmem_wait_ld_regs(vb);
            tmem_ld16(src + 16u * (i + 2), va);
            acc = out_dot16_wb(vb, w + 16 * (i + 1), acc);
          }
          tmem_wait_ld_regs(va);
          tmem_ld16(src + 16u * 7, vb);
          acc = out_dot16_wb(va, w + 16 * 6, acc);
          tmem_wait_ld_regs(vb);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_at_relaxed(d1_empty, 0);  // all of D1 read: the next job may overwrite it
        ++u1;
        if (go) acc = out_dot16_wb(vb, w + 16 * 7, acc);
      }
      float* pt = part + (t & 1) * 2 * kTileM;
      pt[h * kTileM + row] = __uint_as_float((uint32_t)acc) + __uint_as_float((uint32_t)(acc >> 32));
      // the two halves of every row meet here; a stop is decided together
      if (!named_bar_and(1, kPairEpi * 32, ok)) break;
      if (h == 0) {
        const int64_t g = (2 * ((int64_t)pair_id + (int64_t)t * n_pairs) + rank) * kTileM + row;
        if (g < a.rows) a.scores[g] = (pt[row] + pt[kTileM + row]) + __ldg(params + p.b_last_off);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no arrival or product of either CTA is still aimed at the other
  if (warp == 0) tmem_dealloc_pair(tmem, 512);
}

// Per batch, before the scorer: normalised bf16 template rows (instance row i
// holds the z-scored instance features at their feature positions 6 ..
// 6+d_inst and zeros elsewhere; request row r likewise for the request block)
// and, for every (request, instance) pair, the 16-byte first chunk of its
// feature row holding the six z-scored pair features (Sec. 4.1 Features;
// Algorithm 4 Normalize) with zeros in columns 6 and 7.
template <typename I>  // index type: 32-bit when every index fits, else 64-bit
__global__ void k_norm_rows(const int64_t* __restrict__ tok_off, const int32_t* __restrict__ hits,
                            uint4* __restrict__ pairx, int n_inst, int d_inst, const float* __restrict__ inst,
                            int n_req, int d_req, const float* __restrict__ req, const float* __restrict__ mean,
                            const float* __restrict__ stdv, int d_pad, uint16_t* __restrict__ xin,
                            uint16_t* __restrict__ xrq) {
  // items: eight template columns of an instance row, of a request row, then
  // one (request, instance) pair
  const I G = (I)(d_pad / 8);
  const I ni = (I)n_inst * G, nr = (I)n_req * G, np = (I)n_req * (I)n_inst;
  for (I e = (I)blockIdx.x * blockDim.x + threadIdx.x; e < ni + nr + np; e += (I)gridDim.x * blockDim.x) {
    if (e < ni + nr) {
      const bool is_inst = e < ni;
      const I f = is_inst ? e : e - ni;
      const I row = f / G;
      const int c0 = (int)(f - row * G) * 8;
      const int off = is_inst ? kPair : kPair + d_inst, dk = is_inst ? d_inst : d_req;
      const float* src = is_inst ? inst + (int64_t)row * d_inst : req + (int64_t)row * d_req;
      uint32_t w[4];
#pragma unroll
      for (int u = 0; u < 8; u += 2) {
        uint32_t pr = 0;
#pragma unroll
        for (int v = 0; v < 2; ++v) {
          const int k = c0 + u + v - off;
          const uint16_t b = (k >= 0 && k < dk) ? bf16_bits(zscore(src[k], mean[off + k], stdv[off + k])) : (uint16_t)0;
          pr |= (uint32_t)b << (16 * v);
        }
        w[u / 2] = pr;
      }
      uint16_t* dst = (is_inst ? xin : xrq) + (int64_t)row * d_pad + c0;
      *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
      const I g = e - ni - nr;
      const I r = g / (I)n_inst;
      const int64_t L = __ldg(tok_off + r + 1) - __ldg(tok_off + r);
      const int h = __ldg(hits + g);
      uint16_t f[kPair];
#pragma unroll
      for (int k = 0; k < kPair; ++k)
        f[k] = bf16_bits(zscore(raw_feature(k, L, h, nullptr, 0, nullptr), __ldg(mean + k), __ldg(stdv + k)));
      pairx[g] = make_uint4(f[0] | ((uint32_t)f[1] << 16), f[2] | ((uint32_t)f[3] << 16),
                            f[4] | ((uint32_t)f[5] << 16), 0u);
    }
  }
}

// Instance template rows (computed when the snapshot or the normaliser
// changes): row i holds the z-scored instance features of instance i, bf16,
// at their feature positions 6 .. 6+d_inst, zeros elsewhere (Algorithm 4
// Normalize).
__global__ void k_inst_templates(int n_inst, int d_inst, const float* __restrict__ inst,
                                 const float* __restrict__ mean, const float* __restrict__ stdv, int d_pad,
                                 uint16_t* __restrict__ xin) {
  const int n = n_inst * d_pad;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n; e += gridDim.x * blockDim.x) {
    const int i = e / d_pad, k = e - i * d_pad - kPair;
    xin[e] = (k >= 0 && k < d_inst)
                 ? bf16_bits(zscore(inst[(int64_t)i * d_inst + k], mean[kPair + k], stdv[kPair + k]))
                 : (uint16_t)0;
  }
}

// Feature image for the pipelined scorer: row g = r * n_inst + i of the batch
// as its bf16 feature row [pair(6) || inst || req || 0-pad] (Sec. 4.1
// Features; Algorithm 4 Normalize), tile t of 128 rows at t * xbytes in the
// 128-byte-swizzled K-major layout of the MMA operand, rows past the batch
// zero.  One CTA per tile: it forms the request template rows of the requests
// it touches and the pair-feature chunk of each row in shared memory; a
// 16-byte chunk of a feature row is then the OR of an instance-template chunk
// (computed with the snapshot), a request-template chunk and, for chunk 0,
// the pair chunk.  Values are bit-identical to the template path.
__global__ void __launch_bounds__(256) k_feature_image(const int64_t* __restrict__ tok_off,
                                                       const int32_t* __restrict__ hits, int n_inst,
                                                       const uint16_t* __restrict__ xin, int d_inst, int d_req,
                                                       const float* __restrict__ req, const float* __restrict__ mean,
                                                       const float* __restrict__ stdv, int d_pad, int64_t rows,
                                                       int64_t n_tiles, int nr_max, uint8_t* __restrict__ ximg) {
  extern __shared__ uint4 fz4[];
  uint4* zr = fz4;                                     // [nr_max][d_pad / 8] request template chunks
  __shared__ uint4 zp[kTileM];                         // pair chunk of each row
  __shared__ int row_i[kTileM];                        // instance of each tile row
  __shared__ int row_q[kTileM];                        // its request, relative to the tile's first
  const int cpr = d_pad / 8;
  const int64_t xbytes = (int64_t)kTileM * d_pad * 2;
  pdl_wait();  // hit lengths from the prefix kernel
  for (int64_t t = blockIdx.x; t < n_tiles; t += gridDim.x) {
    const int64_t g0 = t * kTileM;
    const int nrow = (int)(g0 + kTileM < rows ? kTileM : rows - g0);
    const int64_t r_lo = g0 / n_inst;
    const int i0 = (int)(g0 - r_lo * n_inst);
    if (threadIdx.x < kTileM) {
      const int m = threadIdx.x, q = (i0 + m) / n_inst;
      row_q[m] = q;
      row_i[m] = i0 + m - q * n_inst;
      uint16_t f[kPair];
#pragma unroll
      for (int k = 0; k < kPair; ++k) f[k] = 0;
      if (m < nrow) {
        const int64_t r = r_lo + q;
        const int64_t L = __ldg(tok_off + r + 1) - __ldg(tok_off + r);
        const int h = __ldg(hits + g0 + m);
#pragma unroll
        for (int k = 0; k < kPair; ++k)
          f[k] = bf16_bits(zscore(raw_feature(k, L, h, nullptr, 0, nullptr), __ldg(mean + k), __ldg(stdv + k)));
      }
      zp[m] = make_uint4(f[0] | ((uint32_t)f[1] << 16), f[2] | ((uint32_t)f[3] << 16), f[4] | ((uint32_t)f[5] << 16),
                         0u);
    }
    const int q_last = (i0 + nrow - 1) / n_inst;  // requests r_lo .. r_lo + q_last
    uint16_t* zr16 = reinterpret_cast<uint16_t*>(zr);
    for (int e = threadIdx.x; e < (q_last + 1) * d_pad; e += blockDim.x) {
      const int rl = e / d_pad, k = e - rl * d_pad - kPair - d_inst;
      zr16[e] = (k >= 0 && k < d_req) ? bf16_bits(zscore(__ldg(req + (r_lo + rl) * d_req + k),
                                                         __ldg(mean + kPair + d_inst + k),
                                                         __ldg(stdv + kPair + d_inst + k)))
                                      : (uint16_t)0;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < kTileM * cpr; e += blockDim.x) {
      const int m = e / cpr, c = e - m * cpr;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (m < nrow) {
        const uint4 ti = __ldg(reinterpret_cast<const uint4*>(xin + (int64_t)row_i[m] * d_pad) + c);
        const uint4 tq = zr[row_q[m] * cpr + c];
        const uint4 tp = c == 0 ? zp[m] : make_uint4(0u, 0u, 0u, 0u);
        v = make_uint4(ti.x | tq.x | tp.x, ti.y | tq.y | tp.y, ti.z | tq.z | tp.z, ti.w | tq.w | tp.w);
      }
      *reinterpret_cast<uint4*>(ximg + t * xbytes + sw128_offset(m, 8 * c, kTileM)) = v;
    }
    __syncthreads();
  }
  pdl_trigger();  // the scorer may start once every CTA is here
}

}  // namespace

bool plan_tc(const MlpDesc& m, TcPlan& p, bool allow_pair, bool allow_pipe) {
  p = TcPlan{};
  if (!m.bf16 || m.n_layers < 2) return false;
  p.n_tc = m.n_layers - 1;
  int amax = 0, cb = 0, outmax = 0;
  int64_t off = 0;
  int q = 0;
  p.d_pad = ((m.w[0] + 63) / 64) * 64;
  for (int l = 0; l < p.n_tc; ++l) {
    const int in = m.w[l], out = m.w[l + 1];
    if (out % 64 != 0 || out > 512) return false;
    if (in > 512) return false;
    p.in_pad[l] = ((in + 63) / 64) * 64;
    p.out[l] = out;
    p.nc[l] = out <= 256 ? out : 256;
    if (out % p.nc[l] != 0) return false;
    p.img_off[l] = off;
    const int nk = p.in_pad[l] / 64, nn = out / p.nc[l];
    for (int nci = 0; nci < nn; ++nci)
      for (int kb = 0; kb < nk; ++kb) {
        if (q >= kMaxChunks) return false;
        p.chunk_off[q] = off + ((int64_t)nci * nk + kb) * p.nc[l] * 128;
        p.chunk_len[q] = p.nc[l] * 128;
        ++q;
      }
    off += (int64_t)out * p.in_pad[l] * 2;
    amax = std::max(amax, p.in_pad[l]);
    cb = std::max(cb, p.nc[l] * 128);
    outmax = std::max(outmax, out);
  }
  // the operand tile must also hold every hidden output written by an epilogue
  for (int l = 0; l + 1 < p.n_tc; ++l) amax = std::max(amax, p.out[l]);
  p.chunks = q;
  p.img_bytes = off;
  p.chunk_bytes = cb;
  p.a_bytes = kTileM * amax * 2;
  const int fixed = 1024 + 64;
  const int avail = kMaxSmem - fixed - p.a_bytes;
  const int smax = avail / (cb + 16);
  if (p.chunks <= smax) {
    p.resident = 1;
    p.stages = p.chunks;
  } else {
    p.resident = 0;
    p.stages = std::min(smax, 8);
    if (p.stages < 2) return false;
  }
  p.smem = p.a_bytes + p.stages * cb + (2 * p.stages + 1) * 8 + 16 + 1024;
  p.tmem_cols = 32;
  while ((int)p.tmem_cols < outmax) p.tmem_cols <<= 1;
  p.w_last_off = m.woff[m.n_layers - 1];
  p.b_last_off = m.boff[m.n_layers - 1];
  // pipelined variant: two hidden layers of <= 256, all weights resident
  p.pipe = 0;
  if (allow_pipe && p.n_tc == 2 && p.out[0] <= 256 && p.out[1] <= 256 && p.nc[0] == p.out[0] &&
      p.nc[1] == p.out[1]) {
    const int64_t need = 1024 + (int64_t)p.chunks * cb + kXB * (int64_t)p.d_pad * kTileM * 2 + 2 * kTileM * 128 +
                         8 * 32 + 2 * 256 * 32 + 2 * kTileM * 4 + 256 * 2 + (12 + kWBars) * 8 + 16;
    if (need <= kMaxSmem) {
      p.pipe = 1;
      p.pipe_smem = (int)need;
    }
  }
  // wide variant (when the pipelined one does not apply): two hidden layers of
  // multiples of 128, a feature tile of at most 128 columns.  Its image uses
  // 128-row N-chunks, so the per-tile stream of [128 x 64] slices (layer 1
  // jobs, then layer 2 jobs, K-blocks inner) is the image itself, contiguous;
  // stages hold Q slices (Q in 4, 2, 1 dividing the slices per tile)
  // pair variant (before the wide one): two hidden layers of multiples of 256
  // (at most 512, so that the packed layer-1 activations and one 256-column
  // accumulator fill the 512 TMEM columns), a feature tile of at most 128
  // columns.  Each CTA of a pair streams its half of every [256 x 64] slice
  // (16 KB: the image's per-rank streams); a stage holds Q half-slices, Q the
  // largest divisor of the per-tile stream up to 6 that leaves two stages.
  // (or three hidden layers of exactly 256: the second runs as a compaction
  // job into the TMEM columns the first left free, the third is the output job)
  p.pair = 0;
  const bool two = p.n_tc == 2 && p.out[0] % 256 == 0 && p.out[1] % 256 == 0;
  const bool three = p.n_tc == 3 && p.out[0] == 256 && p.out[1] == 256 && p.out[2] == 256;
  if (allow_pair && !p.pipe && (two || three) && p.d_pad <= 128) {
    const int HL = p.out[p.n_tc - 1];
    const int nk0 = p.in_pad[0] / 64;
    int per_tile = 0, jobs = 0;
    for (int l = 0; l < p.n_tc; ++l) {
      per_tile += (p.out[l] / 256) * (p.in_pad[l] / 64);
      jobs += p.out[l] / 256;
    }
    // alignment, feature tile, ONE, bias operands, bf16 output weights, row
    // partials, barriers, TMEM holder and abort flag
    const int64_t fixed = 1024 + (int64_t)nk0 * kTileM * 128 + 8 * 32 + (int64_t)jobs * kTileM * 32 +
                          (int64_t)HL * 2 + 4 * kTileM * 4 + 10 * 8 + 16;
    for (int Q = 6; Q >= 1 && !p.pair; --Q) {
      if (per_tile % Q) continue;
      const int64_t stages = (kMaxSmem - fixed) / ((int64_t)Q * kTileM * 128 + 16);
      if (stages < 2) continue;
      p.pair_q = Q;
      p.pair_stages = (int)std::min<int64_t>(stages, 12);
      p.pair_smem = (int)(fixed + (int64_t)p.pair_stages * ((int64_t)Q * kTileM * 128 + 16));
      p.pair_slices = per_tile;
      p.pair = 1;
    }
    if (p.pair) {
      int64_t woff = 0;
      for (int l = 0; l < p.n_tc; ++l) {
        p.nc[l] = 128;
        p.img_off[l] = woff;
        woff += (int64_t)p.out[l] * p.in_pad[l] * 2;
      }
      p.img_bytes = woff;  // = 2 ranks x per_tile half-slices x 16 KB
      return true;
    }
  }
  p.wide = 0;
  if (!p.pipe && p.n_tc == 2 && p.out[0] % 128 == 0 && p.out[1] % 128 == 0 && p.d_pad <= 128) {
    int64_t woff = 0;
    q = 0;
    for (int l = 0; l < 2; ++l) {
      p.nc[l] = 128;
      p.img_off[l] = woff;
      const int nk = p.in_pad[l] / 64, nn = p.out[l] / 128;
      for (int nci = 0; nci < nn; ++nci)
        for (int kb = 0; kb < nk; ++kb) {
          p.chunk_off[q] = woff + ((int64_t)nci * nk + kb) * 128 * 128;
          p.chunk_len[q] = 128 * 128;
          ++q;
        }
      woff += (int64_t)p.out[l] * p.in_pad[l] * 2;
    }
    p.chunks = q;
    p.img_bytes = woff;
    p.chunk_bytes = 128 * 128;
    const int H1 = p.out[0], H2 = p.out[1];
    const int per_tile = (H1 / 128) * (p.in_pad[0] / 64) + (H2 / 128) * (H1 / 64);
    const int64_t fixed = 1024 + (int64_t)(p.d_pad / 64) * kTileM * 128 + 256 + (int64_t)(H1 + H2) * 32 +
                          (int64_t)H2 * 2 + 4 * kTileM * 4 + 16 * 8 + 16;
    for (int Q = 4; Q >= 1 && !p.wide; Q >>= 1) {
      if (per_tile % Q) continue;
      const int64_t stages = (kMaxSmem - fixed - 256) / ((int64_t)Q * kTileM * 128 + 16);
      if (stages < 2) continue;
      p.wide_q = Q;
      p.wide_stages = (int)std::min<int64_t>(stages, 12);
      p.wide_smem = (int)(fixed + (int64_t)p.wide_stages * ((int64_t)Q * kTileM * 128 + 16));
      p.wide = 1;
    }
    // the generic kernel keeps working on this layout (128-row chunks)
    const int avail = kMaxSmem - (1024 + 64) - p.a_bytes;
    const int smax = avail / (p.chunk_bytes + 16);
    p.resident = p.chunks <= smax ? 1 : 0;
    p.stages = p.resident ? p.chunks : std::min(smax, 8);
    p.smem = p.a_bytes + p.stages * p.chunk_bytes + (2 * p.stages + 1) * 8 + 16 + 1024;
  }
  return true;
}

// The bf16 feature rows the tensor-core scorers read for the last batch, row
// r * n_inst + i of [rows, d], decoded from where they live: the feature
// image's MMA-layout tiles (pipelined scorer), or the pair chunk OR-ed with
// the instance and request template rows (the other tensor-core scorers,
// exactly as their tile builders combine them).
__global__ void k_read_features(int64_t row0, int64_t n_rows, int d, int d_pad, int n_inst, int pipe,
                                const uint8_t* __restrict__ ximg, const uint4* __restrict__ pairx,
                                const uint16_t* __restrict__ xin, const uint16_t* __restrict__ xrq,
                                uint16_t* __restrict__ out) {
  const int64_t total = n_rows * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = row0 + e / d;
    const int k = (int)(e % d);
    uint16_t v;
    if (pipe) {
      const int64_t t = g / kTileM;
      const int m = (int)(g - t * kTileM);
      const int64_t xbytes = (int64_t)(d_pad / 64) * kTileM * 128;
      v = *reinterpret_cast<const uint16_t*>(ximg + t * xbytes + sw128_offset(m, k, kTileM));
    } else {
      const int64_t r = g / n_inst, i = g - r * n_inst;
      const uint16_t* pc = reinterpret_cast<const uint16_t*>(pairx + g);
      v = (uint16_t)(xin[i * d_pad + k] | xrq[r * d_pad + k] | (k < 8 ? pc[k] : 0));
    }
    out[e] = v;
  }
}

cudaError_t launch_read_features(int64_t row0, int64_t n_rows, int d, const TcPlan& p, int n_inst,
                                 const uint8_t* ximg, const uint4* pairx, const uint16_t* xin, const uint16_t* xrq,
                                 uint16_t* out, cudaStream_t s) {
  if (n_rows <= 0) return cudaSuccess;
  const int grid = (int)std::min<int64_t>((n_rows * d + 255) / 256, 4096);
  k_read_features<<<grid, 256, 0, s>>>(row0, n_rows, d, p.d_pad, n_inst, p.pipe, ximg, pairx, xin, xrq, out);
  return cudaGetLastError();
}

cudaError_t launch_norm_rows(const int64_t* tok_off, const int32_t* hits, uint4* pairx, int n_inst, int d_inst,
                             const float* inst, int n_req, int d_req, const float* req, const float* mean,
                             const float* stdv, int d_pad, uint16_t* xin, uint16_t* xrq, int sms, cudaStream_t s) {
  const int64_t n = (int64_t)(n_inst + n_req) * d_pad + (int64_t)n_req * n_inst;
  if (n <= 0) return cudaSuccess;
  const int grid = (int)std::min<int64_t>((n + 255) / 256, (int64_t)sms * 8);
  if (n + (int64_t)grid * 256 < (1LL << 31))
    k_norm_rows<uint32_t><<<grid, 256, 0, s>>>(tok_off, hits, pairx, n_inst, d_inst, inst, n_req, d_req, req, mean,
                                               stdv, d_pad, xin, xrq);
  else
    k_norm_rows<int64_t><<<grid, 256, 0, s>>>(tok_off, hits, pairx, n_inst, d_inst, inst, n_req, d_req, req, mean,
                                              stdv, d_pad, xin, xrq);
  return cudaGetLastError();
}

cudaError_t launch_inst_templates(int n_inst, int d_inst, const float* inst, const float* mean, const float* stdv,
                                  int d_pad, uint16_t* xin, int sms, cudaStream_t s) {
  const int n = n_inst * d_pad;
  if (n <= 0) return cudaSuccess;
  const int grid = std::min((n + 255) / 256, sms * 4);
  k_inst_templates<<<grid, 256, 0, s>>>(n_inst, d_inst, inst, mean, stdv, d_pad, xin);
  return cudaGetLastError();
}

cudaError_t launch_feature_image(const int64_t* tok_off, const int32_t* hits, int n_inst, const uint16_t* xin,
                                 int d_inst, int n_req, int d_req, const float* req, const float* mean,
                                 const float* stdv, int d_pad, uint8_t* ximg, int sms, cudaStream_t s) {
  const int64_t rows = (int64_t)n_req * n_inst;
  if (rows <= 0) return cudaSuccess;
  const int64_t n_tiles = (rows + kTileM - 1) / kTileM;
  const int nr_max = (kTileM + n_inst - 1) / n_inst + 1;  // requests a tile can touch
  const size_t smem = (size_t)nr_max * d_pad * sizeof(uint16_t);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_feature_image, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  const int grid = (int)std::min<int64_t>(n_tiles, (int64_t)sms * 8);
  return launch_chained(k_feature_image, dim3(grid), dim3(256), smem, s, 1, tok_off, hits, n_inst, xin, d_inst, d_req,
                        req, mean, stdv, d_pad, rows, n_tiles, nr_max, ximg);
}

int pair_max_clusters(const TcPlan& p) {
  if (!p.pair) return 0;
  auto kern = p.n_tc == 3 ? k_score_pair<true> : k_score_pair<false>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p.pair_smem) != cudaSuccess)
    return 0;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(std::max(2, sms & ~1));
  cfg.blockDim = dim3(kThreadsPair);
  cfg.dynamicSmemBytes = (size_t)p.pair_smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_score_tc(const MlpDesc& m, const TcPlan& p, const Published* pub, const int32_t* sel,
                            int n_req, int n_inst, const uint4* pairx, const uint8_t* ximg, int32_t* choice,
                            float* best,
                            const uint16_t* xin, const uint16_t* xrq, int d_inst, int d_req, const float* mean,
                            const float* stdv, float* scores, int* err, int sms, cudaStream_t s) {
  const int64_t rows = (int64_t)n_req * n_inst;
  if (rows <= 0) return cudaSuccess;
  TcArgs a{};
  a.p = p;
  a.img0 = pub[0].img;
  a.img1 = pub[1].img;
  a.params0 = pub[0].params;
  a.params1 = pub[1].params;
  a.sel = sel;
  for (int l = 0; l < m.n_layers; ++l) a.boff[l] = m.boff[l];
  a.w_last_off = p.w_last_off;
  a.n_req = n_req;
  a.n_inst = n_inst;
  a.d = m.w[0];
  a.d_inst = d_inst;
  a.d_req = d_req;
  a.pairx = pairx;
  a.ximg = ximg;
  a.choice = choice;
  a.best = best;
  a.fuse_argmin = (p.pipe && choice && best && n_inst <= 32 && 32 % n_inst == 0) ? 1 : 0;
  a.xin = xin;
  a.xrq = xrq;
  a.mean = mean;
  a.stdv = stdv;
  a.scores = scores;
  a.err = err;
  a.rows = rows;
  a.n_tiles = (int)((rows + kTileM - 1) / kTileM);
  const int grid = std::min(a.n_tiles, sms);
  if (p.pipe) {
    cudaError_t e = cudaFuncSetAttribute(k_score_tc_pipe, cudaFuncAttributeMaxDynamicSharedMemorySize, p.pipe_smem);
    if (e != cudaSuccess) return e;
    return launch_chained(k_score_tc_pipe, dim3(grid), dim3(kThreadsPipe), (size_t)p.pipe_smem, s, 1, a);
  } else if (p.pair) {
    // the image is in the pair layout, which no other scorer reads
    if (!scores) return cudaErrorInvalidValue;
    auto kern = p.n_tc == 3 ? k_score_pair<true> : k_score_pair<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p.pair_smem);
    if (e != cudaSuccess) return e;
    const int tile_pairs = (a.n_tiles + 1) / 2;
    const int fit = p.pair_clusters > 0 ? p.pair_clusters : sms / 2;
    const int pairs = std::max(1, std::min(tile_pairs, fit));
    return launch_chained(kern, dim3(2 * pairs), dim3(kThreadsPair), (size_t)p.pair_smem, s, 2, a);
  } else if (p.wide && scores) {
    cudaError_t e = cudaFuncSetAttribute(k_score_wide, cudaFuncAttributeMaxDynamicSharedMemorySize, p.wide_smem);
    if (e != cudaSuccess) return e;
    return launch_chained(k_score_wide, dim3(grid), dim3(kThreadsWide), (size_t)p.wide_smem, s, 1, a);
  } else {
    cudaError_t e = cudaFuncSetAttribute(k_score_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
    if (e != cudaSuccess) return e;
    k_score_tc<<<grid, kThreadsTc, p.smem, s>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace ls
