// Tensor-core GEMM for the bf16 training step (Sec. 4.3.2 online learning):
//   D[m, n] = sum_k A(m, k) * B(n, k),  A(m, k) = A[m*sam + k*sak],
//                                      B(n, k) = B[n*sbn + k*sbk]
// with fp32 operands in global memory rounded to bf16 (round to nearest even)
// while they are staged into shared memory.  Arbitrary strides make the
// transposed operands of the backward pass (dW = dZ^T A, dX = dZ W) plain
// strided reads.  One CTA computes a 128 x ntile tile with the accumulator in
// tensor memory; K runs in chunks of 64 through two staging buffers (the next
// chunk is staged while the MMAs of the current one run); blockIdx.z splits
// K (partials reduced by the caller).  Epilogues: store (partial), forward
// (Z = D + bias, A_next = bf16(ReLU(Z))), ReLU mask (dZ_prev = D * [Z > 0]),
// or row minimum of squared distances na[m] + nb[n] - 2 D[m, n] over the
// CTA's columns (the replay pool's nearest-neighbour search, Sec. 4.3.2).
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
using namespace sm100;

namespace {

constexpr int kM = 128;
constexpr int kT = 256;  // threads: 8 warps, 2 per TMEM lane quadrant

struct TcGemmArgs {
  int M, N, K;
  const float* A;
  int64_t sam, sak;
  const float* B;
  int64_t sbn, sbk;
  int ntile, kper, epi;
  float* C;
  int64_t ldc, split_stride;
  const float* bias;
  float* act;
  int64_t ld_act;
  int hidden;
  const float* zprev;
  int64_t ld_zprev;
  const float* na;   // epilogue 3: row and column squared norms
  const float* nb;
  int64_t self_off;  // epilogue 3: column row + self_off is skipped
  const int64_t* rows_dev;  // epilogue 3: rows / columns in use (device, nullable)
  const int64_t* cols_dev;
  int* err;
  uint32_t tmem_cols;
};

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void sts32(uint8_t* p, uint32_t v) {
  asm volatile("st.shared.b32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}

// Stage rows [row0, row0 + R) x k [k0, k0 + 64) of a strided fp32 operand as
// a bf16 [R x 64] K-major 128B-swizzled tile; out-of-range elements are 0.
// Every thread first issues all of its loads (R/16 float4 or equivalent), then
// converts and stores, so a chunk costs about one memory latency.
template <int R>
__device__ __forceinline__ void stage(uint8_t* tile, const float* src, int64_t s_row, int64_t s_k, int row0,
                                      int nrow, int64_t k0, int64_t kend, bool vec) {
  constexpr int PER = R * 16 / kT;  // float4-sized pieces per thread
  if (s_k == 1) {
    // piece = 4 consecutive k of one row: e -> (r = e / 16, q = e % 16)
    float4 v[PER];
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int e = threadIdx.x + u * kT;
      const int r = e >> 4, k = (e & 15) * 4;
      const int64_t kk = k0 + k;
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (row0 + r < nrow) {
        const float* p = src + (int64_t)(row0 + r) * s_row + kk;
        if (vec && kk + 3 < kend) {
          v[u] = __ldg(reinterpret_cast<const float4*>(p));
        } else {
          if (kk < kend) v[u].x = __ldg(p);
          if (kk + 1 < kend) v[u].y = __ldg(p + 1);
          if (kk + 2 < kend) v[u].z = __ldg(p + 2);
          if (kk + 3 < kend) v[u].w = __ldg(p + 3);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int e = threadIdx.x + u * kT;
      const int r = e >> 4, k = (e & 15) * 4;
      uint8_t* dst = tile + sw128_offset(r, k, R);
      asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(smem_u32(dst)), "r"(pack2(v[u].x, v[u].y)),
                   "r"(pack2(v[u].z, v[u].w))
                   : "memory");
    }
  } else {
    // rows contiguous: piece = k pair (k, k+1) of 2 consecutive rows:
    // e -> (r = 2 * (e % (R/2)), k = 2 * (e / (R/2)))
    float2 lo[PER], hi[PER];
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int e = threadIdx.x + u * kT;
      const int r = 2 * (e % (R / 2)), k = 2 * (e / (R / 2));
      const int64_t kk = k0 + k;
      lo[u] = make_float2(0.f, 0.f);
      hi[u] = make_float2(0.f, 0.f);
      const float* p = src + (int64_t)(row0 + r) * s_row + kk * s_k;
      const bool r0ok = row0 + r < nrow, r1ok = row0 + r + 1 < nrow;
      if (kk < kend) {
        if (r0ok) lo[u].x = __ldg(p);
        if (r1ok) lo[u].y = __ldg(p + s_row);
      }
      if (kk + 1 < kend) {
        if (r0ok) hi[u].x = __ldg(p + s_k);
        if (r1ok) hi[u].y = __ldg(p + s_k + s_row);
      }
    }
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int e = threadIdx.x + u * kT;
      const int r = 2 * (e % (R / 2)), k = 2 * (e / (R / 2));
      sts32(tile + sw128_offset(r, k, R), pack2(lo[u].x, hi[u].x));
      sts32(tile + sw128_offset(r + 1, k, R), pack2(lo[u].y, hi[u].y));
    }
  }
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

template <int NTILE>
__global__ void __launch_bounds__(kT) k_gemm_tc(const __grid_constant__ TcGemmArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int a_bytes = kM * 128, b_bytes = NTILE * 128;
  uint8_t* As[2] = {smem, smem + a_bytes};
  uint8_t* Bs[2] = {smem + 2 * a_bytes, smem + 2 * a_bytes + b_bytes};
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 2 * a_bytes + 2 * b_bytes);  // [2]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bar + 2);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.y * kM, n0 = blockIdx.x * g.ntile;
  if ((g.rows_dev && m0 >= *g.rows_dev) || (g.epi == 3 && g.cols_dev && n0 >= *g.cols_dev)) {
    // nothing of this tile is in use (row-minimum partials: +inf)
    const int r = m0 + 32 * (warp & 3) + lane;
    if (g.epi == 3 && r < g.M) g.C[(int64_t)r * g.ldc + 2 * blockIdx.x + (warp >> 2)] = INFINITY;
    return;
  }
  const int64_t kbeg = (int64_t)blockIdx.z * g.kper;
  const int64_t kend = kbeg + g.kper < g.K ? kbeg + g.kper : g.K;
  const int nchunks = kend > kbeg ? (int)((kend - kbeg + 63) / 64) : 0;

  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, g.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t idesc = idesc_bf16_f32(kM, NTILE);
  const bool vec_a = g.sak == 1 && (g.sam % 4) == 0 && (reinterpret_cast<uintptr_t>(g.A) & 15) == 0;
  const bool vec_b = g.sbk == 1 && (g.sbn % 4) == 0 && (reinterpret_cast<uintptr_t>(g.B) & 15) == 0;
  bool ok = true;

  for (int c = 0; c < nchunks; ++c) {
    const int b = c & 1;
    if (c >= 2 && !mbar_wait(&bar[b], (uint32_t)(((c - 2) >> 1) & 1))) ok = false;
    const int64_t k0 = kbeg + (int64_t)c * 64;
    stage<kM>(As[b], g.A, g.sam, g.sak, m0, g.M, k0, kend, vec_a);
    stage<NTILE>(Bs[b], g.B, g.sbn, g.sbk, n0, g.N, k0, kend, vec_b);
    fence_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t ab = smem_u32(As[b]), bb = smem_u32(Bs[b]);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        umma_bf16(tmem, sdesc_sw128(ab + 32u * j), sdesc_sw128(bb + 32u * j), idesc, (c | j) ? 1u : 0u);
      umma_commit(&bar[b]);
    }
    __syncwarp();
  }
  if (nchunks > 0) {
    const int b = (nchunks - 1) & 1;
    if (!mbar_wait(&bar[b], (uint32_t)(((nchunks - 1) >> 1) & 1))) ok = false;
    // the other buffer's last commit (if any) completed before this one
  }
  if (!ok) latch_error(g.err, LS_ERR_TIMEOUT);
  tc_fence_after();

  const int q4 = warp & 3, ch = warp >> 2;
  const int row = m0 + 32 * q4 + lane;
  const int half = NTILE / 2;
  const uint32_t lane_addr = (uint32_t)(32 * q4) << 16;
  const bool row_ok = row < g.M;
  float rmin = INFINITY;
  const float row_norm = g.epi == 3 && row_ok ? __ldg(g.na + row) : 0.0f;
  for (int c0 = ch * half; c0 < (ch + 1) * half; c0 += 16) {
    uint32_t v[16];
    if (nchunks > 0) {
      tmem_ld16(tmem + lane_addr + (uint32_t)c0, v);
      tmem_wait_ld();
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = 0u;
    }
    const int nb = n0 + c0;            // first column of this group
    const bool full = nb + 16 <= g.N;  // all 16 columns in range
    // side inputs of the group (bias, or the pre-activation for the mask),
    // all loaded before any use
    float side[16];
    if (g.epi == 1) {
      if (full && (reinterpret_cast<uintptr_t>(g.bias + nb) & 15) == 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 b4 = __ldg(reinterpret_cast<const float4*>(g.bias + nb) + q);
          side[4 * q] = b4.x; side[4 * q + 1] = b4.y; side[4 * q + 2] = b4.z; side[4 * q + 3] = b4.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) side[j] = nb + j < g.N ? __ldg(g.bias + nb + j) : 0.0f;
      }
    } else if (g.epi == 3) {
#pragma unroll
      for (int j = 0; j < 16; ++j) side[j] = nb + j < g.N ? __ldg(g.nb + nb + j) : INFINITY;
    } else if (g.epi == 2) {
      const float* zp = g.zprev + (int64_t)row * g.ld_zprev + nb;
      if (row_ok && full && (reinterpret_cast<uintptr_t>(zp) & 15) == 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 z4 = __ldg(reinterpret_cast<const float4*>(zp) + q);
          side[4 * q] = z4.x; side[4 * q + 1] = z4.y; side[4 * q + 2] = z4.z; side[4 * q + 3] = z4.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) side[j] = (row_ok && nb + j < g.N) ? __ldg(zp + j) : 0.0f;
      }
    }
    if (!row_ok) continue;
    if (g.epi == 3) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float dist = row_norm + side[j] - 2.0f * __uint_as_float(v[j]);
        if ((int64_t)(nb + j) != (int64_t)row + g.self_off) rmin = fminf(rmin, dist);
      }
      continue;
    }
    float out[16], act[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const float acc = __uint_as_float(v[j]);
      if (g.epi == 0) {
        out[j] = acc;
      } else if (g.epi == 1) {
        out[j] = acc + side[j];
        act[j] = round_bf16(out[j] > 0.0f ? out[j] : 0.0f);
      } else {
        out[j] = side[j] > 0.0f ? acc : 0.0f;
      }
    }
    float* crow = g.C + (g.epi == 0 ? (int64_t)blockIdx.z * g.split_stride : 0) + (int64_t)row * g.ldc + nb;
    float* arow = g.epi == 1 && g.hidden ? g.act + (int64_t)row * g.ld_act + nb : nullptr;
    if (full && (reinterpret_cast<uintptr_t>(crow) & 15) == 0 &&
        (!arow || (reinterpret_cast<uintptr_t>(arow) & 15) == 0)) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        reinterpret_cast<float4*>(crow)[q] = make_float4(out[4 * q], out[4 * q + 1], out[4 * q + 2], out[4 * q + 3]);
        if (arow)
          reinterpret_cast<float4*>(arow)[q] = make_float4(act[4 * q], act[4 * q + 1], act[4 * q + 2], act[4 * q + 3]);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (nb + j < g.N) {
          crow[j] = out[j];
          if (arow) arow[j] = act[j];
        }
    }
  }
  if (g.epi == 3 && row_ok) g.C[(int64_t)row * g.ldc + 2 * blockIdx.x + ch] = rmin;
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, g.tmem_cols);
}

template <int NTILE>
cudaError_t run_tc(dim3 grid, int smem, const TcGemmArgs& g, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<NTILE>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  k_gemm_tc<NTILE><<<grid, kT, smem, s>>>(g);
  return cudaGetLastError();
}

}  // namespace

// Picks the tile width and launches; returns cudaErrorInvalidValue when the
// shape is not worth a tensor-core tile (the caller then uses CUDA cores).
cudaError_t launch_gemm_tc(int M, int N, int K, const float* A, int64_t sam, int64_t sak, const float* B,
                           int64_t sbn, int64_t sbk, int splits, int epi, float* C, int64_t ldc,
                           int64_t split_stride, const float* bias, float* act, int64_t ld_act, int hidden,
                           const float* zprev, int64_t ld_zprev, int* err, int sms, cudaStream_t s,
                           const int64_t* rows_dev) {
  if (M < 64 || N < 32 || K < 1) return cudaErrorInvalidValue;
  const int mt = (M + kM - 1) / kM;
  int ntile = 256;
  while (ntile > 64 && (int64_t)mt * ((N + ntile - 1) / ntile) * splits < sms) ntile /= 2;
  while (ntile > 64 && ntile / 2 >= N) ntile /= 2;
  TcGemmArgs g{};
  g.M = M; g.N = N; g.K = K;
  g.A = A; g.sam = sam; g.sak = sak;
  g.B = B; g.sbn = sbn; g.sbk = sbk;
  g.ntile = ntile;
  g.kper = (int)((((int64_t)K + splits - 1) / splits + 63) / 64 * 64);
  g.epi = epi;
  g.C = C; g.ldc = ldc; g.split_stride = split_stride;
  g.bias = bias; g.act = act; g.ld_act = ld_act; g.hidden = hidden;
  g.zprev = zprev; g.ld_zprev = ld_zprev;
  g.rows_dev = rows_dev;
  g.err = err;
  g.tmem_cols = 32;
  while ((int)g.tmem_cols < ntile) g.tmem_cols <<= 1;
  const int zs = (int)(((int64_t)K + g.kper - 1) / g.kper);
  const int smem = 1024 + 2 * kM * 128 + 2 * ntile * 128 + 64;
  dim3 grid((N + ntile - 1) / ntile, mt, zs);
  cudaError_t e2 = cudaSuccess;
  switch (ntile) {
    case 256: e2 = run_tc<256>(grid, smem, g, s); break;
    case 128: e2 = run_tc<128>(grid, smem, g, s); break;
    case 64: e2 = run_tc<64>(grid, smem, g, s); break;
    default: return cudaErrorInvalidValue;
  }
  return e2;
}

cudaError_t launch_rowmin_tc(int M, int N, int K, const float* A, int64_t lda, const float* B, int64_t ldb,
                             const float* na, const float* nb, int64_t self_off, float* part, int64_t ldp,
                             const int64_t* rows_dev, const int64_t* cols_dev, int* parts_used, int* err, int sms,
                             cudaStream_t s) {
  if (M < 64 || N < 32 || K < 1) return cudaErrorInvalidValue;
  const int mt = (M + kM - 1) / kM;
  int ntile = 256;
  while (ntile > 64 && (int64_t)mt * ((N + ntile - 1) / ntile) < sms) ntile /= 2;
  while (ntile > 64 && ntile / 2 >= N) ntile /= 2;
  const int nt = (N + ntile - 1) / ntile;
  if (2 * nt > ldp) return cudaErrorInvalidValue;
  TcGemmArgs g{};
  g.M = M; g.N = N; g.K = K;
  g.A = A; g.sam = lda; g.sak = 1;
  g.B = B; g.sbn = ldb; g.sbk = 1;
  g.ntile = ntile;
  g.kper = (int)(((int64_t)K + 63) / 64 * 64);
  g.epi = 3;
  g.C = part; g.ldc = ldp;
  g.na = na; g.nb = nb; g.self_off = self_off;
  g.rows_dev = rows_dev; g.cols_dev = cols_dev;
  g.err = err;
  g.tmem_cols = 32;
  while ((int)g.tmem_cols < ntile) g.tmem_cols <<= 1;
  const int smem = 1024 + 2 * kM * 128 + 2 * ntile * 128 + 64;
  dim3 grid(nt, mt, 1);
  *parts_used = 2 * nt;
  switch (ntile) {
    case 256: return run_tc<256>(grid, smem, g, s);
    case 128: return run_tc<128>(grid, smem, g, s);
    case 64: return run_tc<64>(grid, smem, g, s);
    default: return cudaErrorInvalidValue;
  }
}

int gemm_tc_splits_used(int K, int splits) {
  const int64_t kper = ((((int64_t)K + splits - 1) / splits + 63) / 64) * 64;
  return (int)(((int64_t)K + kper - 1) / kper);
}

}  // namespace ls
