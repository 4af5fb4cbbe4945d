// Measurement kernels for the roofline ceilings (random 8-byte gathers, fp32
// FMA issue, streaming reads); declared in lodestar_probe.h.  Not part of the
// routing path.
#include "blockhash.cuh"
#include "common.cuh"
#include "lodestar.h"
#include "lodestar_probe.h"

namespace ls {
namespace {

constexpr int kProbeThreads = 256;

__global__ void __launch_bounds__(kProbeThreads) k_probe_gather(const uint64_t* __restrict__ table, uint64_t mask,
                                                                 int per_thread, uint64_t seed, uint64_t* out) {
  const uint64_t t = (uint64_t)blockIdx.x * kProbeThreads + threadIdx.x;
  const uint64_t stride = (uint64_t)gridDim.x * kProbeThreads;
  uint64_t acc = 0;
  for (int i = 0; i < per_thread; i += 8) {
    uint64_t v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint64_t g = (uint64_t)(i + u) * stride + t;
      v[u] = i + u < per_thread ? __ldcg(table + (bh::mix64(seed + g) & mask)) : 0;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) acc ^= v[u];
  }
  out[t] = acc;
}

__global__ void __launch_bounds__(kProbeThreads) k_probe_fma(int64_t iters, float* out) {
  const int t = blockIdx.x * kProbeThreads + threadIdx.x;
  float a[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) a[u] = (float)(t + u) * 1e-7f;
  const float m = 0.999999f, c = 1e-7f;
  for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < 8; ++u) a[u] = fmaf(a[u], m, c);
  }
  float s = 0.0f;
#pragma unroll
  for (int u = 0; u < 8; ++u) s += a[u];
  out[t] = s;
}

__global__ void __launch_bounds__(kProbeThreads) k_probe_read(const uint4* __restrict__ buf, int64_t n16, int passes,
                                                               uint4* out) {
  const int64_t t = (int64_t)blockIdx.x * kProbeThreads + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * kProbeThreads;
  uint4 acc = make_uint4(0u, 0u, 0u, 0u);
  for (int p = 0; p < passes; ++p) {
    for (int64_t i = t; i < n16; i += 4 * stride) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = i + u * stride < n16 ? __ldcg(buf + i + u * stride) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        acc.x ^= v[u].x;
        acc.y ^= v[u].y;
        acc.z ^= v[u].z;
        acc.w ^= v[u].w;
      }
    }
  }
  out[t] = acc;
}

int probe_fail(const char* msg) {
  set_last_error(msg);
  return LS_ERR_ARG;
}

int launched() {
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return LS_OK;
  set_last_error(cudaGetErrorString(e));
  return LS_ERR_CUDA;
}

}  // namespace
}  // namespace ls

extern "C" {

int ls_probe_gather(const uint64_t* table, int64_t n_slots, int32_t blocks, int32_t per_thread, uint64_t seed,
                    uint64_t* out, void* stream) {
  if (!table || !out || n_slots < 2 || (n_slots & (n_slots - 1)) != 0 || blocks < 1 || per_thread < 1)
    return ls::probe_fail("ls_probe_gather: bad argument");
  ls::k_probe_gather<<<blocks, ls::kProbeThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      table, (uint64_t)(n_slots - 1), per_thread, seed, out);
  return ls::launched();
}

int ls_probe_fma(int32_t blocks, int64_t iters, float* out, void* stream) {
  if (!out || blocks < 1 || iters < 1) return ls::probe_fail("ls_probe_fma: bad argument");
  ls::k_probe_fma<<<blocks, ls::kProbeThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(iters, out);
  return ls::launched();
}

int ls_probe_read(const void* buf, int64_t n16, int32_t passes, int32_t blocks, void* out, void* stream) {
  if (!buf || !out || n16 < 1 || passes < 1 || blocks < 1 || (reinterpret_cast<uintptr_t>(buf) & 15))
    return ls::probe_fail("ls_probe_read: bad argument");
  ls::k_probe_read<<<blocks, ls::kProbeThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint4*>(buf), n16, passes, static_cast<uint4*>(out));
  return ls::launched();
}

}  // extern "C"
