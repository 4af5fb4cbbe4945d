// ls_prefix_hits_static: prefix hit lengths with scratch taken from a static
// device array instead of a context's allocations.  Callers that cannot
// allocate while routing (stream capture, a latency-critical routing thread,
// a plugin whose host process owns all device memory) use it; every other
// caller uses the context path of ls_route_batch.  Same kernels as the
// two-phase prefix mode: hash + block-0 screen, then the walk.
#include <mutex>

#include "common.cuh"
#include "lodestar.h"

namespace ls {
namespace {

constexpr int64_t kStaticBlocks = LS_STATIC_MAX_BLOCKS;
constexpr int64_t kStaticPairs = LS_STATIC_MAX_PAIRS;
constexpr size_t kKeysBytes = (size_t)kStaticBlocks * sizeof(uint64_t);
constexpr size_t kWorkBytes = (size_t)kStaticPairs * sizeof(uint32_t);
static_assert(kKeysBytes % 256 == 0 && kWorkBytes % 256 == 0, "scratch parts keep 256-byte alignment");

// Layout: keys [kStaticBlocks] | work [kStaticPairs] | work_n, err (int32 each).
static __device__ __align__(256) unsigned char g_scratch[LS_STATIC_SCRATCH_BYTES];

struct DevScratch {
  unsigned char* base = nullptr;
  int sms = 0;
};
constexpr int kMaxDevices = 64;
std::mutex g_mu;
DevScratch g_dev[kMaxDevices];

// Address of this device's copy of g_scratch, looked up once per device (with
// that device current), and its SM count.
bool device_scratch(DevScratch& out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    set_last_error("ls_prefix_hits_static: no usable current device");
    return false;
  }
  std::lock_guard<std::mutex> g(g_mu);
  DevScratch& d = g_dev[dev];
  if (!d.base) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) {
      set_last_error("ls_prefix_hits_static: cudaGetSymbolAddress failed");
      return false;
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) {
      set_last_error("ls_prefix_hits_static: cannot read the SM count");
      return false;
    }
    d.base = static_cast<unsigned char*>(p);
    d.sms = sms;
  }
  out = d;
  return true;
}

}  // namespace
}  // namespace ls

extern "C" int ls_prefix_hits_static(int32_t n_req, const int32_t* tok, const int64_t* tok_off, int64_t n_tokens,
                                     const uint64_t* tables, int64_t slots_per_instance, int32_t n_inst,
                                     int32_t* hits_out, void* stream) {
  using namespace ls;
  if (n_req < 0 || n_inst < 1 || n_tokens < 0) {
    set_last_error("ls_prefix_hits_static: n_req >= 0, n_inst >= 1 and n_tokens >= 0 required");
    return LS_ERR_ARG;
  }
  if (n_req == 0) return LS_OK;
  if (!tok || !tok_off || !tables || !hits_out) {
    set_last_error("ls_prefix_hits_static: NULL argument");
    return LS_ERR_ARG;
  }
  if (slots_per_instance < 16 || slots_per_instance > (int64_t(1) << 31) ||
      (slots_per_instance & (slots_per_instance - 1)) != 0) {
    set_last_error("ls_prefix_hits_static: slots_per_instance must be a power of two in [16, 2^31]");
    return LS_ERR_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(tables) & 15) != 0) {
    set_last_error("ls_prefix_hits_static: tables must be 16-byte aligned");
    return LS_ERR_ARG;
  }
  if (n_tokens / LS_BLOCK_TOKENS > kStaticBlocks) {
    set_last_error("ls_prefix_hits_static: batch has more block keys than LS_STATIC_MAX_BLOCKS");
    return LS_ERR_ARG;
  }
  if ((int64_t)n_req * n_inst > kStaticPairs) {
    set_last_error("ls_prefix_hits_static: n_req * n_inst exceeds LS_STATIC_MAX_PAIRS");
    return LS_ERR_ARG;
  }
  DevScratch d;
  if (!device_scratch(d)) return LS_ERR_CUDA;
  uint64_t* keys = reinterpret_cast<uint64_t*>(d.base);
  uint32_t* work = reinterpret_cast<uint32_t*>(d.base + kKeysBytes);
  int* work_n = reinterpret_cast<int*>(d.base + kKeysBytes + kWorkBytes);
  int* err = work_n + 1;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const uint32_t mask = (uint32_t)(slots_per_instance - 1);
  cudaError_t e = cudaMemsetAsync(work_n, 0, 2 * sizeof(int), s);
  if (e == cudaSuccess)
    e = launch_hash_screen(n_req, tok, tok_off, keys, kStaticBlocks, err, tables, mask, slots_per_instance, n_inst,
                           hits_out, work, work_n, d.sms, nullptr, s);
  if (e == cudaSuccess)
    e = launch_probe_walk(n_inst, tok_off, keys, kStaticBlocks, tables, mask, slots_per_instance, hits_out, work,
                          work_n, d.sms, s);
  if (e != cudaSuccess) {
    set_last_error(cudaGetErrorString(e));
    return LS_ERR_CUDA;
  }
  return LS_OK;
}
