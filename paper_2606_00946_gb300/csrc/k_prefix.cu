// Prefix tracker kernels: block hashing, table inserts, and the fused
// hash + probe that yields the prefix hit length of every (request, instance)
// pair (Sec. 2: prefix reuse is strictly sequential; Sec. 4.1 Features (2)).
//
// Block key definition (this library's reading; the paper only says that
// gateways index cached prefixes with radix trees or hash tables, Sec. 2):
//   mix64  = SplitMix64 output finaliser;  G = 0x9E3779B97F4A7C15
//   c_b    = mix64( XOR_{j<8} mix64(w_{b,j} + (j+1) G) )       (content)
//   s_{-1} = G,  s_b = s_{b-1} * G + c_b  (mod 2^64)            (prefix state)
//   key_b  = mix64(s_b), 0 mapped to 1                           (table key)
// The prefix state is a linear recurrence, so a CTA computes the keys of 256
// consecutive blocks with one parallel scan instead of a serial chain.
#include <algorithm>
#include <climits>

#include "blockhash.cuh"

namespace ls {
namespace {
using namespace bh;

constexpr int kThreads = 256;           // threads per CTA = blocks per chunk
constexpr int kWarps = kThreads / 32;

// One CTA per sequence: keys of every full block.  Keys of sequence s go to
// keys_out[key_off[s] + b], or, with key_off == nullptr, to the slot
// floor((tok_off[s] - tok_off[0]) / 16) + b (distinct for every (s, b)
// because the blocks of a sequence lie inside its own token range); slots at
// or beyond `cap` are not written and latch LS_ERR_ARG.
// With tables != nullptr the CTA then screens block 0 of its request against
// every instance: h = 0 on a miss, h = 1 on a hit, and hits with more blocks
// join the work list of k_probe_walk.
template <int NT>
__global__ void __launch_bounds__(NT) k_hash_blocks(int n_seq, const int32_t* __restrict__ tok,
                                                    const int64_t* __restrict__ tok_off,
                                                    uint64_t* __restrict__ keys_out,
                                                    const int64_t* __restrict__ key_off, int64_t cap, int* err,
                                                    const uint64_t* __restrict__ tables, uint32_t mask,
                                                    int64_t slots, int n_inst, int32_t* __restrict__ hits,
                                                    uint32_t* __restrict__ work, int* work_n, DevState* st) {
  constexpr int W = NT / 32;
  __shared__ uint64_t wtot[W], wpre[W], carry, key0;
  route_snapshot(st);
  const int64_t tbase = tok_off[0];
  const int lane = threadIdx.x & 31;
  for (int s = blockIdx.x; s < n_seq; s += gridDim.x) {
    const int64_t t0 = tok_off[s];
    const int64_t nb = (tok_off[s + 1] - t0) / kBlockTok;
    const int32_t* base = tok + t0;
    const bool aligned = ((reinterpret_cast<uintptr_t>(base) & 15) == 0);
    const int64_t k0 = key_off ? key_off[s] : (t0 - tbase) / kBlockTok;
    uint64_t* out = keys_out + k0;
    if (!key_off && threadIdx.x == 0 && k0 + nb > cap) latch_error(err, LS_ERR_ARG);
    if (threadIdx.x == 0) carry = kG;
    __syncthreads();
    for (int64_t c0 = 0; c0 < nb; c0 += NT) {
      const int n = (int)(nb - c0 < NT ? nb - c0 : NT);
      const int t = threadIdx.x;
      const uint64_t s_in = carry;
      uint64_t c = t < n ? block_content(base + (c0 + t) * kBlockTok, aligned) : 0ull;
      uint64_t st = chain_scan<NT>(c, s_in, wtot, wpre);
      const uint64_t key = key_of(st);
      if (t < n && (key_off || k0 + c0 + t < cap)) out[c0 + t] = key;
      if (c0 == 0 && t == 0) key0 = key;
      if (t == n - 1) carry = st;
      __syncthreads();
    }
    if (tables) {
      const int64_t row = (int64_t)s * n_inst;
      for (int ib = 0; ib < n_inst; ib += NT) {
        const int i = ib + threadIdx.x;
        bool more = false;
        if (i < n_inst) {
          const bool hit = nb > 0 && k0 < cap && table_contains_v(tables + (int64_t)i * slots, mask, key0);
          hits[row + i] = hit ? 1 : 0;
          more = hit && nb > 1;
        }
        const unsigned bal = __ballot_sync(kFull, more);
        int slot = 0;
        if (lane == 0 && bal) slot = atomicAdd(work_n, __popc(bal));
        slot = __shfl_sync(kFull, slot, 0);
        if (more) work[slot + __popc(bal & ((1u << lane) - 1u))] = (uint32_t)(row + i);
      }
    }
    __syncthreads();
  }
}

// Pairs that hit block 0: one warp per pair walks blocks 1, 2, ... 32 at a
// time (32 independent lookups in flight); the first miss ends the walk.
__global__ void k_probe_walk(int n_inst, const int64_t* __restrict__ tok_off,
                             const uint64_t* __restrict__ keys, int64_t cap,
                             const uint64_t* __restrict__ tables, uint32_t mask, int64_t slots,
                             int32_t* __restrict__ hits, const uint32_t* __restrict__ work,
                             const int* __restrict__ work_n) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int n = *work_n;
  const int64_t tbase = tok_off[0];
  for (int64_t e = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; e < n; e += warps) {
    const uint32_t g = work[e];
    const int r = (int)(g / (uint32_t)n_inst), i = (int)(g - (uint32_t)r * (uint32_t)n_inst);
    const int64_t t0 = tok_off[r];
    const int64_t nb = (tok_off[r + 1] - t0) / kBlockTok;
    const int64_t k0 = (t0 - tbase) / kBlockTok;
    const uint64_t* tab = tables + (int64_t)i * slots;
    int64_t h = nb;
    for (int64_t p = 1; p < nb; p += 32) {
      const int64_t b = p + lane;
      const bool miss = b < nb && (k0 + b >= cap || !table_contains_v(tab, mask, keys[k0 + b]));
      const unsigned bal = __ballot_sync(kFull, miss);
      if (bal) {
        h = p + __ffs(bal) - 1;
        break;
      }
    }
    if (lane == 0) hits[g] = (int32_t)h;
  }
}

// Insert keys into per-instance tables.  Thread per key; the owning instance
// is found by binary search in key_off.  A table holding more than max_keys
// distinct keys, or a probe sequence that visits every slot, latches
// LS_ERR_TABLE_FULL (the loop is bounded by the table size).
__global__ void k_table_insert(const uint64_t* __restrict__ keys, const int64_t* __restrict__ key_off,
                               int n_inst, int64_t n_keys, uint64_t* tables, uint32_t mask,
                               int64_t slots, int32_t* counts, int64_t max_keys, int* err) {
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n_keys;
       k += (int64_t)gridDim.x * blockDim.x) {
    int lo = 0, hi = n_inst - 1;
    while (lo < hi) {
      int mid = (lo + hi + 1) >> 1;
      if (key_off[mid] <= k) lo = mid; else hi = mid - 1;
    }
    uint64_t key = keys[k];
    if (key == 0) key = 1;
    unsigned long long* tab = reinterpret_cast<unsigned long long*>(tables + (int64_t)lo * slots);
    uint32_t s = (uint32_t)key & mask;
    bool done = false;
    for (uint32_t n = 0; n <= mask; ++n) {
      unsigned long long prev = atomicCAS(tab + s, 0ull, (unsigned long long)key);
      if (prev == 0ull) {
        int cnt = atomicAdd(counts + lo, 1);
        if (cnt >= max_keys) latch_error(err, LS_ERR_TABLE_FULL);
        done = true;
        break;
      }
      if (prev == key) { done = true; break; }
      s = (s + 1) & mask;
    }
    if (!done) latch_error(err, LS_ERR_TABLE_FULL);
  }
}

// Fused hash + probe.  One CTA per request (grid-stride).  The request's
// blocks are hashed 256 at a time into shared memory; every instance still
// matching probes them, and hashing stops as soon as no instance matches.
//  - block 0 is screened with one probe per instance (most pairs end there);
//  - then, round by round, the instances still matching share the CTA's 256
//    threads: each gets a window of W = 256 / n_matching consecutive blocks
//    (power of two), all windows are probed at once, and the first miss of
//    each window is found with a shared-memory atomicMin.
__global__ void __launch_bounds__(kThreads) k_prefix_match(int n_req, const int32_t* __restrict__ tok,
                                                           const int64_t* __restrict__ tok_off,
                                                           const uint64_t* __restrict__ tables,
                                                           uint32_t mask, int64_t slots, int n_inst,
                                                           int32_t* __restrict__ hits, DevState* st) {
  __shared__ uint64_t keys[kThreads];
  route_snapshot(st);
  __shared__ uint64_t wtot[kWarps], wpre[kWarps], carry;
  __shared__ int n_alive, n_list;
  extern __shared__ int32_t dyn[];
  int32_t* hv = dyn;                  // [n_inst] hit length so far
  int32_t* dead = dyn + n_inst;       // [n_inst] 1 once the first miss is found
  int32_t* lst = dyn + 2 * n_inst;    // [n_inst] instances with work in this chunk
  int32_t* fm = dyn + 3 * n_inst;     // [n_inst] first miss of list entry k in this round
  const int t = threadIdx.x;

  for (int r = blockIdx.x; r < n_req; r += gridDim.x) {
    const int64_t t0 = tok_off[r];
    const int64_t nb = (tok_off[r + 1] - t0) / kBlockTok;
    const int32_t* base = tok + t0;
    const bool aligned = ((reinterpret_cast<uintptr_t>(base) & 15) == 0);
    for (int i = t; i < n_inst; i += kThreads) { hv[i] = 0; dead[i] = 0; }
    if (t == 0) { carry = kG; n_alive = n_inst; }
    __syncthreads();

    for (int64_t c0 = 0; c0 < nb; c0 += kThreads) {
      if (n_alive == 0) break;  // uniform: read after a barrier
      const int n = (int)(nb - c0 < kThreads ? nb - c0 : kThreads);
      const uint64_t s_in = carry;
      uint64_t c = t < n ? block_content(base + (c0 + t) * kBlockTok, aligned) : 0ull;
      uint64_t st = chain_scan<kThreads>(c, s_in, wtot, wpre);
      if (t < n) keys[t] = key_of(st);
      if (t == n - 1) carry = st;
      if (t == 0) n_list = 0;
      __syncthreads();

      if (c0 == 0) {
        for (int i = t; i < n_inst; i += kThreads) {
          const bool hit = table_contains_v(tables + (int64_t)i * slots, mask, keys[0]);
          hv[i] = hit ? 1 : 0;
          dead[i] = hit ? 0 : 1;
        }
        __syncthreads();
      }
      // list of instances still matching with blocks left in this chunk
      for (int i = t; i < n_inst; i += kThreads)
        if (!dead[i] && hv[i] < c0 + n) {
          const int k = atomicAdd(&n_list, 1);
          lst[k] = i;
          fm[k] = INT_MAX;
        }
      __syncthreads();
      while (n_list > 0) {
        const int nl = n_list;
        int logw = 0;
        while (logw < 8 && (nl << (logw + 1)) <= kThreads) ++logw;
        const int W = 1 << logw;
        for (int e = t; e < nl * W; e += kThreads) {
          const int k = e >> logw;
          const int i = lst[k];
          const int b = (int)(hv[i] - c0) + (e & (W - 1));
          if (b < n && !table_contains_v(tables + (int64_t)i * slots, mask, keys[b])) atomicMin(&fm[k], b);
        }
        __syncthreads();
        if (t == 0) n_list = 0;
        __syncthreads();
        for (int k = t; k < nl; k += kThreads) {
          const int i = lst[k];
          if (fm[k] != INT_MAX) {
            hv[i] = (int32_t)(c0 + fm[k]);
            dead[i] = 1;
          } else {
            const int64_t nv = (int64_t)hv[i] + W;
            hv[i] = (int32_t)(nv < c0 + n ? nv : c0 + n);
          }
        }
        __syncthreads();
        // next list: staged in fm (its values are consumed), then moved to lst
        for (int k = t; k < nl; k += kThreads) {
          const int i = lst[k];
          if (!dead[i] && hv[i] < c0 + n) fm[atomicAdd(&n_list, 1)] = i;
        }
        __syncthreads();
        const int nn = n_list;
        for (int k = t; k < nn; k += kThreads) {
          lst[k] = fm[k];
          fm[k] = INT_MAX;
        }
        __syncthreads();
      }
      if (t == 0) n_alive = 0;
      __syncthreads();
      int alive = 0;
      for (int i = t; i < n_inst; i += kThreads) alive += dead[i] ? 0 : 1;
      if (alive) atomicAdd(&n_alive, alive);
      __syncthreads();
    }
    for (int i = t; i < n_inst; i += kThreads) hits[(int64_t)r * n_inst + i] = hv[i];
    __syncthreads();
  }
}

int grid_for(int64_t n) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t g = n;
  const int64_t cap = (int64_t)sms * 16;
  return (int)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

cudaError_t launch_hash_blocks(int n_seq, const int32_t* tok, const int64_t* tok_off,
                               uint64_t* keys_out, const int64_t* key_off, int64_t cap, int* err,
                               cudaStream_t s) {
  if (n_seq <= 0) return cudaSuccess;
  k_hash_blocks<kThreads><<<grid_for(n_seq), kThreads, 0, s>>>(n_seq, tok, tok_off, keys_out, key_off, cap, err,
                                                             nullptr, 0, 0, 0, nullptr, nullptr, nullptr, nullptr);
  return cudaGetLastError();
}

cudaError_t launch_hash_screen(int n_req, const int32_t* tok, const int64_t* tok_off, uint64_t* keys,
                               int64_t cap, int* err, const uint64_t* tables, uint32_t mask, int64_t slots,
                               int n_inst, int32_t* hits, uint32_t* work, int* work_n, int sms,
                               DevState* st, cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  constexpr int NT = 128;
  const int grid = std::min(n_req, sms * 16);
  k_hash_blocks<NT><<<grid, NT, 0, s>>>(n_req, tok, tok_off, keys, nullptr, cap, err, tables, mask, slots, n_inst,
                                        hits, work, work_n, st);
  return cudaGetLastError();
}

cudaError_t launch_probe_walk(int n_inst, const int64_t* tok_off, const uint64_t* keys, int64_t cap,
                              const uint64_t* tables, uint32_t mask, int64_t slots, int32_t* hits,
                              const uint32_t* work, const int* work_n, int sms, cudaStream_t s) {
  k_probe_walk<<<sms * 8, 256, 0, s>>>(n_inst, tok_off, keys, cap, tables, mask, slots, hits, work, work_n);
  return cudaGetLastError();
}

cudaError_t launch_table_insert(const uint64_t* keys, const int64_t* key_off, int n_inst,
                                int64_t n_keys, uint64_t* tables, uint32_t mask, int64_t slots,
                                int32_t* counts, int64_t max_keys, int* err, cudaStream_t s) {
  if (n_keys <= 0 || n_inst <= 0) return cudaSuccess;
  int64_t blocks = (n_keys + 255) / 256;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (blocks > (int64_t)sms * 32) blocks = (int64_t)sms * 32;
  k_table_insert<<<(int)blocks, 256, 0, s>>>(keys, key_off, n_inst, n_keys, tables, mask, slots,
                                             counts, max_keys, err);
  return cudaGetLastError();
}

cudaError_t launch_prefix_match(int n_req, const int32_t* tok, const int64_t* tok_off,
                                const uint64_t* tables, uint32_t mask, int64_t slots, int n_inst,
                                int32_t* hits, DevState* st, cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  const size_t smem = (size_t)n_inst * 4 * sizeof(int32_t);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_prefix_match, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  k_prefix_match<<<grid_for(n_req), kThreads, smem, s>>>(n_req, tok, tok_off, tables, mask, slots,
                                                         n_inst, hits, st);
  return cudaGetLastError();
}

}  // namespace ls
