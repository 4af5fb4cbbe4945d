// Prefix index over all instances: one open-addressing table maps a block key
// to the bitmask of instances whose cache holds that block (the gateway's
// single logical prefix index of Sec. 4.2, in hash-table form as Sec. 2
// allows).  Hit lengths then need one lookup per (request, block) instead of
// one per (request, block, instance):
//   alive_b = AND_{b' <= b} mask(key_b')   (bits of instances still matching)
//   h_i     = number of leading blocks b with bit i of alive_b set
// which is exactly "leading blocks all cached on instance i, stop at the first
// miss" (Sec. 2: prefix reuse is strictly sequential).
//
// One warp per request: each round hashes the next 32 blocks of the prompt
// (one per lane; the chained prefix state is a warp-wide scan of the linear
// recurrence), looks the 32 keys up at once, and a warp-wide prefix AND of
// their instance masks gives, per lane, the instances still matching every
// block up to it.  An instance that stops matching in the round gets its hit
// length from one ballot; the lane that owns the instance keeps it and the
// row is written once, coalesced, at the end.  The walk stops at the first
// round after which no instance matches, so tokens past the longest hit plus
// one round are never read.  Walks differ in length by orders of magnitude,
// so warps take requests from a shared counter (a warp that finishes a short
// walk takes the next request) rather than a fixed share each.
#include "blockhash.cuh"
#include "sm100.cuh"

namespace ls {
namespace {
using namespace bh;

constexpr int kNT = 128;

// Slot of `key` in the index (linear probing in aligned 4-slot buckets), -1 if absent.
__device__ __forceinline__ int64_t index_find(const uint64_t* __restrict__ gkeys, uint64_t gmask_slots,
                                              uint64_t key) {
  uint64_t s = key & gmask_slots;
  uint32_t first = (uint32_t)(s & 3u);
  uint64_t b = s & ~(uint64_t)3;
  for (uint64_t n = 0; n <= (gmask_slots >> 2) + 1; ++n) {
    const ulonglong2* q = reinterpret_cast<const ulonglong2*>(gkeys + b);
    const ulonglong2 v01 = __ldg(q), v23 = __ldg(q + 1);
    const uint64_t v[4] = {v01.x, v01.y, v23.x, v23.y};
#pragma unroll
    for (uint32_t j = 0; j < 4; ++j) {
      if (j < first) continue;
      if (v[j] == key) return (int64_t)(b + j);
      if (v[j] == 0) return -1;
    }
    first = 0;
    b = (b + 4) & gmask_slots;
  }
  return -1;
}

// With one mask word (at most 64 instances) the index stores each key next to
// its mask, entry e = (ent[2e], ent[2e+1]) = (key, mask), so one 32-byte
// bucket of two entries answers a probe: mask of `key`, 0 if absent.
__device__ __forceinline__ uint64_t index_mask_w1(const uint64_t* __restrict__ ent, uint64_t mslots, uint64_t key) {
  uint64_t s = key & mslots;
  uint32_t first = (uint32_t)(s & 1);
  uint64_t b = s & ~(uint64_t)1;
  for (uint64_t n = 0; n <= (mslots >> 1) + 1; ++n) {
    const ulonglong2* q = reinterpret_cast<const ulonglong2*>(ent + 2 * b);
    const ulonglong2 e0 = __ldg(q), e1 = __ldg(q + 1);
    if (first == 0) {
      if (e0.x == key) return e0.y;
      if (e0.x == 0) return 0;
    }
    if (e1.x == key) return e1.y;
    if (e1.x == 0) return 0;
    first = 0;
    b = (b + 2) & mslots;
  }
  return 0;
}

template <int W>
__global__ void __launch_bounds__(kNT, W <= 4 ? 8 : 1) k_prefix_index(int n_req, const int32_t* __restrict__ tok,
                                                      const int64_t* __restrict__ tok_off,
                                                      const uint64_t* __restrict__ gkeys,
                                                      const uint64_t* __restrict__ gmask, uint64_t gmask_slots,
                                                      int n_inst, int32_t* __restrict__ hits, DevState* st) {
  sm100::pdl_wait();  // the previous kernel of the stream is complete
  route_snapshot(st);
  const int lane = threadIdx.x & 31;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  // G^(lane+1): the factor by which the state entering a round reaches lane
  // `lane` (kept in shared memory: one load per round, no registers held)
  __shared__ uint64_t s_glane[32];
  if (threadIdx.x < 32) {
    uint64_t g = 1, b = kG;
    for (unsigned e = (unsigned)lane + 1; e; e >>= 1) {
      if (e & 1) g *= b;
      b *= b;
    }
    s_glane[lane] = g;
  }
  __syncthreads();
  for (int64_t r = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; r < n_req;) {
    const int64_t t0 = tok_off[r];
    const int64_t nb = (tok_off[r + 1] - t0) / kBlockTok;
    const int32_t* base = tok + t0;
    const uintptr_t ab = reinterpret_cast<uintptr_t>(base);
    const int align = (ab & 15) == 0 ? 16 : (ab & 7) == 0 ? 8 : 4;
    uint64_t alive[W];
    int32_t hreg[W][2];  // hit length of instances 64w + lane and 64w + 32 + lane
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const int lo = 64 * w;
      alive[w] = n_inst >= lo + 64 ? ~0ull : (n_inst > lo ? ((1ull << (n_inst - lo)) - 1ull) : 0ull);
      hreg[w][0] = hreg[w][1] = 0;
    }
    uint64_t state = kG;  // s_{-1}
    bool any = n_inst > 0;
    // tokens of the lane's block in the coming round, requested one round
    // ahead so that their load overlaps the index probes of the current round
    uint32_t tw[16];
    if (lane < nb) block_load(base + (int64_t)lane * kBlockTok, align, tw);
    for (int64_t p = 0; p < nb && any; p += 32) {
      const int64_t b = p + lane;
      const bool in = b < nb;
      // inclusive scan: B = sum_{j <= lane} G^(lane - j) c_j, then s = G^(lane+1) s_in + B
      uint64_t B = in ? block_hash(tw) : 0ull;
      if (b + 32 < nb) block_load(base + (b + 32) * kBlockTok, align, tw);
#pragma unroll
      for (int k = 0; k < 5; ++k) {
        const int off = 1 << k;
        const uint64_t o = __shfl_up_sync(kFull, B, off);
        if (lane >= off) B = gpow(off) * o + B;
      }
      const uint64_t s = s_glane[lane] * state + B;
      const int last = (int)(nb - p < 32 ? nb - p : 32) - 1;
      state = __shfl_sync(kFull, s, last);
      uint64_t pa[W];
      if (in && W == 1) {
        pa[0] = index_mask_w1(gkeys, gmask_slots, key_of(s));
      } else if (in) {
        const int64_t slot = index_find(gkeys, gmask_slots, key_of(s));
#pragma unroll
        for (int w = 0; w < W; ++w) pa[w] = slot >= 0 ? __ldg(gmask + slot * W + w) : 0ull;
      } else {
#pragma unroll
        for (int w = 0; w < W; ++w) pa[w] = 0ull;
      }
      any = false;
#pragma unroll
      for (int w = 0; w < W; ++w) {
        uint64_t x = pa[w];
#pragma unroll
        for (int k = 0; k < 5; ++k) {
          const uint64_t y = __shfl_up_sync(kFull, x, 1 << k);
          if (lane >= (1 << k)) x &= y;
        }
        x &= alive[w];
        const uint64_t end = __shfl_sync(kFull, x, 31);
        uint64_t died = alive[w] & ~end;
        while (died) {
          const int bit = __ffsll((long long)died) - 1;
          const int cnt = __popc(__ballot_sync(kFull, (x >> bit) & 1ull));
          if (lane == (bit & 31)) {
            if (bit >> 5) hreg[w][1] = (int32_t)(p + cnt);
            else hreg[w][0] = (int32_t)(p + cnt);
          }
          died &= died - 1;
        }
        alive[w] = end;
        any = any || end != 0;
      }
    }
    int32_t* hrow = hits + (int64_t)r * n_inst;
#pragma unroll
    for (int w = 0; w < W; ++w)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int bit = 32 * h + lane, i = 64 * w + bit;
        // instances matching every full block (or requests without a full block)
        if (i < n_inst) hrow[i] = ((alive[w] >> bit) & 1ull) ? (int32_t)nb : hreg[w][h];
      }
    // the next request: from the counter (after each warp's first), else a fixed stride
    if (st) {
      uint32_t nx = 0;
      if (lane == 0) nx = atomicAdd(&st->walk_next, 1u);
      r = warps + (int64_t)__shfl_sync(kFull, nx, 0);
    } else {
      r += warps;
    }
  }
  // the counter starts at 0 for the next walk: reset by the last block to finish
  if (st && last_block(&st->done[DONE_WALK]) && threadIdx.x == 0) st->walk_next = 0u;
  sm100::pdl_trigger();  // the next kernel may start once every CTA is here
}

// Insert (instance, key) pairs: thread per key, instance by binary search in
// key_off.  A new key takes a slot (CAS on 0); the instance's bit is OR-ed into
// the slot's mask; a bit set for the first time counts one distinct key of
// that instance (more than max_keys latches LS_ERR_TABLE_FULL, as does a
// probe sequence that finds no room).  With W == 1 keys and masks share the
// interleaved entry array gkeys (gmask unused).
__global__ void k_index_insert(const uint64_t* __restrict__ keys, const int64_t* __restrict__ key_off,
                               int n_inst, int64_t n_keys, uint64_t* gkeys, uint64_t* gmask, int W,
                               uint64_t gmask_slots, int32_t* counts, int64_t max_keys, int* err) {
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n_keys;
       k += (int64_t)gridDim.x * blockDim.x) {
    int lo = 0, hi = n_inst - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (key_off[mid] <= k) lo = mid; else hi = mid - 1;
    }
    uint64_t key = keys[k];
    if (key == 0) key = 1;
    unsigned long long* tab = reinterpret_cast<unsigned long long*>(gkeys);
    const int kstride = W == 1 ? 2 : 1;
    uint64_t s = key & gmask_slots;
    int64_t slot = -1;
    for (uint64_t n = 0; n <= gmask_slots; ++n) {
      const unsigned long long prev = atomicCAS(tab + s * kstride, 0ull, (unsigned long long)key);
      if (prev == 0ull || prev == key) { slot = (int64_t)s; break; }
      s = (s + 1) & gmask_slots;
    }
    if (slot < 0) { latch_error(err, LS_ERR_TABLE_FULL); continue; }
    const unsigned long long bit = 1ull << (lo & 63);
    unsigned long long* mword = W == 1 ? tab + 2 * slot + 1
                                       : reinterpret_cast<unsigned long long*>(gmask + slot * W + (lo >> 6));
    const unsigned long long old = atomicOr(mword, bit);
    if (!(old & bit)) {
      const int cnt = atomicAdd(counts + lo, 1);
      if (cnt >= max_keys) latch_error(err, LS_ERR_TABLE_FULL);
    }
  }
}

}  // namespace

int index_words(int max_instances) { return max_instances <= 64 ? 1 : max_instances <= 128 ? 2 : max_instances <= 256 ? 4 : max_instances <= 512 ? 8 : 0; }

cudaError_t launch_prefix_index(int n_req, const int32_t* tok, const int64_t* tok_off, const uint64_t* gkeys,
                                const uint64_t* gmask, int W, uint64_t gmask_slots, int n_inst, int32_t* hits,
                                int sms, DevState* st, cudaStream_t s) {
  if (n_req <= 0) return cudaSuccess;
  void (*k)(int, const int32_t*, const int64_t*, const uint64_t*, const uint64_t*, uint64_t, int, int32_t*,
            DevState*) = nullptr;
  switch (W) {
    case 1: k = k_prefix_index<1>; break;
    case 2: k = k_prefix_index<2>; break;
    case 4: k = k_prefix_index<4>; break;
    case 8: k = k_prefix_index<8>; break;
    default: return cudaErrorInvalidValue;
  }
  // as many warps as are resident at once (they then take requests from the
  // counter); with no state to keep the counter in, one warp per request
  static int resident[9] = {};
  if (!resident[W]) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kNT, 0) != cudaSuccess || per_sm < 1) {
      cudaGetLastError();
      per_sm = 1;
    }
    resident[W] = per_sm;
  }
  const int want = (n_req + kNT / 32 - 1) / (kNT / 32);
  const int grid = std::max(1, std::min(want, st ? sms * resident[W] : sms * 16));
  return launch_chained(k, dim3(grid), dim3(kNT), 0, s, 1, n_req, tok, tok_off, gkeys, gmask, gmask_slots, n_inst,
                        hits, st);
}

cudaError_t launch_index_insert(const uint64_t* keys, const int64_t* key_off, int n_inst, int64_t n_keys,
                                uint64_t* gkeys, uint64_t* gmask, int W, uint64_t gmask_slots, int32_t* counts,
                                int64_t max_keys, int* err, int sms, cudaStream_t s) {
  if (n_keys <= 0 || n_inst <= 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((n_keys + 255) / 256, (int64_t)sms * 32);
  k_index_insert<<<(int)blocks, 256, 0, s>>>(keys, key_off, n_inst, n_keys, gkeys, gmask, W, gmask_slots, counts,
                                             max_keys, err);
  return cudaGetLastError();
}

}  // namespace ls
