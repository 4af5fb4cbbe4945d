// Block-hash and table-lookup device helpers shared by the prefix kernels.
//   mix64  = SplitMix64 output finaliser;  G = 0x9E3779B97F4A7C15
//   c_b    = mix64( XOR_{j<8} mix64(w_{b,j} + (j+1) G) )       (content)
//   s_{-1} = G,  s_b = s_{b-1} * G + c_b  (mod 2^64)            (prefix state)
//   key_b  = mix64(s_b), 0 mapped to 1                           (table key)
#pragma once

#include "common.cuh"

namespace ls {
namespace bh {

constexpr unsigned kFull = 0xffffffffu;

__host__ __device__ constexpr uint64_t gpow(uint64_t e) {
  uint64_t r = 1, b = kG;
  while (e) {
    if (e & 1) r *= b;
    b *= b;
    e >>= 1;
  }
  return r;
}

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t word_mix(uint32_t lo, uint32_t hi, int j) {
  uint64_t w = (uint64_t)lo | ((uint64_t)hi << 32);
  return mix64(w + (uint64_t)(j + 1) * kG);
}

// Content hash of the 16 tokens at p.  `aligned`: p is 16-byte aligned.
__device__ __forceinline__ uint64_t block_content(const int32_t* p, bool aligned) {
  uint64_t acc = 0;
  if (aligned) {
    const int4* q = reinterpret_cast<const int4*>(p);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      int4 t = __ldg(q + v);
      acc ^= word_mix((uint32_t)t.x, (uint32_t)t.y, 2 * v);
      acc ^= word_mix((uint32_t)t.z, (uint32_t)t.w, 2 * v + 1);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      acc ^= word_mix((uint32_t)__ldg(p + 2 * j), (uint32_t)__ldg(p + 2 * j + 1), j);
  }
  return mix64(acc);
}

// The same content hash in two steps, so that a block's tokens can be
// requested well before they are hashed.  `align`: 16, 8 or 4, the largest
// power of two (up to 16) dividing the byte address of p.
__device__ __forceinline__ void block_load(const int32_t* p, int align, uint32_t (&w)[16]) {
  if (align == 16) {
    const int4* q = reinterpret_cast<const int4*>(p);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int4 t = __ldg(q + v);
      w[4 * v] = (uint32_t)t.x;
      w[4 * v + 1] = (uint32_t)t.y;
      w[4 * v + 2] = (uint32_t)t.z;
      w[4 * v + 3] = (uint32_t)t.w;
    }
  } else if (align == 8) {
    const int2* q = reinterpret_cast<const int2*>(p);
#pragma unroll
    for (int v = 0; v < 8; ++v) {
      const int2 t = __ldg(q + v);
      w[2 * v] = (uint32_t)t.x;
      w[2 * v + 1] = (uint32_t)t.y;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 16; ++j) w[j] = (uint32_t)__ldg(p + j);
  }
}
__device__ __forceinline__ uint64_t block_hash(const uint32_t (&w)[16]) {
  uint64_t acc = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) acc ^= word_mix(w[2 * j], w[2 * j + 1], j);
  return mix64(acc);
}

// Prefix state after this thread's block, for a chunk whose first block
// follows state s_in.  Thread t holds content c (0 for threads past the last
// block: they come after every real block, so they change nothing).
// Inclusive scan of B_t = sum_{j<=t} G^(t-j) c_j, state_t = G^(t+1) s_in + B_t.
template <int NT>
__device__ __forceinline__ uint64_t chain_scan(uint64_t c, uint64_t s_in, uint64_t* wtot,
                                               uint64_t* wpre) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint64_t B = c;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const int off = 1 << k;
    uint64_t o = __shfl_up_sync(kFull, B, off);
    if (lane >= off) B = gpow(off) * o + B;  // left span times G^(right span)
  }
  if (lane == 31) wtot[warp] = B;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint64_t e = s_in;
    for (int w = 0; w < NT / 32; ++w) {
      wpre[w] = e;
      e = gpow(32) * e + wtot[w];
    }
  }
  __syncthreads();
  uint64_t gl = 1, base = kG;  // G^(lane+1)
  for (unsigned e = (unsigned)lane + 1; e; e >>= 1) {
    if (e & 1) gl *= base;
    base *= base;
  }
  return gl * wpre[warp] + B;
}

__device__ __forceinline__ uint64_t key_of(uint64_t state) {
  uint64_t k = mix64(state);
  return k ? k : 1ull;
}

// Open-addressing membership (linear probing from key & mask, 0 = empty slot),
// read one aligned 32-byte bucket (4 slots, two 16-byte loads) per step: the
// probe sequence from slot s is s, s+1, ... so only slots at or after s count
// in the first bucket, which is visited again in full if the walk wraps
// around.  Tables have >= 16 slots.
__device__ __forceinline__ bool table_contains_v(const uint64_t* __restrict__ tab, uint32_t mask,
                                                 uint64_t key) {
  uint32_t s = (uint32_t)key & mask;
  uint32_t first = s & 3u;
  uint32_t b = s & ~3u;
  for (uint32_t n = 0; n <= (mask >> 2) + 1; ++n) {
    const ulonglong2* q = reinterpret_cast<const ulonglong2*>(tab + b);
    const ulonglong2 v01 = __ldg(q), v23 = __ldg(q + 1);
    const uint64_t v[4] = {v01.x, v01.y, v23.x, v23.y};
#pragma unroll
    for (uint32_t j = 0; j < 4; ++j) {
      if (j < first) continue;
      if (v[j] == key) return true;
      if (v[j] == 0) return false;
    }
    first = 0;
    b = (b + 4) & mask;
  }
  return false;
}

}  // namespace bh
}  // namespace ls
