// Weight publish (Sec. 4.3.1 P2: training never writes the weights routing
// reads; a new version becomes visible to routing in one atomic switch).
//
// One launch fills the buffer routes are not reading, 1 - st->cur, from the
// master weights:
//   params  fp32 flat copy, weights rounded to bf16 in bf16 mode, biases exact;
//   wt      per-layer transposed weights W^T [in, out] (CUDA-core scorer only);
//   img     bf16 hidden-layer weights pre-swizzled into the tensor-core operand
//           layout: N-chunks of nc rows x K-blocks of 64 columns, 128-byte
//           swizzle, one 16-byte chunk (8 columns) per thread.  For the pair
//           scorer a job is 256 output rows, rows 128 r .. 128 r + 127 of it
//           (an N-chunk, [128 x 64] per K-block: a 16 KB half-slice) belong to
//           rank r, and rank r's half-slices of a tile (the jobs of layer 1,
//           then of each later layer, K-blocks inner) are contiguous;
//   bounds  the staged feature bounds (Algorithm 4 [l, u]), lo [d] then hi [d].
// The last block to finish bumps the version and then flips st->cur, so a
// route that sees the new index sees a complete buffer.
#include "common.cuh"
#include "sm100.cuh"

namespace ls {
namespace {

struct PubArgs {
  MlpDesc m;
  const float* master;
  float* params[2];
  float* wt[2];
  uint8_t* img[2];
  float* bounds[2];
  const float* bounds_stage;
  int64_t n_bounds;                      // 2 d
  int64_t n_params;
  int64_t n_wt;                          // elements of the transposed copy (0: not kept)
  int n_tc;                              // tensor-core layers (0: no image)
  int in_pad[LS_MAX_LAYERS], nc[LS_MAX_LAYERS];
  int64_t img_off[LS_MAX_LAYERS];
  int64_t grp_end[LS_MAX_LAYERS];        // cumulative 8-column groups of the image, per layer
  int pair;                              // pair-scorer layout
  int pair_slices;                       // 16 KB half-slices per rank per tile
  int pair_q0[LS_MAX_LAYERS];            // first half-slice of layer l's jobs within a tile
  DevState* st;
};

__device__ __forceinline__ uint32_t bf16x2_bits(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__global__ void __launch_bounds__(256) k_publish(const __grid_constant__ PubArgs a) {
  const int cur = *reinterpret_cast<volatile int32_t*>(&a.st->cur);
  const int tgt = cur == 0 ? 1 : 0;
  const MlpDesc& m = a.m;
  float* __restrict__ pp = a.params[tgt];
  float* __restrict__ wt = a.wt[tgt];
  uint8_t* __restrict__ img = a.img[tgt];
  float* __restrict__ bnd = a.bounds[tgt];
  const int64_t n_img = a.n_tc ? a.grp_end[a.n_tc - 1] : 0;
  // work items: the flat parameters 4 at a time, then the transposed copy,
  // the image groups and the bounds one at a time
  const int64_t n_p4 = (a.n_params + 3) / 4;
  const int64_t total = n_p4 + a.n_wt + n_img + a.n_bounds;
  for (int64_t it = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; it < total;
       it += (int64_t)gridDim.x * blockDim.x) {
    const int64_t e = it - n_p4 + a.n_params;  // element index of the items past the parameters
    if (it < n_p4) {
      const int64_t e0 = 4 * it;
      float v[4];
      if (e0 + 4 <= a.n_params) {
        const float4 q = __ldg(reinterpret_cast<const float4*>(a.master + e0));
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] = e0 + j < a.n_params ? __ldg(a.master + e0 + j) : 0.0f;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t ej = e0 + j;
        int l = 0;
        while (l + 1 < m.n_layers && ej >= m.woff[l + 1]) ++l;
        if (m.bf16 && ej < m.boff[l]) v[j] = round_bf16(v[j]);
      }
      if (e0 + 4 <= a.n_params) {
        *reinterpret_cast<float4*>(pp + e0) = make_float4(v[0], v[1], v[2], v[3]);
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (e0 + j < a.n_params) pp[e0 + j] = v[j];
      }
    } else if (e < a.n_params + a.n_wt) {
      const int64_t t = e - a.n_params;
      int l = 0;
      while (l + 1 < m.n_layers && t >= m.wtoff[l + 1]) ++l;
      const int out = m.w[l + 1], in = m.w[l];
      const int64_t u = t - m.wtoff[l];
      const int k = (int)(u / out), o = (int)(u - (int64_t)k * out);
      const float v = __ldg(a.master + m.woff[l] + (int64_t)o * in + k);
      wt[t] = m.bf16 ? round_bf16(v) : v;
    } else if (e >= a.n_params + a.n_wt + n_img) {
      const int64_t t = e - (a.n_params + a.n_wt + n_img);
      bnd[t] = __ldg(a.bounds_stage + t);
    } else {
      const int64_t g = e - a.n_params - a.n_wt;
      int l = 0;
      while (g >= a.grp_end[l]) ++l;
      const int64_t gl = g - (l ? a.grp_end[l - 1] : 0);
      const int in = m.w[l], gpr = a.in_pad[l] / 8, nc = a.nc[l];
      const int o = (int)(gl / gpr), k0 = (int)(gl - (int64_t)o * gpr) * 8;
      const float* src = a.master + m.woff[l] + (int64_t)o * in;
      float v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = k0 + j < in ? __ldg(src + k0 + j) : 0.0f;
      const int nci = o / nc, orow = o - nci * nc;
      int64_t off;
      if (a.pair) {  // nc == 128: N-chunk nci is rank nci % 2's half of 256-column job nci / 2
        const int j = nci >> 1, r = nci & 1, nk = a.in_pad[l] / 64;
        const int q = a.pair_q0[l] + j * nk + (k0 >> 6);
        off = ((int64_t)r * a.pair_slices + q) * (128 * 128) + sm100::sw128_offset(orow, k0 & 63, 128);
      } else {
        off = a.img_off[l] + (int64_t)nci * (a.in_pad[l] / 64) * nc * 128 + sm100::sw128_offset(orow, k0, nc);
      }
      uint4 q;
      q.x = bf16x2_bits(v[0], v[1]);
      q.y = bf16x2_bits(v[2], v[3]);
      q.z = bf16x2_bits(v[4], v[5]);
      q.w = bf16x2_bits(v[6], v[7]);
      *reinterpret_cast<uint4*>(img + off) = q;
    }
  }
  // last_block: barrier, then thread 0 fences (cumulative over the block's
  // writes) before it arrives; the flip below comes after every block's writes
  if (last_block(&a.st->done[DONE_PUB]) && threadIdx.x == 0) {
    const uint64_t ver = a.st->version + 1;
    a.st->pub_version[tgt] = ver;
    a.st->version = ver;
    __threadfence();
    *reinterpret_cast<volatile int32_t*>(&a.st->cur) = tgt;
  }
}

}  // namespace

cudaError_t launch_publish(const MlpDesc& m, const TcPlan* tc, const float* master, const Published* pub,
                           int want_wt, const float* bounds_stage, DevState* st, int sms, cudaStream_t s) {
  PubArgs a{};
  a.m = m;
  a.master = master;
  for (int b = 0; b < 2; ++b) {
    a.params[b] = pub[b].params;
    a.wt[b] = pub[b].wt;
    a.img[b] = pub[b].img;
    a.bounds[b] = pub[b].bounds;
  }
  a.bounds_stage = bounds_stage;
  a.n_bounds = 2 * (int64_t)m.w[0];
  int64_t n_params = 0, n_wt = 0;
  for (int l = 0; l < m.n_layers; ++l) {
    n_params += (int64_t)m.w[l + 1] * m.w[l] + m.w[l + 1];
    n_wt += (int64_t)m.w[l + 1] * m.w[l];
  }
  a.n_params = n_params;
  a.n_wt = want_wt ? n_wt : 0;
  a.n_tc = tc ? tc->n_tc : 0;
  int64_t groups = 0;
  for (int l = 0; l < a.n_tc; ++l) {
    a.in_pad[l] = tc->in_pad[l];
    a.nc[l] = tc->nc[l];
    a.img_off[l] = tc->img_off[l];
    groups += (int64_t)tc->out[l] * (tc->in_pad[l] / 8);
    a.grp_end[l] = groups;
  }
  if (tc && tc->pair) {
    a.pair = 1;
    a.pair_slices = tc->pair_slices;
    int q0 = 0;
    for (int l = 0; l < tc->n_tc; ++l) {
      a.pair_q0[l] = q0;
      q0 += (tc->out[l] / 256) * (tc->in_pad[l] / 64);
    }
  }
  a.st = st;
  const int64_t total = (a.n_params + 3) / 4 + a.n_wt + groups + a.n_bounds;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((total + 255) / 256, (int64_t)sms * 4));
  k_publish<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace ls
