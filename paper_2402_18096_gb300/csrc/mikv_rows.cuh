// mikv_rows.cuh — warp-level building blocks shared by the standalone kernels and the fused step
// kernel: the (score, id) demotion order, the combination of split-attention partials and the
// importance weight of a slot.
#pragma once

#include "mikv_device.cuh"

namespace mikv {

// Total order of (score, id): ascending score, then ascending id. -0 is folded into +0.
__device__ __forceinline__ unsigned long long order_key(float s, int32_t id) {
  uint32_t u = __float_as_uint(s == 0.f ? 0.f : s);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (uint32_t)(id ^ (int32_t)0x80000000);
}

// Warp that owns unit U when n_units units are split into n_warps equal contiguous shares.
__device__ __forceinline__ int owner_warp(long long U, long long n_units, int n_warps) {
  int w = (int)(((U + 1) * n_warps - 1) / n_units);
  while (w > 0 && (long long)w * n_units / n_warps > U) --w;
  while (w + 1 < n_warps && (long long)(w + 1) * n_units / n_warps <= U) ++w;
  return w;
}

// The split partials of query head jh of KV head bh: warps w0..w1 of the attention kernel wrote slots
// w + bh, each a normalised output with its (max, sum). merge_stats_warp gives every lane (M, L) = (max
// logit, sum of exp(logit - M)); merge_output_warp gives lane l the output of channels 4l..4l+3, the
// partials weighted by exp(max - M) * sum, over L. The per-slot statistics are read by all lanes at once
// and broadcast with shuffles, so a merge costs a few dependent loads whatever the slot count.
__device__ __forceinline__ float merge_weight(const float* part_ml, int G, int bh, int jh, int w0, int i, float M) {
  constexpr float kLog2e = 1.4426950408889634f;
  const size_t slot = (size_t)(w0 + i + bh);
  const float ms = part_ml[(slot * G + jh) * 2];
  return ms == -INFINITY ? 0.f : fast_exp2((ms - M) * kLog2e) * part_ml[(slot * G + jh) * 2 + 1];
}

__device__ __forceinline__ void merge_stats_warp(const float* part_ml, int G, int bh, int jh, int w0, int w1, int lane,
                                                 float& M, float& L) {
  const int n = w1 - w0 + 1;
  M = -INFINITY;
  for (int c0 = 0; c0 < n; c0 += 32) {
    const int i = c0 + lane;
    if (i < n) M = fmaxf(M, part_ml[((size_t)(w0 + i + bh) * G + jh) * 2]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float Lp = 0.f;
  for (int c0 = lane; c0 < n; c0 += 32) Lp += merge_weight(part_ml, G, bh, jh, w0, c0, M);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Lp += __shfl_xor_sync(0xffffffffu, Lp, off);
  L = Lp;
}

__device__ __forceinline__ void merge_output_warp(const float* part_o, const float* part_ml, int G, int bh, int jh,
                                                  int w0, int w1, int lane, float M, float L, float (&out)[4]) {
  const int n = w1 - w0 + 1;
  float O[4] = {0.f, 0.f, 0.f, 0.f};
  for (int c0 = 0; c0 < n; c0 += 32) {
    const float wt = c0 + lane < n ? merge_weight(part_ml, G, bh, jh, w0, c0 + lane, M) : 0.f;
    const int cnt = min(32, n - c0);
    int k = 0;
    for (; k + 4 <= cnt; k += 4) {  // four partials' loads in flight, summed in slot order
      float4 po[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        po[u] = reinterpret_cast<const float4*>(part_o + ((size_t)(w0 + c0 + k + u + bh) * G + jh) * kHeadDim)[lane];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float ws = __shfl_sync(0xffffffffu, wt, k + u);
        O[0] += ws * po[u].x;
        O[1] += ws * po[u].y;
        O[2] += ws * po[u].z;
        O[3] += ws * po[u].w;
      }
    }
    for (; k < cnt; ++k) {
      const float ws = __shfl_sync(0xffffffffu, wt, k);
      const float4 po = reinterpret_cast<const float4*>(part_o + ((size_t)(w0 + c0 + k + bh) * G + jh) * kHeadDim)[lane];
      O[0] += ws * po.x;
      O[1] += ws * po.y;
      O[2] += ws * po.z;
      O[3] += ws * po.w;
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) out[i] = O[i] / L;
}

// Both steps at once when the head has at most NB partials: every load (each partial's statistics and output)
// is issued before any is used, so the merge costs one round of loads; the arithmetic, and its order, is that of
// merge_stats_warp followed by merge_output_warp, so the bits are the same. More partials take those two.
template <int NB>
__device__ __forceinline__ void merge_head_warp(const float* part_o, const float* part_ml, int G, int bh, int jh,
                                                int w0, int w1, int lane, float& M, float& L, float (&out)[4]) {
  constexpr float kLog2e = 1.4426950408889634f;
  const int n = w1 - w0 + 1;
  if (n > NB || n > 32) {
    merge_stats_warp(part_ml, G, bh, jh, w0, w1, lane, M, L);
    merge_output_warp(part_o, part_ml, G, bh, jh, w0, w1, lane, M, L, out);
    return;
  }
  float4 po[NB];
#pragma unroll
  for (int k = 0; k < NB; ++k)
    if (k < n) po[k] = __ldcg(reinterpret_cast<const float4*>(part_o + ((size_t)(w0 + k + bh) * G + jh) * kHeadDim) + lane);
  float ms = -INFINITY, ls = 0.f;
  if (lane < n) {
    const float2 v = __ldcg(reinterpret_cast<const float2*>(part_ml + ((size_t)(w0 + lane + bh) * G + jh) * 2));
    ms = v.x;
    ls = v.y;
  }
  M = ms;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  const float wt = lane < n && ms != -INFINITY ? fast_exp2((ms - M) * kLog2e) * ls : 0.f;
  float Lp = wt;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Lp += __shfl_xor_sync(0xffffffffu, Lp, off);
  L = Lp;
  float O[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int k = 0; k < NB; ++k) {
    if (k < n) {
      const float ws = __shfl_sync(0xffffffffu, wt, k);
      O[0] += ws * po[k].x;
      O[1] += ws * po[k].y;
      O[2] += ws * po[k].z;
      O[3] += ws * po[k].w;
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) out[i] = O[i] / L;
}

// Importance weight of one slot for one query head: exp(s - M) / L, as exp2((s - M) log2 e) times the
// reciprocal of L (the same arithmetic in the fused step tail and in mikv_update_importance).
__device__ __forceinline__ float importance_weight(float s, float M, float inv_L) {
  constexpr float kLog2e = 1.4426950408889634f;
  return fast_exp2((s - M) * kLog2e) * inv_L;
}

}  // namespace mikv
