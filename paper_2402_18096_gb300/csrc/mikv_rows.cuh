// mikv_rows.cuh — warp-level building blocks shared by the standalone kernels and the fused step
// kernel: Eq. 1 quantization of one 128-channel row into the packed layout, the (score, id) demotion
// order, and the combination of split-attention partials.
#pragma once

#include "mikv_device.cuh"

namespace mikv {

// Bit position of channel c (= 16 m + u) in a plane of f-bit fields: 16-bit unit and bit offset.
__device__ __forceinline__ void field_pos(int c, int f, int& unit, int& bit) {
  const int u = c & 15, m = c >> 4;
  if (f == 1) {
    unit = u & 7;
    bit = 8 * (u >> 3) + m;
  } else {
    const int P = 16 / f;
    unit = 8 * (2 * (m / P) + (u >> 3)) + (u & 7);
    bit = f * (m % P);
  }
}

// Quantize one row (Eq. 1) held as fp32 values x[4] of channels 4 lane .. 4 lane + 3 of each lane, with
// one warp. Writes 16 * BITS bytes of packed codes to `codes` and 128 / GROUP (alpha, beta) fp16 pairs to
// `params`. `buf` is 32 words of this warp's shared memory. Every rounding is explicit (fsub/fdiv
// round-to-nearest, fp16 round-down / round-up, round-half-even to int), so codes and parameters are
// bit-identical to an IEEE fp32 evaluation. BITS in {2, 3, 4, 8}.
template <int BITS, int GROUP>
__device__ __forceinline__ void quantize_values_warp(const float (&x)[4], uint8_t* codes, __half2* params,
                                                     uint32_t* buf, int lane) {
  constexpr int QMAX = (1 << BITS) - 1;
  constexpr int LANES = GROUP / 4;  // lanes per quantization group
  constexpr int WORDS = 4 * BITS;   // 32-bit words of one packed row
  if (lane < WORDS) buf[lane] = 0u;
  __syncwarp();
  float mn = fminf(fminf(x[0], x[1]), fminf(x[2], x[3]));
  float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
#pragma unroll
  for (int off = 1; off < LANES; off <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  // Eq. 1: beta = min, alpha = (max - min) / (2^N - 1), stored in fp16 with outward rounding.
  const __half beta16 = __float2half_rd(mn);
  const float beta = __half2float(beta16);
  const float span = __fsub_rn(mx, beta);
  const __half alpha16 = span == 0.f ? __float2half_rn(1.f) : __float2half_ru(__fdiv_rn(span, (float)QMAX));
  const float alpha = __half2float(alpha16);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    int code = __float2int_rn(__fdiv_rn(__fsub_rn(x[e], beta), alpha));
    code = code < 0 ? 0 : (code > QMAX ? QMAX : code);
    const int c = 4 * lane + e;
    int unit, bit;
    field_pos(c, BITS == 3 ? 2 : BITS, unit, bit);
    const uint32_t fmask = BITS == 3 ? 3u : (uint32_t)QMAX;
    atomicOr(&buf[unit >> 1], (((uint32_t)code & fmask) << bit) << (16 * (unit & 1)));
    if (BITS == 3) {
      field_pos(c, 1, unit, bit);
      atomicOr(&buf[8 + (unit >> 1)], (((uint32_t)code >> 2) << bit) << (16 * (unit & 1)));
    }
  }
  __syncwarp();
  if (lane < WORDS) reinterpret_cast<uint32_t*>(codes)[lane] = buf[lane];
  if ((lane & (LANES - 1)) == 0) params[(4 * lane) / GROUP] = __halves2half2(alpha16, beta16);
}

// Quantize one bf16 row (Eq. 1, Eq. 3): lane l owns channels 4l..4l+3 of `src`; keys pass `bal` (fp32
// [128], or nullptr = 1), multiplied in before the quantizer.
template <int BITS, int GROUP>
__device__ __forceinline__ void quantize_row_warp(const __nv_bfloat16* src, const float* bal, uint8_t* codes,
                                                  __half2* params, uint32_t* buf, int lane) {
  const uint2 raw = *reinterpret_cast<const uint2*>(src + 4 * lane);
  float x[4] = {__uint_as_float(raw.x << 16), __uint_as_float(raw.x & 0xffff0000u),
                __uint_as_float(raw.y << 16), __uint_as_float(raw.y & 0xffff0000u)};
  if (bal) {  // Eq. 3: keys times the balancer before the quantizer
    const float4 b = *reinterpret_cast<const float4*>(bal + 4 * lane);
    x[0] = __fmul_rn(x[0], b.x);
    x[1] = __fmul_rn(x[1], b.y);
    x[2] = __fmul_rn(x[2], b.z);
    x[3] = __fmul_rn(x[3], b.w);
  }
  quantize_values_warp<BITS, GROUP>(x, codes, params, buf, lane);
}

// fp32 dequantization of channels 4 lane .. 4 lane + 3 of one packed row of `bits`-bit codes (bits in
// {2, 4, 8}, one plane) with (alpha, beta) per group of `group` channels: x = alpha * code + beta, the
// product exact in fp32 and the sum rounded once (one fma).
__device__ __forceinline__ void dequantize_values_warp(const uint8_t* codes, const __half2* params, int bits,
                                                       int group, int lane, float (&x)[4]) {
  const uint16_t* units = reinterpret_cast<const uint16_t*>(codes);
  const uint32_t mask = (1u << bits) - 1u;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int c = 4 * lane + e;
    int unit, bit;
    field_pos(c, bits, unit, bit);
    const uint32_t code = ((uint32_t)units[unit] >> bit) & mask;
    const float2 ab = __half22float2(params[c / group]);
    x[e] = __fmaf_rn(ab.x, (float)code, ab.y);
  }
}

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

// Importance weight of one slot for one query head: exp(s - M) / L, as exp2((s - M) log2 e) times the
// reciprocal of L (the same arithmetic in the fused step tail and in mikv_update_importance).
__device__ __forceinline__ float importance_weight(float s, float M, float inv_L) {
  constexpr float kLog2e = 1.4426950408889634f;
  return fast_exp2((s - M) * kLog2e) * inv_L;
}

}  // namespace mikv
