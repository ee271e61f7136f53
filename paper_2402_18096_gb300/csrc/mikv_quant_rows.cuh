// mikv_quant_rows.cuh — Eq. 1 quantization into the packed retained layout (group-wise asymmetric codes
// with fp16 scale and zero, keys times the Eq. 3 balancer): the scale / zero / code helpers every
// quantizer uses (so the bulk kernel, the fused step tail and the coded important set produce the same
// bits), the one-warp-per-row quantizer of a single 128-channel row, and the fp32 dequantization of a
// coded important row (Sec. 3.3).
#pragma once

#include "mikv_device.cuh"

namespace mikv {

// Bit position of channel c (= 16 m + u) in a plane of f-bit fields: 16-bit unit and bit offset.
__device__ __forceinline__ void field_pos(int c, int f, int& unit, int& bit) {
  const int u = c & 15, m = c >> 4;
  if (f == 1) {  // the two channels u and u + 8 of a unit alternate: their bits for m sit at 2 m and 2 m + 1
    unit = u & 7;
    bit = 2 * m + (u >> 3);
  } else {
    const int P = 16 / f;
    unit = 8 * (2 * (m / P) + (u >> 3)) + (u & 7);
    bit = f * (m % P);
  }
}

// Packs four F-bit fields (channels 4 lane .. 4 lane + 3, field values in code[]) into the row's 32-bit
// words at `row`. In the layout of field_pos the fields of channels 4 lane and 4 lane + 1 fall into one
// word and those of 4 lane + 2 and 4 lane + 3 into the next, for every F the layout uses (1, 2, 4, 8);
// the lanes that share that pair of words differ only in the lane bits of R, so an OR butterfly over
// those bits assembles the words, and the lanes with those bits clear store them (8 bytes each).
template <int F>
__device__ __forceinline__ void pack_fields(const uint32_t (&code)[4], uint32_t* row, int lane) {
  constexpr int R = F == 1 ? 0x1E : F == 2 ? 0x1C : F == 4 ? 0x0C : 0x04;
  uint32_t w0 = 0u, w1 = 0u;
  int word0 = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    int unit, bit;
    field_pos(4 * lane + e, F, unit, bit);
    if (e == 0) word0 = unit >> 1;
    const uint32_t f = code[e] << (bit + 16 * (unit & 1));
    if (e < 2)
      w0 |= f;
    else
      w1 |= f;
  }
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    if (R & off) {
      w0 |= __shfl_xor_sync(0xffffffffu, w0, off);
      w1 |= __shfl_xor_sync(0xffffffffu, w1, off);
    }
  }
  if ((lane & R) == 0) *reinterpret_cast<uint2*>(row + word0) = make_uint2(w0, w1);
}

// Eq. 1 scale and zero of a group with minimum mn and maximum mx: beta = min, alpha = (max - min) /
// (2^N - 1), stored in fp16 with outward rounding (beta down, alpha up) so the stored grid covers the
// group; a group with zero span gets alpha = 1 (every code 0). Also the fp32 values of the stored pair
// and the IEEE reciprocal of alpha.
struct Eq1Params {
  __half alpha16, beta16;
  float alpha, beta, ralpha;
};

template <int QMAX>
__device__ __forceinline__ Eq1Params eq1_params(float mn, float mx) {
  Eq1Params p;
  p.beta16 = __float2half_rd(mn);
  p.beta = __half2float(p.beta16);
  const float span = __fsub_rn(mx, p.beta);
  p.alpha16 = span == 0.f ? __float2half_rn(1.f) : __float2half_ru(__fdiv_rn(span, (float)QMAX));
  p.alpha = __half2float(p.alpha16);
  p.ralpha = __frcp_rn(p.alpha);
  return p;
}

// Eq. 1 code of x: round-half-even of the IEEE quotient (x - beta) / alpha, clamped to [0, QMAX].
// eq1_code_fast takes the product (x - beta) * (1 / alpha) (both factors IEEE-rounded), which lies within
// 2^-15 of the true quotient for quotients below 256 while the IEEE quotient lies within 2^-17 of it, and
// rounds it half to even by adding 2^23 (the fp32 sum is an integer; its low mantissa bits are the code).
// The two agree unless the product is within 2^-13 of a half-integer (or not finite): such elements set
// `redo`, and eq1_code_exact decides them with the division.
template <int QMAX>
__device__ __forceinline__ uint32_t eq1_code_fast(float x, const Eq1Params& p, bool& redo) {
  const float q = __fmul_rn(__fsub_rn(x, p.beta), p.ralpha);
  const float y = __fadd_rn(q, 8388608.f);
  const float fr = __fsub_rn(q, __fsub_rn(y, 8388608.f));  // q - rint(q), exact
  redo |= !(fabsf(fr) < 0.5f - 0x1p-13f);
  return min(__float_as_uint(y) - 0x4B000000u, (uint32_t)QMAX);
}

template <int QMAX>
__device__ __forceinline__ uint32_t eq1_code_exact(float x, const Eq1Params& p) {
  const int c = __float2int_rn(__fdiv_rn(__fsub_rn(x, p.beta), p.alpha));
  return (uint32_t)(c < 0 ? 0 : (c > QMAX ? QMAX : c));
}

// Quantize one row (Eq. 1) held as fp32 values x[4] of channels 4 lane .. 4 lane + 3 of each lane, with
// one warp. Writes 16 * BITS bytes of packed codes to `codes` (8-byte aligned) and 128 / GROUP
// (alpha, beta) fp16 pairs to `params`. Every rounding is explicit (fsub/fdiv round-to-nearest, fp16
// round-down / round-up, round-half-even to int), so codes and parameters are bit-identical to an IEEE
// fp32 evaluation of Eq. 1. BITS in {2, 3, 4, 8}; 3-bit codes are two planes (low 2 bits, then the high bit).
template <int BITS, int GROUP>
__device__ __forceinline__ void quantize_values_warp(const float (&x)[4], uint8_t* codes, __half2* params,
                                                     int lane) {
  constexpr int QMAX = (1 << BITS) - 1;
  constexpr int LANES = GROUP / 4;  // lanes per quantization group
  float mn = fminf(fminf(x[0], x[1]), fminf(x[2], x[3]));
  float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
#pragma unroll
  for (int off = 1; off < LANES; off <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  const Eq1Params p = eq1_params<QMAX>(mn, mx);
  uint32_t code[4];
  bool redo = false;
#pragma unroll
  for (int e = 0; e < 4; ++e) code[e] = eq1_code_fast<QMAX>(x[e], p, redo);
  if (redo) {
#pragma unroll
    for (int e = 0; e < 4; ++e) code[e] = eq1_code_exact<QMAX>(x[e], p);
  }
  uint32_t* row = reinterpret_cast<uint32_t*>(codes);
  if constexpr (BITS == 3) {
    const uint32_t lo[4] = {code[0] & 3u, code[1] & 3u, code[2] & 3u, code[3] & 3u};
    const uint32_t hb[4] = {code[0] >> 2, code[1] >> 2, code[2] >> 2, code[3] >> 2};
    pack_fields<2>(lo, row, lane);
    pack_fields<1>(hb, row + 8, lane);
  } else {
    pack_fields<BITS>(code, row, lane);
  }
  if ((lane & (LANES - 1)) == 0) params[(4 * lane) / GROUP] = __halves2half2(p.alpha16, p.beta16);
}

// Channels 4 lane .. 4 lane + 3 of a bf16 row (8 bytes, `raw`) as fp32, times the key balancer `bal`
// (fp32 [128]) when one is given (Eq. 3: keys are balanced before the quantizer).
__device__ __forceinline__ void row_values(uint2 raw, const float* bal, int lane, float (&x)[4]) {
  x[0] = __uint_as_float(raw.x << 16);
  x[1] = __uint_as_float(raw.x & 0xffff0000u);
  x[2] = __uint_as_float(raw.y << 16);
  x[3] = __uint_as_float(raw.y & 0xffff0000u);
  if (bal) {
    const float4 b = *reinterpret_cast<const float4*>(bal + 4 * lane);
    x[0] = __fmul_rn(x[0], b.x);
    x[1] = __fmul_rn(x[1], b.y);
    x[2] = __fmul_rn(x[2], b.z);
    x[3] = __fmul_rn(x[3], b.w);
  }
}

// Quantize one bf16 row (Eq. 1, Eq. 3): lane l owns channels 4l..4l+3 of `src`; keys pass `bal` (fp32
// [128], or nullptr = 1), multiplied in before the quantizer.
template <int BITS, int GROUP>
__device__ __forceinline__ void quantize_row_warp(const __nv_bfloat16* src, const float* bal, uint8_t* codes,
                                                  __half2* params, int lane) {
  float x[4];
  row_values(*reinterpret_cast<const uint2*>(src + 4 * lane), bal, lane, x);
  quantize_values_warp<BITS, GROUP>(x, codes, params, lane);
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

}  // namespace mikv
