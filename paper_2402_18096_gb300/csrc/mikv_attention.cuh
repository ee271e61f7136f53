// mikv_attention.cuh — split-K flash-decoding over the mixed-precision KV cache (sm_103a): the kernel
// templates. Each mikv_attn_h*.cu instantiates them for one important-set precision; mikv_attention.cu
// holds the work plan, the merge kernel and the dispatch.
//
// Computes, per (batch b, KV head h) and the G query heads that share it, softmax attention of the
// new query over the important set (bf16 K/V, attended with q) and the retained set (N-bit codes,
// keys balanced and attended with q / balancer), Eq. 3-4 of arxiv 2402.18096; the two sets are one
// unordered set for attention (Sec. 3.4), so they are streamed separately and merged by the online
// softmax.
//
// Work decomposition. Every (b, h) owns the same sequence of "units": an important unit is one block
// of 16 bf16 tokens (8 KB of K and V), a retained unit is up to eight blocks of 16 coded
// tokens (about the same bytes). The two kinds are interleaved evenly inside each head's sequence, the
// sequences of all heads are concatenated, and every warp of the persistent grid takes one contiguous,
// equal share. A warp therefore streams a balanced mix of bandwidth-heavy and ALU-heavy units and
// touches one or two heads (a few, for small caches); it writes one partial (max, sum, output) per head
// it touched, and a merge kernel combines the partials of each query head.
//
// Per warp: a private shared-memory ring (2 stages by default) fed by TMA (lane 0 issues 2-D tensor copies: bf16
// rows and packed codes with hardware swizzle, one box per array per unit, (alpha, beta) pairs as
// 16-byte rows; one mbarrier per stage, every wait bounded in time). No cross-warp synchronisation.
//
// A coded important set (Sec. 3.3, Table 3: INT8 / INT4 / INT2 codes, groups of 64) is streamed in
// units laid out like retained units and attended with the same block code, with exact value codes
// and its logits stored for the importance update.
//
// Per 16-token block: ldmatrix yields mma.sync fragments directly (the ABI's code layout is built for
// this); tokens sit on M for QK^T and channels on M for PV, query heads on N. Codes become exact fp16
// integers with one LOP3 each (the code bits OR-ed under an fp16 exponent that makes the code's lowest
// bit weigh 1) and one HSUB2. Keys are then dequantized (alpha * c + beta, HFMA2) for QK^T; for PV the
// value scale is folded into the probabilities (p * alpha per token and group) and the zero into one
// extra MMA row (sum of p * beta per group), so values need no HFMA2. Online softmax in fp32;
// movmatrix turns probabilities into the PV operand without shared memory.
//
// With one query head per KV head (G = 1, bf16 important set, per-token retained keys) the N columns that no
// head would use carry the quantization groups instead (the mha_* functions): the keys' alpha and beta are
// applied per group after the MMA in fp32, and the values' beta sums, alpha sums and normaliser come from one
// correction MMA.
#pragma once

#include <math.h>

#include "mikv_device.cuh"
#include "mikv_internal.h"
#include "mikv_rows.cuh"

namespace mikv {
namespace {

// Launch shape (compile-time tuning knobs; the defaults are the measured best on GB300).
#ifndef MIKV_ATTN_WARPS
#define MIKV_ATTN_WARPS 12
#endif
#ifndef MIKV_ATTN_STAGES
#define MIKV_ATTN_STAGES 2
#endif
#ifndef MIKV_ATTN_CTAS
#define MIKV_ATTN_CTAS 1
#endif
#ifndef MIKV_QK_ACC
#define MIKV_QK_ACC 2
#endif
#ifndef MIKV_LO_PAIR
#define MIKV_LO_PAIR 1
#endif
#ifndef MIKV_PAIR_ACC
#define MIKV_PAIR_ACC 1
#endif
#ifndef MIKV_MHA_PATH
#define MIKV_MHA_PATH 1
#endif
// L2 prefetch of the first head's query and balancer rows before the grid-dependency wait (0 turns it off).
#ifndef MIKV_Q_PREFETCH
#define MIKV_Q_PREFETCH 1
#endif
constexpr int kWarps = MIKV_ATTN_WARPS;     // independent warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kNS = MIKV_ATTN_STAGES;       // ring stages per warp
constexpr bool kLoPair = MIKV_LO_PAIR != 0;  // retained blocks processed two at a time
constexpr int kPairAcc = MIKV_PAIR_ACC;      // QK^T accumulators per block when paired
constexpr int kStageBytes = kUnitBytes;
constexpr int kHiBlockBytes = 8192;         // K and V of 16 tokens: 4 boxes of 16 rows x 64 bf16
constexpr int kCtasPerSm = MIKV_ATTN_CTAS;
constexpr int kQkAcc = MIKV_QK_ACC;         // independent accumulators of the QK^T MMA chain
constexpr int kUnitsPerWarp = 24;    // share the grid sizing starts from; the plan then fills every warp slot
                                     // it can (min(units, slots) warps)
constexpr float kLog2e = 1.4426950408889634f;

__host__ __device__ constexpr int smem_bytes() { return 1024 + kWarps * kNS * kStageBytes + kWarps * kNS * 8; }

// Position in the concatenated unit sequence. Unit i of a head (of n_u units, hu of them important)
// is important when floor((i+1) hu / n_u) > floor(i hu / n_u): important units are spread evenly.
// The cursor keeps r = (i hu) mod n_u and h = floor(i hu / n_u) so each step is O(1).
struct Cursor {
  int bh, i, r, h;
};

struct UnitKind {
  bool hi;
  int index;  // important block index, or retained unit index
};

__device__ __forceinline__ Cursor cursor_at(int u, int hu, int n_u) {
  Cursor c;
  c.bh = u / n_u;
  c.i = u - c.bh * n_u;
  const long long p = (long long)c.i * hu;
  c.h = (int)(p / n_u);
  c.r = (int)(p - (long long)c.h * n_u);
  return c;
}

__device__ __forceinline__ UnitKind cursor_kind(const Cursor& c, int hu, int n_u) {
  UnitKind k;
  k.hi = c.r + hu >= n_u;
  k.index = k.hi ? c.h : c.i - c.h;
  return k;
}

__device__ __forceinline__ void cursor_next(Cursor& c, int hu, int n_u) {
  const bool hi = c.r + hu >= n_u;
  c.r += hu - (hi ? n_u : 0);
  c.h += hi ? 1 : 0;
  if (++c.i == n_u) {
    ++c.bh;
    c.i = c.r = c.h = 0;
  }
}

// Running softmax state of heads 2t, 2t+1: reference max m (warp-uniform per head), sum l of
// exp(logit - m) over this thread's tokens, and mx, the largest logit this thread has seen.
struct Softmax {
  float m[2], l[2], mx[2];
};

template <int Q>
__device__ __forceinline__ void sum_acc(const float (&accs)[Q][4], float (&acc)[4]) {
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    float v = accs[0][e];
#pragma unroll
    for (int q = 1; q < Q; ++q) v += accs[q][e];
    acc[e] = v;
  }
}

// Online-softmax update for NK 16-token blocks. s[k] holds scaled logits of (token g, head 2t),
// (g, 2t+1), (g+8, 2t), (g+8, 2t+1) of block k (-inf past the end); returns unnormalised
// probabilities in p.
// o (output) and ob (zero-row and alpha sums) are running sums at the current reference max m: all are
// rescaled when m moves. The reference is only moved (one cross-lane reduction) when some logit exceeds it by
// more than kLazy; otherwise the block reuses the old reference, so probabilities stay below e^kLazy.
constexpr float kLazy = 4.f;

// ODD: whether head 2t + 1 can exist (G > 1). With one query head per KV head only column 0 of the MMA tiles
// (lanes with t = 0, head 0) is real, so the odd column's statistics and probabilities are skipped (its
// probabilities are 0, which keeps the column's output sums at 0).
template <int NB, int NK, bool ODD = true>
__device__ __forceinline__ void softmax_blocks(const float (&s)[NK][4], Softmax& st, float (&o)[8][4],
                                               float (&ob)[NB][4], float (&p)[NK][4]) {
  float bm0 = fmaxf(s[0][0], s[0][2]), bm1 = ODD ? fmaxf(s[0][1], s[0][3]) : -INFINITY;
#pragma unroll
  for (int k = 1; k < NK; ++k) {
    bm0 = fmaxf(bm0, fmaxf(s[k][0], s[k][2]));
    if (ODD) bm1 = fmaxf(bm1, fmaxf(s[k][1], s[k][3]));
  }
  st.mx[0] = fmaxf(st.mx[0], bm0);
  if (ODD) st.mx[1] = fmaxf(st.mx[1], bm1);
  if (__any_sync(0xffffffffu, bm0 > st.m[0] + kLazy || (ODD && bm1 > st.m[1] + kLazy))) {
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, off));
      if (ODD) bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, off));
    }
    const float mn0 = fmaxf(st.m[0], bm0), mn1 = ODD ? fmaxf(st.m[1], bm1) : st.m[1];
    const float c0 = mn0 == st.m[0] ? 1.f : fast_exp2((st.m[0] - mn0) * kLog2e);
    const float c1 = !ODD || mn1 == st.m[1] ? 1.f : fast_exp2((st.m[1] - mn1) * kLog2e);
    st.l[0] *= c0;
    if (ODD) st.l[1] *= c1;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      o[mt][0] *= c0;
      o[mt][2] *= c0;
      if (ODD) {
        o[mt][1] *= c1;
        o[mt][3] *= c1;
      }
    }
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      ob[i][0] *= c0;
      ob[i][2] *= c0;
      if (ODD) {
        ob[i][1] *= c1;
        ob[i][3] *= c1;
      }
    }
    st.m[0] = mn0;
    st.m[1] = mn1;
  }
  const float ml0 = st.m[0] * kLog2e, ml1 = st.m[1] * kLog2e;
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    p[k][0] = fast_exp2(fmaf(s[k][0], kLog2e, -ml0));
    p[k][2] = fast_exp2(fmaf(s[k][2], kLog2e, -ml0));
    st.l[0] += p[k][0] + p[k][2];
    if (ODD) {
      p[k][1] = fast_exp2(fmaf(s[k][1], kLog2e, -ml1));
      p[k][3] = fast_exp2(fmaf(s[k][3], kLog2e, -ml1));
      st.l[1] += p[k][1] + p[k][3];
    } else {
      p[k][1] = p[k][3] = 0.f;
    }
  }
}

// Scale raw dot products, mask tokens >= valid, and store important-set logits.
template <int G>
__device__ __forceinline__ void finish_logits(const float (&acc)[4], float scale, int valid, int g, int t,
                                              float* logit_base, int hi_stride, int slot0, float (&s)[4]) {
  s[0] = acc[0] * scale;
  s[1] = acc[1] * scale;
  s[2] = acc[2] * scale;
  s[3] = acc[3] * scale;
  if (valid < 16) {
    if (g >= valid) s[0] = s[1] = -INFINITY;
    if (g + 8 >= valid) s[2] = s[3] = -INFINITY;
  }
  if (logit_base) {
    const int h0 = 2 * t, h1 = 2 * t + 1;
    if (h0 < G) {
      if (g < valid) logit_base[(size_t)h0 * hi_stride + slot0 + g] = s[0];
      if (g + 8 < valid) logit_base[(size_t)h0 * hi_stride + slot0 + g + 8] = s[2];
    }
    if (h1 < G) {
      if (g < valid) logit_base[(size_t)h1 * hi_stride + slot0 + g] = s[1];
      if (g + 8 < valid) logit_base[(size_t)h1 * hi_stride + slot0 + g + 8] = s[3];
    }
  }
}

// ---------------------------------------------------------------------- code extraction
//
// A 32-bit fragment register holds two 16-bit units (two channels or two tokens) whose codes sit at
// the same bit positions. OR-ing the masked code bits under the fp16 exponent of 2^(10 - pos) gives
// the exact value 2^(10 - pos) + code (the code's lowest bit then weighs 1); HSUB2 of that power of
// two leaves the exact code. Positions 10 and up lie in the exponent field and are shifted down first.

__device__ __forceinline__ uint32_t exact_codes(uint32_t x_with_magic, uint32_t magic2) {
  return h2_as_u32(__hsub2(u32_as_h2(x_with_magic), u32_as_h2(magic2)));
}

__device__ __forceinline__ uint32_t mag2(int j) {  // fp16 pair 2^(10 - 2j), j = 0..4
  return j == 0 ? 0x64006400u : j == 1 ? 0x5C005C00u : j == 2 ? 0x54005400u : j == 3 ? 0x4C004C00u : 0x44004400u;
}

// 2-bit code j (0..7) of each unit of r (r10 = r >> 10): exact fp16 pair.
__device__ __forceinline__ uint32_t code2(uint32_t r, uint32_t r10, int j) {
  if (j < 5) return exact_codes(and_or(r, 0x00030003u << (2 * j), mag2(j)), mag2(j));
  const int jj = j - 5;
  return exact_codes(and_or(r10, 0x00030003u << (2 * jj), mag2(jj)), mag2(jj));
}

// 4-bit code p (0..3) of each unit of r (r8 = r >> 8): exact fp16 pair (magics 2^10 and 2^6).
__device__ __forceinline__ uint32_t code4(uint32_t r, uint32_t r8, int p) {
  const uint32_t src = p < 2 ? r : r8;
  const int pp = p & 1;
  const uint32_t mag = pp ? 0x54005400u : 0x64006400u;
  return exact_codes(and_or(src, 0x000F000Fu << (4 * pp), mag), mag);
}

// 8-bit code: the low (hi = 0) or high (hi = 1) byte of each unit of r, under the exponent of 1024.
__device__ __forceinline__ uint32_t code8(uint32_t r, int hi) {
  return exact_codes(prmt(r, 0x64646464u, hi ? 0x4341u : 0x4240u), 0x64006400u);
}

// 3-bit code with its low bits at [p, p + 2) of r and its high bit at p + 2 of hs (each unit), OR-ed under
// `magic`, the fp16 exponent that makes bit p weigh 1: the pair holds magic + code exactly. In the 1-bit plane
// the bits of the two channels u and u + 8 of a unit alternate (bit 2 m + (u div 8) for channel 16 m + u), so
// one shift of the plane word lines up the high bit of every code of a channel with its low bits.
__device__ __forceinline__ uint32_t or_code3(uint32_t r, uint32_t hs, int p, uint32_t magic) {
  return and_or(hs, 0x00040004u << p, and_or(r, 0x00030003u << p, magic));
}

// Key codes (exact) of k-step ks, N = 3: kr = a fragment register of the 2-bit plane (its codes for ks at bits
// 2 ks), kr8 = kr >> 8; he / he8 the 1-bit plane word shifted so that the high bits of ks <= 3 / ks >= 4 land
// at 2 ks + 2 / 2 (ks - 4) + 2.
__device__ __forceinline__ uint32_t kcode3(uint32_t kr, uint32_t kr8, uint32_t he, uint32_t he8, int ks) {
  const int j = ks & 3;
  return exact_codes(or_code3(ks < 4 ? kr : kr8, ks < 4 ? he : he8, 2 * j, mag2(j)), mag2(j));
}

// Value codes, N = 3, take a code offset M in {64, 16} like vcode2: code mt is read at bit 4 + 2 (mt & 1) of the
// words shifted by 4 - 4 (mt div 2) (the low bits) and by two more (the high bit).
__host__ __device__ constexpr float voff3(int mt) { return (mt & 1) ? 16.f : 64.f; }

// Value codes (N = 2, 4) skip the subtraction: the code is placed at a mantissa position where it
// weighs 1 under a magic M in {4, 16, 64}, so the fp16 pair holds M + code exactly. The PV sums then
// carry M * sum(p * alpha) per channel on top of the wanted sum; that term is measured by a ones-row
// MMA on the same fp16 operands and removed in write_partial. M stays small (<= 64) so the removal
// costs only a few bits of the fp32 accumulator.
// N = 2: code j of r sits at bits 2j of each unit. Codes 0..2 are read from r << 4 (bits 4, 6, 8), codes
// 3, 4 from r itself (bits 6, 8), codes 5..7 from r >> 6 (bits 4, 6, 8): offsets 64, 16, 4, 16, 4, 64, 16, 4.
__device__ __forceinline__ uint32_t vcode2(uint32_t rl4, uint32_t r, uint32_t rr6, int j) {
  const uint32_t src = j < 3 ? rl4 : (j < 5 ? r : rr6);
  const int pos = j < 3 ? j + 2 : (j < 5 ? j : j - 3);  // 2-bit field index of the code in src
  return and_or(src, 0x00030003u << (2 * pos), mag2(pos));
}
__host__ __device__ constexpr float voff2(int j) {
  return (j == 0 || j == 5) ? 64.f : (j == 2 || j == 4 || j == 7) ? 4.f : 16.f;
}
// N = 4: nibble p of r at bits 4p. Nibbles 0 and 1 are read at bits 4..7 of r << 4 and r (M = 64),
// nibbles 2 and 3 at bits 6..9 of r >> 2 and r >> 6 (M = 16).
__device__ __forceinline__ uint32_t vcode4(const uint32_t (&sh)[4], int p) {
  return p < 2 ? and_or(sh[p], 0x00F000F0u, 0x54005400u) : and_or(sh[p], 0x03C003C0u, 0x4C004C00u);
}
__host__ __device__ constexpr float voff4(int p) { return p < 2 ? 64.f : 16.f; }

template <int BITS>
__host__ __device__ constexpr float voff(int mt) {
  return BITS == 2 ? voff2(mt) : BITS == 4 ? voff4(mt & 3) : BITS == 3 ? voff3(mt) : 0.f;
}

// The code fragments of one 16-token block (N = 2, 3, 4). KeyFrag: the QK^T A operand (tokens g, g + 8 on M,
// channels on K) with exact codes; ValFrag: the PV A operand (channels on M, tokens 2t, 2t+1, 2t+8, 2t+9 on K) with
// the codes offset by voff (or exact). `rows` is the block's first code row in the stage (pitch U.pitch bytes).
template <int BITS, int PITCH>
struct KeyFrag {
  static constexpr int NR = BITS == 4 ? 8 : 4;
  uint32_t kr[NR], kh[NR];
  uint32_t he0, he1, ho0, ho1, he0s, he1s, ho0s, ho1s;  // N = 3 only

  __device__ __forceinline__ void load(uint32_t rows, int lane) {
    const int r8 = lane & 7, j = lane >> 3;
    const int tok = r8 + 8 * (j & 1);
    uint32_t kb0 = 0, kb1 = 0;
    if (BITS == 4) {
      const int o0 = tok * 64 + 16 * (j >> 1), sw = ((tok >> 1) & 3) << 4;
      uint32_t r0[4], r1[4];
      ldsm_x4(rows + (o0 ^ sw), r0);
      ldsm_x4(rows + ((o0 + 32) ^ sw), r1);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        kr[i] = r0[i];
        kr[(NR == 8 ? 4 : 0) + i] = r1[i];
      }
    } else {
      // N = 2: 32-byte tokens under the 64B swizzle (bits 4..5 ^= bits 7..8); N = 3: 48-byte tokens, unswizzled
      const int o0 = tok * PITCH + 16 * (j >> 1), sw = BITS == 2 ? ((tok >> 2) & 3) << 4 : 0;
      uint32_t r0[4];
      ldsm_x4(rows + (o0 ^ sw), r0);
#pragma unroll
      for (int i = 0; i < 4; ++i) kr[i] = r0[i];
      if (BITS == 3) ldsm_x2(rows + (lane & 15) * PITCH + 32, kb0, kb1);
    }
#pragma unroll
    for (int i = 0; i < NR; ++i) kh[i] = kr[i] >> (BITS == 2 ? 10 : 8);
    // N = 3: the 1-bit plane words of tokens g (kb0) and g + 8 (kb1) shifted so that the high bit of code ks sits
    // two bits above its low bits: channels 2t, 2t+1 use the even bits (<< 2 for ks <= 3, >> 6 for ks >= 4),
    // channels 2t+8, 2t+9 the odd bits (<< 1, >> 7)
    he0 = kb0 << 2, he1 = kb1 << 2, ho0 = kb0 << 1, ho1 = kb1 << 1;
    he0s = kb0 >> 6, he1s = kb1 >> 6, ho0s = kb0 >> 7, ho1s = kb1 >> 7;
  }

  // exact codes of k-step ks (channels 16 ks .. 16 ks + 15) as fp16 pairs
  __device__ __forceinline__ void code(int ks, uint32_t (&c)[4]) const {
    if (BITS == 4) {
      const int ri = (ks >> 2) * 4, p = ks & 3;
#pragma unroll
      for (int i = 0; i < 4; ++i) c[i] = code4(kr[ri + i], kh[ri + i], p);
    } else if (BITS == 2) {
#pragma unroll
      for (int i = 0; i < 4; ++i) c[i] = code2(kr[i], kh[i], ks);
    } else {
      c[0] = kcode3(kr[0], kh[0], he0, he0s, ks);
      c[1] = kcode3(kr[1], kh[1], he1, he1s, ks);
      c[2] = kcode3(kr[2], kh[2], ho0, ho0s, ks);
      c[3] = kcode3(kr[3], kh[3], ho1, ho1s, ks);
    }
  }
};

template <int BITS, int PITCH, bool EXACT>
struct ValFrag {
  static constexpr int NR = BITS == 4 ? 8 : 4;
  uint32_t vr[NR];
  uint32_t vb0, vb1;  // N = 3: the 1-bit plane words of tokens (2t, 2t+1) and (2t+8, 2t+9)

  __device__ __forceinline__ void load(uint32_t rows, int lane) {
    const int r8 = lane & 7, j = lane >> 3;
    const int tok = r8 + 8 * (j >> 1);
    vb0 = vb1 = 0;
    if (BITS == 4) {
      const int o0 = tok * 64 + 16 * (j & 1), sw = ((tok >> 1) & 3) << 4;
      uint32_t r0[4], r1[4];
      ldsm_x4_t(rows + (o0 ^ sw), r0);
      ldsm_x4_t(rows + ((o0 + 32) ^ sw), r1);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        vr[i] = r0[i];
        vr[(NR == 8 ? 4 : 0) + i] = r1[i];
      }
    } else {
      const int o0 = tok * PITCH + 16 * (j & 1), sw = BITS == 2 ? ((tok >> 2) & 3) << 4 : 0;
      uint32_t r0[4];
      ldsm_x4_t(rows + (o0 ^ sw), r0);
#pragma unroll
      for (int i = 0; i < 4; ++i) vr[i] = r0[i];
      if (BITS == 3) ldsm_x2_t(rows + (lane & 15) * PITCH + 32, vb0, vb1);
    }
  }

  // codes of channels 16 mt .. 16 mt + 15 (EXACT: exact codes; else the codes plus voff<BITS>(mt))
  __device__ __forceinline__ void code(int mt, uint32_t (&a)[4]) const {
    if (BITS == 4) {
      const int ri = (mt >> 2) * 4, pp = mt & 3;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t w = vr[ri + i];
        if (EXACT) {
          a[i] = code4(w, w >> 8, pp);
        } else {
          const uint32_t c4[4] = {w << 4, w, w >> 2, w >> 6};  // shared by the four mt of this word
          a[i] = vcode4(c4, pp);
        }
      }
    } else if (BITS == 2) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (EXACT)
          a[i] = code2(vr[i], vr[i] >> 10, mt);
        else
          a[i] = vcode2(vr[i] << 4, vr[i], vr[i] >> 6, mt);  // the shifted copies are shared by all mt
      }
    } else {
      // vr[0], vr[2]: channel g (tokens 2t, 2t+1 and 2t+8, 2t+9), whose high bits are the even bits of vb0, vb1;
      // vr[1], vr[3]: channel g + 8, the odd bits
      const int k = mt >> 1, s = 4 - 4 * k;  // codes 2k, 2k+1 read at bits 4, 6 of the words shifted by s
      auto sh = [](uint32_t x, int n) { return n >= 0 ? x << n : x >> -n; };
      const uint32_t r4[4] = {sh(vr[0], s), sh(vr[1], s), sh(vr[2], s), sh(vr[3], s)};
      const uint32_t h4[4] = {sh(vb0, s + 2), sh(vb0, s + 1), sh(vb1, s + 2), sh(vb1, s + 1)};
      const int p = 4 + 2 * (mt & 1);
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = or_code3(r4[i], h4[i], p, mag2(p >> 1));
    }
  }
};

// ---------------------------------------------------------------------- one important block

template <int G, int NB>
__device__ __forceinline__ void process_hi(uint32_t blk, int valid, int slot0, const uint32_t (&qb)[8][2],
                                           float scale, float* logit_base, int hi_stride, Softmax& st,
                                           float (&o)[8][4], float (&ob)[NB][4], int lane) {
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;
  float accs[kQkAcc][4];
#pragma unroll
  for (int q = 0; q < kQkAcc; ++q) accs[q][0] = accs[q][1] = accs[q][2] = accs[q][3] = 0.f;
  const int krow = r8 + 8 * (j & 1);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int chunk = 2 * (ks & 3) + (j >> 1);
    uint32_t a[4];
    ldsm_x4(blk + (ks >> 2) * 2048 + krow * 128 + ((chunk ^ (krow & 7)) << 4), a);
    mma_bf16(accs[ks % kQkAcc], a, qb[ks][0], qb[ks][1]);
  }
  float acc[4];
  sum_acc(accs, acc);
  float s[1][4], p[1][4];
  finish_logits<G>(acc, scale, valid, g, t, logit_base, hi_stride, slot0, s[0]);
  softmax_blocks<NB, 1, (G > 1)>(s, st, o, ob, p);
  const uint32_t pb0 = movmatrix_t(pack_bf16(p[0][0], p[0][1]));
  const uint32_t pb1 = movmatrix_t(pack_bf16(p[0][2], p[0][3]));
  {
    // row 4 of the zero-row sums: the bf16 probabilities exactly as the PV MMA uses them (normaliser)
    const uint32_t one = g == 4 ? 0x3F803F80u : 0u;
    const uint32_t a[4] = {one, 0u, one, 0u};
    mma_bf16(ob[0], a, pb0, pb1);
  }
  uint32_t m01 = 0xffffffffu, m89 = 0xffffffffu;
  if (valid < 16) {
    m01 = (2 * t < valid ? 0x0000ffffu : 0u) | (2 * t + 1 < valid ? 0xffff0000u : 0u);
    m89 = (2 * t + 8 < valid ? 0x0000ffffu : 0u) | (2 * t + 9 < valid ? 0xffff0000u : 0u);
  }
  const int vtok = r8 + 8 * (j >> 1);
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int chunk = 2 * (mt & 3) + (j & 1);
    uint32_t a[4];
    ldsm_x4_t(blk + 4096 + (mt >> 2) * 2048 + vtok * 128 + ((chunk ^ (vtok & 7)) << 4), a);
    if (valid < 16) {  // rows past the end may hold any bits: zero them (P is 0 there, NaN * 0 is not)
      a[0] &= m01;
      a[1] &= m01;
      a[2] &= m89;
      a[3] &= m89;
    }
    mma_bf16(o[mt], a, pb0, pb1);
  }
}

// ---------------------------------------------------------------------- one retained block

// Key side of coded block b of a unit (retained, or coded important with logit_base set): scaled
// logits s, -inf past valid; important-set logits are also stored at logit_base[head][slot0 + token].
// KCH (per-channel retained keys, App. C): qh holds the query scaled by the group's per-channel alpha,
// the codes enter the MMA as exact integers, and kbias[hd] (sum over channels of q * beta for heads 2t,
// 2t+1) is added to the dot products; no per-token key parameters.
template <int BITS, int GROUP, int G, int QACC, bool KCH = false>
__device__ __forceinline__ void lo_logits(uint32_t unit, int b, int valid, const uint32_t (&qh)[8][2], float scale,
                                          float (&s)[4], int lane, float* logit_base = nullptr, int hi_stride = 0,
                                          int slot0 = 0, const float* kbias = nullptr) {
  constexpr LoUnit U = KCH ? lo_unit_layout_kch(BITS, GROUP) : lo_unit_layout(BITS, GROUP);
  constexpr int NG = kHeadDim / GROUP;
  constexpr int PR = U.param_row;
  // this block's rows inside the unit's sections
  const uint32_t ka = unit + U.k_a + b * 16 * U.pitch;
  const uint32_t kp = unit + U.k_p + b * 16 * PR;
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;

  uint32_t pk0[NG], pk1[NG];
  if constexpr (!KCH) {
    lds_vec<NG>(kp + g * PR, pk0);
    lds_vec<NG>(kp + (g + 8) * PR, pk1);
  }
  float accs[QACC][4];
#pragma unroll
  for (int q = 0; q < QACC; ++q) accs[q][0] = accs[q][1] = accs[q][2] = accs[q][3] = 0.f;
  if constexpr (BITS == 8) {
    // 128-byte token rows under the 128B swizzle; channels 32 i .. 32 i + 31 (ks = 2 i, 2 i + 1) share
    // one ldmatrix: each 16-bit unit holds the code of ks = 2 i (low byte) and ks = 2 i + 1 (high byte)
    const int tok = r8 + 8 * (j & 1);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint32_t r[4];
      ldsm_x4(ka + tok * 128 + (((2 * i + (j >> 1)) ^ (tok & 7)) << 4), r);
#pragma unroll
      for (int hb = 0; hb < 2; ++hb) {
        const int ks = 2 * i + hb, gi = (16 * ks) / GROUP;
        const __half2 p0 = u32_as_h2(pk0[gi]), p1 = u32_as_h2(pk1[gi]);
        const __half2 al0 = __low2half2(p0), be0 = __high2half2(p0);
        const __half2 al1 = __low2half2(p1), be1 = __high2half2(p1);
        const uint32_t a[4] = {h2_as_u32(__hfma2(u32_as_h2(code8(r[0], hb)), al0, be0)),
                               h2_as_u32(__hfma2(u32_as_h2(code8(r[1], hb)), al1, be1)),
                               h2_as_u32(__hfma2(u32_as_h2(code8(r[2], hb)), al0, be0)),
                               h2_as_u32(__hfma2(u32_as_h2(code8(r[3], hb)), al1, be1))};
        mma_f16(accs[ks % QACC], a, qh[ks][0], qh[ks][1]);
      }
    }
    float acc[4];
    sum_acc(accs, acc);
    finish_logits<G>(acc, scale, valid, g, t, logit_base, hi_stride, slot0, s);
    return;
  }

  // ---- keys of tokens g and g+8
  KeyFrag<BITS, U.pitch> kf;
  kf.load(ka, lane);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int gi = (16 * ks) / GROUP;
    // (alpha, alpha) and (beta, beta) of tokens g and g + 8: half-broadcasts the HFMA2 operand selectors absorb
    uint32_t c[4];
    kf.code(ks, c);
    if constexpr (KCH) {
      mma_f16(accs[ks % QACC], c, qh[ks][0], qh[ks][1]);
    } else {
      const __half2 p0 = u32_as_h2(pk0[gi]), p1 = u32_as_h2(pk1[gi]);
      const __half2 al0 = __low2half2(p0), be0 = __high2half2(p0);
      const __half2 al1 = __low2half2(p1), be1 = __high2half2(p1);
      const uint32_t a[4] = {h2_as_u32(__hfma2(u32_as_h2(c[0]), al0, be0)), h2_as_u32(__hfma2(u32_as_h2(c[1]), al1, be1)),
                             h2_as_u32(__hfma2(u32_as_h2(c[2]), al0, be0)), h2_as_u32(__hfma2(u32_as_h2(c[3]), al1, be1))};
      mma_f16(accs[ks % QACC], a, qh[ks][0], qh[ks][1]);
    }
  }
  float acc[4];
  sum_acc(accs, acc);
  if constexpr (KCH) {
    acc[0] += kbias[0];
    acc[1] += kbias[1];
    acc[2] += kbias[0];
    acc[3] += kbias[1];
  }
  finish_logits<G>(acc, scale, valid, g, t, logit_base, hi_stride, slot0, s);
}

// Per-channel keys (App. C): from the group's (alpha, beta) pairs of the key channels (512 bytes at kp),
// the query fragments scaled per channel, qk = q * alpha, and the per-head bias sum_c q_c beta_c (one MMA
// per k-step whose row 0 holds beta; lanes 4 t .. 4 t + 3 all receive heads 2t, 2t+1).
__device__ __forceinline__ void kch_prepare(uint32_t kp, const uint32_t (&qh)[8][2], uint32_t (&qk)[8][2],
                                            float (&kbias)[2], int lane) {
  const int g = lane >> 2, t = lane & 3;
  float cb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    uint32_t be[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int c = 16 * ks + 8 * r + 2 * t;  // channels c, c + 1 of this fragment
      const uint32_t p0 = lds32(kp + 4 * c), p1 = lds32(kp + 4 * c + 4);
      qk[ks][r] = h2_as_u32(__hmul2(u32_as_h2(qh[ks][r]), u32_as_h2(prmt(p0, p1, 0x5410u))));
      be[r] = prmt(p0, p1, 0x7632u);
    }
    const uint32_t a[4] = {g == 0 ? be[0] : 0u, 0u, g == 0 ? be[1] : 0u, 0u};
    mma_f16(cb, a, qh[ks][0], qh[ks][1]);
  }
  kbias[0] = __shfl_sync(0xffffffffu, cb[0], t);
  kbias[1] = __shfl_sync(0xffffffffu, cb[1], t);
}

// Value side of coded block b: o, ob += P (this block's probabilities p) times the block's values.
// EXACT (coded important blocks): codes enter the MMA as exact integers, so the block adds nothing to
// the alpha sums that remove the retained set's code offsets.
template <int BITS, int GROUP, int NB, bool EXACT, bool KCH = false>
__device__ __forceinline__ void lo_values(uint32_t unit, int b, int valid, const float (&p)[4], float (&o)[8][4],
                                          float (&ob)[NB][4], int lane) {
  static_assert(!(EXACT && BITS == 3), "coded important sets use 8-, 4- or 2-bit codes");
  constexpr LoUnit U = KCH ? lo_unit_layout_kch(BITS, GROUP) : lo_unit_layout(BITS, GROUP);
  constexpr int NG = kHeadDim / GROUP;
  constexpr int PR = U.param_row;
  const uint32_t va = unit + U.v_a + b * 16 * U.pitch;
  const uint32_t vp = unit + U.v_p + b * 16 * PR;
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;
  const uint32_t pb0 = movmatrix_t(pack_f16(p[0], p[1]));  // (P[2t][head g], P[2t+1][head g])
  const uint32_t pb1 = movmatrix_t(pack_f16(p[2], p[3]));  // tokens 2t+8, 2t+9

  // ---- values of tokens (2t, 2t+1) and (2t+8, 2t+9), channels 16 mt + g and 16 mt + 8 + g
  const int vtok = r8 + 8 * (j >> 1);
  ValFrag<BITS == 8 ? 2 : BITS, U.pitch, EXACT> vf;
  if constexpr (BITS != 8) vf.load(va, lane);
  // (alpha, beta) of the four tokens for every group; zero past the end (exact zeros in the sums)
  const int t0 = 2 * t, t1 = 2 * t + 1, t8 = 2 * t + 8, t9 = 2 * t + 9;
  uint32_t pv0[NG], pv1[NG], pv8[NG], pv9[NG];
  lds_vec<NG>(vp + t0 * PR, pv0);
  lds_vec<NG>(vp + t1 * PR, pv1);
  lds_vec<NG>(vp + t8 * PR, pv8);
  lds_vec<NG>(vp + t9 * PR, pv9);
  // zero rows: row r < 4 of the beta operand holds, for this thread's tokens, beta of the group that
  // contains channels 32 r .. 32 r + 31 (a granularity the important and retained sets share)
  uint32_t bw0 = 0, bw1 = 0, bw8 = 0, bw9 = 0;
  if (g < 4) {
    const int pidx = (32 * g) / GROUP;
    bw0 = lds32(vp + t0 * PR + 4 * pidx);
    bw1 = lds32(vp + t1 * PR + 4 * pidx);
    bw8 = lds32(vp + t8 * PR + 4 * pidx);
    bw9 = lds32(vp + t9 * PR + 4 * pidx);
  }
  if (valid < 16) {
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
      if (t0 >= valid) pv0[gi] = 0u;
      if (t1 >= valid) pv1[gi] = 0u;
      if (t8 >= valid) pv8[gi] = 0u;
      if (t9 >= valid) pv9[gi] = 0u;
    }
    if (t0 >= valid) bw0 = 0u;
    if (t1 >= valid) bw1 = 0u;
    if (t8 >= valid) bw8 = 0u;
    if (t9 >= valid) bw9 = 0u;
  }
  {
    // rows 0..3: sum over tokens of p * beta per 32-channel slice; row 4: sum of the fp16 probabilities
    // exactly as the code MMAs use them (the normaliser of the output)
    uint32_t a0 = prmt(bw0, bw1, 0x7632u), a2 = prmt(bw8, bw9, 0x7632u);
    if (g == 4) a0 = a2 = 0x3C003C00u;
    const uint32_t a[4] = {a0, 0u, a2, 0u};
    mma_f16(ob[0], a, pb0, pb1);
  }
  uint32_t pa0[NG], pa1[NG];  // p * alpha per group: B operand of the code MMAs
#pragma unroll
  for (int gi = 0; gi < NG; ++gi) {
    pa0[gi] = h2_as_u32(__hmul2(u32_as_h2(pb0), u32_as_h2(prmt(pv0[gi], pv1[gi], 0x5410u))));
    pa1[gi] = h2_as_u32(__hmul2(u32_as_h2(pb1), u32_as_h2(prmt(pv8[gi], pv9[gi], 0x5410u))));
  }
  if (!EXACT) {
    // sum of p * alpha per group, from the same fp16 operands as the code MMAs: ones in rows 0..7
    // (even groups) or 8..15 (odd groups), so ob[1 + gi / 2] holds two groups per fragment
    constexpr uint32_t kOne = 0x3C003C00u;
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
      const uint32_t e = (gi & 1) ? 0u : kOne, d = (gi & 1) ? kOne : 0u;
      const uint32_t a[4] = {e, d, e, d};
      mma_f16(ob[1 + gi / 2], a, pa0[gi], pa1[gi]);
    }
  }
  if constexpr (BITS == 8) {
    // channels 32 i .. 32 i + 31 (mt = 2 i, 2 i + 1) share one transposed ldmatrix, as for the keys
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint32_t r[4];
      ldsm_x4_t(va + vtok * 128 + (((2 * i + (j & 1)) ^ (vtok & 7)) << 4), r);
#pragma unroll
      for (int hb = 0; hb < 2; ++hb) {
        const int mt = 2 * i + hb, gi = (16 * mt) / GROUP;
        const uint32_t a[4] = {code8(r[0], hb), code8(r[1], hb), code8(r[2], hb), code8(r[3], hb)};
        mma_f16(o[mt], a, pa0[gi], pa1[gi]);
      }
    }
    return;
  }
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int gi = (16 * mt) / GROUP;
    uint32_t a[4];
    vf.code(mt, a);
    mma_f16(o[mt], a, pa0[gi], pa1[gi]);  // sums p * alpha * (code + offset)
  }
}

// NK consecutive coded blocks b .. b + NK - 1 of a unit (n_left = valid tokens from block b on, at
// least 16 (NK - 1) + 1): the key sides first, one softmax update over all NK blocks, then the value
// sides, so the dependency chains of the blocks overlap. HI: blocks of a coded important set (logits
// stored for the importance update, exact value codes); slot0 = important slot of block b's first row.
template <int BITS, int GROUP, int G, int NB, int NK, bool HI, bool KCH = false>
__device__ __forceinline__ void process_coded(uint32_t unit, int b, int n_left, const uint32_t (&qh)[8][2],
                                              float scale, Softmax& st, float (&o)[8][4], float (&ob)[NB][4],
                                              int lane, float* logit_base = nullptr, int hi_stride = 0,
                                              int slot0 = 0, const float* kbias = nullptr) {
  float s[NK][4], p[NK][4];
#pragma unroll
  for (int k = 0; k < NK; ++k)
    lo_logits<BITS, GROUP, G, NK == 1 ? kQkAcc : kPairAcc, KCH>(unit, b + k, min(16, n_left - 16 * k), qh, scale,
                                                                s[k], lane, HI ? logit_base : nullptr, hi_stride,
                                                                slot0 + 16 * k, kbias);
  softmax_blocks<NB, NK, (G > 1)>(s, st, o, ob, p);
#pragma unroll
  for (int k = 0; k < NK; ++k)
    lo_values<BITS, GROUP, NB, HI, KCH>(unit, b + k, min(16, n_left - 16 * k), p[k], o, ob, lane);
}

// Write this warp's partial for one head: the output normalised by the sum of the rounded probabilities
// the MMAs used (row 4 of the zero-row sums), so rounding the probabilities to bf16 / fp16 only perturbs
// the weights of a convex combination; and the true max and fp32 sum of its tokens (the sum is kept at
// the reference max m while streaming and rescaled here to the largest logit seen).
template <int BITS, int GROUP, int G, int NB>
__device__ __forceinline__ void write_partial(const AttnArgs& a, int slot, Softmax& st, const float (&o)[8][4],
                                              const float (&ob)[NB][4], int lane) {
  const int g = lane >> 2, t = lane & 3;
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], off);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], off);
    st.mx[0] = fmaxf(st.mx[0], __shfl_xor_sync(0xffffffffu, st.mx[0], off));
    st.mx[1] = fmaxf(st.mx[1], __shfl_xor_sync(0xffffffffu, st.mx[1], off));
  }
  float c[2];
#pragma unroll
  for (int hd = 0; hd < 2; ++hd)  // m <= mx <= m + kLazy; equal (also both -inf) gives 1
    c[hd] = st.mx[hd] == st.m[hd] ? 1.f : fast_exp2((st.m[hd] - st.mx[hd]) * kLog2e);
  float bz0[4], bz1[4];  // sum p * beta over channels 32 r .. 32 r + 31, heads 2t, 2t+1: lane 4 r + t
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    bz0[r] = __shfl_sync(0xffffffffu, ob[0][0], r * 4 + t);
    bz1[r] = __shfl_sync(0xffffffffu, ob[0][1], r * 4 + t);
  }
  const float inv[2] = {1.f / __shfl_sync(0xffffffffu, ob[0][0], 16 + t),   // row 4, lane 16 + t
                        1.f / __shfl_sync(0xffffffffu, ob[0][1], 16 + t)};
#pragma unroll
  for (int hd = 0; hd < 2; ++hd) {
    const int head = 2 * t + hd;
    if (head < G) {
      float* po = a.part_o + ((size_t)slot * G + head) * kHeadDim;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const int gi = (16 * mt) / GROUP;
        float z = hd ? bz1[mt >> 1] : bz0[mt >> 1];
        z = fmaf(-voff<BITS>(mt), ob[1 + gi / 2][2 * (gi & 1) + hd], z);
        po[16 * mt + g] = (o[mt][hd] + z) * inv[hd];
        po[16 * mt + 8 + g] = (o[mt][2 + hd] + z) * inv[hd];
      }
      if (g == 0) {
        a.part_ml[((size_t)slot * G + head) * 2] = st.mx[hd];
        a.part_ml[((size_t)slot * G + head) * 2 + 1] = st.l[hd] * c[hd];
      }
    }
  }
}

// ---------------------------------------------------------------------- one query head per KV head (G = 1)
//
// With G = 1 only one of the eight columns of the QK^T and PV tiles would hold a query head. This path (bf16
// important set, per-token retained keys) gives the other columns work, indexed by the quantization group
// (NG = 128 / group groups per row):
//  - keys: column n of the query operand holds the balanced query on the channels of group n mod NG and zeros
//    elsewhere, so the MMA over exact key codes gives every token one partial dot product per group. The token's
//    (alpha, beta) then enter in fp32, s = scale * sum_g (alpha_g (q . code)_g + beta_g (sum of q over g)): no key
//    element is dequantized (Eq. 1 and Eq. 3-4 regrouped per group).
//  - values: column n < NG of the probability operand holds p * alpha of group n, column NG holds p, and one
//    more MMA, whose row n < NG holds beta of group n and row NG ones, gives the beta sums, the alpha sums that
//    remove the code offsets, and the normaliser (the sum of the probabilities as the MMAs used them).
// Every lane then holds the logits of its tokens g and g + 8 (the important blocks replicate the query over all
// columns; the group sums of a retained block are complete in every lane, after one shuffle when NG = 4), which
// is what movmatrix needs to place the probabilities of every column.

constexpr uint32_t kOnesF16 = 0x3C003C00u, kOnesBf16 = 0x3F803F80u;

// Per-head query operands. Lane (g, t) holds channels 16 ks + 2t (+1) (r = 0) and 16 ks + 2t + 8 (+9) (r = 1) of
// every k-step: qb, the bf16 query, in every column (important blocks); qh, the fp16 balanced query q / b (Eq. 4),
// in the columns of its group (retained blocks); qs0 / qs1, the fp32 sums of qh over the groups of this lane's
// columns 2t and 2t + 1.
template <int GROUP>
__device__ __forceinline__ void mha_query(const AttnArgs& a, int b, int h, int lane, uint32_t (&qb)[8][2],
                                          uint32_t (&qh)[8][2], float& qs0, float& qs1) {
  constexpr int NG = kHeadDim / GROUP;
  const int g = lane >> 2, t = lane & 3;
  const __nv_bfloat16* qp = static_cast<const __nv_bfloat16*>(a.q) + (size_t)(b * a.heads_q + h) * kHeadDim;
  // Every row of lanes needs the same fragments: lane (g, t) loads and divides (Eq. 4) those of k-step ks = g only,
  // every load before any division (the divisions branch), and the fragments reach the other rows by shuffles.
  uint32_t qw[2], fw[2];
  float2 bal[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int c = 16 * g + 2 * t + 8 * r;
    qw[r] = *reinterpret_cast<const uint32_t*>(qp + c);
    bal[r] = a.balancer ? *reinterpret_cast<const float2*>(a.balancer + h * kHeadDim + c) : make_float2(1.f, 1.f);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const float q0 = __uint_as_float(qw[r] << 16), q1 = __uint_as_float(qw[r] & 0xffff0000u);
    fw[r] = pack_f16(__fdiv_rn(q0, bal[r].x), __fdiv_rn(q1, bal[r].y));
  }
  float cs[8];  // this lane's four channels of each k-step
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const bool mine = g % NG == (16 * ks) / GROUP;
    cs[ks] = 0.f;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      qb[ks][r] = __shfl_sync(0xffffffffu, qw[r], 4 * ks + t);
      const uint32_t f = __shfl_sync(0xffffffffu, fw[r], 4 * ks + t);
      qh[ks][r] = mine ? f : 0u;
      cs[ks] += __low2float(u32_as_h2(f)) + __high2float(u32_as_h2(f));
    }
  }
  float gs[NG];
#pragma unroll
  for (int i = 0; i < NG; ++i) gs[i] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {  // k-step sums over the four lanes t (the same bits in each), then per group
    float v = cs[ks];
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    v += __shfl_xor_sync(0xffffffffu, v, 2);
    gs[(16 * ks) / GROUP] += v;
  }
  qs0 = gs[(2 * t) % NG];
  qs1 = gs[(2 * t + 1) % NG];
}

// Online-softmax update for NK blocks of the G = 1 path: s[k] = logits of tokens g and g + 8 of block k (the same
// in the four lanes of a row); p = unnormalised probabilities. All four columns of o and ob belong to the one
// head and are rescaled together when the reference max moves (lazily, as in softmax_blocks).
template <int NK>
__device__ __forceinline__ void mha_softmax(const float (&s)[NK][2], Softmax& st, float (&o)[8][4], float (&ob)[4],
                                            float (&p)[NK][2]) {
  float bm = fmaxf(s[0][0], s[0][1]);
#pragma unroll
  for (int k = 1; k < NK; ++k) bm = fmaxf(bm, fmaxf(s[k][0], s[k][1]));
  st.mx[0] = fmaxf(st.mx[0], bm);
  if (__any_sync(0xffffffffu, bm > st.m[0] + kLazy)) {
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, off));
    const float mn = fmaxf(st.m[0], bm);
    const float c = mn == st.m[0] ? 1.f : fast_exp2((st.m[0] - mn) * kLog2e);
    st.l[0] *= c;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
#pragma unroll
      for (int e = 0; e < 4; ++e) o[mt][e] *= c;
#pragma unroll
    for (int e = 0; e < 4; ++e) ob[e] *= c;
    st.m[0] = mn;
  }
  const float ml = st.m[0] * kLog2e;
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    p[k][0] = fast_exp2(fmaf(s[k][0], kLog2e, -ml));
    p[k][1] = fast_exp2(fmaf(s[k][1], kLog2e, -ml));
    st.l[0] += p[k][0] + p[k][1];
  }
}

// One bf16 important block on the G = 1 path: logits (stored for the importance update), softmax, PV, and the
// block's probabilities (as the bf16 MMA uses them) into the normaliser, entry (NG, NG) of the correction tile.
template <int NG>
__device__ __forceinline__ void mha_hi(uint32_t blk, int valid, int slot0, const uint32_t (&qb)[8][2], float scale,
                                       float* logit_base, Softmax& st, float (&o)[8][4], float (&ob)[4], int lane) {
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;
  float accs[kQkAcc][4];
#pragma unroll
  for (int q = 0; q < kQkAcc; ++q) accs[q][0] = accs[q][1] = accs[q][2] = accs[q][3] = 0.f;
  const int krow = r8 + 8 * (j & 1);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int chunk = 2 * (ks & 3) + (j >> 1);
    uint32_t a[4];
    ldsm_x4(blk + (ks >> 2) * 2048 + krow * 128 + ((chunk ^ (krow & 7)) << 4), a);
    mma_bf16(accs[ks % kQkAcc], a, qb[ks][0], qb[ks][1]);
  }
  float acc[4];
  sum_acc(accs, acc);
  float s[1][2], p[1][2];
  s[0][0] = g < valid ? acc[0] * scale : -INFINITY;
  s[0][1] = g + 8 < valid ? acc[2] * scale : -INFINITY;
  if (logit_base && t == 0) {
    if (g < valid) logit_base[slot0 + g] = s[0][0];
    if (g + 8 < valid) logit_base[slot0 + g + 8] = s[0][1];
  }
  mha_softmax<1>(s, st, o, ob, p);
  const uint32_t pb0 = movmatrix_t(pack_bf16(p[0][0], p[0][0]));  // tokens 2t, 2t+1, every column
  const uint32_t pb1 = movmatrix_t(pack_bf16(p[0][1], p[0][1]));  // tokens 2t+8, 2t+9
  {
    const uint32_t one = g == NG ? kOnesBf16 : 0u;
    const uint32_t a[4] = {one, 0u, one, 0u};
    mma_bf16(ob, a, g == NG ? pb0 : 0u, g == NG ? pb1 : 0u);
  }
  uint32_t m01 = 0xffffffffu, m89 = 0xffffffffu;
  if (valid < 16) {
    m01 = (2 * t < valid ? 0x0000ffffu : 0u) | (2 * t + 1 < valid ? 0xffff0000u : 0u);
    m89 = (2 * t + 8 < valid ? 0x0000ffffu : 0u) | (2 * t + 9 < valid ? 0xffff0000u : 0u);
  }
  const int vtok = r8 + 8 * (j >> 1);
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int chunk = 2 * (mt & 3) + (j & 1);
    uint32_t a[4];
    ldsm_x4_t(blk + 4096 + (mt >> 2) * 2048 + vtok * 128 + ((chunk ^ (vtok & 7)) << 4), a);
    if (valid < 16) {  // rows past the end may hold any bits: zero them (P is 0 there, NaN * 0 is not)
      a[0] &= m01;
      a[1] &= m01;
      a[2] &= m89;
      a[3] &= m89;
    }
    mma_bf16(o[mt], a, pb0, pb1);
  }
}

// Logits of retained block b (tokens g, g + 8; -inf past valid) on the G = 1 path.
template <int BITS, int GROUP, int QACC>
__device__ __forceinline__ void mha_lo_logits(uint32_t unit, int b, int valid, const uint32_t (&qh)[8][2], float qs0,
                                              float qs1, float scale, float (&s)[2], int lane) {
  constexpr LoUnit U = lo_unit_layout(BITS, GROUP);
  constexpr int NG = kHeadDim / GROUP;
  constexpr int PR = U.param_row;
  const uint32_t ka = unit + U.k_a + b * 16 * U.pitch;
  const uint32_t kp = unit + U.k_p + b * 16 * PR;
  const int g = lane >> 2, t = lane & 3;
  // (alpha, beta) of tokens g and g + 8 for the groups of columns 2t, 2t + 1
  uint32_t pg[2], p8[2];
  if constexpr (NG == 1) {
    pg[0] = pg[1] = lds32(kp + g * PR);
    p8[0] = p8[1] = lds32(kp + (g + 8) * PR);
  } else {
    const int off = NG == 4 ? 8 * (t & 1) : 0;
    lds_vec<2>(kp + g * PR + off, pg);
    lds_vec<2>(kp + (g + 8) * PR + off, p8);
  }
  float accs[QACC][4];
#pragma unroll
  for (int q = 0; q < QACC; ++q) accs[q][0] = accs[q][1] = accs[q][2] = accs[q][3] = 0.f;
  KeyFrag<BITS, U.pitch> kf;
  kf.load(ka, lane);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    uint32_t c[4];
    kf.code(ks, c);
    mma_f16(accs[ks % QACC], c, qh[ks][0], qh[ks][1]);
  }
  float acc[4];
  sum_acc(accs, acc);
  const __half2 g0 = u32_as_h2(pg[0]), e0 = u32_as_h2(p8[0]);
  float sg = fmaf(__low2float(g0), acc[0], __high2float(g0) * qs0);
  float s8 = fmaf(__low2float(e0), acc[2], __high2float(e0) * qs0);
  if constexpr (NG >= 2) {
    const __half2 g1 = u32_as_h2(pg[1]), e1 = u32_as_h2(p8[1]);
    sg += fmaf(__low2float(g1), acc[1], __high2float(g1) * qs1);
    s8 += fmaf(__low2float(e1), acc[3], __high2float(e1) * qs1);
  }
  if constexpr (NG == 4) {  // lanes t and t ^ 1 hold the group pairs (0, 1) and (2, 3)
    sg += __shfl_xor_sync(0xffffffffu, sg, 1);
    s8 += __shfl_xor_sync(0xffffffffu, s8, 1);
  }
  s[0] = g < valid ? sg * scale : -INFINITY;
  s[1] = g + 8 < valid ? s8 * scale : -INFINITY;
}

// Values of retained block b on the G = 1 path: o += the block's codes (plus voff) times the group-column
// probability operand; the correction tile ob += beta sums, alpha sums and the normaliser.
template <int BITS, int GROUP>
__device__ __forceinline__ void mha_lo_values(uint32_t unit, int b, int valid, const float (&p)[2], float (&o)[8][4],
                                              float (&ob)[4], int lane) {
  constexpr LoUnit U = lo_unit_layout(BITS, GROUP);
  constexpr int NG = kHeadDim / GROUP;
  constexpr int PR = U.param_row;
  const uint32_t va = unit + U.v_a + b * 16 * U.pitch;
  const uint32_t vp = unit + U.v_p + b * 16 * PR;
  const int g = lane >> 2, t = lane & 3;
  const uint32_t pb0 = movmatrix_t(pack_f16(p[0], p[0]));  // tokens 2t, 2t+1, every column
  const uint32_t pb1 = movmatrix_t(pack_f16(p[1], p[1]));  // tokens 2t+8, 2t+9
  ValFrag<BITS, U.pitch, false> vf;
  vf.load(va, lane);
  // (alpha, beta) of group g (lanes g < NG; the others read group 0 and do not use it) for the four tokens
  const uint32_t gp = vp + 4 * (g < NG ? g : 0);
  uint32_t w0 = lds32(gp + (2 * t) * PR), w1 = lds32(gp + (2 * t + 1) * PR);
  uint32_t w8 = lds32(gp + (2 * t + 8) * PR), w9 = lds32(gp + (2 * t + 9) * PR);
  if (valid < 16) {  // exact zeros past the end
    if (2 * t >= valid) w0 = 0u;
    if (2 * t + 1 >= valid) w1 = 0u;
    if (2 * t + 8 >= valid) w8 = 0u;
    if (2 * t + 9 >= valid) w9 = 0u;
  }
  uint32_t B0, B1, A0, A2;
  if (g < NG) {
    B0 = h2_as_u32(__hmul2(u32_as_h2(pb0), u32_as_h2(prmt(w0, w1, 0x5410u))));
    B1 = h2_as_u32(__hmul2(u32_as_h2(pb1), u32_as_h2(prmt(w8, w9, 0x5410u))));
    A0 = prmt(w0, w1, 0x7632u);
    A2 = prmt(w8, w9, 0x7632u);
  } else {
    B0 = g == NG ? pb0 : 0u;
    B1 = g == NG ? pb1 : 0u;
    A0 = A2 = g == NG ? kOnesF16 : 0u;
  }
  {
    const uint32_t a[4] = {A0, 0u, A2, 0u};
    mma_f16(ob, a, B0, B1);
  }
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    uint32_t a[4];
    vf.code(mt, a);
    mma_f16(o[mt], a, B0, B1);  // column g < NG: sums p * alpha_g * (code + offset)
  }
}

template <int BITS, int GROUP, int NK>
__device__ __forceinline__ void mha_coded(uint32_t unit, int b, int n_left, const uint32_t (&qh)[8][2], float qs0,
                                          float qs1, float scale, Softmax& st, float (&o)[8][4], float (&ob)[4],
                                          int lane) {
  float s[NK][2], p[NK][2];
#pragma unroll
  for (int k = 0; k < NK; ++k)
    mha_lo_logits<BITS, GROUP, NK == 1 ? kQkAcc : kPairAcc>(unit, b + k, min(16, n_left - 16 * k), qh, qs0, qs1,
                                                             scale, s[k], lane);
  mha_softmax<NK>(s, st, o, ob, p);
#pragma unroll
  for (int k = 0; k < NK; ++k) mha_lo_values<BITS, GROUP>(unit, b + k, min(16, n_left - 16 * k), p[k], o, ob, lane);
}

// The partial of the G = 1 path (same content as write_partial): channel c of tile mt (group gi) is read from column
// gi, out = (o - voff * alpha sum + beta sum) / normaliser, with the sums taken from the correction tile.
template <int BITS, int GROUP>
__device__ __forceinline__ void mha_write_partial(const AttnArgs& a, int slot, Softmax& st, const float (&o)[8][4],
                                                  const float (&ob)[4], int lane) {
  constexpr int NG = kHeadDim / GROUP;
  const int g = lane >> 2, t = lane & 3;
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {  // over the rows g (the four lanes of a row hold the same tokens)
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], off);
    st.mx[0] = fmaxf(st.mx[0], __shfl_xor_sync(0xffffffffu, st.mx[0], off));
  }
  const float c = st.mx[0] == st.m[0] ? 1.f : fast_exp2((st.m[0] - st.mx[0]) * kLog2e);
  // correction tile entry (r, n) sits in lane 4 r + n / 2, element n & 1 (rows r < 8)
  const float inv = 1.f / __shfl_sync(0xffffffffu, ob[NG & 1], 4 * NG + NG / 2);
  float za[NG], zb[NG];
#pragma unroll
  for (int gi = 0; gi < NG; ++gi) {
    za[gi] = __shfl_sync(0xffffffffu, ob[gi & 1], 4 * NG + gi / 2);  // sum of p * alpha of group gi
    zb[gi] = __shfl_sync(0xffffffffu, ob[NG & 1], 4 * gi + NG / 2);  // sum of p * beta of group gi
  }
  float* po = a.part_o + (size_t)slot * kHeadDim;
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int gi = (16 * mt) / GROUP;
    if (t == gi / 2) {
      const float z = fmaf(-voff<BITS>(mt), za[gi], zb[gi]);
      po[16 * mt + g] = (o[mt][gi & 1] + z) * inv;
      po[16 * mt + 8 + g] = (o[mt][2 + (gi & 1)] + z) * inv;
    }
  }
  if (lane == 0) {
    a.part_ml[(size_t)slot * 2] = st.mx[0];
    a.part_ml[(size_t)slot * 2 + 1] = st.l[0] * c;
  }
}

template <int BITS, int GROUP, int HB, bool KCH>
__device__ __forceinline__ void issue_unit(const AttnArgs& a, const Cursor& c, uint32_t dst, uint32_t bar, uint64_t pol) {
  constexpr LoUnit U = KCH ? lo_unit_layout_kch(BITS, GROUP) : lo_unit_layout(BITS, GROUP);
  const UnitKind k = cursor_kind(c, a.hi_units, a.n_u);
  if constexpr (HB != 16) {
    if (k.hi) {
      constexpr LoUnit H = lo_unit_layout(HB, kHiGroup);
      const long long row = (long long)c.bh * a.hi_stride + 16 * H.blocks * k.index;  // first slot
      mbar_arrive_expect_tx(bar, H.tx);
      const int crow = (int)(row * H.pitch / H.map_w), prow = (int)(row * H.param_row / H.param_w);
      tma_load_2d(dst + H.k_a, &a.map_k_hi, 0, crow, bar, pol);
      tma_load_2d(dst + H.v_a, &a.map_v_hi, 0, crow, bar, pol);
      tma_load_2d(dst + H.k_p, &a.map_k_hp, 0, prow, bar, pol);
      tma_load_2d(dst + H.v_p, &a.map_v_hp, 0, prow, bar, pol);
      return;
    }
  }
  MIKV_DEBUG_ASSERT(c.bh < a.batch * a.heads_kv && c.i < a.n_u, a.status);
  MIKV_DEBUG_ASSERT(k.hi ? 16 * k.index < a.hi_stride : 16 * U.blocks * k.index < a.lo_cap, a.status);
  if (k.hi) {
    const int row = c.bh * a.hi_stride + 16 * k.index;
    mbar_arrive_expect_tx(bar, kHiBlockBytes);
    tma_load_2d(dst, &a.map_k_hi, 0, row, bar, pol);
    tma_load_2d(dst + 2048, &a.map_k_hi, 64, row, bar, pol);
    tma_load_2d(dst + 4096, &a.map_v_hi, 0, row, bar, pol);
    tma_load_2d(dst + 6144, &a.map_v_hi, 64, row, bar, pol);
  } else {
    // one box per array covers the whole unit (U.blocks blocks of 16 rows); rows past this head's
    // retained length are masked by the consumer, rows past the array are zero-filled by TMA
    const long long row = (long long)c.bh * a.lo_cap + 16 * U.blocks * k.index;  // first token row
    mbar_arrive_expect_tx(bar, U.tx);
    const int crow = (int)(row * U.pitch / U.map_w), prow = (int)(row * U.param_row / U.param_w);
    tma_load_2d(dst + U.k_a, &a.map_k_lo, 0, crow, bar, pol);
    tma_load_2d(dst + U.v_a, &a.map_v_lo, 0, crow, bar, pol);
    if constexpr (KCH) {  // the group's key (alpha, beta) pairs: four 128-byte rows per group of 64 tokens
      const long long grp = (long long)c.bh * (a.lo_cap / kKchGroup) + (16 * U.blocks * k.index) / kKchGroup;
      tma_load_2d(dst + U.k_p, &a.map_k_par, 0, (int)(4 * grp), bar, pol);
    } else {
      tma_load_2d(dst + U.k_p, &a.map_k_par, 0, prow, bar, pol);
    }
    tma_load_2d(dst + U.v_p, &a.map_v_par, 0, prow, bar, pol);
  }
}

// The copies of issue_unit as L2 prefetches (issued before the kernel may read the cache).
template <int BITS, int GROUP, int HB, bool KCH>
__device__ __forceinline__ void prefetch_unit(const AttnArgs& a, const Cursor& c) {
  constexpr LoUnit U = KCH ? lo_unit_layout_kch(BITS, GROUP) : lo_unit_layout(BITS, GROUP);
  const UnitKind k = cursor_kind(c, a.hi_units, a.n_u);
  if constexpr (HB != 16) {
    if (k.hi) {
      constexpr LoUnit H = lo_unit_layout(HB, kHiGroup);
      const long long row = (long long)c.bh * a.hi_stride + 16 * H.blocks * k.index;  // first slot
      const int crow = (int)(row * H.pitch / H.map_w), prow = (int)(row * H.param_row / H.param_w);
      tma_prefetch_2d(&a.map_k_hi, 0, crow);
      tma_prefetch_2d(&a.map_v_hi, 0, crow);
      tma_prefetch_2d(&a.map_k_hp, 0, prow);
      tma_prefetch_2d(&a.map_v_hp, 0, prow);
      return;
    }
  }
  if (k.hi) {
    const int row = c.bh * a.hi_stride + 16 * k.index;
    tma_prefetch_2d(&a.map_k_hi, 0, row);
    tma_prefetch_2d(&a.map_k_hi, 64, row);
    tma_prefetch_2d(&a.map_v_hi, 0, row);
    tma_prefetch_2d(&a.map_v_hi, 64, row);
  } else {
    // one box per array covers the whole unit (U.blocks blocks of 16 rows); rows past this head's
    // retained length are masked by the consumer, rows past the array are zero-filled by TMA
    const long long row = (long long)c.bh * a.lo_cap + 16 * U.blocks * k.index;  // first token row
    const int crow = (int)(row * U.pitch / U.map_w), prow = (int)(row * U.param_row / U.param_w);
    tma_prefetch_2d(&a.map_k_lo, 0, crow);
    tma_prefetch_2d(&a.map_v_lo, 0, crow);
    if constexpr (KCH) {  // the group's key (alpha, beta) pairs: four 128-byte rows per group of 64 tokens
      const long long grp = (long long)c.bh * (a.lo_cap / kKchGroup) + (16 * U.blocks * k.index) / kKchGroup;
      tma_prefetch_2d(&a.map_k_par, 0, (int)(4 * grp));
    } else {
      tma_prefetch_2d(&a.map_k_par, 0, prow);
    }
    tma_prefetch_2d(&a.map_v_par, 0, prow);
  }
}

// The step's new token for important slot `slot` of head bh (fused insertion, bf16 important set): its key and
// value rows replace row slot % 16 of the staged 16-token unit (the 128B-swizzled boxes of 64 channels x 16
// rows, keys at +0 / +2048, values at +4096 / +6144) and are written to the cache with its id and a zero score.
// Lane l carries channels 4 l .. 4 l + 3 of both rows.
__device__ __forceinline__ void insert_row(const AttnArgs& a, int bh, int slot, uint32_t stage, int lane) {
  const uint2 kw = reinterpret_cast<const uint2*>(a.ins_k + (size_t)bh * kHeadDim)[lane];
  const uint2 vw = reinterpret_cast<const uint2*>(a.ins_v + (size_t)bh * kHeadDim)[lane];
  const int r = slot & 15, box = lane >> 4, chunk = (lane & 15) >> 1;
  const uint32_t off = box * 2048 + r * 128 + ((chunk ^ (r & 7)) << 4) + (lane & 1) * 8;
  asm volatile("st.shared.v2.u32 [%0], {%1, %2};" ::"r"(stage + off), "r"(kw.x), "r"(kw.y) : "memory");
  asm volatile("st.shared.v2.u32 [%0], {%1, %2};" ::"r"(stage + 4096 + off), "r"(vw.x), "r"(vw.y) : "memory");
  const size_t row = (size_t)bh * a.hi_stride + slot;
  reinterpret_cast<uint2*>(a.ins_k_hi + row * kHeadDim)[lane] = kw;
  reinterpret_cast<uint2*>(a.ins_v_hi + row * kHeadDim)[lane] = vw;
  if (lane == 0) {
    a.ins_hi_tok[row] = a.ins_tok;
    a.ins_acc[row] = 0.f;
  }
  __syncwarp();
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

template <int BITS, int GROUP, int HB, int G, bool KCH = false>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) attention_kernel(const __grid_constant__ AttnArgs a) {
  constexpr LoUnit U = KCH ? lo_unit_layout_kch(BITS, GROUP) : lo_unit_layout(BITS, GROUP);
  constexpr LoUnit H = lo_unit_layout(HB == 16 ? 2 : HB, kHiGroup);
  static_assert(U.total <= kStageBytes && H.total <= kStageBytes, "unit too large for a stage");
  static_assert(!KCH || HB == 16, "per-channel retained keys need a bf16 important set");
  // one query head per KV head with a bf16 important set and per-token retained keys: the group-column path
  constexpr bool MHA = MIKV_MHA_PATH && G == 1 && HB == 16 && !KCH;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wg = blockIdx.x * kWarps + warp;
  if (wg >= a.n_warps) return;  // no block-wide synchronisation follows
  const uint32_t ring = base + warp * kNS * kStageBytes;
  const uint32_t bars = base + kWarps * kNS * kStageBytes + warp * kNS * 8;
  const int u0 = (int)((long long)wg * a.n_units / a.n_warps);
  const int u1 = (int)((long long)(wg + 1) * a.n_units / a.n_warps);
  const int hu = a.hi_units, n_u = a.n_u;
  Cursor ci = cursor_at(u0, hu, n_u);  // next unit to issue (lane 0)
  const uint64_t pol = l2_evict_first();  // the cache is streamed once per launch
  if (lane == 0) {
    for (int s = 0; s < kNS; ++s) mbar_init(bars + 8 * s, 1);
    fence_mbar_init();
    prefetch_tensormap(&a.map_k_hi);
    prefetch_tensormap(&a.map_v_hi);
    if (HB != 16) {
      prefetch_tensormap(&a.map_k_hp);
      prefetch_tensormap(&a.map_v_hp);
    }
    if (a.lo_blocks > 0) {  // the retained-set maps are only encoded when the retained arrays exist
      prefetch_tensormap(&a.map_k_lo);
      prefetch_tensormap(&a.map_v_lo);
      prefetch_tensormap(&a.map_k_par);
      prefetch_tensormap(&a.map_v_par);
    }
  }
  // warm L2 with this warp's first units while the previous kernel drains (reads only; L2 stays coherent with
  // its writes). Prefetching further ahead than the ring during the stream measured slower on every shape.
  if (lane == 0) {
    Cursor cp = cursor_at(u0, hu, n_u);
    for (int k = 0; k < kNS && u0 + k < u1; ++k) {
      prefetch_unit<BITS, GROUP, HB, KCH>(a, cp);
      cursor_next(cp, hu, n_u);
    }
  }
  // the first head's query rows (G x 256 bytes) and balancer row (512 bytes) into L2, every line of both
  if (MIKV_Q_PREFETCH && u0 < u1) {
    const int b0 = ci.bh / a.heads_kv, h0 = ci.bh - b0 * a.heads_kv;
    const char* qrow =
        reinterpret_cast<const char*>(static_cast<const __nv_bfloat16*>(a.q) + (size_t)(b0 * a.heads_q + h0 * G) * kHeadDim);
    constexpr int nq = 2 * G + 1;  // the rows need not start on a line
    static_assert(nq + 5 <= 32, "one line per lane");
    if (lane < nq) prefetch_l2(qrow + (lane < 2 * G ? 128 * lane : 256 * G - 1));
    if (!KCH && a.balancer && lane >= nq && lane < nq + 5) {
      const char* brow = reinterpret_cast<const char*>(a.balancer + h0 * kHeadDim);
      prefetch_l2(brow + (lane - nq < 4 ? 128 * (lane - nq) : 4 * kHeadDim - 1));
    }
  }
  grid_dependency_wait();  // the cache and the query come from the kernels before this one
  allow_dependent_launch();
  if (lane == 0) {
    for (int k = 0; k < kNS && u0 + k < u1; ++k) {
      issue_unit<BITS, GROUP, HB, KCH>(a, ci, ring + k * kStageBytes, bars + 8 * k, pol);
      cursor_next(ci, hu, n_u);
    }
  }
  __syncwarp();

  const int g = lane >> 2, t = lane & 3;
  uint32_t qb[8][2], qh[8][2];
  constexpr int NB = 1 + (kHeadDim / GROUP + 1) / 2;  // beta rows + alpha-sum pairs
  Softmax st;
  float o[8][4], ob[NB][4];
  __shared__ int s_ins[kWarps];  // each warp's insertion slot of its current head (fused insertion; kept out of
                                 // the register file)
  if (lane == 0) s_ins[warp] = -1;
  float* logit_base = nullptr;
  float qs0 = 0.f, qs1 = 0.f;  // G = 1 path: sums of the balanced query over the groups of columns 2t, 2t + 1
  Cursor cc = cursor_at(u0, hu, n_u);  // unit being consumed
  int cur = -1;
  bool failed = false;
  int u = u0;
  for (; u < u1; ++u) {
    if (cc.bh != cur) {
      if (cur >= 0) {
        if constexpr (MHA)
          mha_write_partial<BITS, GROUP>(a, wg + cur, st, o, ob[0], lane);
        else
          write_partial<BITS, GROUP, G, NB>(a, wg + cur, st, o, ob, lane);
      }
      cur = cc.bh;
      const int b = cur / a.heads_kv, h = cur - b * a.heads_kv;
      // query fragments (B operand: head g; channels 16 ks + 2t (+1) and 16 ks + 2t + 8 (+9))
      if constexpr (MHA) {
        mha_query<GROUP>(a, b, h, lane, qb, qh, qs0, qs1);
      } else {
        // Column g < G holds query head g. The RQ = 8 / G rows of lanes g' = g + G j (j < RQ) share head g's
        // fragments: row g' loads and divides (Eq. 4) the k-steps ks = j (mod RQ), every load before any division
        // (the divisions branch), and the fragments reach row g by shuffles; rows g >= G then hold zeros.
        constexpr int RQ = 8 / G;
        const int hq = g % G, j = g / G;
        const __nv_bfloat16* qp =
            static_cast<const __nv_bfloat16*>(a.q) + (size_t)(b * a.heads_q + h * G + hq) * kHeadDim;
        uint32_t qw[8 / RQ][2], fw[8 / RQ][2];
        float2 bal[8 / RQ][2];
#pragma unroll
        for (int m = 0; m < 8 / RQ; ++m)
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            const int c = 16 * (j + RQ * m) + 2 * t + 8 * r;
            qw[m][r] = *reinterpret_cast<const uint32_t*>(qp + c);
            bal[m][r] = !KCH && a.balancer ? *reinterpret_cast<const float2*>(a.balancer + h * kHeadDim + c)
                                           : make_float2(1.f, 1.f);
          }
#pragma unroll
        for (int m = 0; m < 8 / RQ; ++m)
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            const float q0 = __uint_as_float(qw[m][r] << 16), q1 = __uint_as_float(qw[m][r] & 0xffff0000u);
            if constexpr (KCH)  // per-channel retained keys are not balanced
              fw[m][r] = pack_f16(q0, q1);
            else
              fw[m][r] = pack_f16(__fdiv_rn(q0, bal[m][r].x), __fdiv_rn(q1, bal[m][r].y));
          }
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
#pragma unroll
          for (int r = 0; r < 2; ++r) {  // k-step ks of head g: row g + G (ks mod RQ), its entry ks div RQ
            const int src = 4 * ((g < G ? g : 0) + G * (ks % RQ)) + t;
            const uint32_t wq = __shfl_sync(0xffffffffu, qw[ks / RQ][r], src);
            const uint32_t wf = __shfl_sync(0xffffffffu, fw[ks / RQ][r], src);
            qb[ks][r] = g < G ? wq : 0u;
            qh[ks][r] = g < G ? wf : 0u;
          }
      }
      logit_base = a.hi_logits ? a.hi_logits + (size_t)(b * a.heads_q + h * G) * a.hi_stride : nullptr;
      if (HB == 16 && a.ins_slots) {
        __syncwarp();
        if (lane == 0) {
          const int sl = a.ins_slots[cur];
          const bool ok = sl >= 0 && sl < a.hi_cap;  // an out-of-range slot inserts nothing
          if (!ok) MIKV_BOUNDS_FAIL(a.status);
          s_ins[warp] = ok ? sl : -1;
        }
        __syncwarp();
      }
      st.m[0] = st.m[1] = -INFINITY;
      st.l[0] = st.l[1] = 0.f;
      st.mx[0] = st.mx[1] = -INFINITY;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
#pragma unroll
      for (int i = 0; i < NB; ++i) ob[i][0] = ob[i][1] = ob[i][2] = ob[i][3] = 0.f;
    }
    const int s = (u - u0) % kNS;
    const uint32_t use = (u - u0) / kNS;
    if (!mbar_wait(bars + 8 * s, use & 1)) {
      record_error(a.status, kErrFullTimeout);
      failed = true;
      break;
    }
    const uint32_t stage = ring + s * kStageBytes;
    const UnitKind k = cursor_kind(cc, hu, n_u);
    if (k.hi) {
      if constexpr (HB == 16) {
        if (a.ins_slots) {
          const int sl = s_ins[warp];
          if (sl >= 0 && (sl >> 4) == k.index) insert_row(a, cur, sl, stage, lane);
        }
        if constexpr (MHA)
          mha_hi<kHeadDim / GROUP>(stage, min(16, a.hi_cap - 16 * k.index), 16 * k.index, qb, a.sm_scale, logit_base,
                                   st, o, ob[0], lane);
        else
          process_hi<G, NB>(stage, min(16, a.hi_cap - 16 * k.index), 16 * k.index, qb, a.sm_scale, logit_base,
                            a.hi_stride, st, o, ob, lane);
      } else {
        const int first = k.index * H.blocks;
        const int nb = min(H.blocks, a.hi_blocks - first);
        int b = 0;
        if (kLoPair)
          for (; b + 1 < nb; b += 2)
            process_coded<HB, kHiGroup, G, NB, 2, true>(stage, b, a.hi_cap - 16 * (first + b), qh, a.sm_scale, st,
                                                        o, ob, lane, logit_base, a.hi_stride, 16 * (first + b));
        for (; b < nb; ++b)
          process_coded<HB, kHiGroup, G, NB, 1, true>(stage, b, a.hi_cap - 16 * (first + b), qh, a.sm_scale, st, o,
                                                      ob, lane, logit_base, a.hi_stride, 16 * (first + b));
      }
    } else {
      const int first = k.index * U.blocks;
      const int nb = min(U.blocks, a.lo_blocks - first);
      int b = 0;
      if constexpr (KCH) {
        uint32_t qk[8][2];
        float kbias[2];
        kch_prepare(stage + U.k_p, qh, qk, kbias, lane);
        for (; b + 1 < nb; b += 2)
          process_coded<BITS, GROUP, G, NB, 2, false, true>(stage, b, a.n_lo - 16 * (first + b), qk, a.sm_scale, st,
                                                            o, ob, lane, nullptr, 0, 0, kbias);
      } else if constexpr (MHA) {
        if (kLoPair)
          for (; b + 1 < nb; b += 2)
            mha_coded<BITS, GROUP, 2>(stage, b, a.n_lo - 16 * (first + b), qh, qs0, qs1, a.sm_scale, st, o, ob[0],
                                      lane);
        for (; b < nb; ++b)
          mha_coded<BITS, GROUP, 1>(stage, b, a.n_lo - 16 * (first + b), qh, qs0, qs1, a.sm_scale, st, o, ob[0], lane);
      } else {
        if (kLoPair)
          for (; b + 1 < nb; b += 2)
            process_coded<BITS, GROUP, G, NB, 2, false>(stage, b, a.n_lo - 16 * (first + b), qh, a.sm_scale, st, o,
                                                        ob, lane);
        for (; b < nb; ++b)
          process_coded<BITS, GROUP, G, NB, 1, false>(stage, b, a.n_lo - 16 * (first + b), qh, a.sm_scale, st, o,
                                                      ob, lane);
      }
    }
    cursor_next(cc, hu, n_u);
    __syncwarp();
    if (lane == 0 && u + kNS < u1) {
      fence_proxy_async();  // our generic reads of this stage precede the next asynchronous write
      issue_unit<BITS, GROUP, HB, KCH>(a, ci, stage, bars + 8 * s, pol);
      cursor_next(ci, hu, n_u);
    }
  }
  if (failed) {
    // leave no copy in flight into this warp's ring: wait (bounded) for every unit still issued
    if (lane == 0)
      for (int v = u; v < u1 && v < u + kNS; ++v) {
        const int s = (v - u0) % kNS;
        if (!mbar_wait(bars + 8 * s, ((v - u0) / kNS) & 1)) record_error(a.status, kErrDrainTimeout);
      }
    return;
  }
  if (cur >= 0) {
    if constexpr (MHA)
      mha_write_partial<BITS, GROUP>(a, wg + cur, st, o, ob[0], lane);
    else
      write_partial<BITS, GROUP, G, NB>(a, wg + cur, st, o, ob, lane);
  }
}

template <int BITS, int GROUP, int HB, int G, bool KCH = false>
cudaError_t launch_kernel(const AttnArgs& a, int grid, cudaStream_t st) {
  auto kern = attention_kernel<BITS, GROUP, HB, G, KCH>;
  static bool configured = false;
  const int smem = smem_bytes();
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_chained(kern, dim3(grid), dim3(kThreads), smem, st, a);
}

template <int BITS, int GROUP, int HB, bool KCH>
cudaError_t dispatch_g(const AttnArgs& a, int G, int grid, cudaStream_t st) {
  switch (G) {
    case 1: return launch_kernel<BITS, GROUP, HB, 1, KCH>(a, grid, st);
    case 2: return launch_kernel<BITS, GROUP, HB, 2, KCH>(a, grid, st);
    case 4: return launch_kernel<BITS, GROUP, HB, 4, KCH>(a, grid, st);
    case 8: return launch_kernel<BITS, GROUP, HB, 8, KCH>(a, grid, st);
  }
  return cudaErrorInvalidValue;
}

template <int BITS, int HB, bool KCH>
cudaError_t dispatch_group(const AttnArgs& a, int group, int G, int grid, cudaStream_t st) {
  switch (group) {
    case 32: return dispatch_g<BITS, 32, HB, KCH>(a, G, grid, st);
    case 64: return dispatch_g<BITS, 64, HB, KCH>(a, G, grid, st);
    case 128: return dispatch_g<BITS, 128, HB, KCH>(a, G, grid, st);
  }
  return cudaErrorInvalidValue;
}

// Every (retained bits, group, G) kernel for one important-set precision HB (16 = bf16), with per-token
// or (KCH) per-channel retained keys.
template <int HB, bool KCH = false>
cudaError_t launch_attention_hb(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st) {
  switch (bits) {
    case 2: return dispatch_group<2, HB, KCH>(a, group, G, grid, st);
    case 3: return dispatch_group<3, HB, KCH>(a, group, G, grid, st);
    case 4: return dispatch_group<4, HB, KCH>(a, group, G, grid, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace
}  // namespace mikv
