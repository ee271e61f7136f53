// mikv_attention.cu — split-K flash-decoding over the mixed-precision KV cache (sm_103a).
//
// Computes, per (batch b, KV head h) and the G query heads that share it, softmax attention of the
// new query over the important set (bf16 K/V, attended with q) and the retained set (N-bit codes,
// keys balanced and attended with q / balancer), Eq. 3-4 of arxiv 2402.18096; the two sets are one
// unordered set for attention (Sec. 3.4), so they are streamed separately and merged by the online
// softmax.
//
// Design (per CTA: 4 consumer warps + 1 producer warp, 2 CTAs per SM, persistent over work items):
//  * work item = (b, h, context split); splits are contiguous ranges of 16-token blocks;
//  * the producer lane streams blocks into a 3-stage shared-memory ring with TMA: 2-D tensor copies
//    with hardware swizzle for bf16 rows and packed codes, 1-D bulk copies for (alpha, beta) pairs,
//    completion tracked by mbarriers (every wait is bounded in time);
//  * a consumer warp takes one 16-token block at a time: ldmatrix yields the mma.sync fragments
//    directly (the packed-code layout of the ABI is built for this), codes become fp16 in registers
//    (exact magic-number conversion, then alpha * c + beta), QK^T and PV run on tensor cores with fp32
//    accumulation (tokens on M for QK^T, channels on M for PV, query heads on N), online softmax in
//    fp32; movmatrix turns the probabilities into the PV operand without shared memory;
//  * the 4 warps' partial (max, sum, output) are combined through shared memory and written per item;
//    a merge kernel combines the splits of each query head.
#include <math.h>

#include "mikv_device.cuh"
#include "mikv_internal.h"

namespace mikv {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kStages = 3;
constexpr int kStageBytes = 32768;
constexpr int kHiBlockBytes = 8192;  // K and V of 16 tokens: 4 boxes of 16 rows x 64 bf16
constexpr int kMinBlocksPerSplit = 8;
constexpr int kCtasPerSm = 2;
constexpr int kItemsPerCta = 8;
constexpr float kLog2e = 1.4426950408889634f;

template <int BITS, int GROUP>
struct LoLayout {
  static constexpr int kRowBytes = 16 * BITS;               // packed codes of one row
  static constexpr int kCodeBox = 16 * kRowBytes;           // 16 rows of codes
  static constexpr int kParamRow = 4 * (kHeadDim / GROUP);  // (alpha, beta) fp16 pairs of one row
  static constexpr int kParamBox = 16 * kParamRow;
  static constexpr int kTxBytes = 2 * kCodeBox + 2 * kParamBox;
  static constexpr int kBlockBytes = (kTxBytes + 511) / 512 * 512;  // keeps swizzle atoms aligned
  static constexpr int kPerWarpRaw = kStageBytes / (kConsumerWarps * kBlockBytes);
  static constexpr int kBlocksPerWarp = kPerWarpRaw < 8 ? kPerWarpRaw : 8;
  static constexpr int kK = 0, kV = kCodeBox, kKp = 2 * kCodeBox, kVp = 2 * kCodeBox + kParamBox;
};

__host__ __device__ constexpr int red_bytes(int G) { return kConsumerWarps * G * 130 * 4; }
__host__ __device__ constexpr int smem_bytes(int G) {
  return 1024 + kStages * kStageBytes + red_bytes(G) + 2 * kStages * 8;
}

__device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Stage k of an item with n_hs important stages and n_ls retained stages: alternate while both
// remain so that bandwidth-heavy (important) and ALU-heavy (retained) stages interleave.
__device__ __forceinline__ void stage_kind(int k, int n_hs, int n_ls, bool& hi, int& j) {
  const int m = n_hs < n_ls ? n_hs : n_ls;
  if (k < 2 * m) {
    hi = (k & 1) == 0;
    j = k >> 1;
  } else {
    hi = n_hs > n_ls;
    j = m + (k - 2 * m);
  }
}

__device__ __forceinline__ void split_range(int total, int n_split, int s, int& b0, int& b1) {
  b0 = (int)((long long)total * s / n_split);
  b1 = (int)((long long)total * (s + 1) / n_split);
}

struct Softmax {
  float m[2], l[2];
};

// Online-softmax update for one 16-token block. sacc holds raw q.k for (token g, head 2t),
// (g, 2t+1), (g+8, 2t), (g+8, 2t+1); returns unnormalised probabilities in p.
__device__ __forceinline__ void softmax_block(const float (&s)[4], Softmax& st, float (&o)[8][4],
                                              float (&p)[4]) {
  float bm0 = fmaxf(s[0], s[2]), bm1 = fmaxf(s[1], s[3]);
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, off));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, off));
  }
  const float mn0 = fmaxf(st.m[0], bm0), mn1 = fmaxf(st.m[1], bm1);
  if (__any_sync(0xffffffffu, mn0 > st.m[0] || mn1 > st.m[1])) {
    const float c0 = mn0 == st.m[0] ? 1.f : fast_exp2((st.m[0] - mn0) * kLog2e);
    const float c1 = mn1 == st.m[1] ? 1.f : fast_exp2((st.m[1] - mn1) * kLog2e);
    st.l[0] *= c0;
    st.l[1] *= c1;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      o[mt][0] *= c0;
      o[mt][1] *= c1;
      o[mt][2] *= c0;
      o[mt][3] *= c1;
    }
    st.m[0] = mn0;
    st.m[1] = mn1;
  }
  const float ml0 = st.m[0] * kLog2e, ml1 = st.m[1] * kLog2e;
  p[0] = fast_exp2(fmaf(s[0], kLog2e, -ml0));
  p[1] = fast_exp2(fmaf(s[1], kLog2e, -ml1));
  p[2] = fast_exp2(fmaf(s[2], kLog2e, -ml0));
  p[3] = fast_exp2(fmaf(s[3], kLog2e, -ml1));
  st.l[0] += p[0] + p[2];
  st.l[1] += p[1] + p[3];
}

// Scale raw dot products, mask tokens >= valid, and store important-set logits.
template <int G>
__device__ __forceinline__ void finish_logits(const float (&acc)[4], float scale, int valid, int g, int t,
                                              float* logit_base, int hi_stride, int slot0,
                                              float (&s)[4]) {
  const float ninf = -INFINITY;
  s[0] = g < valid ? acc[0] * scale : ninf;
  s[1] = g < valid ? acc[1] * scale : ninf;
  s[2] = g + 8 < valid ? acc[2] * scale : ninf;
  s[3] = g + 8 < valid ? acc[3] * scale : ninf;
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

// One block of 16 important tokens (bf16, 128B-swizzled boxes: K ch 0-63, K ch 64-127, V, V).
template <int G>
__device__ __forceinline__ void process_hi(uint32_t blk, int valid, int slot0, const uint32_t (&qb)[8][2],
                                           float scale, float* logit_base, int hi_stride, Softmax& st,
                                           float (&o)[8][4], int lane) {
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const int krow = r8 + 8 * (j & 1);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int chunk = 2 * (ks & 3) + (j >> 1);
    uint32_t a[4];
    ldsm_x4(blk + (ks >> 2) * 2048 + krow * 128 + ((chunk ^ (krow & 7)) << 4), a);
    mma_bf16(acc, a, qb[ks][0], qb[ks][1]);
  }
  float s[4], p[4];
  finish_logits<G>(acc, scale, valid, g, t, logit_base, hi_stride, slot0, s);
  softmax_block(s, st, o, p);
  const uint32_t pb0 = movmatrix_t(pack_bf16(p[0], p[1]));
  const uint32_t pb1 = movmatrix_t(pack_bf16(p[2], p[3]));
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
    a[0] &= m01;
    a[1] &= m01;
    a[2] &= m89;
    a[3] &= m89;
    mma_bf16(o[mt], a, pb0, pb1);
  }
}

// One block of 16 retained tokens: packed codes (swizzled boxes), then (alpha, beta) rows.
template <int BITS, int GROUP, int G>
__device__ __forceinline__ void process_lo(uint32_t blk, int valid, const uint32_t (&qh)[8][2], float scale,
                                           Softmax& st, float (&o)[8][4], int lane) {
  using L = LoLayout<BITS, GROUP>;
  constexpr int NG = kHeadDim / GROUP;
  const int g = lane >> 2, t = lane & 3, r8 = lane & 7, j = lane >> 3;

  // ---- keys: codes of tokens g and g+8
  uint32_t kr[BITS == 4 ? 8 : 4];
  uint32_t kb0 = 0, kb1 = 0;
  {
    const int tok = r8 + 8 * (j & 1);
    if (BITS == 4) {
      const int o0 = tok * 64 + 16 * (j >> 1), sw = ((tok >> 1) & 3) << 4;
      uint32_t r0[4], r1[4];
      ldsm_x4(blk + L::kK + (o0 ^ sw), r0);
      ldsm_x4(blk + L::kK + ((o0 + 32) ^ sw), r1);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        kr[i] = r0[i];
        kr[(BITS == 4 ? 4 : 0) + i] = r1[i];
      }
    } else {
      const int o0 = tok * 32 + 16 * (j >> 1), sw = ((tok >> 2) & 1) << 4;
      uint32_t r0[4];
      ldsm_x4(blk + L::kK + (o0 ^ sw), r0);
#pragma unroll
      for (int i = 0; i < 4; ++i) kr[i] = r0[i];
      if (BITS == 3) ldsm_x2(blk + L::kK + 512 + (lane & 15) * 16, kb0, kb1);
    }
  }
  uint32_t pk0[NG], pk1[NG];
#pragma unroll
  for (int gi = 0; gi < NG; ++gi) {
    pk0[gi] = lds32(blk + L::kKp + g * L::kParamRow + 4 * gi);
    pk1[gi] = lds32(blk + L::kKp + (g + 8) * L::kParamRow + 4 * gi);
  }
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int gi = (16 * ks) / GROUP;
    const uint32_t al0 = prmt(pk0[gi], pk0[gi], 0x1010u), be0 = prmt(pk0[gi], pk0[gi], 0x3232u);
    const uint32_t al1 = prmt(pk1[gi], pk1[gi], 0x1010u), be1 = prmt(pk1[gi], pk1[gi], 0x3232u);
    uint32_t x0, x1, x2, x3;
    if (BITS == 4) {
      const int ri = (ks >> 2) * 4, sh = 4 * (ks & 3);
      x0 = and_or(kr[ri + 0] >> sh, 0x000f000fu, 0x64006400u);
      x1 = and_or(kr[ri + 1] >> sh, 0x000f000fu, 0x64006400u);
      x2 = and_or(kr[ri + 2] >> sh, 0x000f000fu, 0x64006400u);
      x3 = and_or(kr[ri + 3] >> sh, 0x000f000fu, 0x64006400u);
    } else {
      const int sh = 2 * ks;
      x0 = and_or(kr[0] >> sh, 0x00030003u, 0x64006400u);
      x1 = and_or(kr[1] >> sh, 0x00030003u, 0x64006400u);
      x2 = and_or(kr[2] >> sh, 0x00030003u, 0x64006400u);
      x3 = and_or(kr[3] >> sh, 0x00030003u, 0x64006400u);
      if (BITS == 3) {
        x0 |= ((kb0 >> ks) << 2) & 0x00040004u;
        x1 |= ((kb1 >> ks) << 2) & 0x00040004u;
        x2 |= ((kb0 >> (8 + ks)) << 2) & 0x00040004u;
        x3 |= ((kb1 >> (8 + ks)) << 2) & 0x00040004u;
      }
    }
    const uint32_t a[4] = {dequant_pair(x0, al0, be0), dequant_pair(x1, al1, be1), dequant_pair(x2, al0, be0),
                           dequant_pair(x3, al1, be1)};
    mma_f16(acc, a, qh[ks][0], qh[ks][1]);
  }
  float s[4], p[4];
  finish_logits<G>(acc, scale, valid, g, t, nullptr, 0, 0, s);
  softmax_block(s, st, o, p);
  const uint32_t pb0 = movmatrix_t(pack_f16(p[0], p[1]));
  const uint32_t pb1 = movmatrix_t(pack_f16(p[2], p[3]));

  // ---- values: codes of tokens (2t, 2t+1) and (2t+8, 2t+9) for channels 16 mt + g (+8)
  uint32_t vr[BITS == 4 ? 8 : 4];
  uint32_t vb0 = 0, vb1 = 0;
  {
    const int tok = r8 + 8 * (j >> 1);
    if (BITS == 4) {
      const int o0 = tok * 64 + 16 * (j & 1), sw = ((tok >> 1) & 3) << 4;
      uint32_t r0[4], r1[4];
      ldsm_x4_t(blk + L::kV + (o0 ^ sw), r0);
      ldsm_x4_t(blk + L::kV + ((o0 + 32) ^ sw), r1);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        vr[i] = r0[i];
        vr[(BITS == 4 ? 4 : 0) + i] = r1[i];
      }
    } else {
      const int o0 = tok * 32 + 16 * (j & 1), sw = ((tok >> 2) & 1) << 4;
      uint32_t r0[4];
      ldsm_x4_t(blk + L::kV + (o0 ^ sw), r0);
#pragma unroll
      for (int i = 0; i < 4; ++i) vr[i] = r0[i];
      if (BITS == 3) ldsm_x2_t(blk + L::kV + 512 + (lane & 15) * 16, vb0, vb1);
    }
  }
  uint32_t pv[4][NG];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int tok = 2 * t + (k & 1) + 8 * (k >> 1);
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
      const uint32_t w = lds32(blk + L::kVp + tok * L::kParamRow + 4 * gi);
      pv[k][gi] = tok < valid ? w : 0u;  // alpha = beta = 0 makes rows past the end exact zeros
    }
  }
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int gi = (16 * mt) / GROUP;
    const uint32_t a01 = prmt(pv[0][gi], pv[1][gi], 0x5410u), b01 = prmt(pv[0][gi], pv[1][gi], 0x7632u);
    const uint32_t a89 = prmt(pv[2][gi], pv[3][gi], 0x5410u), b89 = prmt(pv[2][gi], pv[3][gi], 0x7632u);
    uint32_t y0, y1, y2, y3;
    if (BITS == 4) {
      const int ri = (mt >> 2) * 4, sh = 4 * (mt & 3);
      y0 = and_or(vr[ri + 0] >> sh, 0x000f000fu, 0x64006400u);
      y1 = and_or(vr[ri + 1] >> sh, 0x000f000fu, 0x64006400u);
      y2 = and_or(vr[ri + 2] >> sh, 0x000f000fu, 0x64006400u);
      y3 = and_or(vr[ri + 3] >> sh, 0x000f000fu, 0x64006400u);
    } else {
      const int sh = 2 * mt;
      y0 = and_or(vr[0] >> sh, 0x00030003u, 0x64006400u);
      y1 = and_or(vr[1] >> sh, 0x00030003u, 0x64006400u);
      y2 = and_or(vr[2] >> sh, 0x00030003u, 0x64006400u);
      y3 = and_or(vr[3] >> sh, 0x00030003u, 0x64006400u);
      if (BITS == 3) {
        y0 |= ((vb0 >> mt) << 2) & 0x00040004u;
        y1 |= ((vb0 >> (8 + mt)) << 2) & 0x00040004u;
        y2 |= ((vb1 >> mt) << 2) & 0x00040004u;
        y3 |= ((vb1 >> (8 + mt)) << 2) & 0x00040004u;
      }
    }
    const uint32_t a[4] = {dequant_pair(y0, a01, b01), dequant_pair(y1, a01, b01), dequant_pair(y2, a89, b89),
                           dequant_pair(y3, a89, b89)};
    mma_f16(o[mt], a, pb0, pb1);
  }
}

template <int BITS, int GROUP, int G>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) attention_split_kernel(const __grid_constant__ AttnArgs a) {
  using L = LoLayout<BITS, GROUP>;
  static_assert(L::kBlocksPerWarp >= 1, "retained block too large for a stage");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  float* red = reinterpret_cast<float*>(base_ptr + kStages * kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + kStages * kStageBytes + red_bytes(G));
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&bars[s]), 1);
      mbar_init(smem_u32(&bars[kStages + s]), kConsumerWarps);
    }
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int* abort_v = &abort_flag;

  if (warp == kConsumerWarps) {
    // ------------------------------------------------------------------ producer
    if (lane != 0) return;
    prefetch_tensormap(&a.map_k_hi);
    prefetch_tensormap(&a.map_v_hi);
    if (a.lo_blocks > 0) {  // the retained-set maps are only encoded when the retained arrays exist
      prefetch_tensormap(&a.map_k_lo);
      prefetch_tensormap(&a.map_v_lo);
    }
    uint32_t it = 0;
    uint32_t issued_mask = 0, last_use[kStages] = {0, 0, 0};
    bool failed = false;
    for (int item = blockIdx.x; item < a.n_items && !failed; item += gridDim.x) {
      const int bh = item / a.n_split, sp = item - bh * a.n_split;
      int hb0, hb1, lb0, lb1;
      split_range(a.hi_blocks, a.n_split, sp, hb0, hb1);
      split_range(a.lo_blocks, a.n_split, sp, lb0, lb1);
      const int n_hs = ceil_div(hb1 - hb0, kConsumerWarps);
      const int n_ls = ceil_div(lb1 - lb0, kConsumerWarps * L::kBlocksPerWarp);
      for (int k = 0; k < n_hs + n_ls; ++k, ++it) {
        const int s = it % kStages;
        const uint32_t use = it / kStages;
        const uint32_t full = smem_u32(&bars[s]), empty = smem_u32(&bars[kStages + s]);
        if (*abort_v) { failed = true; break; }
        if (use > 0 && !mbar_wait(empty, (use - 1) & 1)) {
          record_error(a.status, kErrEmptyTimeout);
          *abort_v = 1;
          failed = true;
          break;
        }
        bool hi;
        int jj;
        stage_kind(k, n_hs, n_ls, hi, jj);
        const uint32_t dst = base + s * kStageBytes;
        if (hi) {
          const int first = hb0 + jj * kConsumerWarps;
          const int nb = min(kConsumerWarps, hb1 - first);
          mbar_arrive_expect_tx(full, nb * kHiBlockBytes);
          for (int w = 0; w < nb; ++w) {
            const int row = bh * a.hi_stride + 16 * (first + w);
            const uint32_t blk = dst + w * kHiBlockBytes;
            tma_load_2d(blk, &a.map_k_hi, 0, row, full);
            tma_load_2d(blk + 2048, &a.map_k_hi, 64, row, full);
            tma_load_2d(blk + 4096, &a.map_v_hi, 0, row, full);
            tma_load_2d(blk + 6144, &a.map_v_hi, 64, row, full);
          }
        } else {
          const int first = lb0 + jj * kConsumerWarps * L::kBlocksPerWarp;
          const int nb = min(kConsumerWarps * L::kBlocksPerWarp, lb1 - first);
          mbar_arrive_expect_tx(full, nb * L::kTxBytes);
          for (int i = 0; i < nb; ++i) {
            const int row = bh * a.lo_cap + 16 * (first + i);
            const uint32_t blk = dst + i * L::kBlockBytes;
            tma_load_2d(blk + L::kK, &a.map_k_lo, 0, row, full);
            tma_load_2d(blk + L::kV, &a.map_v_lo, 0, row, full);
            if (BITS == 3) {
              tma_load_2d(blk + L::kK + 512, &a.map_k_lo1, 32, row, full);
              tma_load_2d(blk + L::kV + 512, &a.map_v_lo1, 32, row, full);
            }
            bulk_load(blk + L::kKp, static_cast<const uint8_t*>(a.k_params) + (size_t)row * L::kParamRow,
                      L::kParamBox, full);
            bulk_load(blk + L::kVp, static_cast<const uint8_t*>(a.v_params) + (size_t)row * L::kParamRow,
                      L::kParamBox, full);
          }
        }
        issued_mask |= 1u << s;
        last_use[s] = use;
      }
    }
    if (failed) {
      // Leave no copy in flight into this CTA's shared memory: wait (bounded) for every stage issued.
      for (int s = 0; s < kStages; ++s)
        if ((issued_mask >> s) & 1u)
          if (!mbar_wait(smem_u32(&bars[s]), last_use[s] & 1)) record_error(a.status, kErrDrainTimeout);
    }
    return;
  }

  // -------------------------------------------------------------------- consumers
  const int g = lane >> 2, t = lane & 3;
  uint32_t it = 0;
  for (int item = blockIdx.x; item < a.n_items; item += gridDim.x) {
    const int bh = item / a.n_split, sp = item - bh * a.n_split;
    const int b = bh / a.heads_kv, h = bh - b * a.heads_kv;
    int hb0, hb1, lb0, lb1;
    split_range(a.hi_blocks, a.n_split, sp, hb0, hb1);
    split_range(a.lo_blocks, a.n_split, sp, lb0, lb1);
    const int n_hs = ceil_div(hb1 - hb0, kConsumerWarps);
    const int n_ls = ceil_div(lb1 - lb0, kConsumerWarps * L::kBlocksPerWarp);

    // query fragments (B operand, head g, channels 16 ks + 2t (+1) and 16 ks + 2t + 8 (+9))
    uint32_t qb[8][2], qh[8][2];
    if (g < G) {
      const __nv_bfloat16* qp =
          static_cast<const __nv_bfloat16*>(a.q) + (size_t)(b * a.heads_q + h * G + g) * kHeadDim;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int c = 16 * ks + 2 * t + 8 * r;
          const uint32_t w = *reinterpret_cast<const uint32_t*>(qp + c);
          qb[ks][r] = w;
          const float q0 = __uint_as_float(w << 16), q1 = __uint_as_float(w & 0xffff0000u);
          const float b0 = a.balancer ? a.balancer[h * kHeadDim + c] : 1.f;
          const float b1 = a.balancer ? a.balancer[h * kHeadDim + c + 1] : 1.f;
          qh[ks][r] = pack_f16(__fdiv_rn(q0, b0), __fdiv_rn(q1, b1));  // Eq. 4
        }
    } else {
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) qb[ks][0] = qb[ks][1] = qh[ks][0] = qh[ks][1] = 0u;
    }
    float* logit_base =
        a.hi_logits ? a.hi_logits + (size_t)(b * a.heads_q + h * G) * a.hi_stride : nullptr;

    Softmax st;
    st.m[0] = st.m[1] = -INFINITY;
    st.l[0] = st.l[1] = 0.f;
    float o[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

    for (int k = 0; k < n_hs + n_ls; ++k, ++it) {
      if (*abort_v) continue;
      const int s = it % kStages;
      const uint32_t use = it / kStages;
      if (!mbar_wait(smem_u32(&bars[s]), use & 1)) {
        record_error(a.status, kErrFullTimeout);
        *abort_v = 1;
        continue;
      }
      bool hi;
      int jj;
      stage_kind(k, n_hs, n_ls, hi, jj);
      const uint32_t dst = base + s * kStageBytes;
      if (hi) {
        const int hb = hb0 + jj * kConsumerWarps + warp;
        if (hb < hb1)
          process_hi<G>(dst + warp * kHiBlockBytes, min(16, a.hi_cap - 16 * hb), 16 * hb, qb, a.sm_scale,
                        logit_base, a.hi_stride, st, o, lane);
      } else {
        const int first = lb0 + jj * kConsumerWarps * L::kBlocksPerWarp + warp * L::kBlocksPerWarp;
        for (int i = 0; i < L::kBlocksPerWarp; ++i) {
          const int lb = first + i;
          if (lb >= lb1) break;
          process_lo<BITS, GROUP, G>(dst + (warp * L::kBlocksPerWarp + i) * L::kBlockBytes,
                                     min(16, a.n_lo - 16 * lb), qh, a.sm_scale, st, o, lane);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars[kStages + s]));
    }

    // ---- combine the 4 warps' partials and write this item's (max, sum, output)
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], off);
      st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], off);
    }
    float* rw = red + warp * G * 130;
#pragma unroll
    for (int hd = 0; hd < 2; ++hd) {
      const int head = 2 * t + hd;
      if (head < G) {
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          rw[head * 130 + 16 * mt + g] = o[mt][hd];
          rw[head * 130 + 16 * mt + 8 + g] = o[mt][2 + hd];
        }
        if (g == 0) {
          rw[head * 130 + 128] = st.m[hd];
          rw[head * 130 + 129] = st.l[hd];
        }
      }
    }
    named_bar_sync(1, kConsumerWarps * 32);
    for (int idx = warp * 32 + lane; idx < G * kHeadDim; idx += kConsumerWarps * 32) {
      const int head = idx / kHeadDim, ch = idx - head * kHeadDim;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) M = fmaxf(M, red[(w * G + head) * 130 + 128]);
      float O = 0.f, Ls = 0.f;
      if (M != -INFINITY) {
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) {
          const float mw = red[(w * G + head) * 130 + 128];
          const float wt = mw == -INFINITY ? 0.f : fast_exp2((mw - M) * kLog2e);
          O += wt * red[(w * G + head) * 130 + ch];
          Ls += wt * red[(w * G + head) * 130 + 129];
        }
      }
      a.part_o[((size_t)item * G + head) * kHeadDim + ch] = O;
      if (ch == 0) {
        a.part_ml[((size_t)item * G + head) * 2] = M;
        a.part_ml[((size_t)item * G + head) * 2 + 1] = Ls;
      }
    }
    named_bar_sync(1, kConsumerWarps * 32);
  }
}

template <int OUT_F32>
__global__ void __launch_bounds__(128) merge_kernel(const MergeArgs a, int G) {
  const int bq = blockIdx.x;
  const int b = bq / a.heads_q, hq = bq - b * a.heads_q;
  const int h = hq / G, jh = hq - h * G;
  const int c = threadIdx.x;
  const size_t item0 = (size_t)(b * a.heads_kv + h) * a.n_split;
  float M = -INFINITY;
  for (int s = 0; s < a.n_split; ++s) M = fmaxf(M, a.part_ml[((item0 + s) * G + jh) * 2]);
  float O = 0.f, Ls = 0.f;
  for (int s = 0; s < a.n_split; ++s) {
    const float ms = a.part_ml[((item0 + s) * G + jh) * 2];
    if (ms == -INFINITY) continue;
    const float wt = fast_exp2((ms - M) * kLog2e);
    Ls += wt * a.part_ml[((item0 + s) * G + jh) * 2 + 1];
    O += wt * a.part_o[((item0 + s) * G + jh) * kHeadDim + c];
  }
  const float r = O / Ls;
  if (OUT_F32)
    static_cast<float*>(a.out)[(size_t)bq * kHeadDim + c] = r;
  else
    static_cast<__nv_bfloat16*>(a.out)[(size_t)bq * kHeadDim + c] = __float2bfloat16_rn(r);
  if (c == 0 && a.ml) {
    a.ml[2 * bq] = M;
    a.ml[2 * bq + 1] = Ls;
  }
}

template <int BITS, int GROUP, int G>
cudaError_t launch_split(const AttnArgs& a, int grid, cudaStream_t st) {
  auto kern = attention_split_kernel<BITS, GROUP, G>;
  static bool configured = false;
  const int smem = smem_bytes(G);
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  kern<<<grid, kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

template <int BITS, int GROUP>
cudaError_t dispatch_g(const AttnArgs& a, int G, int grid, cudaStream_t st) {
  switch (G) {
    case 1: return launch_split<BITS, GROUP, 1>(a, grid, st);
    case 2: return launch_split<BITS, GROUP, 2>(a, grid, st);
    case 4: return launch_split<BITS, GROUP, 4>(a, grid, st);
    case 8: return launch_split<BITS, GROUP, 8>(a, grid, st);
  }
  return cudaErrorInvalidValue;
}

template <int BITS>
cudaError_t dispatch_group(const AttnArgs& a, int group, int G, int grid, cudaStream_t st) {
  switch (group) {
    case 32: return dispatch_g<BITS, 32>(a, G, grid, st);
    case 64: return dispatch_g<BITS, 64>(a, G, grid, st);
    case 128: return dispatch_g<BITS, 128>(a, G, grid, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

AttnPlan plan_attention(const mikv_shape& s, int n_lo, int num_sms) {
  AttnPlan p;
  const int hb = (s.hi_cap + 15) / 16, lb = (n_lo + 15) / 16;
  const int bh = s.batch * s.heads_kv;
  const int grid_cap = num_sms * kCtasPerSm;
  const int want = (kItemsPerCta * grid_cap + bh - 1) / bh;
  const int cap = (hb + lb + kMinBlocksPerSplit - 1) / kMinBlocksPerSplit;
  p.n_split = want < cap ? want : cap;
  if (p.n_split < 1) p.n_split = 1;
  p.n_items = bh * p.n_split;
  p.grid = p.n_items < grid_cap ? p.n_items : grid_cap;
  return p;
}

size_t attention_workspace_bytes(const mikv_shape& s, int n_lo_max, int num_sms) {
  const AttnPlan p = plan_attention(s, n_lo_max, num_sms);
  const int G = s.heads_q / s.heads_kv;
  const size_t part = (size_t)p.n_items * G * (kHeadDim + 2) * sizeof(float);
  return kWsHeader + (part + 255) / 256 * 256;
}

cudaError_t launch_attention(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st) {
  switch (bits) {
    case 2: return dispatch_group<2>(a, group, G, grid, st);
    case 3: return dispatch_group<3>(a, group, G, grid, st);
    case 4: return dispatch_group<4>(a, group, G, grid, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_merge(const MergeArgs& a, int G, int out_f32, cudaStream_t st) {
  const int grid = a.batch * a.heads_q;
  if (out_f32)
    merge_kernel<1><<<grid, kHeadDim, 0, st>>>(a, G);
  else
    merge_kernel<0><<<grid, kHeadDim, 0, st>>>(a, G);
  return cudaGetLastError();
}

}  // namespace mikv
