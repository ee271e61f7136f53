// mikv_step.cu — the tail of one decode step, fused into one kernel per (batch b, KV head h):
// combine the attention partials of the G query heads (output and softmax statistics), add this
// step's attention weights to the accumulated importance of every important slot (heavy-hitter
// policy, Fig. 4 / Sec. 3 of arxiv 2402.18096), pick the least important slot by (score, token id),
// and quantize/pack its key and value rows into the next retained row (Eq. 1, Eq. 3).
//
// Each part performs the same arithmetic, in the same order, as the standalone kernels behind
// mikv_decode_attention's merge, mikv_update_importance, mikv_select_demote and mikv_quantize_pack,
// so a step through mikv_decode_step gives the same bits as the four separate calls.
#include <math.h>

#include "mikv_device.cuh"
#include "mikv_internal.h"
#include "mikv_quant_rows.cuh"
#include "mikv_rows.cuh"

namespace mikv {
namespace {

constexpr int kPostThreads = 256;

// Four consecutive important slots of one (b, KV head): the G query heads' logits, the score and the
// token id (hi_stride % 16 == 0 keeps every group 16-byte aligned).
template <int G>
struct SlotQuad {
  float4 lg[G];
  float4 ac;
  int4 tk;
};

template <int G>
__device__ __forceinline__ void load_logits(const float* logit, int hi_stride, int v, SlotQuad<G>& q) {
#pragma unroll
  for (int j = 0; j < G; ++j) q.lg[j] = reinterpret_cast<const float4*>(logit + (size_t)j * hi_stride)[v];
}

// Scores and ids through L2 only: also read before the grid-dependency wait (see step_post_kernel).
template <int G>
__device__ __forceinline__ void load_scores(const float* acc, const int32_t* tok, int v, SlotQuad<G>& q) {
  q.ac = __ldcg(reinterpret_cast<const float4*>(acc) + v);
  q.tk = __ldcg(reinterpret_cast<const int4*>(tok) + v);
}

template <int G>
__device__ __forceinline__ void load_quad(const float* logit, const float* acc, const int32_t* tok, int hi_stride,
                                          int v, SlotQuad<G>& q) {
  load_logits<G>(logit, hi_stride, v, q);
  load_scores<G>(acc, tok, v, q);
}

// Importance update of the slots of q below hi_cap (the arithmetic of update_importance_kernel: the
// weights exp(s - m) / l of the G heads summed in head order, then added to the score), the updated
// scores stored, and the running minimum of (score, id) advanced.
template <int G>
__device__ __forceinline__ void update_quad(float* acc, int hi_cap, int v, SlotQuad<G>& q, const float* s_m,
                                            const float* s_il, unsigned long long& best, int& best_slot) {
  float* ac = &q.ac.x;
  const int32_t* tk = &q.tk.x;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int i = 4 * v + e;
    if (i >= hi_cap) break;
    float add = 0.f;
#pragma unroll
    for (int j = 0; j < G; ++j) add += importance_weight((&q.lg[j].x)[e], s_m[j], s_il[j]);
    ac[e] = ac[e] + add;
    const unsigned long long k = order_key(ac[e], tk[e]);
    if (k < best) {
      best = k;
      best_slot = i;
    }
  }
  reinterpret_cast<float4*>(acc)[v] = q.ac;  // padding slots (>= hi_cap) are written back unchanged
}

static_assert(kPostThreads == 256, "eight warps: one per query head for the merge, one argmin entry per warp");

template <int BITS, int GROUP, int G, int OUT_F32>
__global__ void __launch_bounds__(kPostThreads, 2) step_post_kernel(const StepPostArgs a) {
  __shared__ float s_m[8], s_l[8], s_il[8];
  __shared__ unsigned long long s_best[kPostThreads / 32];
  __shared__ int s_slot[kPostThreads / 32];
  __shared__ int s_victim;
  const int bh = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = bh / a.heads_kv, h = bh - b * a.heads_kv;
  float* acc = a.acc + (size_t)bh * a.hi_stride;
  const int32_t* tok = a.hi_tok + (size_t)bh * a.hi_stride;
  const float* logit = a.hi_logits + (size_t)(b * a.heads_q + h * G) * a.hi_stride;
  const int nv = (a.hi_cap + 3) / 4;  // groups of four slots

  // 0. Scores and ids are read before the grid-dependency wait. This kernel starts only once every block of
  // the attention kernel has passed its own wait, so every kernel before the attention kernel has completed;
  // the attention kernel itself writes one of them: the slot it inserts the new token into (slots[bh], set by
  // the previous step's tail), whose group is read again after the wait. The first groups of this thread go
  // to registers, every line of the rest into L2.
  constexpr int kPre = G <= 4 ? 2 : 1;
  SlotQuad<G> q0, qp;
  const int ins = a.slots[bh];
  if (tid < nv) load_scores<G>(acc, tok, tid, q0);
  if (kPre == 2 && tid + kPostThreads < nv) load_scores<G>(acc, tok, tid + kPostThreads, qp);
  for (int l = kPre * kPostThreads / 8 + tid; l < (nv + 7) / 8; l += kPostThreads) {  // 8 groups per line
    prefetch_l2(acc + 32 * l);
    prefetch_l2(tok + 32 * l);
  }
  grid_dependency_wait();  // logits, partials and the inserted slot come from the attention kernel
  allow_dependent_launch();
  // the first groups' logits are loaded before the statistics, which they do not depend on (two groups each
  // where registers allow: those loads overlap the statistics' loads below)
  if (tid < nv) {
    load_logits<G>(logit, a.hi_stride, tid, q0);
    if (ins >> 2 == tid) load_scores<G>(acc, tok, tid, q0);
  }
  if (kPre == 2 && tid + kPostThreads < nv) {
    load_logits<G>(logit, a.hi_stride, tid + kPostThreads, qp);
    if (ins >> 2 == tid + kPostThreads) load_scores<G>(acc, tok, tid + kPostThreads, qp);
  }

  // 1. softmax statistics (M, L) of query heads h*G .. h*G+G-1 from the split partials (one warp per head)
  const int w0 = owner_warp((long long)bh * a.n_u, a.n_units, a.n_warps);
  const int w1 = owner_warp((long long)(bh + 1) * a.n_u - 1, a.n_units, a.n_warps);
  if (warp < G) {
    float M, L;
    merge_stats_warp(a.part_ml, G, bh, warp, w0, w1, lane, M, L);
    if (lane == 0) {
      s_m[warp] = M;
      s_l[warp] = L;
      s_il[warp] = 1.f / L;
    }
  }
  __syncthreads();

  // 2. importance update and the least important slot (keys are unique: ids are distinct)
  unsigned long long best = ~0ull;
  int best_slot = -1;
  if (tid < nv) update_quad<G>(acc, a.hi_cap, tid, q0, s_m, s_il, best, best_slot);
  if (kPre == 2 && tid + kPostThreads < nv) update_quad<G>(acc, a.hi_cap, tid + kPostThreads, qp, s_m, s_il, best, best_slot);
  constexpr int kInFlight = G <= 4 ? 2 : 1;  // groups loaded before any of them is used
  for (int v = tid + kPre * kPostThreads; v < nv; v += kInFlight * kPostThreads) {
    SlotQuad<G> q1, q2;
    const bool two = kInFlight == 2 && v + kPostThreads < nv;
    load_quad<G>(logit, acc, tok, a.hi_stride, v, q1);
    if (two) load_quad<G>(logit, acc, tok, a.hi_stride, v + kPostThreads, q2);
    update_quad<G>(acc, a.hi_cap, v, q1, s_m, s_il, best, best_slot);
    if (two) update_quad<G>(acc, a.hi_cap, v + kPostThreads, q2, s_m, s_il, best, best_slot);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
    const int os = __shfl_xor_sync(0xffffffffu, best_slot, off);
    if (o < best) {
      best = o;
      best_slot = os;
    }
  }
  if (lane == 0) {
    s_best[warp] = best;
    s_slot[warp] = best_slot;
  }
  __syncthreads();
  if (warp == 0) {  // minimum over the warps' minima (one per lane)
    best = lane < kPostThreads / 32 ? s_best[lane] : ~0ull;
    best_slot = lane < kPostThreads / 32 ? s_slot[lane] : -1;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
      const int os = __shfl_xor_sync(0xffffffffu, best_slot, off);
      if (o < best) {
        best = o;
        best_slot = os;
      }
    }
    if (lane == 0) s_victim = best_slot;
  }
  __syncthreads();

  // 3. the attention output of each query head (warps 2, 3, ... so that warps 0 and 1 demote meanwhile)
  const int jm = (warp + 6) & 7;
  if (jm < G) {
    float r[4];
    merge_output_warp(a.part_o, a.part_ml, G, bh, jm, w0, w1, lane, s_m[jm], s_l[jm], r);
    const size_t bq = (size_t)b * a.heads_q + h * G + jm;
    if (OUT_F32) {
      reinterpret_cast<float4*>(static_cast<float*>(a.out) + bq * kHeadDim)[lane] = make_float4(r[0], r[1], r[2], r[3]);
    } else {
      __nv_bfloat162 v0 = __floats2bfloat162_rn(r[0], r[1]), v1 = __floats2bfloat162_rn(r[2], r[3]);
      uint2 u;
      u.x = *reinterpret_cast<uint32_t*>(&v0);
      u.y = *reinterpret_cast<uint32_t*>(&v1);
      reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.out) + bq * kHeadDim)[lane] = u;
    }
  }
  const int victim = s_victim;
  if (victim < 0 || victim >= a.hi_cap) {  // unreachable for valid scores (hi_cap >= 1, no NaN)
    if (tid == 0) MIKV_BOUNDS_FAIL(a.status);
    return;
  }
  MIKV_DEBUG_ASSERT(a.evict || a.n_lo < a.lo_cap, a.status);
  MIKV_DEBUG_ASSERT(!a.kch || a.hi_cap + a.n_lo % kKchGroup < a.hi_stride, a.status);

  // 4. demote the victim: quantize its key (balanced, Eq. 3) and value rows into retained row n_lo; a
  // coded important row is re-quantized from its fp32 dequantized values (already balanced, Sec. 3.3)
  if (a.evict) {  // eviction (no retained set): the victim's slot only becomes the next insertion slot
    if (tid == 0) a.slots[bh] = victim;
  } else if (a.kch) {  // per-channel keys: the victim waits in bf16 in staging row hi_cap + n_lo % 64
    const size_t src = (size_t)bh * a.hi_stride + victim;
    const size_t dst = (size_t)bh * a.hi_stride + a.hi_cap + (a.n_lo % kKchGroup);
    __nv_bfloat16* k = static_cast<__nv_bfloat16*>(a.k_hi);
    __nv_bfloat16* v = static_cast<__nv_bfloat16*>(a.v_hi);
    if (tid < 32) {
      reinterpret_cast<uint2*>(k + dst * kHeadDim)[tid] = reinterpret_cast<const uint2*>(k + src * kHeadDim)[tid];
    } else if (tid < 64) {
      reinterpret_cast<uint2*>(v + dst * kHeadDim)[tid - 32] = reinterpret_cast<const uint2*>(v + src * kHeadDim)[tid - 32];
    } else if (tid == 64) {
      a.hi_tok[dst] = tok[victim];
      a.slots[bh] = victim;
    }
  } else if (warp < 2) {
    const bool is_v = warp == 1;
    const size_t pos = (size_t)bh * a.lo_cap + a.n_lo;
    const size_t hrow = (size_t)bh * a.hi_stride + victim;
    uint8_t* codes = static_cast<uint8_t*>(is_v ? a.v_codes : a.k_codes) + pos * (16 * BITS);
    __half2* params = static_cast<__half2*>(is_v ? a.v_params : a.k_params) + pos * (kHeadDim / GROUP);
    if (a.hi_bits == 16) {
      const __nv_bfloat16* src = static_cast<const __nv_bfloat16*>(is_v ? a.v_hi : a.k_hi) + hrow * kHeadDim;
      quantize_row_warp<BITS, GROUP>(src, is_v ? nullptr : (a.balancer ? a.balancer + h * kHeadDim : nullptr),
                                     codes, params, lane);
    } else {
      float x[4];
      dequantize_values_warp(static_cast<const uint8_t*>(is_v ? a.v_hi : a.k_hi) + hrow * (16 * a.hi_bits),
                             static_cast<const __half2*>(is_v ? a.v_hi_params : a.k_hi_params) +
                                 hrow * (kHeadDim / kHiGroup),
                             a.hi_bits, kHiGroup, lane, x);
      quantize_values_warp<BITS, GROUP>(x, codes, params, lane);
    }
    if (!is_v && lane == 0) {
      a.lo_tok[pos] = tok[victim];
      a.slots[bh] = victim;
    }
  }
}

template <int BITS, int GROUP, int G>
cudaError_t post_out(const StepPostArgs& a, int out_f32, cudaStream_t st) {
  const int grid = a.batch * a.heads_kv;
  return launch_chained(out_f32 ? step_post_kernel<BITS, GROUP, G, 1> : step_post_kernel<BITS, GROUP, G, 0>, dim3(grid),
                        dim3(kPostThreads), 0, st, a);
}

template <int BITS, int GROUP>
cudaError_t post_g(const StepPostArgs& a, int G, int out_f32, cudaStream_t st) {
  switch (G) {
    case 1: return post_out<BITS, GROUP, 1>(a, out_f32, st);
    case 2: return post_out<BITS, GROUP, 2>(a, out_f32, st);
    case 4: return post_out<BITS, GROUP, 4>(a, out_f32, st);
    case 8: return post_out<BITS, GROUP, 8>(a, out_f32, st);
  }
  return cudaErrorInvalidValue;
}

template <int BITS>
cudaError_t post_group(const StepPostArgs& a, int group, int G, int out_f32, cudaStream_t st) {
  switch (group) {
    case 32: return post_g<BITS, 32>(a, G, out_f32, st);
    case 64: return post_g<BITS, 64>(a, G, out_f32, st);
    case 128: return post_g<BITS, 128>(a, G, out_f32, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_step_post(const StepPostArgs& a, int bits, int group, int G, int out_f32, cudaStream_t st) {
  switch (bits) {
    case 2: return post_group<2>(a, group, G, out_f32, st);
    case 3: return post_group<3>(a, group, G, out_f32, st);
    case 4: return post_group<4>(a, group, G, out_f32, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace mikv
