// mikv_attention.cu — decode attention over the mixed-precision KV cache: the work plan, the merge of
// the split partials, and the dispatch to the kernels of mikv_attention.cuh (instantiated per
// important-set precision in mikv_attn_h16.cu, mikv_attn_h8.cu, mikv_attn_h4.cu, mikv_attn_h2.cu).
#include "mikv_attention.cuh"

namespace mikv {
namespace {

// Combination of the split partials: one warp per query head (4 heads per block), 4 channels per lane.
template <int OUT_F32>
__global__ void __launch_bounds__(128) merge_kernel(const MergeArgs a, int G) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bq = blockIdx.x * 4 + warp;
  grid_dependency_wait();
  allow_dependent_launch();
  if (bq >= a.batch * a.heads_q) return;
  const int b = bq / a.heads_q, hq = bq - b * a.heads_q;
  const int h = hq / G, jh = hq - h * G;
  const int bh = b * a.heads_kv + h;
  const int w0 = owner_warp((long long)bh * a.n_u, a.n_units, a.n_warps);
  const int w1 = owner_warp((long long)(bh + 1) * a.n_u - 1, a.n_units, a.n_warps);
  float r[4], M, L;
  merge_head_warp<12>(a.part_o, a.part_ml, G, bh, jh, w0, w1, lane, M, L, r);
  if (OUT_F32) {
    reinterpret_cast<float4*>(static_cast<float*>(a.out) + (size_t)bq * kHeadDim)[lane] = make_float4(r[0], r[1], r[2], r[3]);
  } else {
    __nv_bfloat162 v0 = __floats2bfloat162_rn(r[0], r[1]), v1 = __floats2bfloat162_rn(r[2], r[3]);
    uint2 u;
    u.x = *reinterpret_cast<uint32_t*>(&v0);
    u.y = *reinterpret_cast<uint32_t*>(&v1);
    reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.out) + (size_t)bq * kHeadDim)[lane] = u;
  }
  if (lane == 0 && a.ml) {
    a.ml[2 * bq] = M;
    a.ml[2 * bq + 1] = L;
  }
}

}  // namespace

AttnPlan plan_attention(const mikv_shape& s, int n_lo, int num_sms) {
  AttnPlan p;
  p.hi_blocks = (s.hi_cap + 15) / 16;
  const int hb = hi_bits_of(s);
  const int kh = hb == 16 ? 1 : lo_unit_layout(hb, kHiGroup).blocks;
  p.hi_units = (p.hi_blocks + kh - 1) / kh;
  p.lo_blocks = (n_lo + 15) / 16;
  const int k = evicting(s) ? 1 : kch_of(s) ? lo_unit_layout_kch(s.bits, s.group).blocks
                                          : lo_unit_layout(s.bits, s.group).blocks;
  p.lo_units = (p.lo_blocks + k - 1) / k;
  p.n_u = p.hi_units + p.lo_units;
  const long long bh = (long long)s.batch * s.heads_kv;
  p.n_units = bh * p.n_u;
  const long long cap = (long long)num_sms * kCtasPerSm * kWarps;
  long long w = (p.n_units + kUnitsPerWarp - 1) / kUnitsPerWarp;
  if (w < cap) w = p.n_units < cap ? p.n_units : cap;  // spread small caches over the whole GPU
  if (w > cap) w = cap;
  if (w < 1) w = 1;
  p.n_warps = (int)w;
  p.grid = (p.n_warps + kWarps - 1) / kWarps;
  p.n_slots = p.n_warps + (int)bh;
  return p;
}

size_t attention_workspace_bytes(const mikv_shape& s, int n_lo_max, int num_sms) {
  // the slot count grows with n_lo only through n_warps, which is capped: size for the cap
  const AttnPlan p = plan_attention(s, n_lo_max, num_sms);
  const long long cap = (long long)num_sms * kCtasPerSm * kWarps;
  const long long slots = cap + (long long)s.batch * s.heads_kv;
  const int G = s.heads_q / s.heads_kv;
  const size_t part = (size_t)(slots > p.n_slots ? slots : p.n_slots) * G * (kHeadDim + 2) * sizeof(float);
  return kWsHeader + (part + 255) / 256 * 256;
}

cudaError_t launch_attention(const AttnArgs& a, int bits, int group, int hi_bits, int G, int grid, cudaStream_t st,
                             bool kch) {
  if (kch) return hi_bits == 16 ? launch_attention_kch(a, bits, group, G, grid, st) : cudaErrorInvalidValue;
  switch (hi_bits) {
    case 16: return launch_attention_h16(a, bits, group, G, grid, st);
    case 8: return launch_attention_h8(a, bits, group, G, grid, st);
    case 4: return launch_attention_h4(a, bits, group, G, grid, st);
    case 2: return launch_attention_h2(a, bits, group, G, grid, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_merge(const MergeArgs& a, int G, int out_f32, cudaStream_t st) {
  const int grid = (a.batch * a.heads_q + 3) / 4;
  return launch_chained(out_f32 ? merge_kernel<1> : merge_kernel<0>, dim3(grid), dim3(128), 0, st, a, G);
}

}  // namespace mikv
