// mikv_internal.h — launch interfaces between the C-ABI layer (mikv_abi.cu) and the kernel
// translation units. Host-side only; not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/mikv.h"

namespace mikv {

// Attention split plan: per (b, kv-head) the important blocks [0, hi_blocks) and retained blocks
// [0, lo_blocks) of 16 tokens are divided into n_split contiguous ranges.
struct AttnPlan {
  int n_split;
  int n_items;  // B * Hkv * n_split
  int grid;     // persistent CTAs
};

struct AttnArgs {
  CUtensorMap map_k_hi, map_v_hi;    // bf16 rows of 128 channels, box 64 x 16, 128B swizzle
  CUtensorMap map_k_lo, map_v_lo;    // packed codes (bits 0..1 plane for N = 3), box row x 16
  CUtensorMap map_k_lo1, map_v_lo1;  // N = 3 only: 1-bit plane, box 16 B x 16
  const void* k_params;
  const void* v_params;
  const void* q;
  const float* balancer;
  float* hi_logits;
  float* part_o;   // [n_items][G][128]
  float* part_ml;  // [n_items][G][2]
  int* status;
  int batch, heads_q, heads_kv, hi_cap, hi_stride, lo_cap, n_lo;
  int hi_blocks, lo_blocks, n_split, n_items;
  float sm_scale;
};

struct MergeArgs {
  const float* part_o;
  const float* part_ml;
  void* out;
  float* ml;
  int batch, heads_q, heads_kv, n_split;
};

AttnPlan plan_attention(const mikv_shape& s, int n_lo, int num_sms);
size_t attention_workspace_bytes(const mikv_shape& s, int n_lo_max, int num_sms);
cudaError_t launch_attention(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
cudaError_t launch_merge(const MergeArgs& a, int G, int out_f32, cudaStream_t st);

cudaError_t launch_quantize_pack(const mikv_shape& s, const mikv_cache& c, const void* k_src,
                                 const void* v_src, const int32_t* src_tok, int n_src,
                                 const int32_t* rows, int n_rows, int lo_start, cudaStream_t st);

cudaError_t launch_balancer(const mikv_shape& s, const void* q_pre, const void* k_pre, int T,
                            float* out, uint32_t* ws_max, cudaStream_t st);

cudaError_t launch_update_importance(const mikv_shape& s, const mikv_cache& c, const float* hi_logits,
                                     const float* ml, cudaStream_t st);

cudaError_t launch_select(int batch, int heads, const float* scores, const int32_t* ids, int n,
                          int stride, int n_demote, int32_t* demoted, int32_t* kept, cudaStream_t st);

cudaError_t launch_insert(const mikv_shape& s, const mikv_cache& c, const void* k_new, const void* v_new,
                          int tok, const int32_t* slots, cudaStream_t st);

cudaError_t launch_gather(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                          const int32_t* src_tok, const float* src_scores, int n_src,
                          const int32_t* rows, int n_rows, cudaStream_t st);

}  // namespace mikv
