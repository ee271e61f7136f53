// mikv_attn_kch.cu — decode-attention kernels with per-channel retained keys (App. C: one (alpha, beta) per
// channel and group of 64 tokens, staged tokens attended in bf16 with the important set) and a bf16
// important set, every (retained bits, value group, query-head group) combination.
#include "mikv_attention.cuh"

namespace mikv {

cudaError_t launch_attention_kch(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st) {
  return launch_attention_hb<16, true>(a, bits, group, G, grid, st);
}

}  // namespace mikv
