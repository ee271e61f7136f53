// mikv_attn_h2.cu — decode-attention kernels for an important set stored in INT2 (groups of 64), every
// (retained bits, group, query-head group) combination; one translation unit per important-set
// precision so the kernel variants compile in parallel.
#include "mikv_attention.cuh"

namespace mikv {

cudaError_t launch_attention_h2(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st) {
  return launch_attention_hb<2>(a, bits, group, G, grid, st);
}

}  // namespace mikv
