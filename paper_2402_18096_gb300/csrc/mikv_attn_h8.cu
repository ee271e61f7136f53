// mikv_attn_h8.cu — decode-attention kernels for an important set stored in INT8 (groups of 64), every
// (retained bits, group, query-head group) combination; one translation unit per important-set
// precision so the kernel variants compile in parallel.
#include "mikv_attention.cuh"

namespace mikv {

cudaError_t launch_attention_h8(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st) {
  return launch_attention_hb<8>(a, bits, group, G, grid, st);
}

}  // namespace mikv
