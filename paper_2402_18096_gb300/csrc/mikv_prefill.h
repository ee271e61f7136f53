// mikv_prefill.h — arguments of the prefill-importance kernels (mikv_prefill.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "mikv_device.cuh"
#include "mikv_internal.h"

namespace mikv {

// Tiles of 128 tokens x 128 channels (bf16) stream through shared memory by TMA.
constexpr int kPfTile = 128;

struct PrefillArgs {
  CUtensorMap map_q;      // q_pre rows [B * Hq * T][128] bf16, box 64 channels x 128 rows, 128B swizzle
  CUtensorMap map_k;      // k_pre rows [B * Hkv * T][128] bf16, same boxes
  CUtensorMap map_q_str;  // the same arrays in boxes of 64 channels x 64 rows (streamed tiles)
  CUtensorMap map_k_str;
  float* stats;       // [B * Hq][T_pad]: log2 of each query's softmax normaliser, log2 sum_t 2^(s_it log2 e);
                      // +inf for the padding queries T .. T_pad - 1
  float* scores;      // [B * Hkv][T]
  int* status;        // workspace status word
  int heads_q, heads_kv, T, T_pad;  // T_pad = T rounded up to a whole tile
  float scale_log2;   // sm_scale * log2(e)
};

// Workspace of mikv_prefill_scores: the status header plus the per-query normalisers (rows padded to whole
// tiles).
inline int prefill_padded(int T) { return (T + kPfTile - 1) / kPfTile * kPfTile; }
inline size_t prefill_workspace_bytes(int batch, int heads_q, int T) {
  const size_t stats = (size_t)batch * heads_q * prefill_padded(T) * sizeof(float);
  return kWsHeader + (stats + 255) / 256 * 256;
}

cudaError_t launch_prefill(const PrefillArgs& a, int batch, cudaStream_t st);

}  // namespace mikv
