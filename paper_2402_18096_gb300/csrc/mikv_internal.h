// mikv_internal.h — launch interfaces between the C-ABI layer (mikv_abi.cu) and the kernel
// translation units. Host-side only; not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/mikv.h"

namespace mikv {

// The library's status word for index checks of the entry points without a workspace (debug builds, -DMIKV_DEBUG;
// nullptr in release builds). Defined in mikv_abi.cu; read by mikv_debug_check.
int* debug_status_word();

// Shared-memory layout of one retained unit: up to `blocks` consecutive 16-token blocks loaded with
// one TMA box per array (codes of K, codes of V, parameters of K, parameters of V; N = 3 adds the
// 1-bit planes). Offsets are in bytes from the unit's stage; each section starts on the alignment its
// swizzle needs (256 B for 32-byte swizzle, 512 B for 64-byte swizzle, 128 B otherwise).
struct LoUnit {
  int blocks;
  int pitch;      // bytes of codes per token (both planes for N = 3), in HBM and in the stage
  int plane_b;    // N = 3: offset of the 1-bit plane inside a token's codes
  int map_w;      // the code arrays are copied as rows of map_w bytes (several tokens per row)
  int param_row;  // bytes of (alpha, beta) pairs per token
  int param_w;    // the parameter arrays are copied as rows of param_w bytes
  int k_a, v_a, k_p, v_p;  // section offsets in the stage
  int total;               // bytes used
  int tx;                  // bytes the TMA boxes deliver
};

constexpr int kUnitBytes = 8192;
constexpr int kHeadDimH = 128;  // head dimension (host-side copy)

__host__ __device__ constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

// A unit's rows of one array are contiguous in HBM (16 n tokens of one head), so TMA copies them as
// wide rows: 64-byte rows with the 64B swizzle for N = 2 (two tokens per row) and N = 4 (one token),
// unswizzled 128-byte rows for N = 3 (48-byte tokens, whose pitch alone spreads ldmatrix rows over all
// banks), 128-byte rows with the 128B swizzle for N = 8 (coded important sets only). Few wide rows per
// unit keep the TMA request rate far below what HBM needs.
__host__ __device__ constexpr LoUnit lo_unit_layout_n(int bits, int group, int n) {
  LoUnit u{};
  u.blocks = n;
  u.pitch = bits == 3 ? 48 : 16 * bits;
  u.plane_b = bits == 3 ? 32 : 0;
  u.map_w = bits == 3 || bits == 8 ? 128 : 64;
  u.param_row = 4 * (128 / group);
  u.param_w = u.param_row == 4 ? 64 : 128;
  const int rows = 16 * n;
  // the 64B / 128B swizzle patterns repeat every 512 / 1024 bytes
  const int code_align = bits == 3 ? 128 : (bits == 8 ? 1024 : 512);
  u.k_a = 0;
  u.v_a = align_up(u.k_a + rows * u.pitch, code_align);
  u.k_p = align_up(u.v_a + rows * u.pitch, 128);
  u.v_p = align_up(u.k_p + rows * u.param_row, 128);
  u.total = u.v_p + rows * u.param_row;
  u.tx = 2 * rows * u.pitch + 2 * rows * u.param_row;
  return u;
}

// Per-channel retained keys (App. C): tokens are grouped by 64; a retained unit is one group (N = 2, 3) or
// half of one (N = 4: two blocks), carrying the group's 128 (alpha, beta) key pairs (512 bytes) in place of
// per-token key parameters; values keep their per-token layout.
constexpr int kKchGroup = 64;

__host__ __device__ constexpr LoUnit lo_unit_layout_kch(int bits, int group) {
  LoUnit u = lo_unit_layout_n(bits, group, bits == 4 ? 2 : 4);
  const int rows = 16 * u.blocks;
  const int code_align = bits == 3 ? 128 : 512;
  u.k_a = 0;
  u.v_a = align_up(rows * u.pitch, code_align);
  u.k_p = align_up(u.v_a + rows * u.pitch, 128);
  u.v_p = align_up(u.k_p + 4 * kHeadDimH, 128);
  u.total = u.v_p + rows * u.param_row;
  u.tx = 2 * rows * u.pitch + 4 * kHeadDimH + rows * u.param_row;
  return u;
}

// The largest unit (at most 8 blocks) that fits one stage.
__host__ __device__ constexpr LoUnit lo_unit_layout(int bits, int group) {
  int n = 8;
  while (n > 1 && lo_unit_layout_n(bits, group, n).total > kUnitBytes) --n;
  return lo_unit_layout_n(bits, group, n);
}

// Group size of a coded important set (Sec. 3.3, Table 3).
constexpr int kHiGroup = 64;

// Attention work plan: per (b, kv-head) a sequence of n_u units (hi_units important units: one bf16
// block of 16 tokens, or lo_unit_layout(hi_bits, 64).blocks coded blocks; lo_units groups of retained
// blocks), all heads concatenated into n_units units and split into n_warps equal contiguous shares;
// warp w writes the partial of head bh into slot w + bh.
struct AttnPlan {
  int hi_blocks, hi_units, lo_blocks, lo_units, n_u;
  int n_units;
  int n_warps;
  int grid;
  int n_slots;
};

struct AttnArgs {
  CUtensorMap map_k_hi, map_v_hi;    // bf16 rows of 128 channels, box 64 x 16, 128B swizzle; or coded
                                     // important rows viewed like retained codes (layout hi_bits, 64)
  CUtensorMap map_k_hp, map_v_hp;    // coded important set: (alpha, beta) rows like map_k_par
  CUtensorMap map_k_lo, map_v_lo;    // packed codes viewed as rows of LoUnit::map_w bytes, box = one unit
  CUtensorMap map_k_par, map_v_par;  // (alpha, beta) pairs viewed as rows of LoUnit::param_w bytes
  const void* q;
  const float* balancer;
  float* hi_logits;
  float* part_o;   // [n_slots][G][128]
  float* part_ml;  // [n_slots][G][2]
  int* status;
  int batch, heads_q, heads_kv, hi_cap, hi_stride, lo_cap, n_lo;
  int hi_blocks, hi_units, lo_blocks, n_u, n_units, n_warps;
  float sm_scale;
  // insertion of a decode step's new token, fused into the attention of a bf16 important set: the unit
  // holding slot ins_slots[b, h] takes the new rows in shared memory, and its warp writes them (and the
  // token id, a zero score) into the cache. ins_slots == nullptr: no insertion.
  const int32_t* ins_slots;
  const __nv_bfloat16* ins_k;  // [B][Hkv][128]
  const __nv_bfloat16* ins_v;
  __nv_bfloat16* ins_k_hi;
  __nv_bfloat16* ins_v_hi;
  int32_t* ins_hi_tok;
  float* ins_acc;
  int ins_tok;
};

struct MergeArgs {
  const float* part_o;
  const float* part_ml;
  void* out;
  float* ml;
  int batch, heads_q, heads_kv;
  int n_u, n_units, n_warps;
};

// Fused tail of a decode step (mikv_step.cu): merge + importance update + argmin + demotion.
struct StepPostArgs {
  const float* part_o;
  const float* part_ml;
  void* out;
  const float* hi_logits;
  float* acc;
  int32_t* hi_tok;  // written only for per-channel keys (staging)
  void* k_hi;
  void* v_hi;
  const float* balancer;
  void* k_codes;
  void* v_codes;
  void* k_params;
  void* v_params;
  int32_t* lo_tok;
  int32_t* slots;
  const void* k_hi_params;  // coded important set: (alpha, beta) of the important rows
  const void* v_hi_params;
  int hi_bits;              // 16 = bf16 important rows; 8, 4, 2 = coded (groups of kHiGroup)
  int evict;                // no retained set: the victim's slot is freed, nothing is demoted
  int kch;                  // per-channel retained keys: the victim is staged at important row hi_cap + n_lo % 64
  int* status;              // the workspace status word (index checks of debug builds)
  int batch, heads_q, heads_kv, hi_cap, hi_stride, lo_cap, n_lo;
  int n_u, n_units, n_warps;
};

cudaError_t launch_step_post(const StepPostArgs& a, int bits, int group, int G, int out_f32, cudaStream_t st);

AttnPlan plan_attention(const mikv_shape& s, int n_lo, int num_sms);
size_t attention_workspace_bytes(const mikv_shape& s, int n_lo_max, int num_sms);
cudaError_t launch_attention(const AttnArgs& a, int bits, int group, int hi_bits, int G, int grid, cudaStream_t st,
                             bool kch = false);
// per-channel retained keys, bf16 important set (mikv_attn_kch.cu)
cudaError_t launch_attention_kch(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
// one translation unit per important-set precision (mikv_attn_h*.cu)
cudaError_t launch_attention_h16(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
cudaError_t launch_attention_h8(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
cudaError_t launch_attention_h4(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
cudaError_t launch_attention_h2(const AttnArgs& a, int bits, int group, int G, int grid, cudaStream_t st);
// effective important-set precision of a shape: 16 for bf16 (hi_bits 0 or 16)
inline int hi_bits_of(const mikv_shape& s) { return s.hi_bits == 0 ? 16 : s.hi_bits; }
// bits == 0: no retained set, demoted tokens are evicted (the H2O baseline). The kernels then run with
// any retained layout (none of its units exist); these give the one they are instantiated with.
inline bool evicting(const mikv_shape& s) { return s.bits == 0; }
// per-channel retained keys (App. C), groups of kKchGroup tokens
inline bool kch_of(const mikv_shape& s) { return s.k_channel_group == kKchGroup; }
inline int lo_bits_of(const mikv_shape& s) { return s.bits == 0 ? 2 : s.bits; }
inline int lo_group_of(const mikv_shape& s) { return s.bits == 0 ? 32 : s.group; }
cudaError_t launch_merge(const MergeArgs& a, int G, int out_f32, cudaStream_t st);

cudaError_t launch_quantize_pack(const mikv_shape& s, const mikv_cache& c, const void* k_src,
                                 const void* v_src, const int32_t* src_tok, int n_src,
                                 const int32_t* rows, int n_rows, int lo_start, cudaStream_t st);

// Per-channel retained keys (App. C): append rows at retained positions p0 .. p0 + n_rows - 1 (quantizing
// every group of 64 that completes, staging the rest in important rows hi_cap ..); with n_rows == 0 and
// p0 = 64 (j + 1), quantize group j from its staged rows.
cudaError_t launch_kch_append(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                              const int32_t* src_tok, int n_src, const int32_t* rows, int n_rows, int p0,
                              cudaStream_t st);

// insert (rows == nullptr, slots/tok used) or gather (rows/n_rows) into a coded important set
cudaError_t launch_hi_quant(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                            const int32_t* src_tok, const float* src_scores, int n_src, const int32_t* rows,
                            int n_rows, const int32_t* slots, int tok, cudaStream_t st);

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

// Launch of a kernel on the decode-step path with programmatic dependent launch allowed: the kernel may be
// scheduled while the previous kernel of the stream finishes (hiding the launch gap), and executes
// grid_dependency_wait() before its first access to memory that other kernels write or read.
template <typename... P, typename... A>
cudaError_t launch_chained(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, A&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<A&&>(args)...);
}

}  // namespace mikv
