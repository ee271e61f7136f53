// mikv_abi.cu — host side of the libmikv C ABI (include/mikv.h): argument validation, tensor-map
// encoding for TMA, workspace layout and kernel dispatch. Nothing here allocates device memory or
// synchronises, except mikv_workspace_check and mikv_noalloc_check, which read a status word on request.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <mutex>

#ifndef MIKV_NVTX
#define MIKV_NVTX 1
#endif
#if MIKV_NVTX
#include <nvtx3/nvToolsExt.h>
#endif

#include "mikv_device.cuh"
#include "mikv_internal.h"
#include "mikv_prefill.h"

using namespace mikv;

namespace {
// One NVTX range per compute entry point, named after the call, around its validation and launches (host time:
// the kernels run later on the stream). Without a tool attached, push and pop return at once; -DMIKV_NVTX=0
// leaves them out.
struct CallRange {
#if MIKV_NVTX
  explicit CallRange(const char* name) { nvtxRangePushA(name); }
  ~CallRange() { nvtxRangePop(); }
#else
  explicit CallRange(const char*) {}
#endif
  CallRange(const CallRange&) = delete;
  CallRange& operator=(const CallRange&) = delete;
};
}  // namespace
#define MIKV_CALL_RANGE() const CallRange mikv_call_range_(__func__)

// The library's own status word for the index checks of debug builds (-DMIKV_DEBUG) in the entry points that take
// no workspace (insertion, gather, quantize/pack). Looked up in the current context on every use.
#ifdef MIKV_DEBUG
static __device__ int g_debug_status;
int* mikv::debug_status_word() {
  void* p = nullptr;
  return cudaGetSymbolAddress(&p, g_debug_status) == cudaSuccess ? static_cast<int*>(p) : nullptr;
}
#else
int* mikv::debug_status_word() { return nullptr; }
#endif

namespace {

mikv_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MIKV_OK : MIKV_ERR_CUDA; }

int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

bool shape_ok(const mikv_shape* s) {
  return s && s->batch > 0 && s->heads_q > 0 && s->heads_kv > 0 && s->heads_q % s->heads_kv == 0 &&
         s->head_dim > 0 && s->bits >= 0 && (s->bits == 0 || s->group > 0) && s->hi_cap >= 0 &&
         s->hi_stride >= s->hi_cap &&
         s->hi_stride % 16 == 0 && s->lo_cap >= 0 && s->lo_cap % 16 == 0;
}

mikv_status shape_supported(const mikv_shape* s) {
  if (!shape_ok(s)) return MIKV_ERR_ARG;
  const int G = s->heads_q / s->heads_kv;
  if (s->head_dim != kHeadDim) return MIKV_ERR_UNSUPPORTED;
  if (s->bits != 0) {  // bits == 0: eviction, no retained set (its group is ignored)
    if (s->bits < 2 || s->bits > 4) return MIKV_ERR_UNSUPPORTED;
    if (s->group != 32 && s->group != 64 && s->group != 128) return MIKV_ERR_UNSUPPORTED;
  }
  if (G != 1 && G != 2 && G != 4 && G != 8) return MIKV_ERR_UNSUPPORTED;
  const int hb = s->hi_bits;
  if (hb != 0 && hb != 16 && hb != 8 && hb != 4 && hb != 2) return MIKV_ERR_UNSUPPORTED;
  if (hb != 0 && hb != 16 && s->hi_group != kHiGroup) return MIKV_ERR_UNSUPPORTED;
  if (s->k_channel_group != 0) {  // per-channel retained keys (App. C)
    if (s->k_channel_group != kKchGroup || (hb != 0 && hb != 16) || s->bits == 0) return MIKV_ERR_UNSUPPORTED;
    if (s->hi_stride < s->hi_cap + kKchGroup || s->lo_cap % kKchGroup) return MIKV_ERR_ARG;
  }
  return MIKV_OK;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// The cache's arrays exist (and, for a coded important set, so do its parameter arrays, 16-byte aligned).
bool cache_ok(const mikv_cache* c, const mikv_shape* s) {
  if (!(c && c->k_hi && c->v_hi && c->hi_tok && c->acc)) return false;
  if (!evicting(*s) && !(c->k_codes && c->v_codes && c->k_params && c->v_params && c->lo_tok)) return false;
  if (hi_bits_of(*s) != 16)
    return c->k_hi_params && c->v_hi_params && aligned(c->k_hi_params, 16) && aligned(c->v_hi_params, 16);
  return true;
}

// ------------------------------------------------------------------ tensor maps

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

struct MapKey {
  const void* ptr;
  uint64_t inner, rows, stride;
  uint32_t bx, by;
  int dtype, swz;
  bool operator==(const MapKey& o) const { return memcmp(this, &o, sizeof(MapKey)) == 0; }
};

// Encoded maps are kept per (pointer, geometry): a layer's cache arrays are reused every step.
bool make_map(CUtensorMap* out, const void* ptr, CUtensorMapDataType dtype, uint64_t inner, uint64_t rows,
              uint64_t stride_bytes, uint32_t bx, uint32_t by, CUtensorMapSwizzle swz) {
  static std::mutex mu;
  static MapKey keys[64];
  static CUtensorMap maps[64];
  static int used = 0, next = 0;
  MapKey k;
  memset(&k, 0, sizeof k);
  k.ptr = ptr;
  k.inner = inner;
  k.rows = rows;
  k.stride = stride_bytes;
  k.bx = bx;
  k.by = by;
  k.dtype = (int)dtype;
  k.swz = (int)swz;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (keys[i] == k) {
      *out = maps[i];
      return true;
    }
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {stride_bytes};
  const cuuint32_t box[2] = {bx, by};
  const cuuint32_t estr[2] = {1, 1};
  CUtensorMap m;
  if (enc(&m, dtype, 2, const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  const int slot = used < 64 ? used++ : (next++ & 63);
  keys[slot] = k;
  maps[slot] = m;
  *out = m;
  return true;
}

// Checks shared by every attention entry point (nothing is launched when they fail).
mikv_status attention_args_ok(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo, const void* q,
                              const void* out, int32_t out_dtype) {
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!cache_ok(cache, shape) || !q || !out || n_lo < 0 || (out_dtype != MIKV_OUT_BF16 && out_dtype != MIKV_OUT_F32))
    return MIKV_ERR_ARG;
  if (n_lo > shape->lo_cap) return MIKV_ERR_CAPACITY;
  if (evicting(*shape) && n_lo != 0) return MIKV_ERR_ARG;
  if (shape->hi_cap + n_lo < 1) return MIKV_ERR_ARG;
  if (!aligned(cache->k_hi, 16) || !aligned(cache->v_hi, 16) || !aligned(cache->k_codes, 16) ||
      !aligned(cache->v_codes, 16) || !aligned(cache->k_params, 16) || !aligned(cache->v_params, 16) ||
      !aligned(q, 4) || (cache->balancer && !aligned(cache->balancer, 16)))
    return MIKV_ERR_ARG;
  return MIKV_OK;
}

struct StepLayout {
  size_t attn, logits, total;
};

StepLayout step_layout(const mikv_shape* s, int n_lo_max) {
  StepLayout L;
  L.attn = attention_workspace_bytes(*s, n_lo_max, num_sms());
  const size_t logits = (size_t)s->batch * s->heads_q * s->hi_stride * sizeof(float);
  L.logits = L.attn;
  L.total = L.logits + (logits + 255) / 256 * 256;
  return L;
}

// Launches the attention kernel and, when `merge` is set, the merge of its partials into out / ml.
// With `merge` unset the partials stay in the workspace and *args_out describes them.
mikv_status attention_impl(const mikv_shape* s, const mikv_cache* c, int32_t n_lo, const void* q, float sm_scale,
                           void* out, int32_t out_dtype, float* hi_logits, float* ml, void* ws, size_t ws_bytes,
                           cudaStream_t st, bool merge = true, AttnArgs* args_out = nullptr,
                           const int32_t* ins_slots = nullptr, const void* ins_k = nullptr,
                           const void* ins_v = nullptr, int32_t ins_tok = 0) {
  const int sms = num_sms();
  // per-channel keys: the n_lo mod 64 staged retained tokens are attended as important rows hi_cap ..
  const bool kch = kch_of(*s);
  const int n_stage = kch ? n_lo % kKchGroup : 0;
  mikv_shape se = *s;
  se.hi_cap += n_stage;
  n_lo -= n_stage;
  const AttnPlan plan = plan_attention(se, n_lo, sms);
  if (ws_bytes < attention_workspace_bytes(*s, n_lo + n_stage, sms)) return MIKV_ERR_WORKSPACE;
  if ((long long)s->batch * s->heads_kv * plan.n_u > 2000000000LL) return MIKV_ERR_UNSUPPORTED;
  const int G = s->heads_q / s->heads_kv;
  AttnArgs a;
  memset(&a, 0, sizeof a);
  const uint64_t hi_rows = (uint64_t)s->batch * s->heads_kv * s->hi_stride;
  const uint64_t lo_rows = (uint64_t)s->batch * s->heads_kv * s->lo_cap;
  const int hb = hi_bits_of(*s);
  bool ok;
  if (hb == 16) {
    ok = make_map(&a.map_k_hi, c->k_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, hi_rows, 2 * kHeadDim, 64, 16,
                  CU_TENSOR_MAP_SWIZZLE_128B) &&
         make_map(&a.map_v_hi, c->v_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, hi_rows, 2 * kHeadDim, 64, 16,
                  CU_TENSOR_MAP_SWIZZLE_128B);
  } else {
    // coded important rows: viewed like retained codes of layout (hb, 64); hi_stride % 16 == 0 keeps
    // every unit row-aligned
    const LoUnit H = lo_unit_layout(hb, kHiGroup);
    const uint64_t code_rows = hi_rows * H.pitch / H.map_w;
    const uint32_t code_box = 16u * H.blocks * H.pitch / H.map_w;
    const CUtensorMapSwizzle swz = hb == 8 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    const uint64_t par_rows = hi_rows * H.param_row / H.param_w;
    const uint32_t par_box = 16u * H.blocks * H.param_row / H.param_w;
    ok = make_map(&a.map_k_hi, c->k_hi, CU_TENSOR_MAP_DATA_TYPE_UINT8, H.map_w, code_rows, H.map_w, H.map_w,
                  code_box, swz) &&
         make_map(&a.map_v_hi, c->v_hi, CU_TENSOR_MAP_DATA_TYPE_UINT8, H.map_w, code_rows, H.map_w, H.map_w,
                  code_box, swz) &&
         make_map(&a.map_k_hp, c->k_hi_params, CU_TENSOR_MAP_DATA_TYPE_UINT8, H.param_w, par_rows, H.param_w,
                  H.param_w, par_box, CU_TENSOR_MAP_SWIZZLE_NONE) &&
         make_map(&a.map_v_hp, c->v_hi_params, CU_TENSOR_MAP_DATA_TYPE_UINT8, H.param_w, par_rows, H.param_w,
                  H.param_w, par_box, CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  if (ok && lo_rows > 0 && !evicting(*s)) {
    // retained arrays: each is viewed as rows of U.map_w (codes) or U.param_w (alpha, beta) bytes, and
    // one box covers a whole unit of 16 * U.blocks tokens (lo_cap % 16 == 0 keeps units row-aligned)
    const LoUnit U = kch ? lo_unit_layout_kch(s->bits, s->group) : lo_unit_layout(s->bits, s->group);
    const uint64_t code_rows = lo_rows * U.pitch / U.map_w;
    const uint32_t code_box = 16u * U.blocks * U.pitch / U.map_w;
    const CUtensorMapSwizzle swz = s->bits == 3 ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_64B;
    const uint64_t par_rows = lo_rows * U.param_row / U.param_w;
    const uint32_t par_box = 16u * U.blocks * U.param_row / U.param_w;
    ok = make_map(&a.map_k_lo, c->k_codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, U.map_w, code_rows, U.map_w, U.map_w,
                  code_box, swz) &&
         make_map(&a.map_v_lo, c->v_codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, U.map_w, code_rows, U.map_w, U.map_w,
                  code_box, swz) &&
         (kch ? make_map(&a.map_k_par, c->k_params, CU_TENSOR_MAP_DATA_TYPE_UINT8, 128,
                         lo_rows / kKchGroup * 4, 128, 128, 4, CU_TENSOR_MAP_SWIZZLE_NONE)  // 512 B per group
              : make_map(&a.map_k_par, c->k_params, CU_TENSOR_MAP_DATA_TYPE_UINT8, U.param_w, par_rows, U.param_w,
                         U.param_w, par_box, CU_TENSOR_MAP_SWIZZLE_NONE)) &&
         make_map(&a.map_v_par, c->v_params, CU_TENSOR_MAP_DATA_TYPE_UINT8, U.param_w, par_rows, U.param_w,
                  U.param_w, par_box, CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  if (!ok) return MIKV_ERR_CUDA;
  a.q = q;
  a.balancer = c->balancer;
  a.hi_logits = hi_logits;
  char* wsb = static_cast<char*>(ws);
  a.status = reinterpret_cast<int*>(wsb);
  a.part_o = reinterpret_cast<float*>(wsb + kWsHeader);
  a.part_ml = a.part_o + (size_t)plan.n_slots * G * kHeadDim;
  a.batch = s->batch;
  a.heads_q = s->heads_q;
  a.heads_kv = s->heads_kv;
  a.hi_cap = se.hi_cap;
  a.hi_stride = s->hi_stride;
  a.lo_cap = s->lo_cap;
  a.n_lo = n_lo;
  a.hi_blocks = plan.hi_blocks;
  a.hi_units = plan.hi_units;
  a.lo_blocks = plan.lo_blocks;
  a.n_u = plan.n_u;
  a.n_units = plan.n_units;
  a.n_warps = plan.n_warps;
  a.sm_scale = sm_scale;
  if (ins_slots) {
    a.ins_slots = ins_slots;
    a.ins_k = static_cast<const __nv_bfloat16*>(ins_k);
    a.ins_v = static_cast<const __nv_bfloat16*>(ins_v);
    a.ins_k_hi = static_cast<__nv_bfloat16*>(c->k_hi);
    a.ins_v_hi = static_cast<__nv_bfloat16*>(c->v_hi);
    a.ins_hi_tok = c->hi_tok;
    a.ins_acc = c->acc;
    a.ins_tok = ins_tok;
  }
  cudaError_t e = launch_attention(a, lo_bits_of(*s), lo_group_of(*s), hb, G, plan.grid, st, kch);
  if (e != cudaSuccess) return MIKV_ERR_CUDA;
  if (args_out) *args_out = a;
  if (!merge) return MIKV_OK;
  MergeArgs m;
  m.part_o = a.part_o;
  m.part_ml = a.part_ml;
  m.out = out;
  m.ml = ml;
  m.batch = s->batch;
  m.heads_q = s->heads_q;
  m.heads_kv = s->heads_kv;
  m.n_u = plan.n_u;
  m.n_units = plan.n_units;
  m.n_warps = plan.n_warps;
  e = launch_merge(m, G, out_dtype == MIKV_OUT_F32, st);
  return cuda_status(e);
}

}  // namespace

extern "C" {

const char* mikv_status_string(mikv_status s) {
  switch (s) {
    case MIKV_OK: return "ok";
    case MIKV_ERR_ARG: return "invalid argument";
    case MIKV_ERR_UNSUPPORTED: return "unsupported configuration";
    case MIKV_ERR_CAPACITY: return "capacity exceeded";
    case MIKV_ERR_CUDA: return "CUDA error";
    case MIKV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case MIKV_ERR_DEVICE: return "a kernel reported an internal failure";
    case MIKV_ERR_SCRATCH: return "problem needs more scratch than the built-in no-allocation buffer holds";
  }
  return "unknown status";
}

size_t mikv_workspace_bytes(const mikv_shape* shape, int32_t op, int32_t n_lo_max) {
  if (shape_supported(shape) != MIKV_OK || n_lo_max < 0) return 0;
  switch (op) {
    case MIKV_WS_ATTENTION: return attention_workspace_bytes(*shape, n_lo_max, num_sms());
    case MIKV_WS_BALANCER: return kWsHeader + 2 * (size_t)shape->heads_kv * kHeadDim * sizeof(uint32_t);
    case MIKV_WS_STEP: return step_layout(shape, n_lo_max).total;
    case MIKV_WS_PREFILL: return prefill_workspace_bytes(shape->batch, shape->heads_q, n_lo_max);
  }
  return 0;
}

mikv_status mikv_workspace_reset(void* workspace, size_t ws_bytes, void* stream) {
  if (!workspace || ws_bytes < kWsHeader) return MIKV_ERR_WORKSPACE;
  return cuda_status(cudaMemsetAsync(workspace, 0, sizeof(int), static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_workspace_check(const void* workspace, void* stream) {
  if (!workspace) return MIKV_ERR_WORKSPACE;
  int v = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&v, workspace, sizeof v, cudaMemcpyDeviceToHost, st) != cudaSuccess) return MIKV_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return MIKV_ERR_CUDA;
  return v == 0 ? MIKV_OK : MIKV_ERR_DEVICE;
}

mikv_status mikv_compute_balancer(const mikv_shape* shape, const void* q_pre, const void* k_pre, int32_t T,
                                  float* balancer_out, void* workspace, size_t ws_bytes, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!q_pre || !k_pre || !balancer_out || T <= 0) return MIKV_ERR_ARG;
  if (!workspace || !aligned(workspace, 256) ||
      ws_bytes < mikv_workspace_bytes(shape, MIKV_WS_BALANCER, 0))
    return MIKV_ERR_WORKSPACE;
  uint32_t* ws = reinterpret_cast<uint32_t*>(static_cast<char*>(workspace) + kWsHeader);
  return cuda_status(launch_balancer(*shape, q_pre, k_pre, T, balancer_out, ws, static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_quantize_pack(const mikv_shape* shape, const mikv_cache* cache, const void* k_src,
                               const void* v_src, const int32_t* src_tok, int32_t n_src, const int32_t* rows,
                               int32_t n_rows, int32_t lo_start, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (evicting(*shape)) return MIKV_ERR_UNSUPPORTED;  // no retained set to write
  if (!cache_ok(cache, shape) || !k_src || !v_src || n_src <= 0 || n_rows < 0 || lo_start < 0 || (n_rows > 0 && !rows))
    return MIKV_ERR_ARG;
  if (!aligned(k_src, 16) || !aligned(v_src, 16)) return MIKV_ERR_ARG;  // rows are read in 16-byte pieces
  if ((int64_t)lo_start + n_rows > shape->lo_cap) return MIKV_ERR_CAPACITY;
  if ((int64_t)shape->batch * shape->heads_kv > 65535)
    return MIKV_ERR_UNSUPPORTED;
  if (kch_of(*shape)) {  // append: complete groups quantized per channel, the rest staged
    if (n_rows == 0) return MIKV_OK;
    if (!rows) return MIKV_ERR_ARG;
    return cuda_status(launch_kch_append(*shape, *cache, k_src, v_src, src_tok, n_src, rows, n_rows, lo_start,
                                         static_cast<cudaStream_t>(stream)));
  }
  return cuda_status(launch_quantize_pack(*shape, *cache, k_src, v_src, src_tok, n_src, rows, n_rows, lo_start,
                                          static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_prefill_scores(const mikv_shape* shape, const void* q_pre, const void* k_pre, int32_t T,
                                float sm_scale, float* scores, void* workspace, size_t ws_bytes, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!q_pre || !k_pre || !scores || T <= 0) return MIKV_ERR_ARG;
  if (!aligned(q_pre, 16) || !aligned(k_pre, 16) || !aligned(scores, 4)) return MIKV_ERR_ARG;
  if ((int64_t)shape->batch * shape->heads_q * T + kPfTile >= 2147483647LL ||
      (int64_t)shape->batch * shape->heads_q > 65535)
    return MIKV_ERR_UNSUPPORTED;
  if (!workspace || !aligned(workspace, 256) || ws_bytes < prefill_workspace_bytes(shape->batch, shape->heads_q, T))
    return MIKV_ERR_WORKSPACE;
  PrefillArgs a;
  memset(&a, 0, sizeof a);
  const uint64_t qrows = (uint64_t)shape->batch * shape->heads_q * T;
  const uint64_t krows = (uint64_t)shape->batch * shape->heads_kv * T;
  if (!make_map(&a.map_q, q_pre, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, qrows, 2 * kHeadDim, 64, kPfTile,
                CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&a.map_k, k_pre, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, krows, 2 * kHeadDim, 64, kPfTile,
                CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&a.map_q_str, q_pre, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, qrows, 2 * kHeadDim, 64, kPfTile / 2,
                CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&a.map_k_str, k_pre, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, kHeadDim, krows, 2 * kHeadDim, 64, kPfTile / 2,
                CU_TENSOR_MAP_SWIZZLE_128B))
    return MIKV_ERR_CUDA;
  char* wsb = static_cast<char*>(workspace);
  a.status = reinterpret_cast<int*>(wsb);
  a.stats = reinterpret_cast<float*>(wsb + kWsHeader);
  a.scores = scores;
  a.heads_q = shape->heads_q;
  a.heads_kv = shape->heads_kv;
  a.T = T;
  a.T_pad = prefill_padded(T);
  a.scale_log2 = sm_scale * 1.4426950408889634f;
  return cuda_status(launch_prefill(a, shape->batch, static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_decode_attention(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo, const void* q,
                                  float sm_scale, void* out, int32_t out_dtype, float* hi_logits, float* ml,
                                  void* workspace, size_t ws_bytes, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = attention_args_ok(shape, cache, n_lo, q, out, out_dtype);
  if (st != MIKV_OK) return st;
  if (!workspace || !aligned(workspace, 256)) return MIKV_ERR_WORKSPACE;
  return attention_impl(shape, cache, n_lo, q, sm_scale, out, out_dtype, hi_logits, ml, workspace, ws_bytes,
                        static_cast<cudaStream_t>(stream));
}

mikv_status mikv_update_importance(const mikv_shape* shape, const mikv_cache* cache, const float* hi_logits,
                                   const float* ml, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!cache_ok(cache, shape) || !hi_logits || !ml) return MIKV_ERR_ARG;
  if (shape->hi_cap == 0) return MIKV_OK;
  return cuda_status(launch_update_importance(*shape, *cache, hi_logits, ml, static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_select_demote(int32_t batch, int32_t heads, const float* scores, const int32_t* ids, int32_t n,
                               int32_t stride, int32_t n_demote, int32_t* demoted, int32_t* kept, void* stream) {
  MIKV_CALL_RANGE();
  if (batch <= 0 || heads <= 0 || !scores || n < 0 || stride < n || n_demote < 0 || n_demote > n) return MIKV_ERR_ARG;
  if (n_demote > 0 && !demoted) return MIKV_ERR_ARG;
  if ((int64_t)batch * heads > 2147483647) return MIKV_ERR_UNSUPPORTED;
  if (n == 0) return MIKV_OK;
  return cuda_status(launch_select(batch, heads, scores, ids, n, stride, n_demote, demoted, kept,
                                   static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_insert_token(const mikv_shape* shape, const mikv_cache* cache, const void* k_new,
                              const void* v_new, int32_t tok, const int32_t* slots, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!cache_ok(cache, shape) || !k_new || !v_new || !slots) return MIKV_ERR_ARG;
  if (shape->hi_cap < 1) return MIKV_ERR_CAPACITY;
  return cuda_status(launch_insert(*shape, *cache, k_new, v_new, tok, slots, static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_gather_hi(const mikv_shape* shape, const mikv_cache* cache, const void* k_src, const void* v_src,
                           const int32_t* src_tok, const float* src_scores, int32_t n_src, const int32_t* rows,
                           int32_t n_rows, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!cache_ok(cache, shape) || !k_src || !v_src || n_src <= 0 || n_rows < 0 || (n_rows > 0 && !rows))
    return MIKV_ERR_ARG;
  if (n_rows > shape->hi_cap) return MIKV_ERR_CAPACITY;
  return cuda_status(launch_gather(*shape, *cache, k_src, v_src, src_tok, src_scores, n_src, rows, n_rows,
                                   static_cast<cudaStream_t>(stream)));
}

mikv_status mikv_decode_step(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo, const void* q,
                             const void* k_new, const void* v_new, int32_t tok, int32_t* slots, float sm_scale,
                             void* out, int32_t out_dtype, void* workspace, size_t ws_bytes, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = shape_supported(shape);
  if (st != MIKV_OK) return st;
  if (!cache_ok(cache, shape) || !q || !k_new || !v_new || !slots || !out || n_lo < 0) return MIKV_ERR_ARG;
  if (shape->hi_cap < 1) return MIKV_ERR_CAPACITY;
  if (!evicting(*shape) && (int64_t)n_lo + 1 > shape->lo_cap) return MIKV_ERR_CAPACITY;
  if (!workspace || !aligned(workspace, 256)) return MIKV_ERR_WORKSPACE;
  const StepLayout L = step_layout(shape, n_lo);
  if (ws_bytes < L.total) return MIKV_ERR_WORKSPACE;
  char* wsb = static_cast<char*>(workspace);
  float* logits = reinterpret_cast<float*>(wsb + L.logits);
  if ((st = attention_args_ok(shape, cache, n_lo, q, out, out_dtype)) != MIKV_OK) return st;
  if (!aligned(k_new, 8) || !aligned(v_new, 8)) return MIKV_ERR_ARG;
  // a bf16 important set takes the new token inside the attention kernel; a coded one quantizes it first
  const bool fused_insert = hi_bits_of(*shape) == 16;
  if (!fused_insert && (st = mikv_insert_token(shape, cache, k_new, v_new, tok, slots, stream)) != MIKV_OK)
    return st;
  // attention without its separate merge: the fused tail below merges, updates, selects and demotes
  AttnArgs a;
  if ((st = attention_impl(shape, cache, n_lo, q, sm_scale, out, out_dtype, logits, nullptr, workspace, L.attn,
                           static_cast<cudaStream_t>(stream), false, &a, fused_insert ? slots : nullptr, k_new,
                           v_new, tok)) != MIKV_OK)
    return st;
  StepPostArgs p;
  p.status = a.status;
  p.part_o = a.part_o;
  p.part_ml = a.part_ml;
  p.out = out;
  p.hi_logits = logits;
  p.acc = cache->acc;
  p.hi_tok = cache->hi_tok;
  p.k_hi = cache->k_hi;
  p.v_hi = cache->v_hi;
  p.balancer = cache->balancer;
  p.k_codes = cache->k_codes;
  p.v_codes = cache->v_codes;
  p.k_params = cache->k_params;
  p.v_params = cache->v_params;
  p.lo_tok = cache->lo_tok;
  p.slots = slots;
  p.k_hi_params = cache->k_hi_params;
  p.v_hi_params = cache->v_hi_params;
  p.hi_bits = hi_bits_of(*shape);
  p.evict = evicting(*shape) ? 1 : 0;
  p.kch = kch_of(*shape) ? 1 : 0;
  p.batch = shape->batch;
  p.heads_q = shape->heads_q;
  p.heads_kv = shape->heads_kv;
  p.hi_cap = shape->hi_cap;
  p.hi_stride = shape->hi_stride;
  p.lo_cap = shape->lo_cap;
  p.n_lo = n_lo;
  p.n_u = a.n_u;
  p.n_units = a.n_units;
  p.n_warps = a.n_warps;
  cudaError_t e = launch_step_post(p, lo_bits_of(*shape), lo_group_of(*shape), shape->heads_q / shape->heads_kv,
                                   out_dtype == MIKV_OUT_F32, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess && p.kch && n_lo % kKchGroup == kKchGroup - 1)  // the victim completed a group
    e = launch_kch_append(*shape, *cache, nullptr, nullptr, nullptr, 0, nullptr, 0, n_lo + 1,
                          static_cast<cudaStream_t>(stream));
  return cuda_status(e);
}

double mikv_cache_fraction(int32_t bits, int32_t group, double ratio, int32_t hi_bits) {
  if (group <= 0) return -1.0;
  const double hi = hi_bits >= 16 ? 1.0 : (hi_bits + 32.0 / group) / 16.0;
  const double lo = (bits + 32.0 / group) / 16.0;
  return ratio * hi + (1.0 - ratio) * lo;
}

int32_t mikv_budget(int32_t T, double ratio) {
  if (T < 0 || !(ratio >= 0.0 && ratio <= 1.0)) return -1;
  return (int32_t)floor(ratio * (double)T + 0.5);
}

size_t mikv_retained_row_bytes(int32_t bits, int32_t group, int32_t head_dim) {
  if (bits <= 0 || group <= 0 || head_dim <= 0 || head_dim % group) return 0;
  return (size_t)head_dim * bits / 8 + (size_t)4 * (head_dim / group);
}

}  // extern "C"

// ---------------------------------------------------------------------------- no-allocation entry
//
// For callers that may not allocate device memory on the decode path (an engine that owns all device
// memory and forbids plugins to call the CUDA allocator, or a serving loop that cannot afford a
// synchronising cudaMalloc): decode attention whose split partials live in a fixed file-scope device
// buffer of the library instead of a caller workspace. The buffer is part of the loaded module, so
// every device that loads the library holds it until the process exits.

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[MIKV_NOALLOC_SCRATCH_BYTES];

// Device address of the buffer in the current context. The name of a __device__ array in host code is only
// a host-side stand-in, so the address must come from the runtime. It is looked up on every call (the lookup
// allocates nothing): an address kept from an earlier call would dangle after cudaDeviceReset or when the
// caller makes another context current. The first lookup in a context loads the library's device code there.
mikv_status noalloc_scratch(void** out) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return MIKV_ERR_CUDA;
  *out = p;
  return MIKV_OK;
}

}  // namespace

extern "C" mikv_status mikv_decode_attention_noalloc(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo,
                                                     const void* q, float sm_scale, void* out, int32_t out_dtype,
                                                     float* hi_logits, float* ml, void* stream) {
  MIKV_CALL_RANGE();
  mikv_status st = attention_args_ok(shape, cache, n_lo, q, out, out_dtype);
  if (st != MIKV_OK) return st;
  const size_t need = attention_workspace_bytes(*shape, n_lo, num_sms());
  if (need > MIKV_NOALLOC_SCRATCH_BYTES) return MIKV_ERR_SCRATCH;
  void* ws = nullptr;
  if ((st = noalloc_scratch(&ws)) != MIKV_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, sizeof(int), s) != cudaSuccess) return MIKV_ERR_CUDA;  // status word starts at 0
  return attention_impl(shape, cache, n_lo, q, sm_scale, out, out_dtype, hi_logits, ml, ws,
                        MIKV_NOALLOC_SCRATCH_BYTES, s);
}

extern "C" mikv_status mikv_noalloc_check(void* stream) {
  void* ws = nullptr;
  mikv_status st = noalloc_scratch(&ws);
  if (st != MIKV_OK) return st;
  return mikv_workspace_check(ws, stream);
}

extern "C" int32_t mikv_debug_enabled(void) {
#ifdef MIKV_DEBUG
  return 1;
#else
  return 0;
#endif
}

extern "C" mikv_status mikv_debug_check(void* stream) {
#ifdef MIKV_DEBUG
  int* w = debug_status_word();
  if (!w) return MIKV_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int v = 0;
  if (cudaMemcpyAsync(&v, w, sizeof v, cudaMemcpyDeviceToHost, st) != cudaSuccess) return MIKV_ERR_CUDA;
  if (cudaMemsetAsync(w, 0, sizeof(int), st) != cudaSuccess) return MIKV_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return MIKV_ERR_CUDA;
  return v == 0 ? MIKV_OK : MIKV_ERR_DEVICE;
#else
  (void)stream;
  return MIKV_OK;
#endif
}
