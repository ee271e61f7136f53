// mikv_quant.cu — demotion of KV rows into the retained set (Eq. 1 with the Eq. 3 key balancer), rows
// entering a coded important set (Sec. 3.3), and the channel balancer itself (Eq. 2), arxiv 2402.18096.
//
// quantize_pack: each warp quantizes four rows of K or of V, eight lanes per row and 16 channels per lane;
// group minima and maxima come from the lane's channels and butterfly shuffles, scale and zero are
// rounded to fp16 outward so the stored grid covers the group's range, codes are round-half-even of the
// IEEE fp32 quotient (x - beta) / alpha (the Eq. 1 helpers of mikv_quant_rows.cuh, shared with the
// one-row quantizer of the step tail), and the packed words are assembled by a reduce-scatter over the
// lanes that share them.
#include "mikv_device.cuh"
#include "mikv_internal.h"
#include "mikv_quant_rows.cuh"

namespace mikv {
namespace {

struct QPArgs {
  const __nv_bfloat16* k_src;
  const __nv_bfloat16* v_src;
  const int32_t* src_tok;
  const int32_t* rows;
  const float* balancer;
  uint8_t* k_codes;
  uint8_t* v_codes;
  __half2* k_params;
  __half2* v_params;
  int32_t* lo_tok;
  int* dbg;  // debug builds: the library's status word for index checks (nullptr otherwise)
  int heads_kv, n_src, n_rows, lo_start, lo_cap;
};

// Bulk quantize/pack (Eq. 1): eight lanes per row and four rows per warp. Lane l8 = lane & 7 of a row owns
// channels 16 l8 .. 16 l8 + 15 (two 16-byte loads), so a group's scale and zero are computed by GROUP / 16
// lanes, and in the packed layout every channel of the lane sits at field index m = l8 of its 16-bit unit:
// the lane's codes form partial words at fixed positions, which a reduce-scatter over the lanes that share
// them turns into whole words, one or two per lane.
constexpr int kQpRowsPerWarp = 4;

// Reduce-scatter of N partial words over lane bits OFF, OFF / 2, ...: in each round a lane keeps the half
// of its words selected by its lane bit and ORs in the partner's copy of that half. After log2(N) rounds
// lane l8 holds the whole word index (bits of l8 from OFF down), as a single value.
template <int N, int OFF>
__device__ __forceinline__ uint32_t reduce_scatter(const uint32_t (&w)[N], int l8) {
  constexpr int H = N / 2;
  const bool up = (l8 & OFF) != 0;
  uint32_t k[H];
#pragma unroll
  for (int i = 0; i < H; ++i) {
    const uint32_t send = up ? w[i] : w[i + H];
    k[i] = (up ? w[i + H] : w[i]) | __shfl_xor_sync(0xffffffffu, send, OFF);
  }
  if constexpr (H == 1) {
    return k[0];
  } else {
    return reduce_scatter<H, OFF / 2>(k, l8);
  }
}

template <int BITS, int GROUP>
__global__ void __launch_bounds__(256) quantize_pack_kernel(const QPArgs a) {
  constexpr int QMAX = (1 << BITS) - 1;
  constexpr int GL = GROUP / 16;  // lanes per quantization group
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, l8 = lane & 7;
  const bool is_v = (w & 1) != 0;
  const int bh = blockIdx.y, h = bh % a.heads_kv;
  const int i = (blockIdx.x * 4 + (w >> 1)) * kQpRowsPerWarp + (lane >> 3);
  const int r = i < a.n_rows ? a.rows[(size_t)bh * a.n_rows + i] : -1;
  const bool valid = r >= 0 && r < a.n_src;  // out-of-range rows are skipped (documented in the ABI)
  if (i < a.n_rows && !valid && l8 == 0 && !is_v) MIKV_BOUNDS_FAIL(a.dbg);
  // invalid rows run the arithmetic on zeros (every lane takes part in the shuffles) and store nothing
  uint4 raw[2] = {make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u)};
  if (valid) {
    const uint4* src = reinterpret_cast<const uint4*>((is_v ? a.v_src : a.k_src) +
                                                      ((size_t)bh * a.n_src + r) * kHeadDim + 16 * l8);
    raw[0] = src[0];
    raw[1] = src[1];
  }
  float x[16];
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const uint32_t wd[4] = {raw[k].x, raw[k].y, raw[k].z, raw[k].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[8 * k + 2 * j] = __uint_as_float(wd[j] << 16);
      x[8 * k + 2 * j + 1] = __uint_as_float(wd[j] & 0xffff0000u);
    }
  }
  if (!is_v && a.balancer) {  // Eq. 3: keys times the balancer before the quantizer (warp-uniform)
    const float4* bal = reinterpret_cast<const float4*>(a.balancer + h * kHeadDim + 16 * l8);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float4 b = bal[k];
      x[4 * k] = __fmul_rn(x[4 * k], b.x);
      x[4 * k + 1] = __fmul_rn(x[4 * k + 1], b.y);
      x[4 * k + 2] = __fmul_rn(x[4 * k + 2], b.z);
      x[4 * k + 3] = __fmul_rn(x[4 * k + 3], b.w);
    }
  }
  float mn = x[0], mx = x[0];
#pragma unroll
  for (int e = 1; e < 16; ++e) {
    mn = fminf(mn, x[e]);
    mx = fmaxf(mx, x[e]);
  }
#pragma unroll
  for (int off = 1; off < GL; off <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  const Eq1Params p = eq1_params<QMAX>(mn, mx);
  uint32_t code[16];
  bool redo = false;
#pragma unroll
  for (int e = 0; e < 16; ++e) code[e] = eq1_code_fast<QMAX>(x[e], p, redo);
  if (redo) {
#pragma unroll
    for (int e = 0; e < 16; ++e) code[e] = eq1_code_exact<QMAX>(x[e], p);
  }

  const size_t pos = (size_t)bh * a.lo_cap + a.lo_start + i;
  uint32_t* row = reinterpret_cast<uint32_t*>((is_v ? a.v_codes : a.k_codes) + pos * (16 * BITS));
  if constexpr (BITS == 4) {
    // channel 16 l8 + u: unit 16 (l8 >> 2) + u, bits 4 (l8 & 3); the lanes with equal l8 >> 2 share
    // words 8 (l8 >> 2) .. + 7, and lane l8 ends with words 2 l8, 2 l8 + 1
    const int sh = 4 * (l8 & 3);
    uint32_t L[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) L[k] = (code[2 * k] << sh) | (code[2 * k + 1] << (16 + sh));
    uint32_t K[2][4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const bool up = (l8 & 2) != 0;
      K[0][k] = (up ? L[k + 4] : L[k]) | __shfl_xor_sync(0xffffffffu, up ? L[k] : L[k + 4], 2);
    }
    uint32_t out[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const bool up = (l8 & 1) != 0;
      out[k] = (up ? K[0][k + 2] : K[0][k]) | __shfl_xor_sync(0xffffffffu, up ? K[0][k] : K[0][k + 2], 1);
    }
    if (valid) *reinterpret_cast<uint2*>(row + 2 * l8) = make_uint2(out[0], out[1]);
  } else {
    // two-bit fields (INT2, and the low bits of INT3): channel 16 l8 + u sits in unit u at bits 2 l8;
    // all eight lanes share words 0..7, and lane l8 ends with word l8
    const int sh = 2 * l8;
    uint32_t L[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) L[k] = ((code[2 * k] & 3u) << sh) | ((code[2 * k + 1] & 3u) << (16 + sh));
    const uint32_t wd = reduce_scatter<8, 4>(L, l8);
    if (valid) row[l8] = wd;
    if constexpr (BITS == 3) {
      // high bits: channel 16 l8 + u sits in unit u & 7 at bit 2 l8 + (u >> 3) (words 8..11 of the row);
      // after two rounds a lane pair holds one word, and the pair's even lane stores it
      uint32_t H[4] = {0u, 0u, 0u, 0u};
#pragma unroll
      for (int u = 0; u < 16; ++u) H[(u & 7) >> 1] |= (code[u] >> 2) << (16 * (u & 1) + 2 * l8 + (u >> 3));
      uint32_t K[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const bool up = (l8 & 4) != 0;
        K[k] = (up ? H[k + 2] : H[k]) | __shfl_xor_sync(0xffffffffu, up ? H[k] : H[k + 2], 4);
      }
      const bool up = (l8 & 2) != 0;
      uint32_t hw = (up ? K[1] : K[0]) | __shfl_xor_sync(0xffffffffu, up ? K[0] : K[1], 2);
      hw |= __shfl_xor_sync(0xffffffffu, hw, 1);
      if (valid && (l8 & 1) == 0) row[8 + (l8 >> 1)] = hw;
    }
  }
  if (valid && l8 % GL == 0)
    ((is_v ? a.v_params : a.k_params) + pos * (kHeadDim / GROUP))[(16 * l8) / GROUP] =
        __halves2half2(p.alpha16, p.beta16);
  if (valid && !is_v && l8 == 0) a.lo_tok[pos] = a.src_tok ? a.src_tok[(size_t)bh * a.n_src + r] : r;
}

template <int BITS>
cudaError_t qp_group(const QPArgs& a, int group, dim3 grid, cudaStream_t st) {
  switch (group) {
    case 32: quantize_pack_kernel<BITS, 32><<<grid, 256, 0, st>>>(a); break;
    case 64: quantize_pack_kernel<BITS, 64><<<grid, 256, 0, st>>>(a); break;
    case 128: quantize_pack_kernel<BITS, 128><<<grid, 256, 0, st>>>(a); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

// ------------------------------------------------------- coded important set (Sec. 3.3, Table 3)

// Rows entering a coded important set, quantized like retained rows (Eq. 1 at hi_bits, groups of
// kHiGroup; keys times the balancer first, Eq. 3). Two modes: insert (rows == nullptr: the new token of
// every (b, h) into slot slots[b][h]) and gather (slot i < n_rows receives source row rows[b][h][i]).
struct HiQArgs {
  const __nv_bfloat16* k_src;
  const __nv_bfloat16* v_src;
  const int32_t* src_tok;
  const float* src_scores;
  const int32_t* rows;
  const int32_t* slots;
  const float* balancer;
  uint8_t* k_hc;
  uint8_t* v_hc;
  __half2* k_hp;
  __half2* v_hp;
  int32_t* hi_tok;
  float* acc;
  int* dbg;  // debug builds: the library's status word for index checks (nullptr otherwise)
  int heads_kv, hi_cap, hi_stride, n_src, n_rows, tok;
};

template <int HB>
__global__ void __launch_bounds__(256) hi_quant_kernel(const HiQArgs a) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  grid_dependency_wait();  // insertion: the slot comes from the previous step's tail
  allow_dependent_launch();
  const int i = blockIdx.x * 4 + (w >> 1);
  const bool is_v = (w & 1) != 0;
  const int bh = blockIdx.y, h = bh % a.heads_kv;
  int slot, r = 0;
  const __nv_bfloat16* src;
  if (a.rows) {
    if (i >= a.n_rows) return;
    r = a.rows[(size_t)bh * a.n_rows + i];
    if (r < 0 || r >= a.n_src) {  // out-of-range rows are skipped, as in quantize_pack
      if (lane == 0 && !is_v) MIKV_BOUNDS_FAIL(a.dbg);
      return;
    }
    slot = i;
    src = (is_v ? a.v_src : a.k_src) + ((size_t)bh * a.n_src + r) * kHeadDim;
  } else {
    if (i > 0) return;
    slot = a.slots[bh];
    if (slot < 0 || slot >= a.hi_cap) {
      if (lane == 0 && !is_v) MIKV_BOUNDS_FAIL(a.dbg);
      return;
    }
    src = (is_v ? a.v_src : a.k_src) + (size_t)bh * kHeadDim;
  }
  const size_t row = (size_t)bh * a.hi_stride + slot;
  quantize_row_warp<HB, kHiGroup>(src, is_v ? nullptr : (a.balancer ? a.balancer + h * kHeadDim : nullptr),
                                  (is_v ? a.v_hc : a.k_hc) + row * (16 * HB),
                                  (is_v ? a.v_hp : a.k_hp) + row * (kHeadDim / kHiGroup), lane);
  if (!is_v && lane == 0) {
    a.hi_tok[row] = a.rows ? (a.src_tok ? a.src_tok[(size_t)bh * a.n_src + r] : r) : a.tok;
    a.acc[row] = a.rows && a.src_scores ? a.src_scores[(size_t)bh * a.n_src + r] : 0.f;
  }
}

// ------------------------------------------------------------- per-channel retained keys (App. C)

// Rows of the retained set with per-channel keys: position p of (b, h) belongs to token group p / 64. New
// rows (source rows rows[b][h][p - p0]) and staged rows (important rows hi_cap + p % 64, positions < p0)
// feed the group kernel; the stage kernel copies the rows of an incomplete last group into staging.
struct KchArgs {
  const __nv_bfloat16* k_src;
  const __nv_bfloat16* v_src;
  const int32_t* src_tok;
  const int32_t* rows;
  __nv_bfloat16* k_hi;
  __nv_bfloat16* v_hi;
  int32_t* hi_tok;
  uint8_t* k_codes;
  uint8_t* v_codes;
  __half2* k_params;  // [B][Hkv][lo_cap / 64][128]
  __half2* v_params;
  int32_t* lo_tok;
  int* dbg;  // debug builds: the library's status word for index checks (nullptr otherwise)
  int heads_kv, hi_cap, hi_stride, lo_cap, n_src, n_rows, p0, p_end, g0;
};

constexpr int kKchThreads = 256;

// Source of position p of head bh: the staged row (p < p0) or the new source row; token id in *tok.
// A source row outside [0, n_src) reads as zeros (the host passes rows from mikv_select_demote).
__device__ __forceinline__ const __nv_bfloat16* kch_row(const KchArgs& a, int bh, int p, bool key, int32_t* tok) {
  if (p < a.p0) {
    const size_t r = (size_t)bh * a.hi_stride + a.hi_cap + (p % kKchGroup);
    if (tok) *tok = a.hi_tok[r];
    return (key ? a.k_hi : a.v_hi) + r * kHeadDim;
  }
  const int r = a.rows[(size_t)bh * a.n_rows + (p - a.p0)];
  if (tok) *tok = (r >= 0 && r < a.n_src) ? (a.src_tok ? a.src_tok[(size_t)bh * a.n_src + r] : r) : -1;
  if (r < 0 || r >= a.n_src) {
    if (key) MIKV_BOUNDS_FAIL(a.dbg);
    return nullptr;
  }
  return (key ? a.k_src : a.v_src) + ((size_t)bh * a.n_src + r) * kHeadDim;
}

// Group g0 + blockIdx.x of (b, h) = blockIdx.y, complete: keys quantized per channel over its 64 tokens
// (Eq. 1 with the same explicitly rounded fp32 steps as the per-token quantizer), values per token.
template <int BITS, int GROUP>
__global__ void __launch_bounds__(kKchThreads) kch_group_kernel(const KchArgs a) {
  __shared__ __align__(16) __nv_bfloat16 sk[kKchGroup][kHeadDim];
  __shared__ __align__(16) __nv_bfloat16 sv[kKchGroup][kHeadDim];
  __shared__ uint32_t cbuf[kKchGroup][4 * BITS];
  __shared__ int32_t stok[kKchGroup];
  constexpr int QMAX = (1 << BITS) - 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j = a.g0 + blockIdx.x, bh = blockIdx.y;
  grid_dependency_wait();  // the group's last row is staged by the step tail before this kernel
  allow_dependent_launch();
  // 1. the group's 64 key and value rows (16-byte chunks) into shared memory; code rows cleared
  for (int i = tid; i < kKchGroup * 16; i += kKchThreads) {
    const int t = i >> 4, ch = i & 15;
    const int p = kKchGroup * j + t;
    int32_t tk = -1;
    const __nv_bfloat16* kr = kch_row(a, bh, p, true, &tk);
    const __nv_bfloat16* vr = kch_row(a, bh, p, false, nullptr);
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(&sk[t][0])[ch] = kr ? reinterpret_cast<const uint4*>(kr)[ch] : z;
    reinterpret_cast<uint4*>(&sv[t][0])[ch] = vr ? reinterpret_cast<const uint4*>(vr)[ch] : z;
    if (ch == 0) stok[t] = tk;
  }
  for (int i = tid; i < kKchGroup * 4 * BITS; i += kKchThreads) (&cbuf[0][0])[i] = 0u;
  __syncthreads();
  // 2. keys: one thread per channel
  if (tid < kHeadDim) {
    const int c = tid;
    float mn = INFINITY, mx = -INFINITY;
    for (int t = 0; t < kKchGroup; ++t) {
      const float x = __bfloat162float(sk[t][c]);
      mn = fminf(mn, x);
      mx = fmaxf(mx, x);
    }
    const __half beta16 = __float2half_rd(mn);
    const float beta = __half2float(beta16);
    const float span = __fsub_rn(mx, beta);
    const __half alpha16 = span == 0.f ? __float2half_rn(1.f) : __float2half_ru(__fdiv_rn(span, (float)QMAX));
    const float alpha = __half2float(alpha16);
    a.k_params[((size_t)bh * (a.lo_cap / kKchGroup) + j) * kHeadDim + c] = __halves2half2(alpha16, beta16);
    int unit, bit, unit1 = 0, bit1 = 0;
    field_pos(c, BITS == 3 ? 2 : BITS, unit, bit);
    if (BITS == 3) field_pos(c, 1, unit1, bit1);
    for (int t = 0; t < kKchGroup; ++t) {
      int code = __float2int_rn(__fdiv_rn(__fsub_rn(__bfloat162float(sk[t][c]), beta), alpha));
      code = code < 0 ? 0 : (code > QMAX ? QMAX : code);
      const uint32_t fmask = BITS == 3 ? 3u : (uint32_t)QMAX;
      atomicOr(&cbuf[t][unit >> 1], (((uint32_t)code & fmask) << bit) << (16 * (unit & 1)));
      if (BITS == 3) atomicOr(&cbuf[t][8 + (unit1 >> 1)], (((uint32_t)code >> 2) << bit1) << (16 * (unit1 & 1)));
    }
  }
  __syncthreads();
  const size_t pos0 = (size_t)bh * a.lo_cap + (size_t)kKchGroup * j;
  for (int i = tid; i < kKchGroup * 4 * BITS; i += kKchThreads)
    reinterpret_cast<uint32_t*>(a.k_codes + pos0 * (16 * BITS))[i] = (&cbuf[0][0])[i];
  // 3. values per token (8 rows per warp) and token ids
  for (int t = warp; t < kKchGroup; t += kKchThreads / 32) {
    quantize_row_warp<BITS, GROUP>(&sv[t][0], nullptr, a.v_codes + (pos0 + t) * (16 * BITS),
                                   a.v_params + (pos0 + t) * (kHeadDim / GROUP), lane);
    if (lane == 0) a.lo_tok[pos0 + t] = stok[t];
  }
}

// Rows of the incomplete last group (positions max(p0, 64 * floor(p_end / 64)) .. p_end - 1) into staging.
__global__ void __launch_bounds__(kKchThreads) kch_stage_kernel(const KchArgs a) {
  const int bh = blockIdx.x;
  const int first = max(a.p0, a.p_end / kKchGroup * kKchGroup);
  for (int i = threadIdx.x; i < (a.p_end - first) * 16; i += kKchThreads) {
    const int p = first + (i >> 4), ch = i & 15;
    int32_t tk = -1;
    const __nv_bfloat16* kr = kch_row(a, bh, p, true, &tk);
    const __nv_bfloat16* vr = kch_row(a, bh, p, false, nullptr);
    const size_t r = (size_t)bh * a.hi_stride + a.hi_cap + (p % kKchGroup);
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(a.k_hi + r * kHeadDim)[ch] = kr ? reinterpret_cast<const uint4*>(kr)[ch] : z;
    reinterpret_cast<uint4*>(a.v_hi + r * kHeadDim)[ch] = vr ? reinterpret_cast<const uint4*>(vr)[ch] : z;
    if (ch == 0) a.hi_tok[r] = tk;
  }
}

template <int BITS>
cudaError_t kch_group_launch(const KchArgs& a, int group, dim3 grid, cudaStream_t st) {
  switch (group) {
    case 32: return launch_chained(kch_group_kernel<BITS, 32>, grid, dim3(kKchThreads), 0, st, a);
    case 64: return launch_chained(kch_group_kernel<BITS, 64>, grid, dim3(kKchThreads), 0, st, a);
    case 128: return launch_chained(kch_group_kernel<BITS, 128>, grid, dim3(kKchThreads), 0, st, a);
  }
  return cudaErrorInvalidValue;
}

// ---------------------------------------------------------------------------- Eq. 2 balancer

// Per (token chunk, batch row, head): column maxima of |x| folded into ws with atomicMax on the bit
// patterns (non-negative floats order like their bits). Rows y < B*Hq are queries, the rest keys.
__global__ void __launch_bounds__(128) absmax_kernel(const __nv_bfloat16* q_pre, const __nv_bfloat16* k_pre,
                                                      int B, int Hq, int Hkv, int T, int chunk,
                                                      uint32_t* ws) {
  const int y = blockIdx.y, c = threadIdx.x;
  const bool is_q = y < B * Hq;
  const int yy = is_q ? y : y - B * Hq;
  const int heads = is_q ? Hq : Hkv;
  const int head = yy % heads;
  const int h = is_q ? head / (Hq / Hkv) : head;
  const __nv_bfloat16* base = (is_q ? q_pre : k_pre) + (size_t)yy * T * kHeadDim + c;
  const int t0 = blockIdx.x * chunk, t1 = min(T, t0 + chunk);
  float m = 0.f;
  for (int t = t0; t < t1; ++t) m = fmaxf(m, fabsf(__bfloat162float(base[(size_t)t * kHeadDim])));
  atomicMax(&ws[(is_q ? 0 : Hkv * kHeadDim) + h * kHeadDim + c], __float_as_uint(m));
}

__global__ void __launch_bounds__(128) balancer_kernel(const uint32_t* ws, int Hkv, float* out) {
  const int h = blockIdx.x, c = threadIdx.x;
  const float mq = __uint_as_float(ws[h * kHeadDim + c]);
  const float mk = __uint_as_float(ws[Hkv * kHeadDim + h * kHeadDim + c]);
  out[h * kHeadDim + c] = (mq == 0.f || mk == 0.f) ? 1.f : __fsqrt_rn(__fdiv_rn(mq, mk));
}

}  // namespace

cudaError_t launch_quantize_pack(const mikv_shape& s, const mikv_cache& c, const void* k_src,
                                 const void* v_src, const int32_t* src_tok, int n_src,
                                 const int32_t* rows, int n_rows, int lo_start, cudaStream_t st) {
  if (n_rows == 0) return cudaSuccess;
  QPArgs a = {};
  a.dbg = debug_status_word();
  a.k_src = static_cast<const __nv_bfloat16*>(k_src);
  a.v_src = static_cast<const __nv_bfloat16*>(v_src);
  a.src_tok = src_tok;
  a.rows = rows;
  a.balancer = c.balancer;
  a.k_codes = static_cast<uint8_t*>(c.k_codes);
  a.v_codes = static_cast<uint8_t*>(c.v_codes);
  a.k_params = static_cast<__half2*>(c.k_params);
  a.v_params = static_cast<__half2*>(c.v_params);
  a.lo_tok = c.lo_tok;
  a.heads_kv = s.heads_kv;
  a.n_src = n_src;
  a.n_rows = n_rows;
  a.lo_start = lo_start;
  a.lo_cap = s.lo_cap;
  const dim3 grid((n_rows + 4 * kQpRowsPerWarp - 1) / (4 * kQpRowsPerWarp), s.batch * s.heads_kv);
  switch (s.bits) {
    case 2: return qp_group<2>(a, s.group, grid, st);
    case 3: return qp_group<3>(a, s.group, grid, st);
    case 4: return qp_group<4>(a, s.group, grid, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_hi_quant(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                            const int32_t* src_tok, const float* src_scores, int n_src, const int32_t* rows,
                            int n_rows, const int32_t* slots, int tok, cudaStream_t st) {
  HiQArgs a = {};
  a.dbg = debug_status_word();
  a.k_src = static_cast<const __nv_bfloat16*>(k_src);
  a.v_src = static_cast<const __nv_bfloat16*>(v_src);
  a.src_tok = src_tok;
  a.src_scores = src_scores;
  a.rows = rows;
  a.slots = slots;
  a.balancer = c.balancer;
  a.k_hc = static_cast<uint8_t*>(c.k_hi);
  a.v_hc = static_cast<uint8_t*>(c.v_hi);
  a.k_hp = static_cast<__half2*>(c.k_hi_params);
  a.v_hp = static_cast<__half2*>(c.v_hi_params);
  a.hi_tok = c.hi_tok;
  a.acc = c.acc;
  a.heads_kv = s.heads_kv;
  a.hi_cap = s.hi_cap;
  a.hi_stride = s.hi_stride;
  a.n_src = n_src;
  a.n_rows = n_rows;
  a.tok = tok;
  const dim3 grid(rows ? (n_rows + 3) / 4 : 1, s.batch * s.heads_kv);
  const int threads = rows ? 256 : 64;
  switch (hi_bits_of(s)) {
    case 8: return launch_chained(hi_quant_kernel<8>, grid, dim3(threads), 0, st, a);
    case 4: return launch_chained(hi_quant_kernel<4>, grid, dim3(threads), 0, st, a);
    case 2: return launch_chained(hi_quant_kernel<2>, grid, dim3(threads), 0, st, a);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_kch_append(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                              const int32_t* src_tok, int n_src, const int32_t* rows, int n_rows, int p0,
                              cudaStream_t st) {
  KchArgs a = {};
  a.dbg = debug_status_word();
  a.k_src = static_cast<const __nv_bfloat16*>(k_src);
  a.v_src = static_cast<const __nv_bfloat16*>(v_src);
  a.src_tok = src_tok;
  a.rows = rows;
  a.k_hi = static_cast<__nv_bfloat16*>(c.k_hi);
  a.v_hi = static_cast<__nv_bfloat16*>(c.v_hi);
  a.hi_tok = c.hi_tok;
  a.k_codes = static_cast<uint8_t*>(c.k_codes);
  a.v_codes = static_cast<uint8_t*>(c.v_codes);
  a.k_params = static_cast<__half2*>(c.k_params);
  a.v_params = static_cast<__half2*>(c.v_params);
  a.lo_tok = c.lo_tok;
  a.heads_kv = s.heads_kv;
  a.hi_cap = s.hi_cap;
  a.hi_stride = s.hi_stride;
  a.lo_cap = s.lo_cap;
  a.n_src = n_src;
  a.n_rows = n_rows;
  a.p0 = p0;  // positions < p0 come from staging
  a.p_end = p0 + n_rows;
  const int bh = s.batch * s.heads_kv;
  // groups completed by this append: j0 = first group touched .. (p_end / 64) - 1; with no new rows, the
  // caller asks for the group that ends at p0 (all of it staged)
  const int j0 = n_rows > 0 ? p0 / kKchGroup : p0 / kKchGroup - 1;
  const int j1 = n_rows > 0 ? a.p_end / kKchGroup : p0 / kKchGroup;
  a.g0 = j0;
  if (j1 > j0) {
    cudaError_t e;
    const dim3 grid(j1 - j0, bh);
    switch (s.bits) {
      case 2: e = kch_group_launch<2>(a, s.group, grid, st); break;
      case 3: e = kch_group_launch<3>(a, s.group, grid, st); break;
      case 4: e = kch_group_launch<4>(a, s.group, grid, st); break;
      default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
  }
  if (n_rows > 0 && a.p_end % kKchGroup != 0) {  // the incomplete last group waits in staging
    kch_stage_kernel<<<bh, kKchThreads, 0, st>>>(a);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

cudaError_t launch_balancer(const mikv_shape& s, const void* q_pre, const void* k_pre, int T, float* out,
                            uint32_t* ws_max, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(ws_max, 0, sizeof(uint32_t) * 2 * s.heads_kv * kHeadDim, st);
  if (e != cudaSuccess) return e;
  const int chunk = 256;
  const dim3 grid((T + chunk - 1) / chunk, s.batch * (s.heads_q + s.heads_kv));
  absmax_kernel<<<grid, kHeadDim, 0, st>>>(static_cast<const __nv_bfloat16*>(q_pre),
                                           static_cast<const __nv_bfloat16*>(k_pre), s.batch, s.heads_q,
                                           s.heads_kv, T, chunk, ws_max);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  balancer_kernel<<<s.heads_kv, kHeadDim, 0, st>>>(ws_max, s.heads_kv, out);
  return cudaGetLastError();
}

}  // namespace mikv
