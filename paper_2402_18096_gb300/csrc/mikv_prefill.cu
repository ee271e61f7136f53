// mikv_prefill.cu — initial importance of the prefill tokens (sm_103a): the attention each token receives
// from the prefill's causal attention, summed over the queries and over the G query heads of its KV head
// (the accumulated-attention, heavy-hitter score MiKV uses to choose the important set, Fig. 4 / Sec. 3 of
// arxiv 2402.18096).
//
// Two passes over the causal score matrix S = sm_scale * Q K^T, each a tiled bf16 contraction on the
// fifth-generation tensor cores (tcgen05.mma, M = N = 128, fp32 accumulators in tensor memory) fed by TMA:
//   1. rows:    per query i, the log2 of its softmax normaliser, c_i = log2 sum_{t <= i} 2^(s_it log2 e)
//               (accumulated online against a reference, as in flash attention, without values);
//   2. columns: per key t, sum over the G query heads and the queries i >= t of 2^(s_it log2 e - c_i).
// A CTA of four warps owns one 128-token tile of its fixed operand (queries in pass 1, keys in pass 2: the M
// side, so that thread r of the CTA owns accumulator row r = TMEM lane r) and streams the 128-token tiles of
// the other operand through a two-stage shared-memory ring (128B-swizzled TMA boxes). One thread issues the
// eight K = 16 MMAs of a tile into one of two TMEM accumulators while all four warps read the other one with
// tcgen05.ld and do the softmax arithmetic (the exponentials, one per score, bound the kernel). Only the
// causal triangle is visited; every wait is bounded in time.
#include <math.h>

#include "mikv_device.cuh"
#include "mikv_prefill.h"
#include "mikv_tcgen05.cuh"

namespace mikv {
namespace {

constexpr int kPfThreads = 128;                       // thread r <-> accumulator row r (TMEM lane r)
constexpr int kPfHalf = kPfTile * 128;                // bytes of one 64-channel box (128 rows x 128 B)
constexpr int kPfTileBytes = 2 * kPfHalf;             // 32 KB: one 128 x 128 bf16 tile
constexpr int kPfStages = 2;
constexpr int kPfTmemCols = 2 * kPfTile;              // two fp32 accumulators of 128 columns
constexpr int kPfSmem = (1 + kPfStages) * kPfTileBytes + 64 + 1024;  // tiles, barriers, alignment
static_assert(kPfTile == 128, "one accumulator row per thread");

struct PfSmem {
  uint32_t fixed, stage0, bar_fixed, bar_full0, bar_mma0;
  __device__ uint32_t stage(int s) const { return stage0 + s * kPfTileBytes; }
  __device__ uint32_t full(int s) const { return bar_full0 + 8 * s; }
  __device__ uint32_t mma(int d) const { return bar_mma0 + 8 * d; }
};

__device__ __forceinline__ PfSmem pf_smem() {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  PfSmem r;
  r.fixed = base;
  r.stage0 = base + kPfTileBytes;
  r.bar_fixed = base + (1 + kPfStages) * kPfTileBytes;
  r.bar_full0 = r.bar_fixed + 8;
  r.bar_mma0 = r.bar_full0 + 8 * kPfStages;
  return r;
}

// One 128 x 128 tile (rows row0 .. row0 + 127 of a map) into dst: two 64-channel boxes.
__device__ __forceinline__ void pf_issue(const CUtensorMap* map, int row0, uint32_t dst, uint32_t bar) {
  mbar_arrive_expect_tx(bar, kPfTileBytes);
  tma_load_2d(dst, map, 0, row0, bar);
  tma_load_2d(dst + kPfHalf, map, 64, row0, bar);
}

// The eight K = 16 MMAs of one tile: D = A (fixed tile) x B (staged tile)^T over the 128 channels.
__device__ __forceinline__ void pf_mma_tile(uint32_t d_tmem, uint32_t a_tile, uint32_t b_tile) {
  constexpr uint32_t idesc = umma_idesc_bf16_f32(kPfTile, kPfTile);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const uint32_t off = (ks >> 2) * kPfHalf + (ks & 3) * 32;  // channels 16 ks .. 16 ks + 15
    umma_bf16(d_tmem, umma_desc_sw128(a_tile + off), umma_desc_sw128(b_tile + off), idesc, ks > 0 ? 1u : 0u);
  }
}

// This thread's accumulator row (128 fp32 columns) of buffer d.
__device__ __forceinline__ void pf_load_row(uint32_t tmem, int d, int warp, float (&v)[kPfTile]) {
  const uint32_t t = tmem + (uint32_t)(d * kPfTile) + ((uint32_t)(32 * warp) << 16);
  tmem_ld32(t, v);
  tmem_ld32(t + 32, v + 32);
  tmem_ld32(t + 64, v + 64);
  tmem_ld32(t + 96, v + 96);
  tmem_wait_ld(v);
  reg_fence(v + 32);
  reg_fence(v + 64);
  reg_fence(v + 96);
}

// The tile loop shared by both passes. Tile n's operand rows come from b_row(n); its accumulator, once the
// MMAs are done, goes to epi(n, v). Returns false when a wait timed out (after draining what is in flight).
template <class BRow, class Epi>
__device__ __forceinline__ bool pf_tiles(const PrefillArgs& a, const CUtensorMap* map_a, int a_row,
                                         const CUtensorMap* map_b, int n_tiles, BRow b_row, Epi epi) {
  __shared__ uint32_t s_tmem;
  __shared__ int s_fail;
  const PfSmem sm = pf_smem();
  const int tid = threadIdx.x, warp = tid >> 5;
  int issued_tma = 0, issued_mma = 0;  // tiles whose copies / MMAs were issued (thread 0)
  if (tid == 0) {
    s_fail = 0;
    mbar_init(sm.bar_fixed, 1);
    for (int s = 0; s < kPfStages; ++s) mbar_init(sm.full(s), 1);
    for (int d = 0; d < 2; ++d) mbar_init(sm.mma(d), 1);
    fence_mbar_init();
    pf_issue(map_a, a_row, sm.fixed, sm.bar_fixed);
    for (; issued_tma < kPfStages && issued_tma < n_tiles; ++issued_tma)
      pf_issue(map_b, b_row(issued_tma), sm.stage(issued_tma), sm.full(issued_tma));
  }
  __syncwarp();
  if (warp == 0) tmem_alloc(smem_u32(&s_tmem), kPfTmemCols);
  tcgen05_before_sync();
  __syncthreads();
  tcgen05_after_sync();
  const uint32_t tmem = s_tmem;
  bool fixed_ok = true;
  if (tid == 0) {
    fixed_ok = mbar_wait(sm.bar_fixed, 0);
    if (fixed_ok && mbar_wait(sm.full(0), 0)) {
      pf_mma_tile(tmem, sm.fixed, sm.stage(0));
      umma_commit(sm.mma(0));
      issued_mma = 1;
    } else {
      s_fail = 1;
    }
  }
  __syncthreads();
  int n = 0;
  for (; n < n_tiles && !s_fail; ++n) {
    const int d = n & 1;
    // the next tile's MMAs into the other accumulator (its last reader finished before the barrier below)
    if (tid == 0 && n + 1 < n_tiles) {
      const int s1 = (n + 1) % kPfStages;
      if (mbar_wait(sm.full(s1), ((n + 1) / kPfStages) & 1)) {
        tcgen05_after_sync();
        pf_mma_tile(tmem + (uint32_t)((d ^ 1) * kPfTile), sm.fixed, sm.stage(s1));
        umma_commit(sm.mma(d ^ 1));
        issued_mma = n + 2;
      } else {
        s_fail = 1;
      }
    }
    // warp-uniform, so that the warp-wide TMEM loads below run converged
    if (!__all_sync(0xffffffffu, mbar_wait(sm.mma(d), (n >> 1) & 1))) {
      s_fail = 1;
    } else {
      tcgen05_after_sync();
      // tile n's stage is free again (its MMAs have completed): tile n + kPfStages goes there
      if (tid == 0 && issued_tma < n_tiles && issued_tma == n + kPfStages) {
        pf_issue(map_b, b_row(issued_tma), sm.stage(n % kPfStages), sm.full(n % kPfStages));
        ++issued_tma;
      }
      float v[kPfTile];
      pf_load_row(tmem, d, warp, v);
      epi(n, v);
    }
    tcgen05_before_sync();
    __syncthreads();
  }
  const bool failed = s_fail != 0;
  if (failed && tid == 0) {
    record_error(a.status, kErrFullTimeout);
    // no copy and no MMA may outlive the CTA: wait (bounded) for those still in flight
    if (!fixed_ok && !mbar_wait(sm.bar_fixed, 0)) record_error(a.status, kErrDrainTimeout);
    for (int t = issued_mma; t < issued_tma; ++t)
      if (!mbar_wait(sm.full(t % kPfStages), (t / kPfStages) & 1)) record_error(a.status, kErrDrainTimeout);
    for (int t = n; t < issued_mma; ++t)
      if (!mbar_wait(sm.mma(t & 1), (t >> 1) & 1)) record_error(a.status, kErrDrainTimeout);
  }
  tcgen05_before_sync();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tcgen05_after_sync();
    tmem_dealloc(tmem, kPfTmemCols);
  }
  return !failed;
}

// Exact maximum of a row of the tile (four independent chains).
__device__ __forceinline__ float pf_row_max(const float (&v)[kPfTile]) {
  float mx[4] = {v[0], v[1], v[2], v[3]};
#pragma unroll
  for (int j = 4; j < kPfTile; ++j) mx[j & 3] = fmaxf(mx[j & 3], v[j]);
  return fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
}

// sum_j 2^(v_j * scale - ref): the exponent formed two columns at a time, four independent partial sums.
__device__ __forceinline__ float pf_exp_sum(const float (&v)[kPfTile], float scale, float ref) {
  const uint64_t s2 = f32x2(scale, scale), r2 = f32x2(-ref, -ref);
  uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
  for (int j = 0; j < kPfTile / 2; ++j) {
    float x0, x1;
    f32x2_split(fma_f32x2(f32x2(v[2 * j], v[2 * j + 1]), s2, r2), x0, x1);
    acc[j & 3] = add_f32x2(acc[j & 3], f32x2(fast_exp2(x0), fast_exp2(x1)));
  }
  float t[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) f32x2_split(acc[k], t[2 * k], t[2 * k + 1]);
  return ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
}

// ------------------------------------------------------------------------------- pass 1: row statistics
//
// Per query row the softmax normaliser is accumulated against a reference r (log2 units): the exact maximum
// of the row's first tile, raised only when a later tile's sum would leave the fp32 range (a logit more than
// 64 above r, rare), so most tiles need no maximum at all. The pair (r, sum_t 2^(s_t - r)) defines the same
// normaliser as the true maximum; the kernel stores its log2, r + log2(sum).

__global__ void __launch_bounds__(kPfThreads, 2) prefill_rows_kernel(const __grid_constant__ PrefillArgs a) {
  const int tid = threadIdx.x;
  const int nq = (a.T + kPfTile - 1) / kPfTile;
  const int qt = nq - 1 - (int)blockIdx.x;  // the longest rows first
  const int bq = blockIdx.y;                // b * Hq + query head
  const int G = a.heads_q / a.heads_kv;
  const int b = bq / a.heads_q, h = (bq - b * a.heads_q) / G;
  const int krow0 = (b * a.heads_kv + h) * a.T;
  const int q = kPfTile * qt + tid;  // this thread's query
  float r = -INFINITY, l = 0.f;
  const bool ok = pf_tiles(
      a, &a.map_q, bq * a.T + kPfTile * qt, &a.map_k, qt + 1, [&](int n) { return krow0 + kPfTile * n; },
      [&](int n, float (&v)[kPfTile]) {
        const int k0 = kPfTile * n;
        if (n == qt || k0 + kPfTile > a.T) {  // keys after the query, or past the prefill, do not count
#pragma unroll
          for (int j = 0; j < kPfTile; ++j)
            if (k0 + j > q || k0 + j >= a.T) v[j] = -INFINITY;
        }
        if (r == -INFINITY) {  // the row's first tile fixes the reference
          const float mx = pf_row_max(v);
          if (mx == -INFINITY) return;
          r = mx * a.scale_log2;
        }
        float sum = pf_exp_sum(v, a.scale_log2, r);
        if (!(sum <= 0x1p64f)) {  // a logit far above the reference: move the reference to this tile's maximum
          const float rn = fmaxf(r, pf_row_max(v) * a.scale_log2);
          sum = pf_exp_sum(v, a.scale_log2, rn);
          l *= fast_exp2(r - rn);
          r = rn;
        }
        l += sum;
      });
  if (ok) a.stats[(size_t)bq * a.T_pad + q] = q < a.T ? r + log2f(l) : INFINITY;
}

// ------------------------------------------------------------------------------ pass 2: column sums

__global__ void __launch_bounds__(kPfThreads, 2) prefill_cols_kernel(const __grid_constant__ PrefillArgs a) {
  __shared__ __align__(16) float s_nc[2][kPfTile];  // minus the log2 normalisers of the current and next tile
  const int tid = threadIdx.x;
  const int nq = (a.T + kPfTile - 1) / kPfTile;
  const int kt = blockIdx.x;  // the keys with the most queries first
  const int bh = blockIdx.y;  // b * Hkv + KV head
  const int G = a.heads_q / a.heads_kv;
  const int b = bh / a.heads_kv, h = bh - b * a.heads_kv;
  const int per_head = nq - kt;  // query tiles kt .. nq - 1 of each query head
  const int n_tiles = G * per_head;
  // query tile n: head j = n / per_head, tile qt = kt + n % per_head
  auto qhead = [&](int n) { return b * a.heads_q + h * G + n / per_head; };
  auto qfirst = [&](int n) { return kPfTile * (kt + (n % per_head)); };
  auto qrow = [&](int n) { return qhead(n) * a.T + qfirst(n); };  // first row in the q map
  // tile n's query tid (padding queries carry +inf: they weigh nothing)
  auto neg_norm = [&](int n) { return -a.stats[(size_t)qhead(n) * a.T_pad + qfirst(n) + tid]; };
  s_nc[0][tid] = neg_norm(0);  // visible after the first barrier inside pf_tiles
  const int key = kPfTile * kt + tid;  // this thread's key
  float cs = 0.f;
  const bool ok = pf_tiles(
      a, &a.map_k, bh * a.T + kPfTile * kt, &a.map_q, n_tiles, qrow, [&](int n, float (&v)[kPfTile]) {
        const float next = n + 1 < n_tiles ? neg_norm(n + 1) : 0.f;
        const int q0 = qfirst(n);
        if (q0 == kPfTile * kt) {  // the diagonal tile: queries before the key do not attend to it
#pragma unroll
          for (int j = 0; j < kPfTile; ++j)
            if (q0 + j < key) v[j] = -INFINITY;
        }
        const float4* nc = reinterpret_cast<const float4*>(s_nc[n & 1]);
        const uint64_t s2 = f32x2(a.scale_log2, a.scale_log2);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int j = 0; j < kPfTile / 4; ++j) {
          const float4 c = nc[j];
          float x0, x1, x2, x3;
          f32x2_split(fma_f32x2(f32x2(v[4 * j], v[4 * j + 1]), s2, f32x2(c.x, c.y)), x0, x1);
          f32x2_split(fma_f32x2(f32x2(v[4 * j + 2], v[4 * j + 3]), s2, f32x2(c.z, c.w)), x2, x3);
          acc[(2 * j) & 3] = add_f32x2(acc[(2 * j) & 3], f32x2(fast_exp2(x0), fast_exp2(x1)));
          acc[(2 * j + 1) & 3] = add_f32x2(acc[(2 * j + 1) & 3], f32x2(fast_exp2(x2), fast_exp2(x3)));
        }
        float t[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) f32x2_split(acc[k], t[2 * k], t[2 * k + 1]);
        cs += ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
        s_nc[(n + 1) & 1][tid] = next;  // read after the barrier that ends this tile
      });
  if (ok && key < a.T) a.scores[(size_t)bh * a.T + key] = cs;
}

}  // namespace

cudaError_t launch_prefill(const PrefillArgs& a, int batch, cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(prefill_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kPfSmem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(prefill_cols_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kPfSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int nt = (a.T + kPfTile - 1) / kPfTile;
  prefill_rows_kernel<<<dim3(nt, batch * a.heads_q), kPfThreads, kPfSmem, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  prefill_cols_kernel<<<dim3(nt, batch * a.heads_kv), kPfThreads, kPfSmem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace mikv
