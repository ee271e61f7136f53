// mikv_prefill.cu — initial importance of the prefill tokens (sm_103a): the attention each token receives
// from the prefill's causal attention, summed over the queries and over the G query heads of its KV head
// (the accumulated-attention, heavy-hitter score MiKV uses to choose the important set, Fig. 4 / Sec. 3 of
// arxiv 2402.18096).
//
// Two passes over the causal score matrix S = sm_scale * Q K^T, each a tiled bf16 contraction on the
// fifth-generation tensor cores (tcgen05.mma, M = 128, N = 64, fp32 accumulators in tensor memory) fed by TMA:
//   1. rows:    per query i, the log2 of its softmax normaliser, c_i = log2 sum_{t <= i} 2^(s_it log2 e)
//               (accumulated online against a reference, as in flash attention, without values);
//   2. columns: per key t, sum over the G query heads and the queries i >= t of 2^(s_it log2 e - c_i).
// A CTA owns one 128-token tile of its fixed operand (queries in pass 1, keys in pass 2: the M side, so that
// epilogue thread r owns accumulator row r = TMEM lane r) and streams 64-token tiles of the other operand.
// Its warps specialise: warp 8 issues the TMA copies (the fixed tile, then a four-stage ring of 128B-swizzled
// streamed tiles, with pass 2's query normalisers), warp 9 issues the eight K = 16 MMAs of each tile into one
// of four TMEM accumulators, and warps 0-7 (two per accumulator lane quarter, one per column half) read
// their accumulator rows with tcgen05.ld, release them, and do the softmax arithmetic (an exponential per
// score). The roles hand tiles over through mbarriers only; every wait is bounded in time and gives up when
// another role has failed. Only the causal triangle is visited.
#include <math.h>

#include "mikv_device.cuh"
#include "mikv_prefill.h"
#include "mikv_tcgen05.cuh"

namespace mikv {
namespace {

constexpr int kPfN = 64;                                // tokens of a streamed tile (the MMA's N)
constexpr int kPfEpiWarps = 8;                          // two per accumulator lane quarter: one per column half
constexpr int kPfCols = kPfN / 2;                       // accumulator columns of one epilogue thread
constexpr int kPfThreads = 32 * (kPfEpiWarps + 2);      // warps 0-7 epilogue, 8 copies, 9 MMAs
constexpr int kPfCopyWarp = kPfEpiWarps, kPfMmaWarp = kPfEpiWarps + 1;
constexpr int kPfFixBytes = kPfTile * kHeadDim * 2;     // 32 KB: the fixed 128 x 128 bf16 tile
constexpr int kPfFixHalf = kPfTile * 128;               // one 64-channel box of it
constexpr int kPfStrBytes = kPfN * kHeadDim * 2;        // 16 KB: a streamed 64 x 128 tile
constexpr int kPfStrHalf = kPfN * 128;
constexpr int kPfStages = 4;                            // streamed tiles in flight
constexpr int kPfAcc = 4;                               // TMEM accumulators of kPfN columns
constexpr int kPfTmemCols = kPfAcc * kPfN;
constexpr int kPfStatBytes = kPfN * 4;                 // pass 2: the streamed queries' log2 normalisers
constexpr int kPfBars = 1 + 5 * kPfStages + 1;          // fixed, full/free/acc-full/acc-empty/stats x 4, drain
constexpr int kPfSmem = kPfFixBytes + kPfStages * (kPfStrBytes + kPfStatBytes) + 8 * kPfBars + 1024;
static_assert(kPfTile == 128 && kPfStages == kPfAcc, "one accumulator row per epilogue thread; shared indices");

struct PfSmem {
  uint32_t fixed, stage0, stat0, bars;
  const uint8_t* gbase;  // generic address of `fixed`
  __device__ uint32_t stage(int s) const { return stage0 + s * kPfStrBytes; }
  __device__ uint32_t stat(int s) const { return stat0 + s * kPfStatBytes; }
  __device__ const float* stat_ptr(int s) const { return reinterpret_cast<const float*>(gbase + (stat(s) - fixed)); }
  __device__ uint32_t bar_fixed() const { return bars; }
  __device__ uint32_t full(int s) const { return bars + 8 * (1 + s); }                 // copy landed
  __device__ uint32_t sfree(int s) const { return bars + 8 * (1 + kPfStages + s); }    // MMAs read it
  __device__ uint32_t tfull(int d) const { return bars + 8 * (1 + 2 * kPfStages + d); }  // accumulator ready
  __device__ uint32_t tempty(int d) const { return bars + 8 * (1 + 3 * kPfStages + d); } // accumulator read
  __device__ uint32_t sdone(int s) const { return bars + 8 * (1 + 4 * kPfStages + s); }   // stats read
  __device__ uint32_t drain() const { return bars + 8 * (1 + 5 * kPfStages); }
};

__device__ __forceinline__ PfSmem pf_smem() {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  PfSmem r;
  r.fixed = base;
  r.gbase = smem_raw + (base - smem_u32(smem_raw));
  r.stage0 = base + kPfFixBytes;
  r.stat0 = r.stage0 + kPfStages * kPfStrBytes;
  r.bars = r.stat0 + kPfStages * kPfStatBytes;
  return r;
}

// Bounded wait that also gives up as soon as another role of the CTA has failed.
__device__ __forceinline__ bool pf_wait(uint32_t bar, uint32_t parity, volatile int* fail) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0 && (*fail || global_timer_ns() - t0 > kWaitLimitNs)) {
      *fail = 1;
      return false;
    }
  }
}

// The eight K = 16 MMAs of one tile: D (128 x 64) = fixed tile x streamed tile^T over the 128 channels.
__device__ __forceinline__ void pf_mma_tile(uint32_t d_tmem, uint32_t fix, uint32_t str) {
  constexpr uint32_t idesc = umma_idesc_bf16_f32(kPfTile, kPfN);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const uint32_t k = (ks & 3) * 32;  // channels 16 ks .. 16 ks + 15 inside their 64-channel box
    umma_bf16(d_tmem, umma_desc_sw128(fix + (ks >> 2) * kPfFixHalf + k),
              umma_desc_sw128(str + (ks >> 2) * kPfStrHalf + k), idesc, ks > 0 ? 1u : 0u);
  }
}

// The pipeline shared by both passes: warp 8 streams the n_tiles tiles (rows str_row(n) of map_str) behind
// the fixed tile (rows fix_row .. + 127 of map_fix), warp 9 multiplies each into one of four TMEM
// accumulators, and warps 0-7 hand accumulator row halves to epi(n, col0, v): warp w gets row 32 (w % 4) +
// lane, columns col0 = 32 (w / 4) .. col0 + 31. Returns false when a wait timed out (after draining what was
// in flight); every role leaves through the final barrier.
// STATS (pass 2): the copy warp also stages each streamed tile's kPfN query normalisers (stats + stat_off(n),
// 16-byte aligned in the padded rows) with the tile; the epilogue warps release them through sdone.
template <bool STATS, class StrRow, class StatOff, class Epi>
__device__ __forceinline__ bool pf_pipeline(const PrefillArgs& a, const CUtensorMap* map_fix, int fix_row,
                                            const CUtensorMap* map_str, int n_tiles, StrRow str_row,
                                            StatOff stat_off, Epi epi) {
  __shared__ uint32_t s_tmem;
  __shared__ int s_fail;
  volatile int* fail = &s_fail;
  const PfSmem sm = pf_smem();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_fail = 0;
    mbar_init(sm.bar_fixed(), 1);
    for (int s = 0; s < kPfStages; ++s) {
      mbar_init(sm.full(s), 1);
      mbar_init(sm.sfree(s), 1);
      mbar_init(sm.tfull(s), 1);
      mbar_init(sm.tempty(s), kPfEpiWarps);  // one arrival per epilogue warp
      mbar_init(sm.sdone(s), kPfEpiWarps);
    }
    mbar_init(sm.drain(), 1);
    fence_mbar_init();
  }
  if (warp == kPfMmaWarp) tmem_alloc(smem_u32(&s_tmem), kPfTmemCols);
  tcgen05_before_sync();
  __syncthreads();
  tcgen05_after_sync();
  const uint32_t tmem = s_tmem;

  if (warp == kPfCopyWarp) {
    if (lane == 0) {  // copies: the fixed tile, then the streamed tiles as stages free up
      int last[kPfStages];
      for (int s = 0; s < kPfStages; ++s) last[s] = -1;
      mbar_arrive_expect_tx(sm.bar_fixed(), kPfFixBytes);
      tma_load_2d(sm.fixed, map_fix, 0, fix_row, sm.bar_fixed());
      tma_load_2d(sm.fixed + kPfFixHalf, map_fix, 64, fix_row, sm.bar_fixed());
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % kPfStages;
        const uint32_t ph = ((t / kPfStages) & 1) ^ 1;
        if (t >= kPfStages && !pf_wait(sm.sfree(s), ph, fail)) break;
        if (STATS && t >= kPfStages && !pf_wait(sm.sdone(s), ph, fail)) break;
        const int row = str_row(t);
        mbar_arrive_expect_tx(sm.full(s), kPfStrBytes + (STATS ? kPfStatBytes : 0));
        tma_load_2d(sm.stage(s), map_str, 0, row, sm.full(s));
        tma_load_2d(sm.stage(s) + kPfStrHalf, map_str, 64, row, sm.full(s));
        if (STATS) bulk_load(sm.stat(s), a.stats + stat_off(t), kPfStatBytes, sm.full(s));
        last[s] = t;
      }
      if (*fail) {  // no copy may outlive the CTA
        if (!mbar_wait(sm.bar_fixed(), 0)) record_error(a.status, kErrDrainTimeout);
        for (int s = 0; s < kPfStages; ++s)
          if (last[s] >= 0 && !mbar_wait(sm.full(s), (last[s] / kPfStages) & 1))
            record_error(a.status, kErrDrainTimeout);
      }
    }
  } else if (warp == kPfMmaWarp) {
    if (lane == 0) {  // MMAs: tile n into accumulator n % 4 once its copy landed and its last reader is done
      if (pf_wait(sm.bar_fixed(), 0, fail)) {
        for (int n = 0; n < n_tiles; ++n) {
          const int s = n % kPfStages;
          const uint32_t ph = (n / kPfStages) & 1;
          if (!pf_wait(sm.full(s), ph, fail) || !pf_wait(sm.tempty(s), ph ^ 1, fail)) break;
          tcgen05_after_sync();
          pf_mma_tile(tmem + (uint32_t)(s * kPfN), sm.fixed, sm.stage(s));
          umma_commit(sm.sfree(s));
          umma_commit(sm.tfull(s));
        }
      }
      umma_commit(sm.drain());  // every MMA issued has completed once this arrives
      if (!mbar_wait(sm.drain(), 0)) record_error(a.status, kErrDrainTimeout);
    }
  } else {  // epilogue warps: accumulator lanes 32 (w % 4) .., columns kPfCols (w / 4) ..
    const int half = warp / 4;
    for (int n = 0; n < n_tiles; ++n) {
      const int d = n % kPfAcc;
      const bool ok = pf_wait(sm.tfull(d), (n / kPfAcc) & 1, fail);
      if (!__all_sync(0xffffffffu, ok)) {
        *fail = 1;
        break;
      }
      tcgen05_after_sync();
      float v[kPfCols];
      tmem_ld32(tmem + (uint32_t)(d * kPfN + kPfCols * half) + ((uint32_t)(32 * (warp & 3)) << 16), v);
      tmem_wait_ld(v);
      tcgen05_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(sm.tempty(d));
      // the staged normalisers: observe their copy's completion directly (it has completed: the MMAs
      // that produced this accumulator waited for it, and the stage is not refilled before sdone)
      if (STATS && !__all_sync(0xffffffffu, pf_wait(sm.full(d), (n / kPfStages) & 1, fail))) {
        *fail = 1;
        break;
      }
      epi(n, kPfCols * half, v, sm.stat_ptr(d) + kPfCols * half);
      if (STATS) {
        __syncwarp();
        if (lane == 0) mbar_arrive(sm.sdone(d));
      }
    }
  }
  tcgen05_before_sync();
  __syncthreads();
  const bool failed = s_fail != 0;
  if (failed && tid == 0) record_error(a.status, kErrFullTimeout);
  if (warp == kPfMmaWarp) {
    __syncwarp();
    tcgen05_after_sync();
    tmem_dealloc(tmem, kPfTmemCols);
  }
  return !failed;
}

// Exact maximum of a row of the tile (four independent chains).
__device__ __forceinline__ float pf_row_max(const float (&v)[kPfCols]) {
  float mx[4] = {v[0], v[1], v[2], v[3]};
#pragma unroll
  for (int j = 4; j < kPfCols; ++j) mx[j & 3] = fmaxf(mx[j & 3], v[j]);
  return fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
}

// sum_j 2^(v_j * scale - ref): the exponent formed two columns at a time, four independent partial sums.
__device__ __forceinline__ float pf_exp_sum(const float (&v)[kPfCols], float scale, float ref) {
  const uint64_t s2 = f32x2(scale, scale), r2 = f32x2(-ref, -ref);
  uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
  for (int j = 0; j < kPfCols / 2; ++j) {
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
  __shared__ float s_r[kPfTile], s_l[kPfTile];  // the second column half's partial of each row
  const int row = tid & (kPfTile - 1);
  const int q = kPfTile * qt + row;  // an epilogue thread's query
  const int kend = min(kPfTile * (qt + 1), a.T);  // keys 0 .. kend - 1 can reach this tile's queries
  float r = -INFINITY, l = 0.f;  // over this thread's column half of every tile
  const bool ok = pf_pipeline<false>(
      a, &a.map_q, bq * a.T + kPfTile * qt, &a.map_k_str, (kend + kPfN - 1) / kPfN,
      [&](int n) { return krow0 + kPfN * n; }, [](int) { return (size_t)0; },
      [&](int n, int col0, float (&v)[kPfCols], const float*) {
        const int k0 = kPfN * n + col0;
        if (k0 + kPfCols > kPfTile * qt) {  // keys after the query, or past the prefill, do not count
#pragma unroll
          for (int j = 0; j < kPfCols; ++j)
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
  if (tid >= kPfTile && tid < 2 * kPfTile) {
    s_r[row] = r;
    s_l[row] = l;
  }
  __syncthreads();
  if (ok && tid < kPfTile) {  // both halves against the larger reference
    const float r2 = s_r[row], rm = fmaxf(r, r2);
    const float lt = (r == -INFINITY ? 0.f : l * fast_exp2(r - rm)) + (r2 == -INFINITY ? 0.f : s_l[row] * fast_exp2(r2 - rm));
    a.stats[(size_t)bq * a.T_pad + q] = q < a.T ? rm + log2f(lt) : INFINITY;
  }
}

// ------------------------------------------------------------------------------ pass 2: column sums

__global__ void __launch_bounds__(kPfThreads, 2) prefill_cols_kernel(const __grid_constant__ PrefillArgs a) {
  const int tid = threadIdx.x;
  const int kt = blockIdx.x;  // the keys with the most queries first
  const int bh = blockIdx.y;  // b * Hkv + KV head
  const int G = a.heads_q / a.heads_kv;
  const int b = bh / a.heads_kv, h = bh - b * a.heads_kv;
  const int per_head = (a.T - kPfTile * kt + kPfN - 1) / kPfN;  // query tiles of each head reaching the keys
  // query tile n: head j = n / per_head, first query kPfTile kt + kPfN (n % per_head)
  auto qhead = [&](int n) { return b * a.heads_q + h * G + n / per_head; };
  auto qfirst = [&](int n) { return kPfTile * kt + kPfN * (n % per_head); };
  __shared__ float s_cs[kPfTile];  // the second column half's sum of each row
  const int row = tid & (kPfTile - 1);
  const int key = kPfTile * kt + row;  // an epilogue thread's key
  float cs = 0.f;
  const bool ok = pf_pipeline<true>(
      a, &a.map_k, bh * a.T + kPfTile * kt, &a.map_q_str, G * per_head,
      [&](int n) { return qhead(n) * a.T + qfirst(n); },
      [&](int n) { return (size_t)qhead(n) * a.T_pad + qfirst(n); },
      [&](int n, int col0, float (&v)[kPfCols], const float* stat) {
        const int q0 = qfirst(n) + col0;
        // the log2 normalisers of these queries, staged with the tile (+inf for padding: they weigh nothing)
        const float4* nc = reinterpret_cast<const float4*>(stat);
        if (q0 < kPfTile * (kt + 1)) {  // the diagonal: queries before the key do not attend to it
#pragma unroll
          for (int j = 0; j < kPfCols; ++j)
            if (q0 + j < key) v[j] = -INFINITY;
        }
        const uint64_t s2 = f32x2(a.scale_log2, a.scale_log2);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int j = 0; j < kPfCols / 4; ++j) {
          const float4 c = nc[j];
          float x0, x1, x2, x3;
          f32x2_split(fma_f32x2(f32x2(v[4 * j], v[4 * j + 1]), s2, f32x2(-c.x, -c.y)), x0, x1);
          f32x2_split(fma_f32x2(f32x2(v[4 * j + 2], v[4 * j + 3]), s2, f32x2(-c.z, -c.w)), x2, x3);
          acc[(2 * j) & 3] = add_f32x2(acc[(2 * j) & 3], f32x2(fast_exp2(x0), fast_exp2(x1)));
          acc[(2 * j + 1) & 3] = add_f32x2(acc[(2 * j + 1) & 3], f32x2(fast_exp2(x2), fast_exp2(x3)));
        }
        float t[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) f32x2_split(acc[k], t[2 * k], t[2 * k + 1]);
        cs += ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
      });
  if (tid >= kPfTile && tid < 2 * kPfTile) s_cs[row] = cs;
  __syncthreads();
  if (ok && tid < kPfTile && key < a.T) a.scores[(size_t)bh * a.T + key] = cs + s_cs[row];
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
