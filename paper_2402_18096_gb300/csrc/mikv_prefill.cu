// mikv_prefill.cu — initial importance of the prefill tokens (sm_103a): the attention each token receives
// from the prefill's causal attention, summed over the queries and over the G query heads of its KV head
// (the accumulated-attention, heavy-hitter score MiKV uses to choose the important set, Fig. 4 / Sec. 3 of
// arxiv 2402.18096).
//
// Two passes over the causal score matrix S = sm_scale * Q K^T, each a tiled bf16 contraction on the tensor
// cores (mma.sync m16n8k16, fp32 accumulation) fed by TMA:
//   1. rows:    per query i, m_i = max_{t <= i} s_it and l_i = sum_{t <= i} exp(s_it - m_i)  (online, as in
//               flash attention, without values);
//   2. columns: per key t, sum over the G query heads and the queries i >= t of exp(s_it - m_i) / l_i.
// A CTA of four warps owns one 64-token tile of its fixed operand (queries in pass 1, keys in pass 2) held in
// registers as MMA A fragments (16 rows per warp), and streams the 64-token tiles of the other operand
// through a double-buffered shared-memory ring (128B-swizzled TMA boxes, one mbarrier per buffer, every
// wait bounded in time). Only the causal triangle is visited.
#include <math.h>

#include "mikv_device.cuh"
#include "mikv_prefill.h"

namespace mikv {
namespace {

constexpr int kPfWarps = 4;
constexpr int kPfThreads = 32 * kPfWarps;
constexpr int kPfTileBytes = kPfTile * kHeadDim * 2;  // 16 KB: two boxes of 64 rows x 128 B
constexpr int kPfHalf = kPfTile * 128;                 // bytes of one 64-channel box
constexpr int kPfSmem = 3 * kPfTileBytes + 64 + 1024;  // fixed tile, two ring buffers, barriers, alignment

__device__ __forceinline__ void pf_fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// One 64 x 128 tile (rows row0 .. row0 + 63 of a map) into dst: two 64-channel boxes.
__device__ __forceinline__ void pf_issue(const CUtensorMap* map, int row0, uint32_t dst, uint32_t bar) {
  mbar_arrive_expect_tx(bar, kPfTileBytes);
  tma_load_2d(dst, map, 0, row0, bar);
  tma_load_2d(dst + kPfHalf, map, 64, row0, bar);
}

// A fragments (16 rows x 128 channels) of rows r0 .. r0 + 15 of a staged tile: a[ks] covers channels
// 16 ks .. 16 ks + 15 (ldmatrix from the 128B-swizzled boxes: 16-byte chunk c of row r sits at c ^ (r & 7)).
__device__ __forceinline__ void pf_load_a(uint32_t tile, int r0, int lane, uint32_t (&a)[8][4]) {
  const int row = r0 + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int chunk = 2 * (ks & 3) + (lane >> 4);
    ldsm_x4(tile + (ks >> 2) * kPfHalf + row * 128 + ((chunk ^ (row & 7)) << 4), a[ks]);
  }
}

// c = A (16 rows) x B^T for tile rows 8 nt .. 8 nt + 7 as the 8 columns: c[0], c[1] = row g, columns
// 2t, 2t+1; c[2], c[3] = row g + 8. B fragments come from the tile rows (K-major) with ldmatrix.
__device__ __forceinline__ void pf_tile_s(const uint32_t (&a)[8][4], uint32_t tile, int nt, int lane,
                                          float (&c)[4]) {
  c[0] = c[1] = c[2] = c[3] = 0.f;
  const int row = 8 * nt + (lane & 7), j = lane >> 3;
#pragma unroll
  for (int kp = 0; kp < 4; ++kp) {  // k-steps 2 kp and 2 kp + 1: four consecutive 16-byte chunks
    const int ks = 2 * kp;
    const int chunk = 2 * (ks & 3) + j;
    uint32_t b[4];
    ldsm_x4(tile + (ks >> 2) * kPfHalf + row * 128 + ((chunk ^ (row & 7)) << 4), b);
    mma_bf16(c, a[ks], b[0], b[1]);
    mma_bf16(c, a[ks + 1], b[2], b[3]);
  }
}

struct PfRing {
  uint32_t fixed, buf0, bar_fixed, bar0;
  __device__ uint32_t buf(int s) const { return buf0 + s * kPfTileBytes; }
  __device__ uint32_t bar(int s) const { return bar0 + 8 * s; }
};

__device__ __forceinline__ PfRing pf_ring() {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
  PfRing r;
  r.fixed = base;
  r.buf0 = base + kPfTileBytes;
  r.bar_fixed = base + 3 * kPfTileBytes;
  r.bar0 = r.bar_fixed + 8;
  return r;
}

// Waits (bounded) for the tiles still in flight into the ring after a failed wait, so that no copy
// outlives the CTA; n_next = the tile whose wait failed (or the first not yet waited for), n_end = tiles
// issued.
__device__ __forceinline__ void pf_drain(const PfRing& r, int n_next, int n_end, int* status) {
  for (int n = n_next; n < n_end; ++n)
    if (!mbar_wait(r.bar(n & 1), (n >> 1) & 1)) record_error(status, kErrDrainTimeout);
}

// ------------------------------------------------------------------------------- pass 1: row statistics

__global__ void __launch_bounds__(kPfThreads) prefill_rows_kernel(const __grid_constant__ PrefillArgs a) {
  __shared__ int s_fail;
  const PfRing ring = pf_ring();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int nq = (a.T + kPfTile - 1) / kPfTile;
  const int qt = nq - 1 - (int)blockIdx.x;  // the longest rows first
  const int bq = blockIdx.y;                // b * Hq + query head
  const int G = a.heads_q / a.heads_kv;
  const int b = bq / a.heads_q, h = (bq - b * a.heads_q) / G;
  const int krow0 = (b * a.heads_kv + h) * a.T;
  const int nk = qt + 1;  // key tiles 0 .. qt: the causal triangle
  if (tid == 0) {
    s_fail = 0;
    mbar_init(ring.bar_fixed, 1);
    mbar_init(ring.bar(0), 1);
    mbar_init(ring.bar(1), 1);
    fence_mbar_init();
    pf_issue(&a.map_q, bq * a.T + kPfTile * qt, ring.fixed, ring.bar_fixed);
    for (int n = 0; n < 2 && n < nk; ++n) pf_issue(&a.map_k, krow0 + kPfTile * n, ring.buf(n), ring.bar(n));
  }
  __syncthreads();
  if (!mbar_wait(ring.bar_fixed, 0)) s_fail = 1;
  __syncthreads();
  int n = 0;
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  const int q0 = kPfTile * qt + 16 * warp + g;  // this thread's query rows q0, q0 + 8
  if (!s_fail) {
    uint32_t qa[8][4];
    pf_load_a(ring.fixed, 16 * warp, lane, qa);
    for (; n < nk; ++n) {
      const int s = n & 1;
      if (!mbar_wait(ring.bar(s), (n >> 1) & 1)) s_fail = 1;
      __syncthreads();
      if (s_fail) break;
      float v[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        pf_tile_s(qa, ring.buf(s), nt, lane, v[nt]);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kPfTile * n + 8 * nt + 2 * t + (e & 1);
          const int q = q0 + 8 * (e >> 1);
          v[nt][e] = (key <= q && key < a.T) ? v[nt][e] * a.scale_log2 : -INFINITY;
        }
      }
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        float mx = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) mx = fmaxf(mx, fmaxf(v[nt][2 * r], v[nt][2 * r + 1]));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float mn = fmaxf(m[r], mx);
        if (mn == -INFINITY) continue;  // no key of this row yet
        float sum = 0.f;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) sum += fast_exp2(v[nt][2 * r] - mn) + fast_exp2(v[nt][2 * r + 1] - mn);
        l[r] = l[r] * fast_exp2(m[r] - mn) + sum;
        m[r] = mn;
      }
      __syncthreads();  // every warp is done with this buffer
      if (tid == 0 && n + 2 < nk) {
        pf_fence_proxy_async();
        pf_issue(&a.map_k, krow0 + kPfTile * (n + 2), ring.buf(s), ring.bar(s));
      }
    }
  }
  if (s_fail) {
    if (tid == 0) {
      record_error(a.status, kErrFullTimeout);
      if (!mbar_wait(ring.bar_fixed, 0)) record_error(a.status, kErrDrainTimeout);
      pf_drain(ring, n, nk < n + 2 ? nk : n + 2, a.status);
    }
    return;
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l[r] += __shfl_xor_sync(0xffffffffu, l[r], 1);
    l[r] += __shfl_xor_sync(0xffffffffu, l[r], 2);
    const int q = q0 + 8 * r;
    if (t == 0 && q < a.T) a.stats[(size_t)bq * a.T + q] = make_float2(m[r], 1.f / l[r]);
  }
}

// ------------------------------------------------------------------------------ pass 2: column sums

__global__ void __launch_bounds__(kPfThreads) prefill_cols_kernel(const __grid_constant__ PrefillArgs a) {
  __shared__ int s_fail;
  __shared__ float2 s_stat[2][kPfTile];
  const PfRing ring = pf_ring();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int nq = (a.T + kPfTile - 1) / kPfTile;
  const int kt = blockIdx.x;  // the keys with the most queries first
  const int bh = blockIdx.y;  // b * Hkv + KV head
  const int G = a.heads_q / a.heads_kv;
  const int b = bh / a.heads_kv, h = bh - b * a.heads_kv;
  const int per_head = nq - kt;  // query tiles kt .. nq - 1 of each query head
  const int n_tiles = G * per_head;
  // query tile n: head j = n / per_head, tile qt = kt + n % per_head
  auto qrow = [&](int n) {
    const int j = n / per_head, qt = kt + (n - j * per_head);
    return ((b * a.heads_q + h * G + j) * a.T) + kPfTile * qt;  // first row in the q map (and in stats)
  };
  auto qfirst = [&](int n) { return kPfTile * (kt + (n % per_head)); };  // its first query index
  if (tid == 0) {
    s_fail = 0;
    mbar_init(ring.bar_fixed, 1);
    mbar_init(ring.bar(0), 1);
    mbar_init(ring.bar(1), 1);
    fence_mbar_init();
    pf_issue(&a.map_k, bh * a.T + kPfTile * kt, ring.fixed, ring.bar_fixed);
    for (int n = 0; n < 2 && n < n_tiles; ++n) pf_issue(&a.map_q, qrow(n), ring.buf(n), ring.bar(n));
  }
  // statistics of the first query tile (queries past T are never used: zero)
  if (tid < kPfTile) {
    const int q = qfirst(0) + tid;
    s_stat[0][tid] = q < a.T ? a.stats[(size_t)qrow(0) + tid] : make_float2(0.f, 0.f);
  }
  __syncthreads();
  if (!mbar_wait(ring.bar_fixed, 0)) s_fail = 1;
  __syncthreads();
  int n = 0;
  float cs[2] = {0.f, 0.f};
  const int k0 = kPfTile * kt + 16 * warp + g;  // this thread's keys k0, k0 + 8
  if (!s_fail) {
    uint32_t ka[8][4];
    pf_load_a(ring.fixed, 16 * warp, lane, ka);
    for (; n < n_tiles; ++n) {
      const int s = n & 1;
      float2 next = make_float2(0.f, 0.f);  // the next tile's statistics, loaded while this one computes
      if (tid < kPfTile && n + 1 < n_tiles) {
        const int q = qfirst(n + 1) + tid;
        if (q < a.T) next = a.stats[(size_t)qrow(n + 1) + tid];
      }
      if (!mbar_wait(ring.bar(s), (n >> 1) & 1)) s_fail = 1;
      __syncthreads();
      if (s_fail) break;
      const int qf = qfirst(n);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        float c[4];
        pf_tile_s(ka, ring.buf(s), nt, lane, c);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = 8 * nt + 2 * t + (e & 1);
          const int q = qf + col, key = k0 + 8 * (e >> 1);
          const float2 st = s_stat[s][col];
          const float p = fast_exp2(fmaf(c[e], a.scale_log2, -st.x)) * st.y;
          cs[e >> 1] += (q >= key && q < a.T) ? p : 0.f;
        }
      }
      if (tid < kPfTile) s_stat[s ^ 1][tid] = next;
      __syncthreads();  // every warp is done with this buffer and its statistics
      if (tid == 0 && n + 2 < n_tiles) {
        pf_fence_proxy_async();
        pf_issue(&a.map_q, qrow(n + 2), ring.buf(s), ring.bar(s));
      }
    }
  }
  if (s_fail) {
    if (tid == 0) {
      record_error(a.status, kErrFullTimeout);
      if (!mbar_wait(ring.bar_fixed, 0)) record_error(a.status, kErrDrainTimeout);
      pf_drain(ring, n, n_tiles < n + 2 ? n_tiles : n + 2, a.status);
    }
    return;
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    cs[r] += __shfl_xor_sync(0xffffffffu, cs[r], 1);
    cs[r] += __shfl_xor_sync(0xffffffffu, cs[r], 2);
    const int key = k0 + 8 * r;
    if (t == 0 && key < a.T) a.scores[(size_t)bh * a.T + key] = cs[r];
  }
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
