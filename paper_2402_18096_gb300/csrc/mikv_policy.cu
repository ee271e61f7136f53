// mikv_policy.cu — the importance policy around the attention kernel (arxiv 2402.18096, Fig. 4 and
// Sec. 3): accumulated-attention (heavy-hitter) score update, choice of the tokens that leave the
// important set, insertion of the new token and the important-set build from prefill rows.
#include "mikv_device.cuh"
#include "mikv_internal.h"
#include "mikv_rows.cuh"

namespace mikv {
namespace {

// acc[b][h][i] += sum over the G query heads j of exp(s_ji - m_j) / l_j.
__global__ void __launch_bounds__(128) update_importance_kernel(float* acc, const float* hi_logits,
                                                                 const float* ml, int Hq, int Hkv,
                                                                 int hi_cap, int hi_stride) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int bh = blockIdx.y;
  if (i >= hi_cap) return;
  const int G = Hq / Hkv, b = bh / Hkv, h = bh - b * Hkv;
  float add = 0.f;
  for (int j = 0; j < G; ++j) {
    const int bq = b * Hq + h * G + j;
    add += importance_weight(hi_logits[(size_t)bq * hi_stride + i], ml[2 * bq], 1.f / ml[2 * bq + 1]);
  }
  acc[(size_t)bh * hi_stride + i] += add;
}

constexpr int kSelThreads = 1024;

// Block-wide exclusive scan of one int per thread; returns the prefix and writes the total.
__device__ int block_exclusive_scan(int v, int* total, int* sh) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) sh[w] = x;
  __syncthreads();
  if (w == 0) {
    int z = lane < (kSelThreads / 32) ? sh[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, z, off);
      if (lane >= off) z += y;
    }
    sh[32 + lane] = z;  // inclusive prefix of warp totals
  }
  __syncthreads();
  const int before = (w > 0 ? sh[32 + w - 1] : 0) + x - v;
  *total = sh[32 + kSelThreads / 32 - 1];
  __syncthreads();
  return before;
}

// One block per (b, h): the n_demote smallest keys leave; both lists come out in ascending index order.
__global__ void __launch_bounds__(kSelThreads) select_kernel(const float* scores, const int32_t* ids, int n,
                                                             int stride, int n_demote, int32_t* demoted,
                                                             int32_t* kept) {
  __shared__ unsigned int hist[256];
  __shared__ int sh[64];
  __shared__ unsigned long long s_best[kSelThreads / 32];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_rank;
  const int bh = blockIdx.x, tid = threadIdx.x;
  const float* sc = scores + (size_t)bh * stride;
  const int32_t* id = ids ? ids + (size_t)bh * stride : nullptr;
  int32_t* dem = demoted + (size_t)bh * n_demote;
  int32_t* kep = kept ? kept + (size_t)bh * (n - n_demote) : nullptr;

  unsigned long long thresh;  // largest key that is demoted
  if (n_demote == 0) {
    thresh = 0ull;  // nothing demoted (keys are never 0: the top bit of a score key is set or ~)
  } else if (n_demote == n) {
    thresh = ~0ull;
  } else if (n_demote == 1) {
    unsigned long long best = ~0ull;
    for (int i = tid; i < n; i += kSelThreads) {
      const unsigned long long k = order_key(sc[i], id ? id[i] : i);
      best = k < best ? k : best;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
      best = o < best ? o : best;
    }
    if ((tid & 31) == 0) s_best[tid >> 5] = best;
    __syncthreads();
    if (tid < 32) {
      best = tid < kSelThreads / 32 ? s_best[tid] : ~0ull;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
        best = o < best ? o : best;
      }
      if (tid == 0) s_prefix = best;
    }
    __syncthreads();
    thresh = s_prefix;
  } else {
    // Radix select of the key of rank n_demote - 1, 8 bits per pass from the top.
    unsigned long long prefix = 0ull;
    int rank = n_demote - 1;
    for (int pass = 0; pass < 8; ++pass) {
      const int shift = 56 - 8 * pass;
      const unsigned long long hi_mask = pass == 0 ? 0ull : (~0ull << (shift + 8));
      for (int i = tid; i < 256; i += kSelThreads) hist[i] = 0u;
      __syncthreads();
      for (int i = tid; i < n; i += kSelThreads) {
        const unsigned long long k = order_key(sc[i], id ? id[i] : i);
        if ((k & hi_mask) == prefix) atomicAdd(&hist[(k >> shift) & 0xffu], 1u);
      }
      __syncthreads();
      if (tid == 0) {
        int acc = 0, dgt = 0;
        for (; dgt < 256; ++dgt) {
          if (acc + (int)hist[dgt] > rank) break;
          acc += (int)hist[dgt];
        }
        s_prefix = prefix | ((unsigned long long)dgt << shift);
        s_rank = rank - acc;
      }
      __syncthreads();
      prefix = s_prefix;
      rank = s_rank;
      __syncthreads();
    }
    thresh = prefix;
  }

  // Ascending-index compaction: thread tid owns indices [tid * per, (tid + 1) * per).
  const int per = (n + kSelThreads - 1) / kSelThreads;
  const int i0 = tid * per, i1 = min(n, i0 + per);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += order_key(sc[i], id ? id[i] : i) <= thresh && n_demote > 0;
  int total;
  int pos = block_exclusive_scan(cnt, &total, sh);
  int kpos = i0 - pos;
  for (int i = i0; i < i1; ++i) {
    const bool d = n_demote > 0 && order_key(sc[i], id ? id[i] : i) <= thresh;
    if (d) {
      if (pos < n_demote) dem[pos] = i;
      ++pos;
    } else {
      if (kep && kpos < n - n_demote) kep[kpos] = i;
      ++kpos;
    }
  }
}

__global__ void __launch_bounds__(64) insert_kernel(__nv_bfloat16* k_hi, __nv_bfloat16* v_hi, int32_t* hi_tok,
                                                    float* acc, const __nv_bfloat16* k_new,
                                                    const __nv_bfloat16* v_new, int tok, const int32_t* slots,
                                                    int hi_cap, int hi_stride, int* dbg) {
  const int bh = blockIdx.x, tid = threadIdx.x;
  grid_dependency_wait();  // the slot comes from the previous step's tail
  allow_dependent_launch();
  const int s = slots[bh];
  if (s < 0 || s >= hi_cap) {  // an out-of-range slot is skipped (recorded in debug builds)
    if (tid == 0) MIKV_BOUNDS_FAIL(dbg);
    return;
  }
  const size_t row = (size_t)bh * hi_stride + s;
  if (tid < 32) {
    reinterpret_cast<uint2*>(k_hi + row * kHeadDim)[tid] =
        reinterpret_cast<const uint2*>(k_new + (size_t)bh * kHeadDim)[tid];
  } else {
    reinterpret_cast<uint2*>(v_hi + row * kHeadDim)[tid - 32] =
        reinterpret_cast<const uint2*>(v_new + (size_t)bh * kHeadDim)[tid - 32];
  }
  if (tid == 0) {
    hi_tok[row] = tok;
    acc[row] = 0.f;
  }
}

__global__ void __launch_bounds__(256) gather_kernel(__nv_bfloat16* k_hi, __nv_bfloat16* v_hi, int32_t* hi_tok,
                                                     float* acc, const __nv_bfloat16* k_src,
                                                     const __nv_bfloat16* v_src, const int32_t* src_tok,
                                                     const float* src_scores, int n_src, const int32_t* rows,
                                                     int n_rows, int hi_stride, int* dbg) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + w, bh = blockIdx.y;
  if (i >= n_rows) return;
  const int r = rows[(size_t)bh * n_rows + i];
  if (r < 0 || r >= n_src) {  // an out-of-range source row is skipped (recorded in debug builds)
    if (lane == 0) MIKV_BOUNDS_FAIL(dbg);
    return;
  }
  const size_t src = ((size_t)bh * n_src + r) * kHeadDim, dst = ((size_t)bh * hi_stride + i) * kHeadDim;
  reinterpret_cast<uint2*>(k_hi + dst)[lane] = reinterpret_cast<const uint2*>(k_src + src)[lane];
  reinterpret_cast<uint2*>(v_hi + dst)[lane] = reinterpret_cast<const uint2*>(v_src + src)[lane];
  if (lane == 0) {
    hi_tok[(size_t)bh * hi_stride + i] = src_tok ? src_tok[(size_t)bh * n_src + r] : r;
    acc[(size_t)bh * hi_stride + i] = src_scores ? src_scores[(size_t)bh * n_src + r] : 0.f;
  }
}

}  // namespace

cudaError_t launch_update_importance(const mikv_shape& s, const mikv_cache& c, const float* hi_logits,
                                     const float* ml, cudaStream_t st) {
  const dim3 grid((s.hi_cap + 127) / 128, s.batch * s.heads_kv);
  update_importance_kernel<<<grid, 128, 0, st>>>(c.acc, hi_logits, ml, s.heads_q, s.heads_kv, s.hi_cap,
                                                 s.hi_stride);
  return cudaGetLastError();
}

cudaError_t launch_select(int batch, int heads, const float* scores, const int32_t* ids, int n, int stride,
                          int n_demote, int32_t* demoted, int32_t* kept, cudaStream_t st) {
  select_kernel<<<batch * heads, kSelThreads, 0, st>>>(scores, ids, n, stride, n_demote, demoted, kept);
  return cudaGetLastError();
}

cudaError_t launch_insert(const mikv_shape& s, const mikv_cache& c, const void* k_new, const void* v_new,
                          int tok, const int32_t* slots, cudaStream_t st) {
  if (hi_bits_of(s) != 16)
    return launch_hi_quant(s, c, k_new, v_new, nullptr, nullptr, 0, nullptr, 0, slots, tok, st);
  return launch_chained(insert_kernel, dim3(s.batch * s.heads_kv), dim3(64), 0, st,
                        static_cast<__nv_bfloat16*>(c.k_hi), static_cast<__nv_bfloat16*>(c.v_hi), c.hi_tok, c.acc,
                        static_cast<const __nv_bfloat16*>(k_new), static_cast<const __nv_bfloat16*>(v_new), tok, slots,
                        s.hi_cap, s.hi_stride, debug_status_word());
}

cudaError_t launch_gather(const mikv_shape& s, const mikv_cache& c, const void* k_src, const void* v_src,
                          const int32_t* src_tok, const float* src_scores, int n_src, const int32_t* rows,
                          int n_rows, cudaStream_t st) {
  if (n_rows == 0) return cudaSuccess;
  if (hi_bits_of(s) != 16)
    return launch_hi_quant(s, c, k_src, v_src, src_tok, src_scores, n_src, rows, n_rows, nullptr, 0, st);
  const dim3 grid((n_rows + 7) / 8, s.batch * s.heads_kv);
  gather_kernel<<<grid, 256, 0, st>>>(static_cast<__nv_bfloat16*>(c.k_hi), static_cast<__nv_bfloat16*>(c.v_hi),
                                      c.hi_tok, c.acc, static_cast<const __nv_bfloat16*>(k_src),
                                      static_cast<const __nv_bfloat16*>(v_src), src_tok, src_scores, n_src, rows,
                                      n_rows, s.hi_stride, debug_status_word());
  return cudaGetLastError();
}

}  // namespace mikv
