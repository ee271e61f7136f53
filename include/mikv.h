/*
 * mikv.h — C ABI of libmikv: the GB300 (sm_103a) decode hot path of MiKV, the importance-aware
 * mixed-precision KV cache of "No Token Left Behind: Reliable KV Cache Compression via
 * Importance-Aware Mixed Precision Quantization" (arxiv 2402.18096).
 *
 * What the library computes, per attention layer and decode step:
 *   - important KV pairs (chosen by accumulated attention score, the heavy-hitter policy the paper
 *     plugs in, Fig. 4 / Sec. 3) stay in bf16 in the "important set";
 *   - all other KV pairs are kept, not evicted, as N-bit (N = 2, 3, 4) per-token group-wise asymmetric
 *     round-to-nearest codes with fp16 scale/zero (Eq. 1, Sec. 3.1) in the "retained set";
 *   - keys are multiplied by a per-channel balancer before quantization and the query is divided by
 *     it (Eq. 2-4, Sec. 3.2);
 *   - attention treats the two sets as one unordered set (permutation invariance, Sec. 3.4);
 *   - optionally (Sec. 3.3, Table 3) the important set itself is kept at reduced precision: INT8,
 *     INT4 or INT2 codes with fp16 scale/zero per 64 channels, quantized like the retained set.
 *
 * Conventions shared by every entry point:
 *   - All array pointers are DEVICE pointers owned by the caller; the library never allocates,
 *     frees or synchronises. Every call enqueues its kernels on `stream` (a cudaStream_t passed as
 *     void*, NULL = legacy default stream) and returns before they run.
 *   - Arguments are validated on the host before anything is launched; a call that returns an error
 *     has launched nothing (MIKV_ERR_CUDA excepted: a launch was attempted and failed).
 *   - bf16 = IEEE bfloat16, fp16 = IEEE binary16, both stored as 2-byte little-endian values.
 *   - Layouts are dense row-major in the index order written next to each argument.
 *   - The head dimension d is 128; the query-head group size G = heads_q / heads_kv is 1, 2, 4 or 8
 *     (grouped-query attention: query head j reads KV head j / G).
 *   - Each compute entry point (balancer, quantize/pack, prefill scores, attention, importance update,
 *     select/demote, insert, gather, decode step) marks its host time with one NVTX range named after
 *     the call (NVTX v3, header-only: inert unless a tool such as Nsight is attached; a build with
 *     -DMIKV_NVTX=0 leaves the ranges out).
 *
 * Packed-code layout of one retained row (d = 128, N bits, 16 * N bytes): channel c is written
 * c = 16 m + u (u = c mod 16, m = c div 16) and a plane is a sequence of little-endian 16-bit units.
 * In a plane of f-bit fields (f in {2, 4, 8}) with P = 16 / f codes per unit, channel c sits in unit
 * 8 * (2 * (m div P) + (u div 8)) + (u mod 8) at bits [f * (m mod P), f * (m mod P) + f). In a plane of
 * 1-bit fields, channel c sits in unit (u mod 8) at bit 2 * m + (u div 8). N = 2, 4 and 8 use one
 * plane of N-bit fields; N = 3 uses a plane of 2-bit fields (code bits 0..1) followed by a plane of
 * 1-bit fields (code bit 2). The quantization parameters of a row are d / group pairs of fp16
 * (alpha, beta), alpha first; the dequantized value is alpha * code + beta.
 */
#ifndef MIKV_H
#define MIKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MIKV_OK = 0,
  MIKV_ERR_ARG = 1,         /* null pointer, negative or inconsistent size */
  MIKV_ERR_UNSUPPORTED = 2, /* valid but not built: d != 128, bits not in {2,3,4}, ... */
  MIKV_ERR_CAPACITY = 3,    /* a write would pass lo_cap / hi_cap */
  MIKV_ERR_CUDA = 4,        /* a CUDA call failed; cudaGetLastError() was consumed */
  MIKV_ERR_WORKSPACE = 5,   /* workspace missing, too small or misaligned */
  MIKV_ERR_DEVICE = 6,      /* a kernel reported a failure through the workspace status word */
  MIKV_ERR_SCRATCH = 7      /* the problem needs more scratch than mikv_decode_attention_noalloc's
                               built-in buffer holds (MIKV_NOALLOC_SCRATCH_BYTES) */
} mikv_status;

/* Shape of one layer's mixed-precision cache. */
typedef struct {
  int32_t batch;     /* B */
  int32_t heads_q;   /* Hq, query heads */
  int32_t heads_kv;  /* Hkv, KV heads; Hq / Hkv in {1, 2, 4, 8} */
  int32_t head_dim;  /* d, must be 128 */
  int32_t bits;      /* N, retained-set code width: 2, 3 or 4 (Eq. 1); 0 = no retained set: demoted
                        tokens are evicted (the importance-based eviction baseline, H2O, Sec. 2.2 /
                        Fig. 2); the retained arrays are then unused and may be NULL, n_lo must be 0 */
  int32_t group;     /* g, channels per quantization group: 32, 64 or 128 (Sec. 3.2 uses d/2); ignored when bits = 0 */
  int32_t hi_cap;    /* important slots attended per head: the budget k plus one staging slot */
  int32_t hi_stride; /* rows per head in the important-set arrays: multiple of 16, >= hi_cap */
  int32_t lo_cap;    /* rows per head in the retained-set arrays: multiple of 16 */
  int32_t hi_bits;   /* important-set precision: 0 or 16 = bf16; 8, 4 or 2 = codes (Sec. 3.3, Table 3) */
  int32_t hi_group;  /* channels per group of a coded important set: 64 (ignored for bf16) */
  int32_t k_channel_group; /* 0: retained keys per token (Eq. 1, groups of `group` channels, balanced).
                              64: retained keys per CHANNEL over groups of 64 consecutive retained tokens
                              (App. C): one fp16 (alpha, beta) per (token group, channel), no balancer;
                              values stay per token. Retained tokens wait in bf16 in staging rows
                              hi_cap .. hi_cap + 63 of the important arrays until their group of 64 is
                              complete: of n_lo retained tokens, n_lo mod 64 are staged (in order) and
                              the rest quantized. Requires a bf16 important set, hi_stride >= hi_cap + 64
                              and lo_cap % 64 == 0; k_params is then fp16 [B][Hkv][lo_cap / 64][d][2]. */
} mikv_shape;

/* Device arrays of one layer's cache. Rows >= hi_cap of the important arrays are padding and are
 * never read as data; retained rows >= the current length likewise. */
typedef struct {
  void* k_hi;           /* bf16 [B][Hkv][hi_stride][d], keys WITHOUT the balancer; or, for a coded
                           important set, uint8 [B][Hkv][hi_stride][16 * hi_bits] codes of BALANCED keys */
  void* v_hi;           /* bf16 [B][Hkv][hi_stride][d]; or uint8 [B][Hkv][hi_stride][16 * hi_bits] */
  int32_t* hi_tok;      /* int32 [B][Hkv][hi_stride], token position held by each slot */
  float* acc;           /* fp32 [B][Hkv][hi_stride], accumulated attention score per slot */
  void* k_codes;        /* uint8 [B][Hkv][lo_cap][16 * bits], codes of balanced keys (Eq. 3) */
  void* v_codes;        /* uint8 [B][Hkv][lo_cap][16 * bits] */
  void* k_params;       /* fp16 [B][Hkv][lo_cap][d / group][2] (alpha, beta) */
  void* v_params;       /* fp16 [B][Hkv][lo_cap][d / group][2] */
  int32_t* lo_tok;      /* int32 [B][Hkv][lo_cap], token position of each retained row */
  const float* balancer; /* fp32 [Hkv][d] channel balancer of this layer (Eq. 2), or NULL = 1 */
  void* k_hi_params;    /* coded important set only (else unused): fp16 [B][Hkv][hi_stride][d / hi_group][2] */
  void* v_hi_params;    /* coded important set only: fp16 [B][Hkv][hi_stride][d / hi_group][2] */
} mikv_cache;

/* Output element type of mikv_decode_attention. */
enum { MIKV_OUT_BF16 = 0, MIKV_OUT_F32 = 1 };

/* Which operation a workspace is sized for (mikv_workspace_bytes). */
enum { MIKV_WS_ATTENTION = 0, MIKV_WS_BALANCER = 1, MIKV_WS_STEP = 2, MIKV_WS_PREFILL = 3 };

/* Human-readable name of a status code (static string). */
const char* mikv_status_string(mikv_status s);

/* Bytes of workspace `op` needs for `shape` with up to `n_lo_max` retained rows per head (the
 * attention split count depends on it; for MIKV_WS_PREFILL the third argument is the prefill length T). Returns 0 for an invalid shape. The workspace must be
 * 256-byte aligned; its first 16 bytes hold a status word that kernels set on an internal failure. */
size_t mikv_workspace_bytes(const mikv_shape* shape, int32_t op, int32_t n_lo_max);

/* Zero the workspace status word (enqueued on `stream`). */
mikv_status mikv_workspace_reset(void* workspace, size_t ws_bytes, void* stream);

/* Synchronise `stream`, read the workspace status word and return MIKV_ERR_DEVICE if a kernel
 * reported a failure (a wait that ran out of its iteration limit), else MIKV_OK. */
mikv_status mikv_workspace_check(const void* workspace, void* stream);

/*
 * Channel balancer, Eq. 2 (Sec. 3.2): balancer[h][c] = sqrt(max |q_pre| / max |k_pre|), the maxima
 * taken over all batch rows b, prefill tokens t < T and, for the query, the G query heads of KV head h
 * (the balanced keys are shared by those heads). A zero maximum on either side gives 1. fp32 IEEE
 * division and square root (bit-exact with a correctly rounded CPU evaluation).
 *   q_pre   bf16 [B][Hq][T][d] prefill queries (after positional embedding)
 *   k_pre   bf16 [B][Hkv][T][d] prefill keys
 *   balancer_out fp32 [Hkv][d]
 *   workspace >= mikv_workspace_bytes(shape, MIKV_WS_BALANCER, 0)
 */
mikv_status mikv_compute_balancer(const mikv_shape* shape, const void* q_pre, const void* k_pre,
                                  int32_t T, float* balancer_out, void* workspace, size_t ws_bytes,
                                  void* stream);

/*
 * Demotion into the retained set: Eq. 1 quantizer with Eq. 3 key balancing, group-wise per token.
 * For every (b, h) and i < n_rows, source row r = rows[b][h][i] (0 <= r < n_src) is quantized and
 * written to retained row lo_start + i:
 *   keys   x = bf16(k_src[b][h][r][c]) * balancer[h][c]  (fp32 product; balancer NULL => x = k)
 *   values x = bf16(v_src[b][h][r][c])
 *   per group of `group` channels: beta16 = fp16 rounded toward -inf of min(x); alpha16 = fp16 rounded
 *   toward +inf of fp32((max(x) - beta16) / (2^N - 1)) (1.0 when max(x) == beta16); code = clamp(
 *   round-half-even(fp32((x - beta16) / alpha16)), 0, 2^N - 1). Codes are packed as in the header.
 *   lo_tok[b][h][lo_start + i] = src_tok ? src_tok[b][h][r] : r.
 *   k_src, v_src  bf16 [B][Hkv][n_src][d], 16-byte aligned (e.g. the important arrays, n_src = hi_stride)
 *   src_tok       int32 [B][Hkv][n_src] or NULL
 *   rows          int32 [B][Hkv][n_rows]   (device; e.g. the output of mikv_select_demote)
 * Errors: MIKV_ERR_ARG if k_src or v_src is not 16-byte aligned; MIKV_ERR_CAPACITY if lo_start + n_rows >
 * lo_cap. Rows outside [0, n_src) are skipped by the kernel. Codes and parameters are bit-exact with an IEEE fp32 evaluation of the formulas above.
 */
/* With per-channel keys (k_channel_group = 64), mikv_quantize_pack APPENDS the rows at retained positions
 * lo_start .. lo_start + n_rows - 1, lo_start being the current retained length: a position whose group of
 * 64 completes is quantized with its group (keys per channel from the staged rows and the new ones, values
 * per token), the others are copied into the staging rows (bf16, keys unbalanced) with their token ids. */
mikv_status mikv_quantize_pack(const mikv_shape* shape, const mikv_cache* cache, const void* k_src,
                               const void* v_src, const int32_t* src_tok, int32_t n_src,
                               const int32_t* rows, int32_t n_rows, int32_t lo_start, void* stream);

/*
 * Initial importance of the prefill tokens: the accumulated attention each key receives from the prefill's
 * causal attention (the heavy-hitter score of Fig. 4 / Sec. 3, here taken over the prefill queries):
 *   scores[b][h][t] = sum over the G query heads j of KV head h and the queries i >= t of
 *                     exp(s_it - m_i) / l_i,  s_it = sm_scale * q_pre[b][hG+j][i] . k_pre[b][h][t],
 *   m_i = max_{t' <= i} s_it', l_i = sum_{t' <= i} exp(s_it' - m_i)  (the causal softmax of row i).
 * These are the scores mikv_select_demote / mikv_gather_hi take to build the cache. Two tensor-core
 * passes over the causal triangle (row statistics, then column sums), fp32 accumulation.
 *   q_pre      bf16 [B][Hq][T][d], 16-byte aligned (prefill queries after the positional embedding)
 *   k_pre      bf16 [B][Hkv][T][d], 16-byte aligned
 *   scores     fp32 [B][Hkv][T]
 *   workspace  >= mikv_workspace_bytes(shape, MIKV_WS_PREFILL, T) bytes, 256-byte aligned (the row
 *              statistics; its status word reports an internal failure as in the other entry points)
 * Only batch, heads_q, heads_kv and head_dim of `shape` are used. Requires B * Hq * T < 2^31.
 */
mikv_status mikv_prefill_scores(const mikv_shape* shape, const void* q_pre, const void* k_pre, int32_t T,
                                float sm_scale, float* scores, void* workspace, size_t ws_bytes, void* stream);

/*
 * Single-token decode attention over the mixed-precision cache (Eq. 3-4; Sec. 3.4):
 *   s_i = sm_scale * q . k_hi[i]                  for the hi_cap important slots (bf16 keys)
 *   s_t = sm_scale * (q / balancer) . k_hat[t]    for retained rows t < n_lo, k_hat = alpha*code+beta
 *   out = sum_j softmax(s)_j * v_j  over both sets (v_hat = alpha * code + beta for retained rows)
 * A coded important set (hi_bits < 16) is attended like the retained set: s_i = sm_scale *
 * (q / balancer) . k_hat[i] with its own codes and parameters, values dequantized likewise.
 * Split-K flash decoding: partial (max, sum, unnormalised output) per context split in fp32, merged
 * into `out`. Arithmetic: fp32 accumulation; dot products on tensor cores with bf16 (important) or
 * fp16 (retained: dequantized codes, q / balancer) operands.
 *   q          bf16 [B][Hq][d]
 *   out        [B][Hq][d], bf16 (out_dtype MIKV_OUT_BF16) or fp32 (MIKV_OUT_F32)
 *   hi_logits  fp32 [B][Hq][hi_stride] or NULL: s_i of every important slot i < hi_cap
 *   ml         fp32 [B][Hq][2] or NULL: (m = max_j s_j, l = sum_j exp(s_j - m))
 *   workspace  >= mikv_workspace_bytes(shape, MIKV_WS_ATTENTION, n_lo) bytes, 256-byte aligned
 * Requires hi_cap + n_lo >= 1, 0 <= n_lo <= lo_cap. Every important slot < hi_cap must hold a token.
 */
mikv_status mikv_decode_attention(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo,
                                  const void* q, float sm_scale, void* out, int32_t out_dtype,
                                  float* hi_logits, float* ml, void* workspace, size_t ws_bytes,
                                  void* stream);

/*
 * Accumulated-attention importance (heavy-hitter) update: for every (b, h) and slot i < hi_cap,
 *   acc[b][h][i] += sum over the G query heads j of KV head h of exp(s_ji - m_j) / l_j
 * with s from hi_logits and (m, l) from ml as written by mikv_decode_attention. fp32.
 * Retained tokens are not tracked: once demoted a token cannot return to high precision.
 */
mikv_status mikv_update_importance(const mikv_shape* shape, const mikv_cache* cache,
                                   const float* hi_logits, const float* ml, void* stream);

/*
 * Demotion choice: per (b, h), the n_demote least important of n entries, ordered by
 * (score ascending, id ascending) — ties on the score demote the older token first.
 *   scores   fp32 [batch][heads][stride] (entries 0..n-1 are read; e.g. cache->acc with
 *            n = hi_cap and stride = hi_stride); scores must not be NaN
 *   ids      int32 [batch][heads][stride] or NULL (id = entry index); ids must be distinct per head
 *   demoted  int32 [batch][heads][n_demote]: entry indices of the demoted set, ascending
 *   kept     int32 [batch][heads][n - n_demote] or NULL: the remaining entries, ascending
 * Bit-exact: the selected set is fully determined by the order above.
 */
mikv_status mikv_select_demote(int32_t batch, int32_t heads, const float* scores,
                               const int32_t* ids, int32_t n, int32_t stride, int32_t n_demote,
                               int32_t* demoted, int32_t* kept, void* stream);

/*
 * New-token insertion (Fig. 4: the new KV pair enters the important set in high precision):
 * slot s = slots[b][h] (0 <= s < hi_cap) of every (b, h) receives k_new[b][h], v_new[b][h]
 * (bf16 [B][Hkv][d], keys without balancer), hi_tok = tok and acc = 0. With a coded important set
 * (hi_bits < 16) the rows are quantized on the way in (Eq. 1 at hi_bits, groups of hi_group; the key
 * multiplied by the balancer first, Eq. 3), exactly as mikv_quantize_pack quantizes retained rows.
 */
mikv_status mikv_insert_token(const mikv_shape* shape, const mikv_cache* cache, const void* k_new,
                              const void* v_new, int32_t tok, const int32_t* slots, void* stream);

/*
 * Important-set build from prefill rows: important slot i < n_rows of (b, h) receives source row
 * r = rows[b][h][i] of k_src/v_src (bf16 [B][Hkv][n_src][d]), hi_tok = src_tok ? src_tok[b][h][r] : r
 * and acc = src_scores ? src_scores[b][h][r] : 0. Requires n_rows <= hi_cap. A coded important set
 * receives the quantized rows (as in mikv_insert_token).
 */
mikv_status mikv_gather_hi(const mikv_shape* shape, const mikv_cache* cache, const void* k_src,
                           const void* v_src, const int32_t* src_tok, const float* src_scores,
                           int32_t n_src, const int32_t* rows, int32_t n_rows, void* stream);

/*
 * One whole decode step of one layer, in order: insert the new token into slots[b][h]
 * (mikv_insert_token), attend (mikv_decode_attention over hi_cap slots and n_lo retained rows),
 * update the importance scores (mikv_update_importance), choose the least important slot
 * (mikv_select_demote, n_demote = 1) and demote it to retained row n_lo (mikv_quantize_pack).
 * On return slots[b][h] holds the slot freed by the demotion (the next step's insertion slot);
 * the retained length becomes n_lo + 1. With bits = 0 (eviction) nothing is demoted: the victim's slot
 * is freed and the retained length stays 0. A coded important slot is demoted from its dequantized values:
 * per channel the fp32 value alpha * code + beta (rounded once), quantized at bits / group; keys are
 * already balanced and are not multiplied by the balancer again (Sec. 3.3).
 *   q, k_new, v_new   bf16 [B][Hq][d], [B][Hkv][d], [B][Hkv][d]
 *   slots             int32 [B][Hkv], in/out
 *   out               as in mikv_decode_attention
 *   workspace         >= mikv_workspace_bytes(shape, MIKV_WS_STEP, n_lo)
 * Errors: MIKV_ERR_CAPACITY if n_lo + 1 > lo_cap.
 */
mikv_status mikv_decode_step(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo,
                             const void* q, const void* k_new, const void* v_new, int32_t tok,
                             int32_t* slots, float sm_scale, void* out, int32_t out_dtype,
                             void* workspace, size_t ws_bytes, void* stream);

/*
 * Decode attention without a caller-provided workspace and without any allocation (there is no
 * counterpart in the paper; this is a deployment convenience).
 *
 * Some callers cannot allocate device memory on the decode path: an inference engine that owns every
 * byte of device memory through its own pool and forbids plugins from calling the CUDA allocator, or a
 * latency-critical serving loop that must not call cudaMalloc (it can synchronise the device). This
 * entry point computes exactly what mikv_decode_attention computes, with the same arguments minus the
 * workspace, and keeps its split partials in a scratch buffer that the library itself declares as a
 * fixed-size device array of MIKV_NOALLOC_SCRATCH_BYTES bytes. Every GPU that loads the library holds
 * that buffer until the process exits.
 *   - Every call looks up the buffer's device address in the current context (cudaGetSymbolAddress,
 *     which allocates nothing). The first call on a device (in a context) also loads the library's device
 *     code there: make that first call before any stream capture.
 *   - The call itself allocates nothing and frees nothing; it zeroes the buffer's status word on
 *     `stream` before launching.
 *   - All calls share the one buffer, which keeps the last call's contents: calls that can overlap on
 *     the GPU (different streams without ordering between them) race on it and must not be issued.
 *   - A problem whose scratch (mikv_workspace_bytes(shape, MIKV_WS_ATTENTION, n_lo)) exceeds the
 *     buffer returns MIKV_ERR_SCRATCH and launches nothing.
 *   - A kernel-side failure (a wait that ran out of its time limit) is recorded in the buffer's status
 *     word, not in the return code (the call returns before the kernels run): mikv_noalloc_check reads it.
 */
#define MIKV_NOALLOC_SCRATCH_BYTES (8u << 20)
mikv_status mikv_decode_attention_noalloc(const mikv_shape* shape, const mikv_cache* cache, int32_t n_lo,
                                          const void* q, float sm_scale, void* out, int32_t out_dtype,
                                          float* hi_logits, float* ml, void* stream);

/* Status of the built-in buffer of mikv_decode_attention_noalloc: synchronises `stream`, reads the buffer's
 * status word (left by the last mikv_decode_attention_noalloc call, which zeroed it first) and returns
 * MIKV_ERR_DEVICE if a kernel reported a failure, else MIKV_OK. Allocates nothing. */
mikv_status mikv_noalloc_check(void* stream);

/*
 * Debug builds. Every kernel that takes an index from device memory (an insertion slot in `slots`, a source row in
 * `rows`, the victim of a step) skips the access when the index is out of range, without error. A library built
 * with -DMIKV_DEBUG also records each such skip, and the internal invariants of the attention work split, as a
 * failure: in the workspace status word for the entry points with a workspace (read by mikv_workspace_check), and
 * in a status word of its own for mikv_insert_token, mikv_gather_hi and mikv_quantize_pack. No kernel traps.
 *   mikv_debug_enabled  1 if this library was built with -DMIKV_DEBUG, else 0. Host-only.
 *   mikv_debug_check    synchronises `stream`, reads and clears the library's own status word and returns
 *                       MIKV_ERR_DEVICE if an index check failed since the last call, else MIKV_OK (always
 *                       MIKV_OK in release builds).
 */
int32_t mikv_debug_enabled(void);
mikv_status mikv_debug_check(void* stream);

/*
 * KV-cache size as a fraction of an all-fp16 cache (the "Cache size" columns of Tables 2-3): a ratio
 * `ratio` of tokens kept at hi_bits (16 = fp16; otherwise hi_bits-bit codes plus fp16 alpha/beta per
 * group) and the rest at `bits`-bit codes plus fp16 alpha/beta per `group` channels:
 *   ratio * (hi_bits >= 16 ? 1 : (hi_bits + 32/group) / 16) + (1 - ratio) * (bits + 32/group) / 16.
 * Host-only, pure.
 */
double mikv_cache_fraction(int32_t bits, int32_t group, double ratio, int32_t hi_bits);

/*
 * Important-set budget from the importance ratio (the "Importance ratio" column of Tables 1-3: the share
 * of tokens kept in high precision): k = floor(ratio * T + 0.5), the ratio times the context length
 * rounded half up, evaluated in IEEE double arithmetic. A cache built for context T keeps k important
 * tokens and attends hi_cap = k + 1 important slots (one staging slot receives each decoded token before
 * the step's demotion frees a slot again). Returns -1 for T < 0 or a ratio outside [0, 1] (NaN included).
 * Host-only, pure.
 */
int32_t mikv_budget(int32_t T, double ratio);

/* Bytes of one retained row (codes + parameters, K or V) and of one important row (K or V). */
size_t mikv_retained_row_bytes(int32_t bits, int32_t group, int32_t head_dim);

#ifdef __cplusplus
}
#endif

#endif /* MIKV_H */
