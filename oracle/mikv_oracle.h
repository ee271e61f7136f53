/*
 * mikv_oracle.h — plain, slow CPU oracle for the MiKV mixed-precision KV-cache decode path
 * ("No Token Left Behind", arxiv 2402.18096).
 *
 * TEST INFRASTRUCTURE ONLY. This code exists so that the tests, the smoke check and the
 * CPU-baseline leg of the benchmark can check the CUDA library against an independent,
 * obviously-correct restatement of the paper. The product path never links or calls it.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Precision: the quantizer (Eq. 1) and the channel balancer (Eq. 2) run in fp32 IEEE arithmetic
 * (round-to-nearest-even, no contraction), because the codes they produce are integers that both
 * sides must decide in the same precision. Attention and dequantized values run in fp64.
 *
 * All pointers are host pointers. bf16 and fp16 values are passed as their raw uint16 bit patterns.
 * Array layouts are row-major with the index order written next to each argument.
 *
 * Packed-code layout (our own definition; the paper does not fix one), head dimension d = 128.
 * Channel c is written c = 16 m + u (u = c mod 16, m = c div 16); a plane is a sequence of
 * little-endian 16-bit units. In a plane of f-bit fields (f in {2, 4, 8}) with P = 16 / f codes per
 * unit, channel c sits in unit 8 * (2 * (m div P) + (u div 8)) + (u mod 8) at bits
 * [f * (m mod P), f * (m mod P) + f). In a plane of 1-bit fields, channel c sits in unit u mod 8 at
 * bit 2 * m + (u div 8). N in {2, 4, 8}: one plane of N-bit fields. N = 3: a plane of 2-bit fields
 * holding bits 0..1 of each code, then a plane of 1-bit fields holding bit 2. A row takes 16 * N
 * bytes. Quantization parameters of a row are d/g pairs of fp16 (alpha, beta), alpha first.
 */
#ifndef MIKV_ORACLE_H
#define MIKV_ORACLE_H
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif

/* fp32 -> fp16 bit pattern with rounding mode: 0 nearest-even, -1 toward -inf, +1 toward +inf. */
uint16_t mikv_ref_f32_to_f16(float f, int mode);
/* fp16 bit pattern -> exact value. */
double mikv_ref_f16_to_f64(uint16_t h);

/* Eq. 1 on one quantization group of g values: codes[g], alpha16, beta16. Returns 0. */
int mikv_ref_quantize_group(const float* x, int g, int bits, int32_t* codes, uint16_t* alpha16,
                            uint16_t* beta16);

/* Bit packing of one row of d codes (layout in the file header). */
int mikv_ref_pack_row(const int32_t* codes, int d, int bits, uint8_t* packed);
int mikv_ref_unpack_row(const uint8_t* packed, int d, int bits, int32_t* codes);

/* Quantize + pack one fp32 row: packed[d*bits/8], params[d/g][2] (alpha16, beta16). */
int mikv_ref_quantize_row(const float* x, int d, int bits, int g, uint8_t* packed, uint16_t* params);
/* Dequantize one packed row to exact values x_hat[d] = alpha16 * c + beta16. */
int mikv_ref_dequantize_row(const uint8_t* packed, const uint16_t* params, int d, int bits, int g,
                            double* x_hat);

/* Eq. 2: balancer[Hkv][d] = sqrt(max|q_pre| / max|k_pre|) per KV head and channel, the maxima taken
 * over batch, prefill tokens and (for q) the G = Hq/Hkv query heads that share the KV head.
 * q_pre bf16 [B][Hq][T][d], k_pre bf16 [B][Hkv][T][d]. A zero maximum gives balancer 1. */
int mikv_ref_balancer(int B, int Hq, int Hkv, int T, int d, const uint16_t* q_pre,
                      const uint16_t* k_pre, float* balancer);

/* Demotion into the retained cache (Eq. 1, Eq. 3): for every (b, h) and i < n_rows, source row
 * r = rows[b][h][i] of k_src/v_src (bf16 [B][Hkv][n_src][d]) is quantized (keys multiplied by the
 * balancer first; balancer NULL means 1) and written to retained position lo_start + i:
 * k_codes/v_codes uint8 [B][Hkv][lo_cap][d*bits/8], k_params/v_params fp16 [B][Hkv][lo_cap][d/g][2],
 * lo_tok [B][Hkv][lo_cap] = src_tok[b][h][r] (or r when src_tok is NULL).
 * Returns 0, or -1 on bad arguments / capacity. */
int mikv_ref_quantize_pack(int B, int Hkv, int d, int bits, int g, int lo_cap, const uint16_t* k_src,
                           const uint16_t* v_src, const int32_t* src_tok, int n_src,
                           const int32_t* rows, int n_rows, int lo_start, const float* balancer,
                           uint8_t* k_codes, uint8_t* v_codes, uint16_t* k_params,
                           uint16_t* v_params, int32_t* lo_tok);

/* Single-token decode attention over the mixed-precision cache (Eq. 3-4; softmax attention).
 * q bf16 [B][Hq][d]. Important set: k_hi/v_hi bf16 [B][Hkv][hi_cap][d], all hi_cap slots attended,
 * keys unbalanced and attended with q. Retained set: positions 0..n_lo-1 of the arrays above,
 * attended with q / balancer. Outputs (fp64): out [B][Hq][d], hi_logits [B][Hq][hi_cap]
 * (scaled logits of the important slots), ml [B][Hq][2] = (max logit m, sum of exp(s - m)).
 * hi_logits and ml may be NULL. Returns 0 or -1. */
int mikv_ref_decode_attention(int B, int Hq, int Hkv, int d, int bits, int g, int hi_cap, int lo_cap,
                              int n_lo, const uint16_t* k_hi, const uint16_t* v_hi,
                              const uint8_t* k_codes, const uint8_t* v_codes,
                              const uint16_t* k_params, const uint16_t* v_params,
                              const float* balancer, const uint16_t* q, double sm_scale,
                              double* out, double* hi_logits, double* ml);

/* Accumulated-attention importance (heavy-hitter score): acc[b][h][i] += sum over the G query heads
 * of KV head h of exp(hi_logits - m) / l. hi_logits [B][Hq][hi_cap], ml [B][Hq][2], acc [B][Hkv][hi_cap]
 * (fp32, updated in place; the sum is formed in fp64 and rounded once). */
int mikv_ref_update_importance(int B, int Hq, int Hkv, int hi_cap, const float* hi_logits,
                               const float* ml, float* acc);

/* Selection of the n_demote least important of n slots per (b, h), ordered by (score ascending,
 * id ascending). scores fp32 [B][Hkv][n]; ids int32 [B][Hkv][n] or NULL (id = slot index).
 * demoted [B][Hkv][n_demote] and kept [B][Hkv][n - n_demote] (may be NULL) list slot indices in
 * ascending slot order. Returns 0 or -1. */
int mikv_ref_select_demote(int B, int Hkv, int n, int n_demote, const float* scores,
                           const int32_t* ids, int32_t* demoted, int32_t* kept);

/* New-token insertion into the important set: for every (b, h), slot s = slots[b][h] receives
 * k_new/v_new [B][Hkv][d] (bf16, unbalanced), hi_tok = tok and acc = 0. */
int mikv_ref_insert_token(int B, int Hkv, int d, int hi_cap, const uint16_t* k_new,
                          const uint16_t* v_new, int tok, const int32_t* slots, uint16_t* k_hi,
                          uint16_t* v_hi, int32_t* hi_tok, float* acc);

/* Important-set build from prefill rows: slot i of (b, h) receives source row rows[b][h][i]
 * (k/v bf16 [B][Hkv][n_src][d]), its token id (src_tok or the row index) and its score
 * (src_scores [B][Hkv][n_src], or 0 when NULL). */
int mikv_ref_gather_hi(int B, int Hkv, int d, int hi_cap, const uint16_t* k_src,
                       const uint16_t* v_src, const int32_t* src_tok, const float* src_scores,
                       int n_src, const int32_t* rows, int n_rows, uint16_t* k_hi, uint16_t* v_hi,
                       int32_t* hi_tok, float* acc);

/* Reduced-precision important set (Sec. 3.3, Table 3): important rows stored as hi_bits-bit codes
 * with fp16 (alpha, beta) per group of hg channels, keys balanced (Eq. 3) and attended with q / balancer.
 * k_hc, v_hc uint8 [B][Hkv][hi_cap][d*hi_bits/8]; k_hp, v_hp fp16 [B][Hkv][hi_cap][d/hg][2].
 * mikv_ref_dequantize_row_f32: x[c] = fp32(alpha16 * code + beta16), the sum rounded once.
 * gather_hi_q / insert_token_q: as gather_hi / insert_token, quantizing the rows.
 * decode_attention_q: as decode_attention with the coded important set.
 * demote_hi_q: slot slots[b][h] is dequantized (fp32) and re-quantized at bits/g into retained
 * position lo_pos (no second balancer multiply); lo_tok receives its token id. */
int mikv_ref_dequantize_row_f32(const uint8_t* packed, const uint16_t* params, int d, int bits, int g,
                                float* x);
int mikv_ref_gather_hi_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, const uint16_t* k_src,
                         const uint16_t* v_src, const int32_t* src_tok, const float* src_scores, int n_src,
                         const int32_t* rows, int n_rows, const float* balancer, uint8_t* k_hc, uint8_t* v_hc,
                         uint16_t* k_hp, uint16_t* v_hp, int32_t* hi_tok, float* acc);
int mikv_ref_insert_token_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, const uint16_t* k_new,
                            const uint16_t* v_new, int tok, const int32_t* slots, const float* balancer,
                            uint8_t* k_hc, uint8_t* v_hc, uint16_t* k_hp, uint16_t* v_hp, int32_t* hi_tok,
                            float* acc);
int mikv_ref_decode_attention_q(int B, int Hq, int Hkv, int d, int hi_bits, int hg, int bits, int g, int hi_cap,
                                int lo_cap, int n_lo, const uint8_t* k_hc, const uint8_t* v_hc,
                                const uint16_t* k_hp, const uint16_t* v_hp, const uint8_t* k_codes,
                                const uint8_t* v_codes, const uint16_t* k_params, const uint16_t* v_params,
                                const float* balancer, const uint16_t* q, double sm_scale, double* out,
                                double* hi_logits, double* ml);
int mikv_ref_demote_hi_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, int bits, int g, int lo_cap,
                         const int32_t* slots, int lo_pos, const uint8_t* k_hc, const uint8_t* v_hc,
                         const uint16_t* k_hp, const uint16_t* v_hp, const int32_t* hi_tok, uint8_t* k_codes,
                         uint8_t* v_codes, uint16_t* k_params, uint16_t* v_params, int32_t* lo_tok);

/* Per-channel retained keys (App. C): keys quantized per channel over groups of 64 retained tokens (one
 * fp16 (alpha, beta) per group and channel, no balancer), values per token; retained tokens wait in bf16
 * in staging rows hi_cap .. hi_cap + 63 of the important arrays until their group is complete.
 * quantize_channel_group: x fp32 [64][d] -> packed [64][d*bits/8] (per-token row layout), params [d][2].
 * append_retained_kch: appends rows at retained positions n_lo.. (staging, then group quantization).
 * decode_attention_kch: attention over n_hi bf16 rows (important + staged) and n_lo_q quantized rows. */
int mikv_ref_quantize_channel_group(const float* x, int d, int bits, uint8_t* packed, uint16_t* params);
int mikv_ref_append_retained_kch(int B, int Hkv, int d, int bits, int g, int hi_cap, int hi_rows, int lo_cap,
                                 int n_lo, const uint16_t* k_src, const uint16_t* v_src, const int32_t* src_tok,
                                 int n_src, const int32_t* rows, int n_rows, uint16_t* k_hi, uint16_t* v_hi,
                                 int32_t* hi_tok, uint8_t* k_codes, uint8_t* v_codes, uint16_t* k_params,
                                 uint16_t* v_params, int32_t* lo_tok);
int mikv_ref_decode_attention_kch(int B, int Hq, int Hkv, int d, int bits, int g, int hi_rows, int n_hi, int lo_cap,
                                  int n_lo_q, const uint16_t* k_hi, const uint16_t* v_hi, const uint8_t* k_codes,
                                  const uint8_t* v_codes, const uint16_t* k_params, const uint16_t* v_params,
                                  const uint16_t* q, double sm_scale, double* out, double* hi_logits, double* ml);

/* Prefill importance (the initial accumulated-attention score of every token): scores[b][h][t] = sum over
 * the G query heads of KV head h and the queries i >= t of the causal softmax weight of key t in row i,
 * s = sm_scale * q . k. q_pre bf16 [B][Hq][T][d], k_pre bf16 [B][Hkv][T][d], scores fp64 [B][Hkv][T]. */
int mikv_ref_prefill_scores(int B, int Hq, int Hkv, int T, int d, const uint16_t* q_pre, const uint16_t* k_pre,
                            double sm_scale, double* scores);

/* Closed-form KV-cache size as a fraction of an all-fp16 cache: ratio r of tokens at hi_bits
 * (16 = fp16, else hi_bits-bit codes with fp16 alpha/beta per group g) plus (1 - r) at bits-bit codes
 * with fp16 alpha/beta per group g. */
double mikv_ref_cache_fraction(int bits, int g, double ratio, int hi_bits);

/* Number of important tokens for importance ratio `ratio` over T tokens (Tables 1-3 "Importance ratio"):
 * the integer nearest ratio * T (double product), halves rounded up. -1 if T < 0 or ratio is outside
 * [0, 1]. */
int mikv_ref_budget(int T, double ratio);

#ifdef __cplusplus
}
#endif
#endif
