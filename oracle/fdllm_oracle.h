/*
 * fdllm_oracle.h -- plain fp64 CPU oracle for Frechet profile commit-set selection.
 *
 * TEST INFRASTRUCTURE ONLY.  This oracle exists to check the CUDA path.  Only the
 * test suite, the smoke check and the benchmark's CPU-baseline / reference arm may
 * load it.  The product path (the CUDA library) never calls, links or includes it,
 * and this oracle includes nothing from the product.
 *
 * Everything is computed in double precision with plain loops, in the order of the
 * paper's Algorithm 1 ("Fast-dLLM++: Frechet Profile Decoding"):
 *   confidence/argmax per masked position -> sort -> scan of L_n, U_n, G_n -> n* -> reveal.
 *
 * Conventions shared with the CUDA library's public interface (not its code):
 *   logits  [B, L, V] row-major, V contiguous; dtype 0 = bf16 (raw uint16 bits), 1 = fp32,
 *           2 = fp64 (exact LM-head products), 3 = IEEE half (raw uint16 bits).
 *   mask    uint8 [B, L], 1 = masked; updated in place by the reveal (committed -> 0).
 *   mode    0 = profile (Frechet), 1 = factor, 2 = threshold.
 *   param   profile: f, with margin delta = 1 - f (matched parameter, Cor. factor-reduction);
 *           factor: f;  threshold: tau.
 */
#ifndef FDLLM_ORACLE_H
#define FDLLM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORACLE_BF16 = 0, ORACLE_FP32 = 1, ORACLE_F64 = 2, ORACLE_F16 = 3 };
enum { ORACLE_PROFILE = 0, ORACLE_FACTOR = 1, ORACLE_THRESHOLD = 2 };

/* Per masked position (b,l): x_hat = lowest v attaining max_v logit, c = max_v softmax(v)
 * (Sec. 3 "Notation", Alg. 1 confidence loop).  conf/tok are written only at masked
 * positions.  Rows whose logits contain NaN, or whose maximum is +inf or -inf, get
 * conf = NaN and tok = -1.  Returns the number of such rows.  nthreads <= 1 runs serially. */
int64_t oracle_confidence(const void *logits, int dtype, int64_t B, int64_t L, int64_t V,
                          const uint8_t *mask, double *conf, int32_t *tok, int nthreads);

/* The Frechet profile quantities of Sec. 3 / Eq. frechet_Ln_Un for a profile already
 * sorted in descending order: for n = 1..m,
 *   L_n = max{0, sum_{j<=n} c_(j) - (n-1)},  U_n = 1 - c_(n),  G_n = L_n - U_n.
 * Outputs are indexed n-1. */
void oracle_frechet_scan(const double *c_sorted, int64_t m, double *Ln, double *Un, double *Gn);

/* Selection from given confidences (Alg. 1 sort, scan, select, reveal).
 * For every batch row b: m = number of masked positions.
 *   m == 0            -> out_n[b] = 0, nothing committed.
 *   any masked conf not in (0, 1] (NaN included) -> out_n[b] = -1, nothing committed.
 *   otherwise         -> n* = max{n : rule accepts n}, or 1 if no n is accepted;
 *                        the n* most confident masked positions (ties: lower position
 *                        first) get out_tokens = tok, out_commit = 1, mask = 0.
 * out_commit is fully written; out_tokens only at committed positions.
 * margin[b] (nullable) = decision margin of the row: the smallest of |rule(n) - bound| at
 * n = n* and n = n*+1 and of the ranking gap that decides which positions fill the first n*
 * ranks (c_(n*) - c_(n*+1); when equal confidences straddle the boundary, the gaps from
 * that tie block to its neighbours); +inf when nothing can flip (m == 0, invalid row).
 * Returns the number of invalid rows. */
int64_t oracle_select_from_conf(const double *conf, const int32_t *tok, int64_t B, int64_t L,
                                uint8_t *mask, int mode, double param, int32_t *out_tokens,
                                uint8_t *out_commit, int32_t *out_n, double *margin);

/* Calibration-robust profile selection (App. C, Eq. robust_L_U) on given confidences:
 * lower confidences c_low_i = max{0, c_hat_i - eta_i} with eta_i = eta_pos[i] when eta_pos
 * is given, else the uniform eta; then the profile rule of Sec. 3 on c_low: rank the masked
 * positions by c_low descending (ties: lower position first), L = max{0, sum c_low - (n-1)},
 * U = 1 - c_low_(n), accept n iff L - U > delta = 1 - param, n* = max accepted or 1.
 * Validity, empty rows, outputs and return value as oracle_select_from_conf.  margin[b] also
 * covers min_i |c_hat_i - eta_i| over the row's masked positions (clipping can reorder). */
int64_t oracle_select_robust_from_conf(const double *conf, const int32_t *tok, int64_t B,
                                       int64_t L, uint8_t *mask, double param, double eta,
                                       const double *eta_pos, int32_t *out_tokens,
                                       uint8_t *out_commit, int32_t *out_n, double *margin);

/* Heterogeneity-bonus terms of a descending profile (Prop. heterogeneity-bonus, Eq.
 * heterogeneity_decomp): for n = 1..m, F_n = (n+1) c_(n) - n (factor core) and
 * B_n = sum_{j=1}^{n-1} (c_(j) - c_(n)) (heterogeneity bonus).  Outputs indexed n-1. */
void oracle_bonus_terms(const double *c_sorted, int64_t m, double *Fn, double *Bn);

/* Per batch row, the masked confidences sorted as in Alg. 1 (descending, ties: lower
 * position first) and, at rank n = 1..m_b: G[b, n-1] (Eq. frechet_Ln_Un), F[b, n-1],
 * Bn[b, n-1] (Eq. heterogeneity_decomp) and order[b, n-1] = the position at rank n.  Ranks
 * beyond m_b hold NaN (order -1).  All arrays [B, L]. */
void oracle_profile_terms(const double *conf, const uint8_t *mask, int64_t B, int64_t L,
                          double *G, double *F, double *Bn, int32_t *order);

/* Counter-based synthetic logits (the stand-in forward pass of the decode loop), bf16 bits
 * [B, L, V] for the rows with mask != 0 (mask NULL: all rows), defined for seed s, step t,
 * row (b, l) and index v by SplitMix64's finaliser mix (Steele, Lea, Flood 2014),
 * G = 0x9E3779B97F4A7C15, k = mix(s ^ mix(t*G ^ mix(b << 32 | l))):
 *   noise x_v = float(sum_j (2 u_j + 1) - 262144) * fl32(sqrt(3)/131072), u_j the four
 *               16-bit fields of mix(k + (v+1) G)   (Irwin-Hall, unit variance)
 *   peak       p = mix(k ^ 0xD1B54A32D192ED03): x_{p mod V} += float(p >> 40) * fl32(peak/2^24)
 *   rounded to bf16 (nearest even). */
void oracle_synth_block_logits(uint16_t *out, const uint8_t *mask, int64_t B, int64_t L,
                               int64_t V, uint64_t seed, uint64_t step, double peak_max);

/* Algorithm 1's outer loop on the synthetic forward pass: for each of gen_len / block_len
 * blocks, start with the block fully masked and repeat {logits of the block's masked rows at
 * the global step; selection (mode, param); reveal} until no position of the block is
 * masked, or max_steps global steps were taken.  out_seq [B, gen_len] receives the
 * committed tokens (-1 where none), out_nfe [n_blocks] the steps per block, out_margin [B]
 * the smallest decision margin each row saw (see oracle_select_from_conf).  Returns the
 * total number of steps. */
int64_t oracle_decode_loop(int64_t B, int64_t gen_len, int64_t block_len, int64_t V, int mode,
                           double param, uint64_t seed, double peak_max, int64_t max_steps,
                           int32_t *out_seq, int32_t *out_nfe, double *out_margin,
                           int nthreads);

/* oracle_confidence followed by oracle_select_from_conf.  conf/tok are caller scratch of
 * B*L entries; they come back holding the per-position confidences and argmax tokens. */
int64_t oracle_select(const void *logits, int dtype, int64_t B, int64_t L, int64_t V,
                      uint8_t *mask, int mode, double param, int32_t *out_tokens,
                      uint8_t *out_commit, int32_t *out_n, double *margin, double *conf,
                      int32_t *tok, int nthreads);

/* The LM head that produces the logits (Sec. 3 "Notation": p_i is the softmax of the logits
 * of position i): for every masked row r, out[r][v] = sum_k hidden[r][k] * w[v][k], summed in
 * k order in double precision from the bf16 inputs (raw uint16 bits, widened exactly), and,
 * when out_abs is not NULL, out_abs[r][v] = sum_k |hidden[r][k] * w[v][k]| (the scale of the
 * rounding error of any fp32 evaluation of the same sum).  Unmasked rows are not written.
 * hidden [rows][H], w [V][H], out and out_abs [rows][V]. */
void oracle_lmhead_logits(const uint16_t *hidden, const uint16_t *w, int64_t rows, int64_t H,
                          int64_t V, const uint8_t *mask, double *out, double *out_abs,
                          int nthreads);

/* Counter-based synthetic hidden states [B, L, H] (bf16 bits) against the bf16 head w [V, H]:
 * the LM-head counterpart of oracle_synth_block_logits, an input generator (test
 * infrastructure, no selection arithmetic).  For row (b, l) with row key k: p = mix(k ^
 * 0xD1B54A32D192ED03), target t = p % V, beta = fl32(float(p >> 40) * fl32(beta_max / 2^24));
 * z_j the Irwin-Hall noise at index j; n2 = |w_t|^2 in fp32 as 32 lane sums (lane i: j = i,
 * i + 32, ... in order) folded by an xor butterfly over offsets 16, 8, 4, 2, 1; scale =
 * beta / n2; h_j = fl32(z_j + fl32(scale * w_tj)), rounded to bf16.  Unmasked rows are left
 * as they are. */
void oracle_synth_block_hidden(uint16_t *out, const uint8_t *mask, int64_t B, int64_t L,
                               int64_t H, int64_t V, const uint16_t *w, uint64_t seed,
                               uint64_t step, double beta_max);

/* IEEE half bit patterns to doubles (the fp16 widening of oracle_confidence). */
void oracle_half_to_double(const uint16_t *h, int64_t n, double *out);

#ifdef __cplusplus
}
#endif

#endif /* FDLLM_ORACLE_H */
