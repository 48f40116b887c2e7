/*
 * fdllm_oracle.c -- plain fp64 CPU oracle for Frechet profile commit-set selection.
 *
 * TEST INFRASTRUCTURE ONLY (see fdllm_oracle.h): slow, obviously correct, and sharing no
 * code with the CUDA library.  Each function follows the paper's definitions in the order
 * of Algorithm 1; nothing is blocked, fused or reordered beyond what those state.
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared [-fopenmp] fdllm_oracle.c -lm
 * (-ffp-contract=off keeps a*b+c unfused so that x86 and Arm hosts round alike.)
 */
#include "fdllm_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* IEEE binary16 bits to double, exactly, from the format's definition: sign, 5 exponent
 * bits with bias 15, 10 fraction bits; exponent 0 holds zero and the subnormals
 * (fraction x 2^-24), exponent 31 the infinities and NaNs. */
static double half_to_double(uint16_t h)
{
    const int sign = (h >> 15) & 1, e = (h >> 10) & 0x1F, frac = h & 0x3FF;
    double v;
    if (e == 0)
        v = ldexp((double)frac, -24);
    else if (e == 31)
        v = frac ? NAN : INFINITY;
    else
        v = ldexp((double)(1024 + frac), e - 25);
    return sign ? -v : v;
}

/* One logit widened to double.  bf16 is the upper half of an IEEE fp32 word, so the
 * widening is exact, as is the half's; fp64 logits (the LM head's exact products) are taken
 * as they are. */
static double logit_at(const void *logits, int dtype, int64_t i)
{
    float f;
    if (dtype == ORACLE_F64)
        return ((const double *)logits)[i];
    if (dtype == ORACLE_F16)
        return half_to_double(((const uint16_t *)logits)[i]);
    if (dtype == ORACLE_BF16) {
        uint32_t u = (uint32_t)((const uint16_t *)logits)[i] << 16;
        memcpy(&f, &u, sizeof f);
    } else {
        f = ((const float *)logits)[i];
    }
    return (double)f;
}

static double bf16_to_double(uint16_t b)
{
    float f;
    uint32_t u = (uint32_t)b << 16;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Sec. 3 "Notation" and the confidence loop of Alg. 1:
 *   x_hat_i = argmax_v p_i(v),  c_i = max_v p_i(v),  p_i = softmax of the logits of row i.
 * With M = max_v x_v and S = sum_v exp(x_v - M), max_v p_i(v) = exp(M - M) / S = 1 / S.
 * Ties in the argmax go to the lowest vocabulary index. */
static int confidence_of_row(const void *logits, int dtype, int64_t base, int64_t V,
                             double *c_out, int32_t *tok_out)
{
    double M = -INFINITY;
    int64_t arg = -1;
    int saw_nan = 0;
    for (int64_t v = 0; v < V; ++v) {
        double x = logit_at(logits, dtype, base + v);
        if (isnan(x)) {
            saw_nan = 1;
            continue;
        }
        if (arg < 0 || x > M) { /* strict '>' keeps the lowest index among equal maxima */
            M = x;
            arg = v;
        }
    }
    if (saw_nan || !isfinite(M)) {
        *c_out = NAN;
        *tok_out = -1;
        return 1;
    }
    double S = 0.0;
    for (int64_t v = 0; v < V; ++v)
        S += exp(logit_at(logits, dtype, base + v) - M);
    *c_out = 1.0 / S;
    *tok_out = (int32_t)arg;
    return 0;
}

int64_t oracle_confidence(const void *logits, int dtype, int64_t B, int64_t L, int64_t V,
                          const uint8_t *mask, double *conf, int32_t *tok, int nthreads)
{
    int64_t bad = 0;
    const int64_t rows = B * L;
#ifdef _OPENMP
    if (nthreads < 1)
        nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : bad) num_threads(nthreads)
#else
    (void)nthreads;
#endif
    for (int64_t r = 0; r < rows; ++r) {
        if (!mask[r])
            continue;
        bad += confidence_of_row(logits, dtype, r * V, V, &conf[r], &tok[r]);
    }
    return bad;
}

/* Sec. 3 "Frechet profile quantities" / Eq. frechet_Ln_Un, in the paper's own form. */
void oracle_frechet_scan(const double *c_sorted, int64_t m, double *Ln, double *Un, double *Gn)
{
    double sum = 0.0;
    for (int64_t n = 1; n <= m; ++n) {
        sum += c_sorted[n - 1];
        double l = sum - (double)(n - 1);
        Ln[n - 1] = l > 0.0 ? l : 0.0;
        Un[n - 1] = 1.0 - c_sorted[n - 1];
        Gn[n - 1] = Ln[n - 1] - Un[n - 1];
    }
}

typedef struct {
    double c;
    int32_t pos;
} candidate;

/* Decision margin contribution of the ranking (for parity checks): the smallest positive
 * confidence gap whose sign decides which positions fill the first n* ranks.  Without a tie
 * at the boundary that is c_(n*) - c_(n*+1).  When a block of equal confidences straddles
 * the boundary (ranks a..b with a <= n* < b), the block is committed partly, in position
 * order, so the gaps to its neighbours above and below decide instead. */
static double ranking_gap(const double *cs, int64_t m, int64_t nstar)
{
    double mg = INFINITY;
    if (nstar >= m)
        return mg;
    const double v = cs[nstar - 1];
    if (cs[nstar] != v) {
        const double gap = v - cs[nstar];
        return gap > 0.0 ? gap : mg;
    }
    int64_t a = nstar, b = nstar; /* 1-based ranks of the tie block */
    while (a > 1 && cs[a - 2] == v)
        --a;
    while (b < m && cs[b] == v)
        ++b;
    if (a > 1 && cs[a - 2] - v < mg)
        mg = cs[a - 2] - v;
    if (b < m && v - cs[b] < mg)
        mg = v - cs[b];
    return mg;
}

/* Alg. 1 sort: c_(1) >= c_(2) >= ...; equal confidences keep the lower position first. */
static int by_confidence_desc(const void *pa, const void *pb)
{
    const candidate *a = (const candidate *)pa, *b = (const candidate *)pb;
    if (a->c > b->c)
        return -1;
    if (a->c < b->c)
        return 1;
    return (a->pos > b->pos) - (a->pos < b->pos);
}

int64_t oracle_select_from_conf(const double *conf, const int32_t *tok, int64_t B, int64_t L,
                                uint8_t *mask, int mode, double param, int32_t *out_tokens,
                                uint8_t *out_commit, int32_t *out_n, double *margin)
{
    int64_t bad = 0;
    candidate *cand = (candidate *)malloc((size_t)L * sizeof(candidate));
    double *cs = (double *)malloc((size_t)L * sizeof(double));
    double *Ln = (double *)malloc((size_t)L * sizeof(double));
    double *Un = (double *)malloc((size_t)L * sizeof(double));
    double *Gn = (double *)malloc((size_t)L * sizeof(double));
    double *q = (double *)malloc((size_t)L * sizeof(double)); /* signed distance to the bound */
    int *ok = (int *)malloc((size_t)L * sizeof(int));

    for (int64_t b = 0; b < B; ++b) {
        const int64_t row0 = b * L;
        int64_t m = 0;
        int invalid = 0;
        for (int64_t l = 0; l < L; ++l) {
            out_commit[row0 + l] = 0;
            if (!mask[row0 + l])
                continue;
            double c = conf[row0 + l];
            if (!(c > 0.0 && c <= 1.0))
                invalid = 1;
            cand[m].c = c;
            cand[m].pos = (int32_t)l;
            ++m;
        }
        if (margin)
            margin[b] = INFINITY;
        if (invalid) {
            out_n[b] = -1;
            ++bad;
            continue;
        }
        if (m == 0) { /* Alg. 1 never reaches a block without masked positions */
            out_n[b] = 0;
            continue;
        }

        qsort(cand, (size_t)m, sizeof(candidate), by_confidence_desc);
        for (int64_t j = 0; j < m; ++j)
            cs[j] = cand[j].c;

        /* Alg. 1 scan: one acceptance test per prefix size n = 1..m. */
        if (mode == ORACLE_PROFILE) {
            const double delta = 1.0 - param; /* matched margin, Cor. factor-reduction */
            oracle_frechet_scan(cs, m, Ln, Un, Gn);
            for (int64_t n = 1; n <= m; ++n) {
                ok[n - 1] = Gn[n - 1] > delta; /* G_n > delta (Sec. 3) */
                q[n - 1] = Gn[n - 1] - delta;
            }
        } else if (mode == ORACLE_FACTOR) {
            const double f = param;
            for (int64_t n = 1; n <= m; ++n) {
                double r = (double)(n + 1) * (1.0 - cs[n - 1]); /* (n+1)(1 - c_(n)) < f */
                ok[n - 1] = r < f;
                q[n - 1] = f - r;
            }
        } else { /* threshold: S = {i : c_i >= tau} (Sec. 2, confidence-aware decoding) */
            const double tau = param;
            for (int64_t n = 1; n <= m; ++n) {
                ok[n - 1] = cs[n - 1] >= tau;
                q[n - 1] = cs[n - 1] - tau;
            }
        }

        /* Alg. 1 select: n* = max{n : accepted}; n* = 1 when the set is empty. */
        int64_t nstar = 0;
        for (int64_t n = 1; n <= m; ++n)
            if (ok[n - 1])
                nstar = n;
        if (nstar == 0)
            nstar = 1;

        /* Alg. 1 reveal: the n* most confident masked positions take their argmax token. */
        for (int64_t j = 0; j < nstar; ++j) {
            const int64_t at = row0 + cand[j].pos;
            out_tokens[at] = tok[at];
            out_commit[at] = 1;
            mask[at] = 0;
        }
        out_n[b] = (int32_t)nstar;

        if (margin) {
            double mg = fabs(q[nstar - 1]);
            if (nstar < m && fabs(q[nstar]) < mg)
                mg = fabs(q[nstar]);
            const double gap = ranking_gap(cs, m, nstar);
            if (gap < mg)
                mg = gap;
            margin[b] = mg;
        }
    }

    free(cand);
    free(cs);
    free(Ln);
    free(Un);
    free(Gn);
    free(q);
    free(ok);
    return bad;
}

int64_t oracle_select_robust_from_conf(const double *conf, const int32_t *tok, int64_t B,
                                       int64_t L, uint8_t *mask, double param, double eta,
                                       const double *eta_pos, int32_t *out_tokens,
                                       uint8_t *out_commit, int32_t *out_n, double *margin)
{
    int64_t bad = 0;
    candidate *cand = (candidate *)malloc((size_t)L * sizeof(candidate));
    double *cs = (double *)malloc((size_t)L * sizeof(double));
    double *Ln = (double *)malloc((size_t)L * sizeof(double));
    double *Un = (double *)malloc((size_t)L * sizeof(double));
    double *Gn = (double *)malloc((size_t)L * sizeof(double));
    const double delta = 1.0 - param; /* matched margin, Cor. factor-reduction */

    for (int64_t b = 0; b < B; ++b) {
        const int64_t row0 = b * L;
        int64_t m = 0;
        int invalid = 0;
        double clip_gap = INFINITY; /* closest distance of a c_hat to its clipping point */
        for (int64_t l = 0; l < L; ++l) {
            out_commit[row0 + l] = 0;
            if (!mask[row0 + l])
                continue;
            const double c_hat = conf[row0 + l];
            if (!(c_hat > 0.0 && c_hat <= 1.0))
                invalid = 1;
            /* App. C takes the allowance eta >= 0; a negative or NaN allowance is read as 0 */
            const double eta_raw = eta_pos ? eta_pos[row0 + l] : eta;
            const double eta_i = eta_raw > 0.0 ? eta_raw : 0.0;
            /* App. C: the lower confidence max{0, c_hat - eta} */
            const double c_low = c_hat - eta_i > 0.0 ? c_hat - eta_i : 0.0;
            if (fabs(c_hat - eta_i) < clip_gap)
                clip_gap = fabs(c_hat - eta_i);
            cand[m].c = c_low;
            cand[m].pos = (int32_t)l;
            ++m;
        }
        if (margin)
            margin[b] = INFINITY;
        if (invalid) {
            out_n[b] = -1;
            ++bad;
            continue;
        }
        if (m == 0) {
            out_n[b] = 0;
            continue;
        }
        qsort(cand, (size_t)m, sizeof(candidate), by_confidence_desc);
        for (int64_t j = 0; j < m; ++j)
            cs[j] = cand[j].c;
        /* Eq. robust_L_U on the top-n prefix: the same scan as Sec. 3 on c_low */
        oracle_frechet_scan(cs, m, Ln, Un, Gn);
        int64_t nstar = 0;
        for (int64_t n = 1; n <= m; ++n)
            if (Gn[n - 1] > delta)
                nstar = n;
        if (nstar == 0)
            nstar = 1;
        for (int64_t j = 0; j < nstar; ++j) {
            const int64_t at = row0 + cand[j].pos;
            out_tokens[at] = tok[at];
            out_commit[at] = 1;
            mask[at] = 0;
        }
        out_n[b] = (int32_t)nstar;
        if (margin) {
            double mg = fabs(Gn[nstar - 1] - delta);
            if (nstar < m && fabs(Gn[nstar] - delta) < mg)
                mg = fabs(Gn[nstar] - delta);
            const double gap = ranking_gap(cs, m, nstar);
            if (gap < mg)
                mg = gap;
            if (clip_gap < mg)
                mg = clip_gap;
            margin[b] = mg;
        }
    }
    free(cand);
    free(cs);
    free(Ln);
    free(Un);
    free(Gn);
    return bad;
}

/* Eq. heterogeneity_decomp, term by term. */
void oracle_bonus_terms(const double *c_sorted, int64_t m, double *Fn, double *Bn)
{
    for (int64_t n = 1; n <= m; ++n) {
        const double cn = c_sorted[n - 1];
        Fn[n - 1] = (double)(n + 1) * cn - (double)n;
        double bonus = 0.0;
        for (int64_t j = 1; j <= n - 1; ++j)
            bonus += c_sorted[j - 1] - cn;
        Bn[n - 1] = bonus;
    }
}

void oracle_profile_terms(const double *conf, const uint8_t *mask, int64_t B, int64_t L,
                          double *G, double *F, double *Bn, int32_t *order)
{
    candidate *cand = (candidate *)malloc((size_t)L * sizeof(candidate));
    double *cs = (double *)malloc((size_t)L * sizeof(double));
    double *Lt = (double *)malloc((size_t)L * sizeof(double));
    double *Ut = (double *)malloc((size_t)L * sizeof(double));
    for (int64_t b = 0; b < B; ++b) {
        const int64_t row0 = b * L;
        int64_t m = 0;
        for (int64_t l = 0; l < L; ++l) {
            G[row0 + l] = NAN;
            F[row0 + l] = NAN;
            Bn[row0 + l] = NAN;
            order[row0 + l] = -1;
            if (!mask[row0 + l])
                continue;
            cand[m].c = conf[row0 + l];
            cand[m].pos = (int32_t)l;
            ++m;
        }
        if (m == 0)
            continue;
        qsort(cand, (size_t)m, sizeof(candidate), by_confidence_desc);
        for (int64_t j = 0; j < m; ++j) {
            cs[j] = cand[j].c;
            order[row0 + j] = cand[j].pos;
        }
        oracle_frechet_scan(cs, m, Lt, Ut, G + row0);
        oracle_bonus_terms(cs, m, F + row0, Bn + row0);
    }
    free(cand);
    free(cs);
    free(Lt);
    free(Ut);
}

int64_t oracle_select(const void *logits, int dtype, int64_t B, int64_t L, int64_t V,
                      uint8_t *mask, int mode, double param, int32_t *out_tokens,
                      uint8_t *out_commit, int32_t *out_n, double *margin, double *conf,
                      int32_t *tok, int nthreads)
{
    int64_t bad_rows = oracle_confidence(logits, dtype, B, L, V, mask, conf, tok, nthreads);
    (void)bad_rows;
    return oracle_select_from_conf(conf, tok, B, L, mask, mode, param, out_tokens, out_commit,
                                   out_n, margin);
}

/* ---- synthetic forward pass and the decode loop (test infrastructure) ---- */

static uint64_t splitmix_mix(uint64_t z)
{
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

/* fp32 -> bf16 bits, round to nearest even (finite inputs). */
static uint16_t bf16_round(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    const uint32_t lsb = (u >> 16) & 1u;
    return (uint16_t)((u + 0x7FFFu + lsb) >> 16);
}

void oracle_synth_block_logits(uint16_t *out, const uint8_t *mask, int64_t B, int64_t L,
                               int64_t V, uint64_t seed, uint64_t step, double peak_max)
{
    const uint64_t G = 0x9E3779B97F4A7C15ull;
    const float noise_scale = (float)(sqrt(3.0) / 131072.0);
    const float peak_scale = (float)(peak_max / 16777216.0);
    for (int64_t b = 0; b < B; ++b)
        for (int64_t l = 0; l < L; ++l) {
            const int64_t row = b * L + l;
            if (mask && !mask[row])
                continue;
            const uint64_t k = splitmix_mix(
                seed ^ splitmix_mix(step * G ^ splitmix_mix(((uint64_t)b << 32) | (uint64_t)l)));
            const uint64_t p = splitmix_mix(k ^ 0xD1B54A32D192ED03ull);
            const int64_t pidx = (int64_t)(p % (uint64_t)V);
            const float height = (float)(p >> 40) * peak_scale;
            for (int64_t v = 0; v < V; ++v) {
                const uint64_t h = splitmix_mix(k + (uint64_t)(v + 1) * G);
                const int32_t s = (int32_t)(2 * (h & 0xFFFF) + 2 * ((h >> 16) & 0xFFFF) +
                                            2 * ((h >> 32) & 0xFFFF) + 2 * ((h >> 48) & 0xFFFF) +
                                            4) -
                                  262144;
                float x = (float)s * noise_scale;
                if (v == pidx)
                    x = x + height;
                out[row * V + v] = bf16_round(x);
            }
        }
}

int64_t oracle_decode_loop(int64_t B, int64_t gen_len, int64_t block_len, int64_t V, int mode,
                           double param, uint64_t seed, double peak_max, int64_t max_steps,
                           int32_t *out_seq, int32_t *out_nfe, double *out_margin,
                           int nthreads)
{
    const int64_t nblocks = gen_len / block_len, Lb = block_len;
    uint16_t *logits = (uint16_t *)malloc((size_t)(B * Lb * V) * sizeof(uint16_t));
    uint8_t *mask = (uint8_t *)malloc((size_t)(B * Lb));
    int32_t *tokens = (int32_t *)malloc((size_t)(B * Lb) * sizeof(int32_t));
    uint8_t *commit = (uint8_t *)malloc((size_t)(B * Lb));
    int32_t *n = (int32_t *)malloc((size_t)B * sizeof(int32_t));
    double *margin = (double *)malloc((size_t)B * sizeof(double));
    double *conf = (double *)malloc((size_t)(B * Lb) * sizeof(double));
    int32_t *tok = (int32_t *)malloc((size_t)(B * Lb) * sizeof(int32_t));
    for (int64_t i = 0; i < B * gen_len; ++i)
        out_seq[i] = -1;
    for (int64_t b = 0; b < B; ++b)
        out_margin[b] = INFINITY;
    int64_t step = 0;
    for (int64_t blk = 0; blk < nblocks; ++blk) {
        int64_t nfe = 0;
        for (int64_t i = 0; i < B * Lb; ++i)
            mask[i] = 1;
        for (;;) { /* while the block contains masked positions (Alg. 1) */
            int any = 0;
            for (int64_t i = 0; i < B * Lb; ++i)
                any |= mask[i];
            if (!any || step >= max_steps)
                break;
            oracle_synth_block_logits(logits, mask, B, Lb, V, seed, (uint64_t)step, peak_max);
            for (int64_t i = 0; i < B * Lb; ++i)
                tokens[i] = -1;
            oracle_select(logits, ORACLE_BF16, B, Lb, V, mask, mode, param, tokens, commit, n,
                          margin, conf, tok, nthreads);
            for (int64_t b = 0; b < B; ++b) {
                if (margin[b] < out_margin[b])
                    out_margin[b] = margin[b];
                for (int64_t l = 0; l < Lb; ++l)
                    if (commit[b * Lb + l])
                        out_seq[b * gen_len + blk * Lb + l] = tokens[b * Lb + l];
            }
            ++step;
            ++nfe;
        }
        out_nfe[blk] = (int32_t)nfe;
    }
    free(logits);
    free(mask);
    free(tokens);
    free(commit);
    free(n);
    free(margin);
    free(conf);
    free(tok);
    return step;
}

void oracle_lmhead_logits(const uint16_t *hidden, const uint16_t *w, int64_t rows, int64_t H,
                          int64_t V, const uint8_t *mask, double *out, double *out_abs,
                          int nthreads)
{
    int64_t r;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 1 ? nthreads : 1)
#endif
    for (r = 0; r < rows; ++r) {
        if (mask && !mask[r])
            continue;
        double *h = (double *)malloc((size_t)H * sizeof(double));
        for (int64_t k = 0; k < H; ++k)
            h[k] = bf16_to_double(hidden[r * H + k]);
        for (int64_t v = 0; v < V; ++v) {
            double sum = 0.0, mag = 0.0;
            for (int64_t k = 0; k < H; ++k) {
                const double t = h[k] * bf16_to_double(w[v * H + k]);
                sum += t;
                mag += fabs(t);
            }
            out[r * V + v] = sum;
            if (out_abs)
                out_abs[r * V + v] = mag;
        }
        free(h);
    }
}

void oracle_synth_block_hidden(uint16_t *out, const uint8_t *mask, int64_t B, int64_t L,
                               int64_t H, int64_t V, const uint16_t *w, uint64_t seed,
                               uint64_t step, double beta_max)
{
    const uint64_t G = 0x9E3779B97F4A7C15ull;
    const float noise_scale = (float)(sqrt(3.0) / 131072.0);
    const float beta_scale = (float)(beta_max / 16777216.0);
    for (int64_t b = 0; b < B; ++b)
        for (int64_t l = 0; l < L; ++l) {
            const int64_t row = b * L + l;
            if (mask && !mask[row])
                continue;
            const uint64_t k = splitmix_mix(
                seed ^ splitmix_mix(step * G ^ splitmix_mix(((uint64_t)b << 32) | (uint64_t)l)));
            const uint64_t p = splitmix_mix(k ^ 0xD1B54A32D192ED03ull);
            const int64_t t = (int64_t)(p % (uint64_t)V);
            const float beta = (float)(p >> 40) * beta_scale;
            const uint16_t *wt = w + t * H;
            float lane[32];
            for (int i = 0; i < 32; ++i) {
                float acc = 0.0f;
                for (int64_t j = i; j < H; j += 32) {
                    const float x = (float)bf16_to_double(wt[j]);
                    const float sq = x * x;
                    acc = acc + sq;
                }
                lane[i] = acc;
            }
            for (int o = 16; o > 0; o >>= 1) {
                float next[32];
                for (int i = 0; i < 32; ++i)
                    next[i] = lane[i] + lane[i ^ o];
                for (int i = 0; i < 32; ++i)
                    lane[i] = next[i];
            }
            const float scale = beta / lane[0];
            for (int64_t j = 0; j < H; ++j) {
                const uint64_t h = splitmix_mix(k + (uint64_t)(j + 1) * G);
                const int32_t sv = (int32_t)(2 * (h & 0xFFFF) + 2 * ((h >> 16) & 0xFFFF) +
                                             2 * ((h >> 32) & 0xFFFF) + 2 * ((h >> 48) & 0xFFFF) +
                                             4) -
                                   262144;
                const float z = (float)sv * noise_scale;
                const float prod = scale * (float)bf16_to_double(wt[j]);
                const float hj = z + prod;
                out[row * H + j] = bf16_round(hj);
            }
        }
}

/* The widening of oracle_confidence's fp16 input, exposed for its pin: n IEEE half bit
 * patterns to doubles. */
void oracle_half_to_double(const uint16_t *h, int64_t n, double *out)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = half_to_double(h[i]);
}
