/*
 * wino_oracle.c -- plain fp64 CPU oracle of the WINO scoring-and-revoke step.
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the benchmark's
 * CPU-baseline / reference leg may load this library.  It shares no code,
 * header, table or constant with the CUDA path.
 *
 * What it computes (arXiv 2605.16941, "Roll Out and Roll Back"):
 *   - the model's token distribution p(y_hat_l = v | Y~) over the whole
 *     vocabulary V for every scored row, as the softmax of the LM-head logits
 *     l_v = <h, w_v> (Sec. 3, Eq. 1; Sec. 4.2.1 Eq. 2; Sec. 4.2.2 Eq. 3);
 *     reported per row as argmax_v p, max_v p and p(target);
 *   - the overall WINO step, Eq. 4 (Sec. 4.2.3): draft every masked position
 *     of the current block whose max-probability exceeds tau1 (Eq. 2), re-mask
 *     every decoded position whose shadow-block probability of its current
 *     token is below tau2 (Eq. 3), keep everything else; plus the at-least-one
 *     rule: when no masked position clears tau1, the single most confident
 *     masked position is drafted (the greedy rule of Eq. 1).
 *
 * Arithmetic: every bf16 input is widened exactly to double; logits are
 * accumulated in double in index order k = 0..d-1 (products of two bf16
 * values are exact in double); the softmax uses libm exp() in double.  The
 * code is deliberately a direct transcription of the definitions: no
 * blocking, no fusion, no reordering beyond looping over rows in parallel.
 *
 * Parity pins: see tests/test_oracle_*.py (closed forms, exact rational
 * brute force, special cases reducing to Eq. 1 greedy decoding and to the
 * tau2 = 0 "only draft" ablation of Sec. 6.3.4, and invariants of Eq. 4).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_ERR_ARG (-1)
#define ORACLE_ERR_NOMEM (-2)

/* A bf16 value is the upper 16 bits of an IEEE-754 binary32 value. */
double oracle_bf16_to_double(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Logits of one row: out[v] = sum_k h[k] * W[v, k], W row-major [V, d].
 * The row h is widened to double once; the sum runs in index order. */
void oracle_logits_row(const uint16_t *h, const uint16_t *W, int64_t d, int64_t V, double *out)
{
    double *hd = (double *)malloc((size_t)d * sizeof(double));
    if (!hd) {
        for (int64_t v = 0; v < V; ++v)
            out[v] = NAN;
        return;
    }
    for (int64_t k = 0; k < d; ++k)
        hd[k] = oracle_bf16_to_double(h[k]);
    for (int64_t v = 0; v < V; ++v) {
        const uint16_t *w = W + v * d;
        double acc = 0.0;
        for (int64_t k = 0; k < d; ++k)
            acc += hd[k] * oracle_bf16_to_double(w[k]);
        out[v] = acc;
    }
    free(hd);
}

/*
 * Per-row softmax statistics over the full vocabulary.
 *   argmax[n]  = smallest v with l_v = max_u l_u
 *   pmax[n]    = max_v p_v = exp(0) / sum_v exp(l_v - m) = 1 / Z
 *   ptarget[n] = p_{target[n]} = exp(l_t - m) / Z, or 0 when target[n] is
 *                outside [0, V) (no target for that row)
 *   gap[n]     = m - (largest logit over v != argmax[n]); 0 on an exact tie
 *   maxlogit[n]= m            (optional output, may be NULL)
 *   logz[n]    = m + log Z    (optional output, may be NULL)
 *   entropy[n] = -sum_v p_v log p_v, the entropy WINO+'s deferral and
 *                sharpening terms use (Sec. 5.3, Eq. 6-7) (optional, may be NULL)
 * Rows are independent; they are spread over nthreads (<= 0: library default).
 */
int oracle_score_rows(const uint16_t *H, const uint16_t *W, int64_t N, int64_t d, int64_t V,
                      const int32_t *target, int32_t *argmax, double *pmax, double *ptarget,
                      double *gap, double *maxlogit, double *logz, double *entropy, int nthreads)
{
    if (!H || !W || !argmax || !pmax || !ptarget || !gap || N < 0 || d < 1 || V < 1)
        return ORACLE_ERR_ARG;
    int err = ORACLE_OK;
#ifdef _OPENMP
    if (nthreads <= 0)
        nthreads = omp_get_max_threads();
#pragma omp parallel num_threads(nthreads)
#endif
    {
        double *logit = (double *)malloc((size_t)V * sizeof(double));
        if (!logit) {
#ifdef _OPENMP
#pragma omp atomic write
#endif
            err = ORACLE_ERR_NOMEM;
        }
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
        for (int64_t n = 0; n < N; ++n) {
            if (!logit)
                continue;
            oracle_logits_row(H + n * d, W, d, V, logit);
            int64_t a = 0;
            double m = logit[0];
            for (int64_t v = 1; v < V; ++v)
                if (logit[v] > m) {
                    m = logit[v];
                    a = v;
                }
            double second = -INFINITY;
            for (int64_t v = 0; v < V; ++v)
                if (v != a && logit[v] > second)
                    second = logit[v];
            double Z = 0.0;
            for (int64_t v = 0; v < V; ++v)
                Z += exp(logit[v] - m);
            argmax[n] = (int32_t)a;
            pmax[n] = 1.0 / Z;
            gap[n] = (V > 1) ? (m - second) : INFINITY;
            int64_t t = target ? (int64_t)target[n] : -1;
            ptarget[n] = (t >= 0 && t < V) ? exp(logit[t] - m) / Z : 0.0;
            if (maxlogit)
                maxlogit[n] = m;
            if (logz)
                logz[n] = m + log(Z);
            if (entropy) {
                double h = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    const double p = exp(logit[v] - m) / Z;
                    if (p > 0.0)
                        h -= p * log(p);
                }
                entropy[n] = h;
            }
        }
        free(logit);
    }
    return err;
}

/*
 * Targets of the scored rows for one step.  Rows are ordered [s][kind][l]
 * (kind 0 = current-block row, kind 1 = shadow-block verification row).
 * A verification row is scored against the token its position holds now,
 * y^(k-1) (Eq. 3); block rows and masked positions have no target (-1).
 */
int oracle_row_targets(const int32_t *tokens, int64_t n_seq, int64_t seq_len, int64_t blk_start,
                       int64_t blk_len, int32_t mask_id, int32_t *target)
{
    if (!tokens || !target || n_seq < 0 || blk_len < 1 || blk_start < 0 || blk_start + blk_len > seq_len)
        return ORACLE_ERR_ARG;
    for (int64_t s = 0; s < n_seq; ++s)
        for (int64_t l = 0; l < blk_len; ++l) {
            int32_t y = tokens[s * seq_len + blk_start + l];
            target[(s * 2 + 0) * blk_len + l] = -1;
            target[(s * 2 + 1) * blk_len + l] = (y == mask_id) ? -1 : y;
        }
    return ORACLE_OK;
}

/* Per-position outcome codes written to flags[] (0 = unchanged). */
#define ORACLE_FLAG_DRAFT 1          /* drafted: pmax > tau1 (Eq. 2)                 */
#define ORACLE_FLAG_DRAFT_FALLBACK 2 /* drafted by the at-least-one rule (Eq. 1)     */
#define ORACLE_FLAG_REMASK 3         /* re-masked: p(current token) < tau2 (Eq. 3)   */
#define ORACLE_FLAG_DRAFT_IS_MASK 4  /* selected for drafting but argmax is MASK     */
#define ORACLE_FLAG_DRAFT_TOP_M 5    /* drafted by the fixed-M rule (Sec. 3)         */

/*
 * One WINO step, Eq. 4, on every sequence's current block [blk_start,
 * blk_start + blk_len), in place on tokens[n_seq, seq_len].
 *   D = { l : y_l == MASK and pmax(block row l) > tau1 }                  (Eq. 2)
 *   if D is empty and some y_l == MASK:
 *       D = { the masked l with the largest pmax(block row l);
 *             the smallest such l on ties }                                (Eq. 1)
 *   R = { l : y_l != MASK and ptarget(shadow row l) < tau2 }              (Eq. 3)
 *   y_l <- argmax(block row l) for l in D; y_l <- MASK for l in R.
 * Both conditions read y^(k-1), so D and R are disjoint and the update is
 * simultaneous.  counts[s] = {drafted (MASK -> token), re-masked, MASKs left
 * in the block}; flags[s * blk_len + l] (optional) gets the outcome codes.
 * With freeze_finished != 0, a sequence whose block has no MASK is not
 * stepped at all: its loop, which runs until the block has no MASK (Sec. 4.2.3), has ended
 * for it.  If last_change (int32 [n_seq, seq_len]) is given, every position
 * whose token this step changes is set to step_index.
 *
 * no_shadow != 0 is WINO+ inference (Sec. 5.3, Sec. 6.1.2): there is no
 * shadow block, the rows are the block rows only ([s][l], row s*blk_len + l),
 * drafting uses the single threshold tau1 with the same at-least-one rule,
 * and R is empty (ptarget may be NULL).
 *
 * draft_m > 0 replaces the drafting rule by naive parallel sampling (Sec. 3,
 * the fixed number of tokens per step of Sec. 6.3.3): D is the min(M, #MASK)
 * masked positions with the largest pmax(block row l), the smallest l first
 * among equal pmax; tau1 is not used.  M = 1 is high-confidence greedy
 * decoding (Eq. 1).  Verification is unchanged (off with no_shadow).
 */
int oracle_draft_verify(int32_t *tokens, int64_t n_seq, int64_t seq_len, int64_t blk_start,
                        int64_t blk_len, int32_t mask_id, double tau1, double tau2,
                        const int32_t *argmax, const double *pmax, const double *ptarget,
                        int32_t *counts, int8_t *flags, int freeze_finished, int no_shadow, int32_t step_index,
                        int32_t *last_change, int64_t draft_m)
{
    if (!tokens || !argmax || !pmax || (!ptarget && !no_shadow) || !counts || n_seq < 0 || blk_len < 1 ||
        blk_start < 0 || blk_start + blk_len > seq_len)
        return ORACLE_ERR_ARG;
    int32_t *prev = (int32_t *)malloc((size_t)blk_len * sizeof(int32_t));
    int8_t *inD = (int8_t *)malloc((size_t)blk_len);
    int8_t *inR = (int8_t *)malloc((size_t)blk_len);
    if (!prev || !inD || !inR) {
        free(prev);
        free(inD);
        free(inR);
        return ORACLE_ERR_NOMEM;
    }
    for (int64_t s = 0; s < n_seq; ++s) {
        int32_t *y = tokens + s * seq_len + blk_start;
        const int64_t row_blk = no_shadow ? s * blk_len : (s * 2 + 0) * blk_len; /* kind 0: Y_cur rows  */
        const int64_t row_shd = (s * 2 + 1) * blk_len;                           /* kind 1: Y_shad rows */
        int64_t n_draft = 0, n_mask = 0;
        for (int64_t l = 0; l < blk_len; ++l) {
            prev[l] = y[l];
            inD[l] = (draft_m <= 0) && (prev[l] == mask_id) && (pmax[row_blk + l] > tau1);
            inR[l] = !no_shadow && (prev[l] != mask_id) && (ptarget[row_shd + l] < tau2);
            n_draft += inD[l];
            n_mask += (prev[l] == mask_id);
        }
        if (freeze_finished && n_mask == 0) {
            for (int64_t l = 0; l < blk_len; ++l)
                if (flags)
                    flags[s * blk_len + l] = 0;
            counts[s * 3 + 0] = counts[s * 3 + 1] = counts[s * 3 + 2] = 0;
            continue;
        }
        int64_t fallback = -1;
        if (draft_m > 0) {
            /* the M most confident masked positions: M times, take the best one not yet taken */
            for (int64_t j = 0; j < draft_m && j < n_mask; ++j) {
                int64_t pick = -1;
                for (int64_t l = 0; l < blk_len; ++l)
                    if (prev[l] == mask_id && !inD[l] && (pick < 0 || pmax[row_blk + l] > pmax[row_blk + pick]))
                        pick = l;
                inD[pick] = 1;
            }
        } else if (n_draft == 0 && n_mask > 0) {
            double best = -INFINITY;
            for (int64_t l = 0; l < blk_len; ++l)
                if (prev[l] == mask_id && (fallback < 0 || pmax[row_blk + l] > best)) {
                    best = pmax[row_blk + l];
                    fallback = l;
                }
            inD[fallback] = 1;
        }
        int32_t drafted = 0, remasked = 0, left = 0;
        for (int64_t l = 0; l < blk_len; ++l) {
            int8_t code = 0;
            int32_t before = y[l];
            if (inD[l]) {
                y[l] = argmax[row_blk + l];
                if (y[l] == mask_id)
                    code = ORACLE_FLAG_DRAFT_IS_MASK;
                else {
                    code = (draft_m > 0) ? ORACLE_FLAG_DRAFT_TOP_M
                                         : (l == fallback) ? ORACLE_FLAG_DRAFT_FALLBACK : ORACLE_FLAG_DRAFT;
                    ++drafted;
                }
            } else if (inR[l]) {
                y[l] = mask_id;
                code = ORACLE_FLAG_REMASK;
                ++remasked;
            }
            left += (y[l] == mask_id);
            if (last_change && y[l] != before)
                last_change[s * seq_len + blk_start + l] = step_index;
            if (flags)
                flags[s * blk_len + l] = code;
        }
        counts[s * 3 + 0] = drafted;
        counts[s * 3 + 1] = remasked;
        counts[s * 3 + 2] = left;
    }
    free(prev);
    free(inD);
    free(inR);
    return ORACLE_OK;
}

/*
 * Whole step as the method runs it once per forward pass: gather the rows'
 * targets from the current state, score every row, apply Eq. 4.  Scratch for
 * the per-row statistics is allocated here; the caller may ask for them back
 * (any of argmax_out/pmax_out/ptarget_out/gap_out may be NULL).
 */
int oracle_step(const uint16_t *H, const uint16_t *W, int64_t d, int64_t V, int32_t *tokens, int64_t n_seq,
                int64_t seq_len, int64_t blk_start, int64_t blk_len, int32_t mask_id, double tau1, double tau2,
                int32_t *counts, int8_t *flags, int32_t *argmax_out, double *pmax_out, double *ptarget_out,
                double *gap_out, int nthreads, int freeze_finished, int no_shadow, int32_t step_index,
                int32_t *last_change, int64_t draft_m)
{
    const int64_t N = n_seq * (no_shadow ? 1 : 2) * blk_len;
    int32_t *target = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *am = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    double *pm = (double *)malloc((size_t)N * sizeof(double));
    double *pt = (double *)malloc((size_t)N * sizeof(double));
    double *gp = (double *)malloc((size_t)N * sizeof(double));
    int rc = ORACLE_ERR_NOMEM;
    if (target && am && pm && pt && gp) {
        if (no_shadow) {  /* block rows only: no row has a target */
            for (int64_t n = 0; n < N; ++n)
                target[n] = -1;
            rc = ORACLE_OK;
        } else {
            rc = oracle_row_targets(tokens, n_seq, seq_len, blk_start, blk_len, mask_id, target);
        }
        if (rc == ORACLE_OK)
            rc = oracle_score_rows(H, W, N, d, V, target, am, pm, pt, gp, NULL, NULL, NULL, nthreads);
        if (rc == ORACLE_OK)
            rc = oracle_draft_verify(tokens, n_seq, seq_len, blk_start, blk_len, mask_id, tau1, tau2, am, pm,
                                     pt, counts, flags, freeze_finished, no_shadow, step_index, last_change,
                                     draft_m);
        if (rc == ORACLE_OK) {
            if (argmax_out)
                memcpy(argmax_out, am, (size_t)N * sizeof(int32_t));
            if (pmax_out)
                memcpy(pmax_out, pm, (size_t)N * sizeof(double));
            if (ptarget_out)
                memcpy(ptarget_out, pt, (size_t)N * sizeof(double));
            if (gap_out)
                memcpy(gap_out, gp, (size_t)N * sizeof(double));
        }
    }
    free(target);
    free(am);
    free(pm);
    free(pt);
    free(gp);
    return rc;
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
