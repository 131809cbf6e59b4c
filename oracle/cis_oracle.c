/*
 * cis_oracle.c -- fp64 CPU oracle for the calibrated-importance-sampling (CIS)
 * token loss of arxiv 2609.32444.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * statement of what the GPU path computes.  Only the test suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it.  It shares no
 * header, helper, table or constant generator with the CUDA library, and the
 * CUDA library never calls it.
 *
 * Every quantity is computed in IEEE double precision with plain loops over
 * the vocabulary: an exact maximum, then a plain sum of exp(z - max) -- no
 * online rescaling, no blocking, no fusion.  Rows are independent, so rows
 * are spread over host threads with OpenMP; each row is still computed by a
 * single thread in index order, so results do not depend on the thread count.
 *
 * Passages followed (section / equation / algorithm of the paper):
 *   - Sec. 2.1 and Sec. 3.1: p_t = softmax(z)_{y_t}, the probability the
 *     training engine gives the sampled token; log p_t = z_y - logsumexp(z).
 *   - Eq. 1: token-level GRPO surrogate with the PPO clip and the mismatch
 *     weight k_t; normaliser (1/G) sum_i 1/|y_i|.
 *   - Algorithm 1 (Sec. 3.3): p = exp(l_train), k = exp(l_train - l_infer),
 *     phi = max(1 - p, kappa), f = min{k, 1 + lambda*phi}; the estimate is
 *     (1/n) sum stopgrad(f_m) l'_m.
 *   - Table 8 (App. C.1): the other weight operators and their defaults:
 *     exact ratio clamped to [1e-6, 1e6]; TIS min(k, C); IcePop k 1{k in
 *     [a, b]}; KPop-dagger k 1{max(KL_B(p||q), KL_B(q||p)) <= phi}, fp64, with
 *     p and q clamped to [1e-8, 1 - 1e-8] (App. D.5, "The KL mask and
 *     probability saturation"); Seq-TIS min(K, C) and Seq-MIS K 1{K in [a, b]}
 *     with K the product of k over a response; no correction.
 *   - Sec. 4.3 / App. C.1: the two-sided band max{min{k, 1 + lambda phi},
 *     (1 + p)/2}, the image of e^eps >= 1/2 under k = p + (1 - p) e^eps.
 *   - Lemma 3.1 / Lemma B.1: eps_t = logit p_t - logit q_t.
 *   - App. D (training statistics): the entropy of the training policy,
 *     -sum_j p_j log p_j per token.
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   - the truncation flag is "k > cap", decided in fp64 in the log domain:
 *     log k = l_w - l_inf (exact in fp64 for fp32 inputs) against log(cap);
 *   - 1 - p is evaluated as -expm1(log p);
 *   - the loss is the negated objective, so d loss / d z = c (softmax - onehot);
 *   - in min(rho*A, clip(rho)*A) a tie takes the unclipped branch, so the
 *     gradient flows at rho = 1 +- c exactly;
 *   - a NaN ratio gives a NaN weight (NaN propagates; min{NaN, cap} is not
 *     read as cap);
 *   - "truncated" means the operator changed the weight: capped, clamped,
 *     lifted (band) or masked (IcePop, KPop, Seq-MIS); for the sequence
 *     operators every token of a response gets the response's flag;
 *   - the sequence operators take the product over the valid tokens of each
 *     response (cu_seqlens), as a sum of log k in index order; a valid token
 *     outside every response gets weight 0; a token with an out-of-range id
 *     is left out of its response's product;
 *   - KPop: 1 - p is 1 - (clamped p), and the mask is "metric > phi".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Weight operators (Table 8 of the paper, plus CIS of Algorithm 1). */
enum {
    OR_MODE_CIS = 0,     /* min{k, 1 + lambda*max(1-p, kappa)}      Algorithm 1  */
    OR_MODE_TIS = 1,     /* min(k, C)                                Table 8      */
    OR_MODE_EXACT = 2,   /* k clamped to [lo, hi]                    Table 8      */
    OR_MODE_NONE = 3,    /* 1                                        Table 8      */
    OR_MODE_BAND = 4,    /* max{min{k, 1 + lambda phi}, (1 + p)/2}   Sec. 4.3     */
    OR_MODE_ICEPOP = 5,  /* k 1{k in [a, b]}                         Table 8      */
    OR_MODE_KPOP = 6,    /* k 1{max binary KL <= phi}                Table 8      */
    OR_MODE_SEQ_TIS = 7, /* min(K, C), K = prod of k over a response Table 8      */
    OR_MODE_SEQ_MIS = 8  /* K 1{K in [a, b]}                         Table 8      */
};

enum { OR_AGG_TOKEN_MEAN = 0, OR_AGG_SEQ_MEAN = 1 };

/* Hyper-parameters, all in double precision. */
typedef struct {
    int32_t mode;
    int32_t agg;
    double lambda;    /* CIS threshold on e^eps, Eq. 4                 */
    double kappa;     /* floor on 1 - p, Algorithm 1                   */
    double tis_cap;   /* C of TIS                                      */
    double exact_lo;  /* clamp of the exact ratio                      */
    double exact_hi;
    double clip_low;  /* PPO clip range [1 - c_low, 1 + c_high], Eq. 1 */
    double clip_high;
    double icepop_lo; /* IcePop band [a, b]                            */
    double icepop_hi;
    double kpop_phi;  /* KPop threshold on the binary KL               */
    double seq_cap;   /* C of Seq-TIS                                  */
    double seq_lo;    /* Seq-MIS band [a, b]                           */
    double seq_hi;
    int64_t n_global; /* > 0: the batch's valid tokens, when these rows
                       * are one shard of it (token mean); 0: these rows' */
    int64_t g_global; /* > 0: the batch's responses with a valid token
                       * (sequence mean); 0: these rows'                */
} oracle_params_t;

static int is_seq_mode(int mode)
{
    return mode == OR_MODE_SEQ_TIS || mode == OR_MODE_SEQ_MIS;
}

/* bf16 is the top half of an IEEE binary32; the upcast is exact. */
static double bf16_to_double(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Logit (t, j): dtype 0 = float32, 1 = bf16 bit patterns, 2 = float64. */
static double logit_at(const void *logits, int dtype, int64_t ld, int64_t t, int64_t j)
{
    if (dtype == 0)
        return (double)((const float *)logits)[t * ld + j];
    if (dtype == 2)
        return ((const double *)logits)[t * ld + j];
    return bf16_to_double(((const uint16_t *)logits)[t * ld + j]);
}

static int row_valid(const uint8_t *mask, int64_t t)
{
    return mask == NULL || mask[t] != 0;
}

/*
 * logsumexp of one row, by its definition: M = max_j z_j, then
 * lse = M + log(sum_j exp(z_j - M)).  Sec. 2.1 / 3.1 (softmax of the logits).
 */
static double row_lse(const void *logits, int dtype, int64_t ld, int64_t t, int64_t V)
{
    double M = -INFINITY;
    int any_nan = 0;
    for (int64_t j = 0; j < V; ++j) {
        double z = logit_at(logits, dtype, ld, t, j);
        if (isnan(z))
            any_nan = 1;
        if (z > M)
            M = z;
    }
    if (any_nan)
        return NAN;
    if (M == -INFINITY)
        return -INFINITY;
    double S = 0.0;
    for (int64_t j = 0; j < V; ++j)
        S += exp(logit_at(logits, dtype, ld, t, j) - M);
    return M + log(S);
}

static void set_threads(int nthreads)
{
#ifdef _OPENMP
    if (nthreads > 0)
        omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/*
 * Sampled-token log-probabilities: lp_t = z_{t,y_t} - lse_t, i.e. log p_t with
 * p_t = softmax(z_t)_{y_t} (Sec. 2.1, Sec. 3.1).  Masked rows are not read and
 * get lp = lse = 0.  Returns 0, or -1 if a valid row has an id outside [0, V)
 * (that row then gets NaN).
 */
int oracle_token_logprobs(const void *logits, int dtype, int64_t T, int64_t V, int64_t ld,
                          const int32_t *ids, const uint8_t *mask, double *lp_out,
                          double *lse_out, int nthreads)
{
    int bad = 0;
    set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 4) reduction(| : bad)
    for (int64_t t = 0; t < T; ++t) {
        double lp = 0.0, lse = 0.0;
        if (row_valid(mask, t)) {
            int32_t y = ids[t];
            if (y < 0 || (int64_t)y >= V) {
                bad = 1;
                lp = NAN;
                lse = NAN;
            } else {
                lse = row_lse(logits, dtype, ld, t, V);
                lp = logit_at(logits, dtype, ld, t, y) - lse;
            }
        }
        lp_out[t] = lp;
        if (lse_out)
            lse_out[t] = lse;
    }
    return bad ? -1 : 0;
}

/*
 * Entropy of each row's softmax, H_t = -sum_j p_tj log p_tj with
 * log p_tj = z_tj - lse_t (the training-side entropy the paper logs, App. D);
 * entries with p = 0 add nothing (0 log 0 = 0).  Masked rows get 0.
 */
void oracle_token_entropy(const void *logits, int dtype, int64_t T, int64_t V, int64_t ld,
                          const uint8_t *mask, double *h_out, int nthreads)
{
    set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 4)
    for (int64_t t = 0; t < T; ++t) {
        double h = 0.0;
        if (row_valid(mask, t)) {
            double lse = row_lse(logits, dtype, ld, t, V);
            for (int64_t j = 0; j < V; ++j) {
                double lpj = logit_at(logits, dtype, ld, t, j) - lse;
                double pj = exp(lpj);
                if (pj != 0.0 || isnan(pj))
                    h -= pj * lpj;
            }
        }
        h_out[t] = h;
    }
}

/*
 * One token's weight, Algorithm 1 and Table 8.
 *   lw   : log p used by the weight (training side), double
 *   linf : log q (inference side, the raw sampling-step value), double
 * Outputs the weight, the truncation flag, log k and eps.
 */
static void token_weight(double lw, double linf, const oracle_params_t *P, double *w,
                         int *trunc, double *logk_out, double *eps_out)
{
    /* Algorithm 1: p <- exp(l_train), k <- exp(l_train - l_infer).
     * 1 - p is evaluated as -expm1(l_train), the same number without the
     * cancellation of 1 - exp(l) when p is close to 1. */
    double logk = lw - linf;
    double k = exp(logk);
    double one_minus_p = -expm1(lw);
    double wt = 1.0;
    int tr = 0;
    switch (P->mode) {
    case OR_MODE_CIS: {
        /* phi <- max(1 - p, kappa);  f <- min{k, 1 + lambda*phi}. */
        double phi = one_minus_p > P->kappa ? one_minus_p : P->kappa;
        double cap = 1.0 + P->lambda * phi;
        wt = isnan(k) ? k : (k < cap ? k : cap);
        tr = logk > log1p(P->lambda * phi);
        break;
    }
    case OR_MODE_TIS: {
        /* Table 8: min(k, C). */
        double cap = P->tis_cap;
        wt = isnan(k) ? k : (k < cap ? k : cap);
        tr = logk > log(cap);
        break;
    }
    case OR_MODE_EXACT: {
        /* Table 8: k, clamped to [lo, hi]. */
        wt = k;
        if (wt > P->exact_hi)
            wt = P->exact_hi;
        if (wt < P->exact_lo)
            wt = P->exact_lo;
        tr = logk > log(P->exact_hi) || logk < log(P->exact_lo);
        break;
    }
    case OR_MODE_BAND: {
        /* Sec. 4.3: the CIS weight, lifted from below to (1 + p)/2. */
        double phi = one_minus_p > P->kappa ? one_minus_p : P->kappa;
        double cap = 1.0 + P->lambda * phi;
        double p = exp(lw);
        double lo = 0.5 * (1.0 + p);
        double capped = isnan(k) ? k : (k < cap ? k : cap);
        wt = isnan(capped) ? capped : (capped > lo ? capped : lo);
        tr = logk > log1p(P->lambda * phi) || logk < log(lo);
        break;
    }
    case OR_MODE_ICEPOP: {
        /* Table 8: k kept on [a, b] (bounds included), else masked to 0. */
        int out = logk < log(P->icepop_lo) || logk > log(P->icepop_hi);
        wt = out ? 0.0 : k;
        tr = out;
        break;
    }
    case OR_MODE_KPOP: {
        /* Table 8 / App. D.5: binary KL both ways, fp64, p and q clamped to
         * [1e-8, 1 - 1e-8]; masked when the larger exceeds phi. */
        const double lo = 1e-8, hi = 1.0 - 1e-8;
        double p = exp(lw), q = exp(linf);
        p = p < lo ? lo : (p > hi ? hi : p);
        q = q < lo ? lo : (q > hi ? hi : q);
        double kl_pq = p * log(p / q) + (1.0 - p) * log((1.0 - p) / (1.0 - q));
        double kl_qp = q * log(q / p) + (1.0 - q) * log((1.0 - q) / (1.0 - p));
        double m = kl_pq > kl_qp ? kl_pq : kl_qp;
        int out = m > P->kpop_phi;
        wt = out ? 0.0 : k;
        tr = out;
        break;
    }
    case OR_MODE_SEQ_TIS:
    case OR_MODE_SEQ_MIS:
        /* sequence operators: the weight comes from the response's product */
        wt = 0.0;
        tr = 0;
        break;
    default: /* OR_MODE_NONE: weight 1. */
        wt = 1.0;
        tr = 0;
        break;
    }
    *w = wt;
    *trunc = tr;
    if (logk_out)
        *logk_out = logk;
    if (eps_out) {
        /* Lemma 3.1: eps = logit p - logit q
         *               = (log p - log(1-p)) - (log q - log(1-q)). */
        double one_minus_q = -expm1(linf);
        *eps_out = (lw - log(one_minus_p)) - (linf - log(one_minus_q));
    }
}

/*
 * The weight of every token of a response from the response's log K =
 * sum of log k over its valid tokens (Table 8: Seq-TIS min(K, C), Seq-MIS
 * K 1{K in [a, b]}).
 */
static void seq_weight(double logK, const oracle_params_t *P, double *w, int *trunc)
{
    double K = exp(logK);
    if (P->mode == OR_MODE_SEQ_TIS) {
        double cap = P->seq_cap;
        *w = isnan(K) ? K : (K < cap ? K : cap);
        *trunc = logK > log(cap);
    } else {
        int out = logK < log(P->seq_lo) || logK > log(P->seq_hi);
        *w = out ? 0.0 : K;
        *trunc = out;
    }
}

/*
 * Weights for T tokens (Algorithm 1 / Table 8).  Masked tokens get w = 0,
 * trunc = 0, logk = eps = 0.  The sequence operators need cu_seqlens (B + 1
 * offsets); `skip` (may be NULL) marks tokens left out of the products.
 * Returns 0, or -1 for a sequence operator without cu_seqlens.
 */
static int weights_impl(const double *lp_w, const double *lp_inf, const uint8_t *mask,
                        const uint8_t *skip, int64_t T, const int32_t *cu_seqlens, int64_t B,
                        const oracle_params_t *P, double *w_out, uint8_t *trunc_out,
                        double *logk_out, double *eps_out)
{
    if (is_seq_mode(P->mode) && cu_seqlens == NULL)
        return -1;
    double *lk = (double *)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
    if (!lk)
        return -2;
    for (int64_t t = 0; t < T; ++t) {
        double w = 0.0, e = 0.0;
        int tr = 0;
        lk[t] = 0.0;
        if (row_valid(mask, t))
            token_weight(lp_w[t], lp_inf[t], P, &w, &tr, &lk[t], &e);
        w_out[t] = w;
        if (trunc_out)
            trunc_out[t] = (uint8_t)tr;
        if (logk_out)
            logk_out[t] = lk[t];
        if (eps_out)
            eps_out[t] = e;
    }
    if (is_seq_mode(P->mode)) {
        for (int64_t i = 0; i < B; ++i) {
            double logK = 0.0;
            for (int64_t t = cu_seqlens[i]; t < cu_seqlens[i + 1]; ++t)
                if (row_valid(mask, t) && !(skip && skip[t]))
                    logK += lk[t];
            double w;
            int tr;
            seq_weight(logK, P, &w, &tr);
            for (int64_t t = cu_seqlens[i]; t < cu_seqlens[i + 1]; ++t)
                if (row_valid(mask, t) && !(skip && skip[t])) {
                    w_out[t] = w;
                    if (trunc_out)
                        trunc_out[t] = (uint8_t)tr;
                }
        }
    }
    free(lk);
    return 0;
}

int oracle_weights(const double *lp_w, const double *lp_inf, const uint8_t *mask, int64_t T,
                   const int32_t *cu_seqlens, int64_t B, const oracle_params_t *P,
                   double *w_out, uint8_t *trunc_out, double *logk_out, double *eps_out)
{
    return weights_impl(lp_w, lp_inf, mask, NULL, T, cu_seqlens, B, P, w_out, trunc_out,
                        logk_out, eps_out);
}

/*
 * Per-token loss scale s_t.
 *   token mean (Algorithm 1): s_t = m_t / n, n = number of valid tokens;
 *   sequence mean (Eq. 1):    s_t = m_t / (G * |y_i|) for token t of response
 *                             i, |y_i| = valid tokens of i, G = responses with
 *                             at least one valid token.  Tokens outside every
 *                             response get 0.
 * n and G are counts over the whole batch (Algorithm 1's 1/n, Eq. 1's 1/G):
 * when these T rows are one shard of a batch, n_global / g_global (> 0) give
 * the batch's counts; 0 means these rows are the batch.
 */
void oracle_loss_scales_global(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                               int64_t B, int agg, int64_t n_global, int64_t g_global,
                               double *s_out)
{
    if (agg == OR_AGG_SEQ_MEAN && cu_seqlens != NULL) {
        int64_t G = 0;
        for (int64_t i = 0; i < B; ++i) {
            int64_t n = 0;
            for (int64_t t = cu_seqlens[i]; t < cu_seqlens[i + 1]; ++t)
                n += row_valid(mask, t);
            G += n > 0;
        }
        if (g_global > 0)
            G = g_global;
        for (int64_t t = 0; t < T; ++t)
            s_out[t] = 0.0;
        for (int64_t i = 0; i < B; ++i) {
            int64_t n = 0;
            for (int64_t t = cu_seqlens[i]; t < cu_seqlens[i + 1]; ++t)
                n += row_valid(mask, t);
            for (int64_t t = cu_seqlens[i]; t < cu_seqlens[i + 1]; ++t)
                s_out[t] = row_valid(mask, t) ? 1.0 / ((double)G * (double)n) : 0.0;
        }
        return;
    }
    int64_t n = 0;
    for (int64_t t = 0; t < T; ++t)
        n += row_valid(mask, t);
    if (n_global > 0)
        n = n_global;
    for (int64_t t = 0; t < T; ++t)
        s_out[t] = (n > 0 && row_valid(mask, t)) ? 1.0 / (double)n : 0.0;
}

void oracle_loss_scales(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens, int64_t B,
                        int agg, double *s_out)
{
    oracle_loss_scales_global(mask, T, cu_seqlens, B, agg, 0, 0, s_out);
}

/*
 * The weighted policy-gradient token loss and its gradient with respect to
 * the logits.
 *
 *   rho_t = exp(l_t - l_old,t)        (update ratio, Eq. 1; = 1 in value when
 *                                      no l_old is given, gradient still flows)
 *   J_t   = w_t * min(rho_t A_t, clip(rho_t, 1-c_low, 1+c_high) A_t)   (Eq. 1)
 *   loss  = -sum_t s_t J_t
 *   w_t   = stopgrad weight of Algorithm 1 / Table 8, from l_old if given,
 *           else from the current l_t (detached)
 *   d loss / d z_tj = c_t (softmax_j - [j == y_t]),
 *   c_t   = s_t w_t A_t rho_t g_t, g_t = 1 if the unclipped branch is taken.
 *
 * Inputs in double (the Python wrapper upcasts fp32 exactly).  lp_old, w_fixed
 * may be NULL.  w_fixed replaces the computed weights (used to freeze them for
 * finite differences).  dz is written for the rows listed in `rows` (nrows of
 * them, dz_out is [nrows, V]); rows == NULL means every row (dz_out [T, V]).
 * Per-token outputs (lp, lse, w, trunc, loss_terms, c, logk) are for all T
 * rows; logk_out and stats_out may be NULL.
 *
 * stats_out[0..3] are the batch statistics the paper logs while training
 * (App. D: how many tokens the correction acted on, the largest |log k_t|)
 * and the truncated excess of Lemma B.2 (k - f, the ratio mass a capped
 * token loses):
 *   [0] n_valid      number of valid tokens;
 *   [1] n_truncated  valid tokens whose weight the operator changed;
 *   [2] max_abs_logk max over valid tokens of |log k_t|, log k_t = l_w - l_inf
 *                    (a token whose log k is not a number -- an out-of-range
 *                    id, a NaN logit -- is left out; 0 when none is left);
 *   [3] trunc_excess sum over truncated tokens of (k_t - w_t), k_t = exp(log
 *                    k_t) the token's own ratio, in index order.
 * Returns 0, -1 if a valid row has an out-of-range id, -3 for a sequence
 * operator without cu_seqlens.
 */
int oracle_loss_fwd_bwd(const void *logits, int dtype, int64_t T, int64_t V, int64_t ld,
                        const int32_t *ids, const double *lp_inf, const double *lp_old,
                        const double *adv, const uint8_t *mask, const int32_t *cu_seqlens,
                        int64_t B, const oracle_params_t *P, const double *w_fixed,
                        const int64_t *rows, int64_t nrows, double *dz_out, double *lp_out,
                        double *lse_out, double *w_out, uint8_t *trunc_out,
                        double *loss_terms, double *c_out, double *loss_out, double *logk_out,
                        double *stats_out, int nthreads)
{
    size_t nT = (size_t)(T > 0 ? T : 1);
    double *s = (double *)malloc(sizeof(double) * nT);
    double *lse = (double *)malloc(sizeof(double) * nT);
    double *cc = (double *)malloc(sizeof(double) * nT);
    double *terms = (double *)malloc(sizeof(double) * nT);
    if (!s || !lse || !cc || !terms) {
        free(s);
        free(lse);
        free(cc);
        free(terms);
        return -2;
    }
    oracle_loss_scales_global(mask, T, cu_seqlens, B, P->agg, P->n_global, P->g_global, s);
    double *lpv = (double *)malloc(sizeof(double) * nT);
    double *lwv = (double *)malloc(sizeof(double) * nT);
    double *wv = (double *)malloc(sizeof(double) * nT);
    uint8_t *trv = (uint8_t *)malloc(nT);
    uint8_t *badv = (uint8_t *)malloc(nT);
    double *lkv = (double *)malloc(sizeof(double) * nT);
    if (!lpv || !lwv || !wv || !trv || !badv || !lkv) {
        free(s);
        free(lse);
        free(cc);
        free(terms);
        free(lpv);
        free(lwv);
        free(wv);
        free(trv);
        free(badv);
        free(lkv);
        return -2;
    }
    int bad = 0;
    set_threads(nthreads);
    /* 1. log p of every valid row (Sec. 2.1) */
#pragma omp parallel for schedule(dynamic, 4) reduction(| : bad)
    for (int64_t t = 0; t < T; ++t) {
        double lp = 0.0, ls = 0.0;
        badv[t] = 0;
        if (row_valid(mask, t)) {
            int32_t y = ids[t];
            if (y < 0 || (int64_t)y >= V) {
                bad = 1;
                badv[t] = 1;
                lp = NAN;
                ls = NAN;
            } else {
                ls = row_lse(logits, dtype, ld, t, V);
                lp = logit_at(logits, dtype, ld, t, y) - ls;
            }
        }
        lse[t] = ls;
        lpv[t] = lp;
        lwv[t] = lp_old ? lp_old[t] : lp;
    }
    /* 2. the weights (Algorithm 1 / Table 8), per token or per response */
    int rc = weights_impl(lwv, lp_inf, mask, badv, T, cu_seqlens, B, P, wv, trv, lkv, NULL);
    if (rc != 0) {
        free(s);
        free(lse);
        free(cc);
        free(terms);
        free(lpv);
        free(lwv);
        free(wv);
        free(trv);
        free(badv);
        free(lkv);
        return rc == -1 ? -3 : -2;
    }
    /* 3. the token terms of Eq. 1 and c_t */
    for (int64_t t = 0; t < T; ++t) {
        double w = 0.0, term = 0.0, c = 0.0;
        int tr = 0;
        if (row_valid(mask, t)) {
            if (badv[t]) {
                term = NAN;
            } else {
                double lp = lpv[t];
                w = w_fixed ? w_fixed[t] : wv[t];
                tr = trv[t];
                /* Eq. 1: rho = pi_theta / p_old, clipped to [1-c_low, 1+c_high]. */
                double rho = lp_old ? exp(lp - lp_old[t]) : 1.0;
                double A = adv[t];
                double rho_c = rho;
                if (rho_c < 1.0 - P->clip_low)
                    rho_c = 1.0 - P->clip_low;
                if (rho_c > 1.0 + P->clip_high)
                    rho_c = 1.0 + P->clip_high;
                double unclipped = rho * A;
                double clipped = rho_c * A;
                int g = unclipped <= clipped; /* the min takes the unclipped branch */
                double obj = g ? unclipped : clipped;
                term = -s[t] * w * obj;
                c = s[t] * w * A * rho * (double)g;
            }
        }
        cc[t] = c;
        terms[t] = term;
        lp_out[t] = lpv[t];
        if (w_out)
            w_out[t] = w;
        if (trunc_out)
            trunc_out[t] = (uint8_t)tr;
        wv[t] = w;
        trv[t] = (uint8_t)tr;
    }
    /* 4. the batch statistics (App. D training statistics; Lemma B.2's k - f),
     * over the valid tokens in index order */
    {
        double n_valid = 0.0, n_trunc = 0.0, max_abs = 0.0, excess = 0.0;
        for (int64_t t = 0; t < T; ++t) {
            if (!row_valid(mask, t))
                continue;
            n_valid += 1.0;
            if (!badv[t] && !isnan(lkv[t]) && fabs(lkv[t]) > max_abs)
                max_abs = fabs(lkv[t]);
            if (trv[t]) {
                n_trunc += 1.0;
                excess += exp(lkv[t]) - wv[t];
            }
        }
        if (stats_out) {
            stats_out[0] = n_valid;
            stats_out[1] = n_trunc;
            stats_out[2] = max_abs;
            stats_out[3] = excess;
        }
        if (logk_out)
            for (int64_t t = 0; t < T; ++t)
                logk_out[t] = !row_valid(mask, t) ? 0.0 : (badv[t] ? NAN : lkv[t]);
    }
    free(lpv);
    free(lwv);
    free(wv);
    free(trv);
    free(badv);
    free(lkv);
    /* loss = -sum_t s_t J_t, summed in index order. */
    double loss = 0.0;
    for (int64_t t = 0; t < T; ++t)
        loss += terms[t];
    if (loss_out)
        *loss_out = loss;
    if (loss_terms)
        memcpy(loss_terms, terms, sizeof(double) * (size_t)T);
    if (lse_out)
        memcpy(lse_out, lse, sizeof(double) * (size_t)T);
    if (c_out)
        memcpy(c_out, cc, sizeof(double) * (size_t)T);

    /* d loss / d z_tj = c_t (softmax_tj - [j == y_t]) for the requested rows. */
    if (dz_out) {
        int64_t nr = rows ? nrows : T;
#pragma omp parallel for schedule(dynamic, 1)
        for (int64_t r = 0; r < nr; ++r) {
            int64_t t = rows ? rows[r] : r;
            double *out = dz_out + r * V;
            int valid = t >= 0 && t < T && row_valid(mask, t);
            int32_t y = valid ? ids[t] : -1;
            if (!valid || y < 0 || (int64_t)y >= V) {
                for (int64_t j = 0; j < V; ++j)
                    out[j] = 0.0;
                continue;
            }
            for (int64_t j = 0; j < V; ++j) {
                double sm = exp(logit_at(logits, dtype, ld, t, j) - lse[t]);
                out[j] = cc[t] * (sm - (j == (int64_t)y ? 1.0 : 0.0));
            }
        }
    }
    free(s);
    free(lse);
    free(cc);
    free(terms);
    return bad ? -1 : 0;
}

/*
 * Mismatch diagnostics from the two engines' full logits (App. A.5 and
 * Sec. 4.3, Fig. 5c-d).  Per position t, with p = softmax(z_train),
 * q = softmax(z_infer), the normalised gauge delta_j = log q_j - log p_j
 * (App. A.5, "Gauge convention") and the sampled token y:
 *   eps_t   = -delta_y + log sum_{j != y} w_j exp(delta_j),
 *             w_j = e^{z_j} / sum_{j' != y} e^{z_j'}   (Lemma 3.1's definition)
 *   logk_t  = log p_y - log q_y,  p_t = p_y
 * and, for the weight operator f of `P` (a token operator) applied to every
 * candidate token j (k_j = p_j / q_j), with g_j = e_j - p the gradient of
 * log p_j with respect to the logits and expectations over y ~ q:
 *   bias2_t = || E_q[(f_y - k_y) g_y] ||^2
 *   dvar_t  = (E_q ||f_y g_y||^2 - ||E_q f_y g_y||^2) - (E_q ||g_y||^2 - ||E_q g_y||^2)
 * Both vectors are formed explicitly (a V-vector per position), not from a
 * closed form.  Masked rows get 0.  Returns 0, or -1 for a sequence operator
 * (the candidates of one position have no response to share).
 */
int oracle_mismatch_diagnostics(const void *z_train, const void *z_infer, int dtype, int64_t T,
                                int64_t V, int64_t ld, const int32_t *ids, const uint8_t *mask,
                                const oracle_params_t *P, double *eps_out, double *logk_out,
                                double *p_out, double *bias2_out, double *dvar_out, int nthreads)
{
    if (is_seq_mode(P->mode))
        return -1;
    set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t t = 0; t < T; ++t) {
        double eps = 0.0, lk = 0.0, pt = 0.0, bias2 = 0.0, dvar = 0.0;
        if (row_valid(mask, t)) {
            const int64_t y = ids[t];
            const double lse = row_lse(z_train, dtype, ld, t, V);
            const double lsei = row_lse(z_infer, dtype, ld, t, V);
            double *lp = (double *)malloc(sizeof(double) * (size_t)V);
            double *lq = (double *)malloc(sizeof(double) * (size_t)V);
            double *bvec = (double *)malloc(sizeof(double) * (size_t)V);
            double *fvec = (double *)malloc(sizeof(double) * (size_t)V);
            double *gvec = (double *)malloc(sizeof(double) * (size_t)V);
            double *pv = (double *)malloc(sizeof(double) * (size_t)V);
            for (int64_t j = 0; j < V; ++j) {
                lp[j] = logit_at(z_train, dtype, ld, t, j) - lse;
                lq[j] = logit_at(z_infer, dtype, ld, t, j) - lsei;
                pv[j] = exp(lp[j]); /* p_j, the training softmax */
            }
            /* eps by Lemma 3.1's definition, in the normalised gauge */
            double Sy = 0.0, acc = 0.0;
            for (int64_t j = 0; j < V; ++j)
                if (j != y)
                    Sy += pv[j];
            for (int64_t j = 0; j < V; ++j)
                if (j != y)
                    acc += pv[j] / Sy * exp(lq[j] - lp[j]);
            eps = -(lq[y] - lp[y]) + log(acc);
            lk = lp[y] - lq[y];
            pt = exp(lp[y]);
            /* E_q[(f - k) g], E_q[f g], E_q[g] as V-vectors; second moments */
            double e_f2g2 = 0.0, e_g2 = 0.0;
            for (int64_t j = 0; j < V; ++j)
                bvec[j] = fvec[j] = gvec[j] = 0.0;
            for (int64_t yy = 0; yy < V; ++yy) {
                const double qy = exp(lq[yy]);
                if (qy == 0.0)
                    continue;
                double f, dummy_e;
                int tr;
                token_weight(lp[yy], lq[yy], P, &f, &tr, NULL, &dummy_e);
                const double ky = exp(lp[yy] - lq[yy]);
                double g2 = 0.0;
                for (int64_t j = 0; j < V; ++j) {
                    const double gj = (j == yy ? 1.0 : 0.0) - pv[j];
                    bvec[j] += qy * (f - ky) * gj;
                    fvec[j] += qy * f * gj;
                    gvec[j] += qy * gj;
                    g2 += gj * gj;
                }
                e_f2g2 += qy * f * f * g2;
                e_g2 += qy * g2;
            }
            double nb = 0.0, nf = 0.0, ng = 0.0;
            for (int64_t j = 0; j < V; ++j) {
                nb += bvec[j] * bvec[j];
                nf += fvec[j] * fvec[j];
                ng += gvec[j] * gvec[j];
            }
            bias2 = nb;
            dvar = (e_f2g2 - nf) - (e_g2 - ng);
            free(lp);
            free(lq);
            free(bvec);
            free(fvec);
            free(gvec);
            free(pv);
        }
        eps_out[t] = eps;
        logk_out[t] = lk;
        p_out[t] = pt;
        bias2_out[t] = bias2;
        dvar_out[t] = dvar;
    }
    return 0;
}

/* Confidence-binned sums (Sec. 4.3, Fig. 5b: the sampled tokens binned by
 * p_t, with E[k_t - f_t] in each bin; App. A.5: logarithmic bins of 1 - p_t).
 * Token t with mask 1 falls in bin b when edges[b] <= key[t] < edges[b + 1],
 * the last bin also taking key[t] == edges[nbins]; a NaN key or one outside
 * [edges[0], edges[nbins]] falls in no bin.  For each bin: the count and, for
 * each of the nv value arrays values[i * T .. i * T + T - 1], the fp64 sum over
 * its tokens, added in token order.  Plain loops: the definition written out. */
void oracle_binned_sums(const float *key, const uint8_t *mask, int64_t T, const double *edges,
                        int nbins, const float *values, int nv, int64_t *counts, double *sums)
{
    for (int b = 0; b < nbins; ++b) {
        counts[b] = 0;
        for (int i = 0; i < nv; ++i)
            sums[(int64_t)i * nbins + b] = 0.0;
    }
    for (int64_t t = 0; t < T; ++t) {
        if (!row_valid(mask, t))
            continue;
        const double x = (double)key[t];
        int bin = -1;
        for (int b = 0; b < nbins; ++b) {
            const int last = b == nbins - 1;
            if (x >= edges[b] && (x < edges[b + 1] || (last && x == edges[b + 1]))) {
                bin = b;
                break;
            }
        }
        if (bin < 0)
            continue;
        counts[bin] += 1;
        for (int i = 0; i < nv; ++i)
            sums[(int64_t)i * nbins + bin] += (double)values[(int64_t)i * T + t];
    }
}
