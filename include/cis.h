/*
 * cis.h -- C ABI of libcis, the GB300 (sm_103a) implementation of the
 * training-side token pass of calibrated importance sampling (CIS),
 * arxiv 2609.32444.
 *
 * The pass, per token t of a batch of T tokens over a vocabulary of V:
 *   1. log-softmax of the training logits z_t and the gather of the sampled
 *      token's log-probability  l_t = log softmax(z_t)_{y_t}     (Sec. 2.1);
 *   2. the mismatch weight w_t from l_t (or l_old,t) and the inference-side
 *      log-probability l_inf,t: CIS min{k, 1 + lambda*max(1-p, kappa)}
 *      (Eq. 4, Algorithm 1), TIS min(k, C), the exact ratio clamped to
 *      [lo, hi], or 1 (Table 8), with k = exp(l_w - l_inf), p = exp(l_w);
 *   3. the weighted, PPO-clipped policy-gradient token loss (Eq. 1), with the
 *      weight detached (stopgrad, Algorithm 1);
 *   4. its gradient with respect to the logits,
 *        dz_tj = c_t (softmax(z_t)_j - [j == y_t]),
 *        c_t   = s_t m_t w_t A_t rho_t g_t,
 *      s_t the normaliser, m_t the mask, A_t the advantage, rho_t the update
 *      ratio and g_t = 0 where the PPO clip is active.
 *
 * Conventions shared by every entry point:
 *   - Pointers marked "device" are CUDA device pointers (or managed memory);
 *     they are owned by the caller and must stay valid until the work queued
 *     on `stream` has finished.  The library never allocates device memory;
 *     scratch space is the caller's `workspace`.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every call is asynchronous on that stream; the return value
 *     covers host-side validation and launch errors only.  Errors that only
 *     the device can see (an out-of-range token id, a bounded wait that ran
 *     out) are OR-ed into a device status word that the caller reads after
 *     synchronising (see cis_status_t).
 *   - Logit rows are row-major with a row stride `ld` >= V elements.  Rows
 *     already line up with their sampled token: the caller shifts the model
 *     output by one position (the token at t is scored from the logits at
 *     t - 1, App. C.4).
 *   - Masked tokens (mask[t] == 0) are not read; they get dz = 0, w = 0,
 *     trunc = 0, lp = 0 and contribute nothing to the loss.  mask == NULL
 *     means every token is valid.  Any non-zero mask byte counts as 1.
 *   - T == 0 is a valid no-op (loss 0).
 *   - Non-finite logits: -inf is allowed anywhere except at the sampled
 *     token; NaN propagates into that row's outputs.
 *   - Environment variables exist for tuning sweeps and tests only.  The
 *     defaults are the measured best.  Other settings change summation
 *     orders, never the tolerances.
 *       CIS_SLICE_KB (8..200, default 80), CIS_CLUSTER (1..8) and
 *       CIS_CLUSTER_THREADS (128, 256, 384 or 512; default 256) set the
 *       fused pass's slice target, cluster size and CTA width.  By default a
 *       row of 40 to 80 KB runs on two CTAs of 128 threads (CIS_SLICE_KB or
 *       CIS_CLUSTER turns that off).  They are read once per process.
 *       CIS_DIAG_WARPS (16 or 24 with one CTA per SM, 8 with two, 4 with
 *       four; default 16) and CIS_DIAG_SLOT_GROUPS (>= 1) set the diagnostics
 *       kernel's width and ring-slot size, and CIS_DIAG_KERNEL=row selects its
 *       one-CTA kernel.  They are read at each call.
 *       CIS_LMHEAD_MC (a bit mask over the LM head's GEMMs: 1 logits, 2 dz,
 *       4 dH, 8 dW; default 15) picks the GEMMs that run on 2-CTA clusters
 *       sharing B tiles by multicast, and CIS_LMHEAD_DUAL=0 runs a chunk's
 *       dH and dW as two launches instead of one.  Neither changes a result
 *       bit.  Read at each call.
 */
#ifndef CIS_H
#define CIS_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CIS_API __attribute__((visibility("default")))
#else
#define CIS_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CIS_OK = 0,
    CIS_ERR_INVALID_ARG = 1,   /* host validation failed; nothing was queued   */
    CIS_ERR_UNSUPPORTED = 2,   /* valid, but not supported here (layout, GPU)   */
    CIS_ERR_CUDA = 3,          /* a CUDA runtime call or launch failed          */
    CIS_ERR_DEVICE_TIMEOUT = 4,/* device status bit: a bounded wait ran out     */
    CIS_ERR_BAD_TOKEN_ID = 8   /* device status bit: some valid y_t not in [0,V)*/
} cis_status_t;

typedef enum { CIS_F32 = 0, CIS_BF16 = 1 } cis_dtype_t;

/* Weight operators: CIS is Eq. 4 with the floor of Algorithm 1; the band is
 * the two-sided ablation of Sec. 4.3; the others are the rows of Table 8.
 * p = exp(lp_train), k = exp(lp_train - lp_infer), phi = max(1 - p, kappa).
 * The sequence operators use K, the product of k over the valid tokens of a
 * response (cu_seqlens), and give every token of the response the same
 * weight. */
typedef enum {
    CIS_MODE_CIS = 0,     /* w = min{k, 1 + lambda*phi}                        */
    CIS_MODE_TIS = 1,     /* w = min(k, tis_cap)                               */
    CIS_MODE_EXACT = 2,   /* w = k clamped to [exact_lo, exact_hi]             */
    CIS_MODE_NONE = 3,    /* w = 1                                             */
    CIS_MODE_BAND = 4,    /* w = max{min{k, 1 + lambda*phi}, (1 + p)/2}        */
    CIS_MODE_ICEPOP = 5,  /* w = k if k in [icepop_lo, icepop_hi], else 0      */
    CIS_MODE_KPOP = 6,    /* w = k if max(KL_B(p||q), KL_B(q||p)) <= kpop_phi,
                           *     else 0; fp64, p and q clamped to
                           *     [1e-8, 1 - 1e-8] (App. D.5)                   */
    CIS_MODE_SEQ_TIS = 7, /* w = min(K, seq_cap)                               */
    CIS_MODE_SEQ_MIS = 8  /* w = K if K in [seq_lo, seq_hi], else 0           */
} cis_mode_t;

/* Loss normaliser: Algorithm 1 averages over the n tokens of the batch; Eq. 1
 * averages each response over its |y_i| tokens and the G responses. */
typedef enum {
    CIS_AGG_TOKEN_MEAN = 0,        /* s_t = 1/n, n = number of valid tokens      */
    CIS_AGG_SEQ_MEAN_TOKEN_MEAN = 1/* s_t = 1/(G |y_i|) from cu_seqlens and mask */
} cis_agg_t;

/* Hyper-parameters.  Defaults (cis_default_params): the deployed values of
 * App. C.1 / Table 8: lambda 2.3, kappa 5e-3, TIS cap 2, exact clamp
 * [1e-6, 1e6], IcePop [0.5, 5], KPop phi 2, Seq-TIS cap 2, Seq-MIS [0.5, 2],
 * PPO clip (0.2, 0.28), token mean. */
typedef struct {
    int32_t mode;      /* cis_mode_t                                         */
    int32_t agg;       /* cis_agg_t                                          */
    double lambda;     /* >= 0: threshold on e^eps is 1 + lambda (Eq. 4)     */
    double kappa;      /* in [0, 1]: floor on 1 - p (Algorithm 1)            */
    double tis_cap;    /* >= 1: C of TIS (Eq. 5 assumes C >= 1)              */
    double exact_lo;   /* > 0: clamp of the exact ratio                      */
    double exact_hi;   /* >= exact_lo                                        */
    double clip_low;   /* in [0, 1): rho clipped below at 1 - clip_low       */
    double clip_high;  /* >= 0: rho clipped above at 1 + clip_high           */
    double icepop_lo;  /* >= 0: IcePop band, bounds included                 */
    double icepop_hi;  /* >= icepop_lo                                       */
    double kpop_phi;   /* >= 0: KPop threshold on the binary KL              */
    double seq_cap;    /* > 0: C of Seq-TIS                                  */
    double seq_lo;     /* >= 0: Seq-MIS band, bounds included                */
    double seq_hi;     /* >= seq_lo                                          */
    /* Token-sharded data parallelism (the rows of one batch split across
     * GPUs at response boundaries): a DEVICE pointer to two int64 values
     * {N, G}, the batch's number of valid tokens and of responses with a
     * valid token, i.e. the sum over shards of what cis_count_valid writes.
     * When set, the loss normaliser uses them (token mean: s_t = 1/N;
     * sequence mean: s_t = 1/(G |y_i|), each response lying in one shard),
     * so that the shards' losses add up to the batch loss and each shard's
     * dlogits are the batch's rows.  NULL (the default): this call's own
     * counts.  Read on the device by the call's first kernel.              */
    const int64_t *global_counts;
} cis_params_t;

/* Reduction outputs of cis_loss_fwd_bwd, written on the device. */
typedef struct {
    double loss;          /* -sum_t s_t m_t w_t min(rho A, clip(rho) A)       */
    double trunc_excess;  /* sum over truncated tokens of (k_t - w_t)         */
    int64_t n_valid;      /* number of tokens with mask != 0                  */
    int64_t n_truncated;  /* tokens whose weight the operator changed: capped,
                           * clamped, lifted (band) or masked                 */
    float max_abs_logk;   /* max over valid tokens of |log k_t|               */
    int32_t status;       /* OR of device status bits (cis_status_t)          */
    double entropy_sum;   /* sum over valid tokens of the softmax entropy H_t
                           * when the call writes entropy_out, else 0; the
                           * batch entropy the paper logs is entropy_sum /
                           * n_valid                                          */
} cis_stats_t;

/* Fills *out with the defaults above.  Host only.  CIS_ERR_INVALID_ARG if out
 * is NULL. */
CIS_API cis_status_t cis_default_params(cis_params_t *out);

/*
 * This call's share of the loss normaliser, for token-sharded runs: writes
 * counts_out[0] = N, the number of tokens with mask != 0 (all T when mask is
 * NULL), and counts_out[1] = G, the number of responses [cu_seqlens[i],
 * cu_seqlens[i+1]) with at least one valid token (0 when cu_seqlens is
 * NULL).  Summed over the shards (an all-reduce of the int64 pair) they are
 * what cis_params_t.global_counts points to.
 *   mask        device uint8 [T] or NULL;  cu_seqlens device int32 [B + 1] or
 *               NULL;  counts_out device int64 [2], written.
 * Asynchronous on `stream`.  CIS_ERR_INVALID_ARG for T < 0, B < 0 or a NULL
 * counts_out; CIS_ERR_UNSUPPORTED for more than 12000 responses.
 */
CIS_API cis_status_t cis_count_valid(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                                     int64_t B, int64_t *counts_out, void *stream);

/* Human-readable name of a status value (static string, never NULL). */
CIS_API const char *cis_status_string(int32_t status);

/*
 * Sampled-token log-probabilities (Sec. 2.1): lp_out[t] = z_{t,y_t} -
 * logsumexp_j z_tj, accumulated in fp32.  One read of the logits.
 *   logits     device, [T, ld] of `dtype`, row-major; only j < V is read.
 *   ids        device int32 [T], sampled token ids.
 *   mask       device uint8 [T] or NULL.
 *   lp_out     device float [T].
 *   lse_out    device float [T] or NULL: logsumexp of each row.
 *   entropy_out device float [T] or NULL: entropy of each row's softmax,
 *              H_t = -sum_j p_tj log p_tj (the training-side entropy the
 *              paper logs, App. D); 0 for masked rows.
 *   dev_status device int32 [1] or NULL: device status bits are OR-ed in
 *              (the caller zeroes it first).
 * Errors: CIS_ERR_INVALID_ARG for NULL required pointers, T < 0, V <= 0,
 * ld < V or an unknown dtype.
 */
CIS_API cis_status_t cis_token_logprobs(const void *logits, int32_t dtype, int64_t T, int64_t V,
                                int64_t ld, const int32_t *ids, const uint8_t *mask,
                                float *lp_out, float *lse_out, float *entropy_out,
                                int32_t *dev_status, void *stream);

/*
 * Weights (Algorithm 1, Eq. 4, Table 8) from fp32 log-probabilities.
 *   lp_train  device float [T]: log p_t, the training-side log-probability
 *             the weight is built from (l_old when updating off the snapshot).
 *   lp_infer  device float [T]: log q_t, the raw value recorded at sampling.
 *   mask      device uint8 [T] or NULL.
 *   cu_seqlens device int32 [B + 1] or NULL: response boundaries (non-
 *             decreasing, cu_seqlens[B] <= T; not checked on the host).
 *             Required by the sequence operators (CIS_ERR_INVALID_ARG
 *             without); ignored by the others.  A valid token outside every
 *             response gets weight 0 under a sequence operator.
 *   w_out     device float [T]: the weight (0 for masked tokens).
 *   trunc_out device uint8 [T] or NULL: 1 where the operator changed the
 *             weight from k (capped, clamped, lifted or masked); under a
 *             sequence operator, the response's flag.
 *   eps_out   device float [T] or NULL: the log-odds displacement
 *             eps = logit p - logit q (Lemma 3.1); +-inf or NaN where p or q
 *             rounds to 1 (the weight itself stays finite).
 * Decisions are taken on log k = lp_train - lp_infer, evaluated exactly.  CIS
 * compares k with the cap, and TIS and EXACT compare log k with the log of the
 * bound.  Each is settled in fp32 where its error bound proves the answer, else
 * in fp64.  The band, IcePop, KPop and the sequence operators (log K summed in
 * fp64) decide in fp64.  Errors:
 * CIS_ERR_INVALID_ARG for NULL required pointers, T < 0, parameters outside
 * the ranges of cis_params_t, or a sequence operator without cu_seqlens.
 */
CIS_API cis_status_t cis_weights(const float *lp_train, const float *lp_infer, const uint8_t *mask,
                         int64_t T, const int32_t *cu_seqlens, int64_t B,
                         const cis_params_t *params, float *w_out, uint8_t *trunc_out,
                         float *eps_out, void *stream);

/* Bytes of device workspace cis_loss_fwd_bwd needs for T tokens and
 * vocabulary V.  Host only.  CIS_ERR_INVALID_ARG if bytes is NULL or T < 0. */
CIS_API cis_status_t cis_loss_workspace_size(int64_t T, int64_t V, size_t *bytes);

/*
 * The fused forward + backward token pass (Eq. 1 with the weight of
 * Algorithm 1 / Table 8, the weight detached).
 *   logits      device, [T, ld] of `dtype` (CIS_BF16 or CIS_F32).
 *   ids         device int32 [T].
 *   lp_infer    device float [T]: log q_t recorded by the inference engine.
 *   lp_old      device float [T] or NULL: log p at the rollout snapshot.
 *               NULL means the current parameters are the snapshot: the
 *               weight is built from the current l_t (detached) and
 *               rho = exp(l_t - stopgrad(l_t)) = 1 in value.
 *   adv         device float [T]: advantage A_t.
 *   mask        device uint8 [T] or NULL.
 *   cu_seqlens  device int32 [B + 1] or NULL: response boundaries, needed for
 *               CIS_AGG_SEQ_MEAN_TOKEN_MEAN (tokens outside every response
 *               then get s_t = 0) and by the sequence operators.  Must be
 *               non-decreasing with cu_seqlens[B] <= T; not checked on the
 *               host.
 *   params      host pointer.
 *   dlogits     device, [T, ld_out] of `dlogits_dtype` (CIS_BF16 rounds to
 *               nearest even, CIS_F32); every element j < V of every row is
 *               written.  May not overlap the logits.
 *   lp_out, w_out, trunc_out  device per-token outputs or NULL.
 *   entropy_out device float [T] or NULL: each row's softmax entropy, taken
 *               in the same pass (a variant of the kernel that keeps one more
 *               sum per row; without it the pass does no entropy work), and
 *               summed into stats_out->entropy_sum.
 *   stats_out   device cis_stats_t* or NULL.
 *   loss_out    device double [1] or NULL: the loss (also in stats_out).
 *   workspace   device, >= cis_loss_workspace_size(T, V) bytes, 256-byte
 *               aligned; its first int32 is the device status word, zeroed
 *               by this call.
 * Sums are deterministic: the same inputs give bit-identical outputs.
 * The sequence operators need every log p of a response before any weight:
 * with lp_old the weights are formed first and the pass is unchanged;
 * without it a forward pass (one more read of the logits) gives the log p.
 * A token with an out-of-range id is left out of its response's product.
 * Errors: CIS_ERR_INVALID_ARG for NULL required pointers, T < 0, V <= 0,
 * ld < V, ld_out < V, bad parameters, a short or misaligned workspace, or
 * CIS_AGG_SEQ_MEAN_TOKEN_MEAN or a sequence operator without cu_seqlens;
 * CIS_ERR_CUDA if a launch fails.
 */
CIS_API cis_status_t cis_loss_fwd_bwd(const void *logits, int32_t dtype, int64_t T, int64_t V,
                              int64_t ld, const int32_t *ids, const float *lp_infer,
                              const float *lp_old, const float *adv, const uint8_t *mask,
                              const int32_t *cu_seqlens, int64_t B,
                              const cis_params_t *params, void *dlogits,
                              int32_t dlogits_dtype, int64_t ld_out, float *lp_out,
                              float *w_out, uint8_t *trunc_out, float *entropy_out,
                              cis_stats_t *stats_out, double *loss_out, void *workspace,
                              size_t workspace_bytes, void *stream);

/*
 * Bytes of device workspace cis_loss_fwd_bwd_host needs for T tokens of V
 * entries, the two element types, chunks of chunk_tokens rows and B responses
 * (B = 0 without cu_seqlens).  Host only.  CIS_ERR_INVALID_ARG on bad values.
 */
CIS_API cis_status_t cis_loss_host_workspace_size(int64_t T, int64_t V, int32_t dtype,
                                                  int32_t dlogits_dtype, int64_t chunk_tokens,
                                                  int64_t B, size_t *bytes);

/*
 * cis_loss_fwd_bwd for callers whose buffers are in host memory.
 *   Every tensor argument is a HOST pointer: logits [T, V] and dlogits [T, V]
 *   (contiguous rows), ids, lp_infer, lp_old, adv, mask, cu_seqlens, and the
 *   outputs lp_out, w_out, trunc_out, entropy_out, stats_out, loss_out.  Page-locked
 *   (pinned) memory lets the copies overlap; pageable memory works but the
 *   copies then serialise.
 *   workspace is DEVICE memory of cis_loss_host_workspace_size(...) bytes,
 *   256-byte aligned: the per-token arrays, the loss workspace and three
 *   staging buffers of chunk_tokens rows in each direction.
 * The rows stream through the GPU in chunks of chunk_tokens: while the fused
 * kernel runs on chunk k (on `stream`), the next chunks are copied in and the
 * previous ones copied out on copy streams the library creates once per
 * device (one per staging buffer and direction).  The first chunk's copy in
 * and the last one's copy out run alone, so small chunks overlap more: at
 * T=16384, V=151936 (bf16), chunks of 512 rows (150 MB) took 30-32 ms per call
 * against 35-42 ms for chunks of 2048.  The
 * normaliser and the loss cover the whole batch, so every output equals that
 * of cis_loss_fwd_bwd.  Asynchronous on `stream`: the host outputs are valid
 * once `stream` has completed the call's work.  Errors: as cis_loss_fwd_bwd,
 * plus CIS_ERR_UNSUPPORTED for a sequence operator without lp_old (its
 * weights would need every row's log p before the first chunk's dlogits).
 */
CIS_API cis_status_t cis_loss_fwd_bwd_host(
    const void *logits, int32_t dtype, int64_t T, int64_t V, const int32_t *ids,
    const float *lp_infer, const float *lp_old, const float *adv, const uint8_t *mask,
    const int32_t *cu_seqlens, int64_t B, const cis_params_t *params, void *dlogits,
    int32_t dlogits_dtype, float *lp_out, float *w_out, uint8_t *trunc_out, float *entropy_out,
    cis_stats_t *stats_out, double *loss_out, int64_t chunk_tokens, void *workspace,
    size_t workspace_bytes, void *stream);

/*
 * Bytes of device workspace cis_lmhead_fused needs with its default
 * vocabulary chunk (dz of one chunk within about 1 GiB).  Host only.
 * CIS_ERR_INVALID_ARG if bytes is NULL, T < 0, V <= 0 or H <= 0.
 */
CIS_API cis_status_t cis_lmhead_workspace_size(int64_t T, int64_t V, int64_t H, size_t *bytes);

/*
 * Bytes of device workspace for vocabulary chunks of `chunk` columns (a
 * positive multiple of 256; wider than V rounded up to 256 counts as that).
 * The workspace grows by 2 * ceil(T / 128) * 128 bytes per chunk column.
 * Host only.  CIS_ERR_INVALID_ARG for a NULL bytes, T < 0, V <= 0, H <= 0 or
 * a chunk that is not a positive multiple of 256.
 */
CIS_API cis_status_t cis_lmhead_workspace_size_chunk(int64_t T, int64_t V, int64_t H,
                                                     int64_t chunk, size_t *bytes);

/*
 * The token pass fused with the LM head: logits z = hidden W^T are computed
 * in tiles on the tensor cores and never written to memory; the weight, the
 * loss and the gradients are those of cis_loss_fwd_bwd (Eq. 1, Algorithm 1,
 * Table 8), taken through the LM head:
 *   dhidden = dz W,   dweight = dz^T hidden,   dz = c (softmax - onehot).
 * The forward sweep keeps per-token softmax statistics only; the gradient
 * sweep recomputes z one vocabulary chunk at a time and holds that chunk's dz
 * (bf16 [ceil(T / 128) * 128, chunk]) in the workspace, read by both
 * gradient products where it lies.
 *   hidden      device bf16 [T, H], contiguous rows, 16-byte aligned.
 *   weight      device bf16 [V, H], contiguous rows, 16-byte aligned.
 *   H           hidden size; a multiple of 256 (else CIS_ERR_UNSUPPORTED).
 *   ids, lp_infer, lp_old, adv, mask, cu_seqlens, B, params: as for
 *               cis_loss_fwd_bwd.
 *   dhidden     device [T, H] of grad_dtype (CIS_F32 or CIS_BF16), written;
 *               16-byte aligned (32-byte aligned buffers take the wider stores).
 *   dweight     device [V, H] of grad_dtype, written (rows of tokens that are
 *               masked contribute nothing); alignment as for dhidden.
 *   lp_out, w_out, trunc_out, entropy_out, stats_out, loss_out: as for
 *               cis_loss_fwd_bwd (the entropy comes from the forward sweep's
 *               tiles).
 *   workspace   device, 1024-byte aligned; its first int32 is the device
 *               status word.  workspace_bytes picks the chunk: the widest
 *               multiple of 256 columns whose cis_lmhead_workspace_size_chunk
 *               fits; CIS_ERR_INVALID_ARG if not even 256 columns fit.
 * dz enters the two gradient products in bf16 (the tensor-core operand type);
 * the products accumulate in fp32 (dhidden across chunks too).  Errors: as
 * for cis_loss_fwd_bwd, plus CIS_ERR_UNSUPPORTED if the tensor-map encoder is
 * unavailable.
 */
CIS_API cis_status_t cis_lmhead_fused(const void *hidden, const void *weight, int64_t T,
                                      int64_t H, int64_t V, const int32_t *ids,
                                      const float *lp_infer, const float *lp_old,
                                      const float *adv, const uint8_t *mask,
                                      const int32_t *cu_seqlens, int64_t B,
                                      const cis_params_t *params, void *dhidden, void *dweight,
                                      int32_t grad_dtype, float *lp_out, float *w_out,
                                      uint8_t *trunc_out, float *entropy_out,
                                      cis_stats_t *stats_out, double *loss_out, void *workspace,
                                      size_t workspace_bytes, void *stream);

/*
 * Mismatch diagnostics from both engines' full logits (App. A.5; Sec. 4.3,
 * Fig. 5c-d), one row per position.  With p = softmax(logits_train),
 * q = softmax(logits_infer), y the sampled token and f the weight operator of
 * params (a token operator) applied to every candidate j (k_j = p_j / q_j):
 *   eps_out   [T] the log-odds displacement of y: -delta_y + log sum_{j != y}
 *             w_j e^{delta_j} with w_j = e^{z_j} / sum_{j' != y} e^{z_j'} and
 *             delta in the normalised gauge log q - log p (Lemma 3.1), which
 *             equals logit p_y - logit q_y.
 *   logk_out  [T] or NULL: log k_y = log p_y - log q_y.
 *   p_out     [T] or NULL: p_y.
 *   bias2_out [T] or NULL: || E_{y~q}[(f_y - k_y) g_y] ||^2, g_y = e_y - p the
 *             gradient of log p_y with respect to the logits.
 *   dvar_out  [T] or NULL: the variance increase of f_y g_y over g_y under
 *             y ~ q (trace of the covariance).
 * All outputs are device float arrays; masked rows get 0, valid rows with an
 * id outside [0, V) get NaN and set CIS_ERR_BAD_TOKEN_ID in dev_status
 * (device int32 or NULL).  logits_* are device [T, ld_*] of dtype (CIS_F32 or
 * CIS_BF16).  The expectations over y ~ q are exact sums over the V
 * candidates; the operator's weight is taken in fp32 per candidate.  Two
 * streaming passes over both tensors.  Errors: CIS_ERR_INVALID_ARG for NULL
 * required pointers, T < 0, V <= 0, ld < V, an unknown dtype, bad parameters
 * or a sequence operator.
 */
CIS_API cis_status_t cis_mismatch_diagnostics(const void *logits_train, const void *logits_infer,
                                              int32_t dtype, int64_t T, int64_t V,
                                              int64_t ld_train, int64_t ld_infer,
                                              const int32_t *ids, const uint8_t *mask,
                                              const cis_params_t *params, float *eps_out,
                                              float *logk_out, float *p_out, float *bias2_out,
                                              float *dvar_out, int32_t *dev_status,
                                              void *stream);

/*
 * Confidence-binned counts and sums (Sec. 4.3, Fig. 5b: the sampled tokens
 * binned by p_t, with E[k_t - f_t] in each bin; App. A.5: logarithmic bins of
 * 1 - p_t).  The key is any per-token value (p, 1 - p, ...); the values are
 * up to CIS_MAX_BIN_VALUES per-token arrays (k - f from the token pass, the
 * diagnostics' bias2 and dvar, ...).  A bin's mean is its sum over its count.
 *   key         device float [T].
 *   mask        device uint8 [T] or NULL; masked tokens fall in no bin.
 *   edges       host double [nbins + 1], strictly ascending, no NaN.  Token t
 *               falls in bin b when edges[b] <= key[t] < edges[b + 1]; the
 *               last bin also takes key[t] == edges[nbins].  A NaN key, or one
 *               outside [edges[0], edges[nbins]], falls in no bin.
 *   nbins       1 .. CIS_MAX_BINS.
 *   values      host array of nvalues device float [T] pointers (NULL if
 *               nvalues is 0).
 *   nvalues     0 .. CIS_MAX_BIN_VALUES.
 *   counts_out  device int64 [nbins].
 *   sums_out    device double [nvalues, nbins] (value-major), fp64 sums; a
 *               NaN value makes its bin's sum NaN.  NULL if nvalues is 0.
 *   workspace   device, 256-byte aligned, at least
 *               cis_binned_sums_workspace_size bytes.
 * Deterministic: fixed-order fp64 sums, the same result on every call.
 * Asynchronous on `stream`.  CIS_ERR_INVALID_ARG on a NULL required pointer,
 * T < 0, nbins or nvalues out of range, edges not strictly ascending or a
 * workspace that is too small or misaligned.
 */
#define CIS_MAX_BINS 64
#define CIS_MAX_BIN_VALUES 4
CIS_API cis_status_t cis_binned_sums(const float *key, const uint8_t *mask, int64_t T,
                                     const double *edges, int32_t nbins,
                                     const float *const *values, int32_t nvalues,
                                     int64_t *counts_out, double *sums_out, void *workspace,
                                     size_t workspace_bytes, void *stream);

/* Bytes of device workspace cis_binned_sums needs.  Host only.
 * CIS_ERR_INVALID_ARG if bytes is NULL, T < 0 or nbins / nvalues are out of
 * range. */
CIS_API cis_status_t cis_binned_sums_workspace_size(int64_t T, int32_t nbins, int32_t nvalues,
                                                    size_t *bytes);

/*
 * Largest T that cis_loss_fwd_bwd_noalloc accepts.
 */
#define CIS_NOALLOC_MAX_TOKENS 65536

/*
 * cis_loss_fwd_bwd without the workspace arguments, for callers that cannot
 * allocate device memory: extensions running inside a host framework that owns
 * all device memory and gives them no allocator (serving engines, training
 * runtimes), and C callers with no device allocator of their own.  The paper
 * has no counterpart; this is an interface convenience around the same pass.
 *   - All other arguments, outputs and errors are those of cis_loss_fwd_bwd.
 *   - The scratch is an array of about 1.3 MiB in the library's static device
 *     memory, sized for CIS_NOALLOC_MAX_TOKENS tokens; every GPU that loads the
 *     library keeps one until the process exits.  T > CIS_NOALLOC_MAX_TOKENS
 *     returns CIS_ERR_UNSUPPORTED before any GPU work.
 *   - Every call looks the array's device address up (cudaGetSymbolAddress)
 *     in the calling thread's current context, so a context that was reset or
 *     replaced since the last call is never written through a stale address.
 *     The first lookup on a device may load the library's device code there:
 *     make the first call on each device before any stream capture on it.
 *   - No allocating routine is called.
 *   - All calls share the array.  Each call resets the status word and
 *     overwrites everything else it reads, so sequential calls are
 *     independent; calls whose GPU work overlaps (different streams or host
 *     threads) race and give wrong results.
 *   - Device status bits are reported in stats_out->status.
 */
CIS_API cis_status_t cis_loss_fwd_bwd_noalloc(const void *logits, int32_t dtype, int64_t T,
                                              int64_t V, int64_t ld, const int32_t *ids,
                                              const float *lp_infer, const float *lp_old,
                                              const float *adv, const uint8_t *mask,
                                              const int32_t *cu_seqlens, int64_t B,
                                              const cis_params_t *params, void *dlogits,
                                              int32_t dlogits_dtype, int64_t ld_out,
                                              float *lp_out, float *w_out, uint8_t *trunc_out,
                                              float *entropy_out, cis_stats_t *stats_out,
                                              double *loss_out, void *stream);

/*
 * Profiling aid.  The next cis_loss_fwd_bwd call made from the calling host
 * thread records `begin_event` on its stream just before its main kernel (the
 * fused vocabulary pass) and `end_event` just after it, then forgets both.
 * The events are cudaEvent_t handles passed as void*, owned by the caller.
 * Passing NULL for both cancels a pending request.  Nothing else changes: the
 * call does the same work.  CIS_ERR_INVALID_ARG if exactly one is NULL.
 */
CIS_API cis_status_t cis_profile_next_call(void *begin_event, void *end_event);

/*
 * Self-test of the failure detection of the kernels' waits.
 *
 * Every wait inside the library's kernels (for bulk copies, tensor-core work
 * or other CTAs of a cluster) polls its mbarrier a bounded number of times,
 * each poll suspending for at most 1 µs (about 2 s in all), then sets
 * CIS_ERR_DEVICE_TIMEOUT in the call's device status word and lets the
 * kernel run to its end, so that the CUDA context stays usable and the host
 * reads the error after a synchronisation.  This call runs one CTA that
 * waits on an mbarrier which nothing ever completes, through the same wait
 * code with a poll limit of `max_polls` (1 .. 2^21), and reports the
 * timeout the same way.
 *
 * Arguments:
 *   - max_polls: the poll limit (each poll waits at most about 1 µs).
 *   - cluster_scope: 0 for the CTA-scope wait (bulk copies into this CTA),
 *     1 for the cluster-scope wait (data from other CTAs of a cluster).
 *   - dev_status: device int32, OR-ed with CIS_ERR_DEVICE_TIMEOUT; the
 *     caller clears and reads it.
 *   - stream: cudaStream_t (NULL: the default stream); asynchronous.
 *
 * CIS_ERR_INVALID_ARG for a null status, a limit out of range or a scope
 * other than 0 or 1.
 */
CIS_API cis_status_t cis_selftest_bounded_wait(uint32_t max_polls, int32_t cluster_scope,
                                               int32_t *dev_status, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* CIS_H */
