// cis_api.cu -- the C ABI of libcis (declared in include/cis.h).
//
// Host side only: argument validation, the workspace layout, the fp64 logs of
// the hyper-parameters the certified decisions need, and the launches.  All
// arithmetic on the token pass runs in the kernels.
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

#include "cis_kernels.h"
#include "cis_nvtx.h"

namespace cis {

static bool finite_or_inf_nonneg(double x) { return x == x && x >= 0.0; }

bool params_ok(const cis_params_t *p)
{
    if (p == nullptr)
        return false;
    if (p->mode < CIS_MODE_CIS || p->mode > CIS_MODE_SEQ_MIS)
        return false;
    if (p->agg != CIS_AGG_TOKEN_MEAN && p->agg != CIS_AGG_SEQ_MEAN_TOKEN_MEAN)
        return false;
    if (!finite_or_inf_nonneg(p->lambda))
        return false;
    if (!(p->kappa >= 0.0 && p->kappa <= 1.0))
        return false;
    if (!(p->tis_cap >= 1.0))
        return false;
    if (!(p->exact_lo > 0.0 && p->exact_hi >= p->exact_lo))
        return false;
    if (!(p->clip_low >= 0.0 && p->clip_low < 1.0))
        return false;
    if (!finite_or_inf_nonneg(p->clip_high))
        return false;
    if (!(p->icepop_lo >= 0.0 && p->icepop_hi >= p->icepop_lo))
        return false;
    if (!finite_or_inf_nonneg(p->kpop_phi))
        return false;
    if (!(p->seq_cap > 0.0))
        return false;
    if (!(p->seq_lo >= 0.0 && p->seq_hi >= p->seq_lo))
        return false;
    return true;
}

DevParams make_dev_params(const cis_params_t &p)
{
    DevParams d;
    d.mode = p.mode;
    d.agg = p.agg;
    d.lam = p.lambda;
    d.kappa = p.kappa;
    d.lam_f = (float)p.lambda;
    d.kappa_f = (float)p.kappa;
    d.tis_cap_f = (float)p.tis_cap;
    d.exact_lo_f = (float)p.exact_lo;
    d.exact_hi_f = (float)p.exact_hi;
    d.rho_lo_f = (float)(1.0 - p.clip_low);
    d.rho_hi_f = (float)(1.0 + p.clip_high);
    d.log_tis_cap = log(p.tis_cap);
    d.log_exact_lo = log(p.exact_lo);
    d.log_exact_hi = log(p.exact_hi);
    d.log_rho_lo = log1p(-p.clip_low);
    d.log_rho_hi = log1p(p.clip_high);
    d.log_tis_cap_f = (float)d.log_tis_cap;
    d.log_exact_lo_f = (float)d.log_exact_lo;
    d.log_exact_hi_f = (float)d.log_exact_hi;
    d.log_rho_lo_f = (float)d.log_rho_lo;
    d.log_rho_hi_f = (float)d.log_rho_hi;
    d.log_icepop_lo = log(p.icepop_lo);
    d.log_icepop_hi = log(p.icepop_hi);
    d.kpop_phi = p.kpop_phi;
    d.seq_cap = p.seq_cap;
    d.log_seq_cap = log(p.seq_cap);
    d.log_seq_lo = log(p.seq_lo);
    d.log_seq_hi = log(p.seq_hi);
    return d;
}

static bool shape_ok(int64_t T, int64_t V, int64_t ld)
{
    return T >= 0 && T <= 0x7fffffffLL && V > 0 && V <= 0x7fffffffLL && ld >= V;
}

static bool dtype_ok(int32_t dt) { return dt == CIS_F32 || dt == CIS_BF16; }

static int dtype_bytes(int32_t dt) { return dt == CIS_BF16 ? 2 : 4; }

static cis_status_t cuda_status(cudaError_t e)
{
    if (e == cudaSuccess)
        return CIS_OK;
    if (e == cudaErrorNotSupported)
        return CIS_ERR_UNSUPPORTED;
    return CIS_ERR_CUDA;
}

// Events requested by cis_profile_next_call, per host thread.
static thread_local cudaEvent_t g_prof_begin = nullptr;
static thread_local cudaEvent_t g_prof_end = nullptr;

}  // namespace cis

using namespace cis;

extern "C" {

CIS_API cis_status_t cis_default_params(cis_params_t *out)
{
    if (out == nullptr)
        return CIS_ERR_INVALID_ARG;
    out->mode = CIS_MODE_CIS;
    out->agg = CIS_AGG_TOKEN_MEAN;
    out->lambda = 2.3;
    out->kappa = 5e-3;
    out->tis_cap = 2.0;
    out->exact_lo = 1e-6;
    out->exact_hi = 1e6;
    out->clip_low = 0.2;
    out->clip_high = 0.28;
    out->icepop_lo = 0.5;
    out->icepop_hi = 5.0;
    out->kpop_phi = 2.0;
    out->seq_cap = 2.0;
    out->seq_lo = 0.5;
    out->seq_hi = 2.0;
    out->global_counts = nullptr;
    return CIS_OK;
}

CIS_API cis_status_t cis_count_valid(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                                     int64_t B, int64_t *counts_out, void *stream)
{
    NvtxRange nvtx_range("cis_count_valid");
    if (T < 0 || B < 0 || counts_out == nullptr || (cu_seqlens == nullptr && B > 0))
        return CIS_ERR_INVALID_ARG;
    const cudaError_t e = launch_count_valid(mask, T, cu_seqlens, B, counts_out,
                                             (cudaStream_t)stream);
    return e == cudaSuccess ? CIS_OK
                            : (e == cudaErrorNotSupported ? CIS_ERR_UNSUPPORTED : CIS_ERR_CUDA);
}

CIS_API const char *cis_status_string(int32_t status)
{
    switch (status) {
    case CIS_OK: return "CIS_OK";
    case CIS_ERR_INVALID_ARG: return "CIS_ERR_INVALID_ARG: invalid argument";
    case CIS_ERR_UNSUPPORTED: return "CIS_ERR_UNSUPPORTED: not supported for these arguments";
    case CIS_ERR_CUDA: return "CIS_ERR_CUDA: a CUDA call or launch failed";
    case CIS_ERR_DEVICE_TIMEOUT: return "CIS_ERR_DEVICE_TIMEOUT: a bounded device wait ran out";
    case CIS_ERR_BAD_TOKEN_ID: return "CIS_ERR_BAD_TOKEN_ID: a valid token id is outside [0, V)";
    case CIS_ERR_DEVICE_TIMEOUT | CIS_ERR_BAD_TOKEN_ID:
        return "CIS_ERR_DEVICE_TIMEOUT | CIS_ERR_BAD_TOKEN_ID";
    default: return "unknown cis status";
    }
}

CIS_API cis_status_t cis_token_logprobs(const void *logits, int32_t dtype, int64_t T, int64_t V,
                                        int64_t ld, const int32_t *ids, const uint8_t *mask,
                                        float *lp_out, float *lse_out, float *entropy_out,
                                        int32_t *dev_status, void *stream)
{
    NvtxRange nvtx_range("cis_token_logprobs");
    if (!shape_ok(T, V, ld) || !dtype_ok(dtype))
        return CIS_ERR_INVALID_ARG;
    if (T == 0)
        return CIS_OK;
    if (logits == nullptr || ids == nullptr || lp_out == nullptr)
        return CIS_ERR_INVALID_ARG;
    PassArgs a = {};
    a.logits = logits;
    a.T = T;
    a.V = V;
    a.ld = ld;
    a.ids = ids;
    a.mask = mask;
    a.lp_out = lp_out;
    a.lse_out = lse_out;
    a.entropy_out = entropy_out;
    a.status = dev_status;
    return cuda_status(launch_token_logprobs(a, dtype, (cudaStream_t)stream));
}

CIS_API cis_status_t cis_weights(const float *lp_train, const float *lp_infer,
                                 const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                                 int64_t B, const cis_params_t *params, float *w_out,
                                 uint8_t *trunc_out, float *eps_out, void *stream)
{
    NvtxRange nvtx_range("cis_weights");
    if (T < 0 || !params_ok(params))
        return CIS_ERR_INVALID_ARG;
    const bool seq = is_seq_mode(params->mode);
    if (seq && (cu_seqlens == nullptr || B < 0))
        return CIS_ERR_INVALID_ARG;
    if (T == 0)
        return CIS_OK;
    if (lp_train == nullptr || lp_infer == nullptr || w_out == nullptr)
        return CIS_ERR_INVALID_ARG;
    const DevParams P = make_dev_params(*params);
    cudaStream_t s = (cudaStream_t)stream;
    // per token first (a sequence operator leaves w = 0, trunc = 0 there), then
    // the responses' weights over their valid tokens
    cudaError_t e = launch_weights(lp_train, lp_infer, mask, T, P, w_out, trunc_out, eps_out, s);
    if (e == cudaSuccess && seq)
        e = launch_seq_weights(nullptr, lp_train, lp_infer, nullptr, 0, mask, cu_seqlens, B, T, P,
                               w_out, trunc_out, s);
    return cuda_status(e);
}

CIS_API cis_status_t cis_loss_workspace_size(int64_t T, int64_t V, size_t *bytes)
{
    (void)V;
    if (bytes == nullptr || T < 0)
        return CIS_ERR_INVALID_ARG;
    *bytes = ws_layout(T).total;
    return CIS_OK;
}

CIS_API cis_status_t cis_loss_fwd_bwd(const void *logits, int32_t dtype, int64_t T, int64_t V,
                                      int64_t ld, const int32_t *ids, const float *lp_infer,
                                      const float *lp_old, const float *adv,
                                      const uint8_t *mask, const int32_t *cu_seqlens, int64_t B,
                                      const cis_params_t *params, void *dlogits,
                                      int32_t dlogits_dtype, int64_t ld_out, float *lp_out,
                                      float *w_out, uint8_t *trunc_out, float *entropy_out,
                                      cis_stats_t *stats_out, double *loss_out, void *workspace,
                                      size_t workspace_bytes, void *stream)
{
    NvtxRange nvtx_range("cis_loss_fwd_bwd");
    if (!shape_ok(T, V, ld) || ld_out < V || !dtype_ok(dtype) || !dtype_ok(dlogits_dtype))
        return CIS_ERR_INVALID_ARG;
    if (!params_ok(params))
        return CIS_ERR_INVALID_ARG;
    if ((params->agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN || is_seq_mode(params->mode)) &&
        (cu_seqlens == nullptr || B < 0))
        return CIS_ERR_INVALID_ARG;
    const WsLayout L = ws_layout(T);
    if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 255) ||
        workspace_bytes < L.total)
        return CIS_ERR_INVALID_ARG;
    if (T > 0 && (logits == nullptr || ids == nullptr || lp_infer == nullptr ||
                  adv == nullptr || dlogits == nullptr))
        return CIS_ERR_INVALID_ARG;
    if (T > 0) {
        const uintptr_t a0 = reinterpret_cast<uintptr_t>(logits);
        const uintptr_t a1 = a0 + (uintptr_t)((T - 1) * ld + V) * dtype_bytes(dtype);
        const uintptr_t b0 = reinterpret_cast<uintptr_t>(dlogits);
        const uintptr_t b1 = b0 + (uintptr_t)((T - 1) * ld_out + V) * dtype_bytes(dlogits_dtype);
        if (a0 < b1 && b0 < a1)
            return CIS_ERR_INVALID_ARG;
    }
    cudaStream_t s = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    PassArgs a = {};
    a.logits = logits;
    a.T = T;
    a.V = V;
    a.ld = ld;
    a.ids = ids;
    a.lp_inf = lp_infer;
    a.lp_old = lp_old;
    a.adv = adv;
    a.mask = mask;
    a.scale = reinterpret_cast<float *>(ws + L.scale);
    a.dz = dlogits;
    a.ld_out = ld_out;
    a.lp_out = lp_out;
    a.w_out = w_out;
    a.trunc_out = trunc_out;
    a.entropy_out = entropy_out;
    a.ws_w = reinterpret_cast<float *>(ws + L.w);
    a.ws_trunc = ws + L.trunc;
    a.ws_logk = reinterpret_cast<float *>(ws + L.logk);
    a.ws_terms = reinterpret_cast<double *>(ws + L.terms);
    a.status = reinterpret_cast<int32_t *>(ws + L.status);
    a.P = make_dev_params(*params);

    a.red_parts = ws + L.parts;
    a.red_ticket = reinterpret_cast<uint32_t *>(ws + L.ticket);
    cudaError_t e = launch_scales(mask, T, cu_seqlens, B, params->agg,
                                  reinterpret_cast<float *>(ws + L.scale), a.status,
                                  a.red_ticket, s, params->global_counts);
    if (e != cudaSuccess)
        return cuda_status(e);
    if (T > 0 && is_seq_mode(params->mode)) {
        // Sequence operator: every log p of a response before any weight.  The
        // fp64 log p goes into the terms array (the pass overwrites it), the
        // responses' weights into the weight and flag arrays, which the pass
        // then reads (and writes back unchanged).
        if (lp_old == nullptr) {
            PassArgs f = a;
            f.lp_inf = nullptr;
            f.lp_out = nullptr;
            f.lse_out = nullptr;
            f.entropy_out = nullptr;  // the fused pass writes it
            f.lp64_out = a.ws_terms;
            if ((e = launch_token_logprobs(f, dtype, s)) != cudaSuccess)
                return cuda_status(e);
        }
        if ((e = cudaMemsetAsync(a.ws_w, 0, 4 * (size_t)T, s)) != cudaSuccess ||
            (e = cudaMemsetAsync(a.ws_trunc, 0, (size_t)T, s)) != cudaSuccess)
            return cuda_status(e);
        if ((e = launch_seq_weights(lp_old ? nullptr : a.ws_terms, lp_old, lp_infer, ids, V, mask,
                                    cu_seqlens, B, T, a.P, a.ws_w, a.ws_trunc, s)) != cudaSuccess)
            return cuda_status(e);
        a.w_in = a.ws_w;
        a.trunc_in = a.ws_trunc;
    }
    cudaEvent_t ev0 = g_prof_begin, ev1 = g_prof_end;
    g_prof_begin = g_prof_end = nullptr;
    if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess)
        return cuda_status(e);
    if (T > 0) {
        if (cluster_path_applies(a, dtype, dlogits_dtype))
            e = launch_cluster_fwd_bwd(a, dtype, dlogits_dtype, s);
        else
            e = launch_rowwise_fwd_bwd(a, dtype, dlogits_dtype, s);
        if (e != cudaSuccess)
            return cuda_status(e);
    }
    if (ev1 && (e = cudaEventRecord(ev1, s)) != cudaSuccess)
        return cuda_status(e);
    return cuda_status(launch_reduce(a, stats_out, loss_out, s));
}

CIS_API cis_status_t cis_profile_next_call(void *begin_event, void *end_event)
{
    if ((begin_event == nullptr) != (end_event == nullptr))
        return CIS_ERR_INVALID_ARG;
    g_prof_begin = static_cast<cudaEvent_t>(begin_event);
    g_prof_end = static_cast<cudaEvent_t>(end_event);
    return CIS_OK;
}

}  // extern "C"
