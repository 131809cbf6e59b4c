// cis_diag.cu -- mismatch diagnostics from the two engines' full logits
// (App. A.5; Sec. 4.3, Fig. 5c-d): per position, the log-odds displacement of
// the sampled token, its log ratio and probability, and -- over the whole
// next-token distribution y ~ q -- the squared bias ||E[(f - k) g]||^2 and the
// variance increase of f g over g, with g = e_y - p the gradient of log p_y
// with respect to the logits and f the weight operator.
//
// One CTA of 512 threads per row, two streaming passes over both rows:
//   pass 1: (max, sum) over j != y of each engine's logits (cis_rowops.cuh),
//           giving log p, log q, their log-odds d_p, d_q, and lse of each;
//   pass 2: p_j, q_j, k_j and f_j for every candidate j, accumulating
//             P2 = sum p^2,  R2 = sum r^2,  RP = sum r p    (r = q f - p)
//             C1 = sum q (f^2 - 1)(1 - 2p),  C2 = sum q (f^2 - 1),
//             C3 = sum q (f - 1),  C4 = sum q^2 (f^2 - 1),
//             C5 = sum q (f - 1) p,  QP = sum q p.
// With sum q = sum p = 1 the expectations reduce to these sums:
//   E_q[(f - k) g]_j = r_j - p_j C3, so bias2 = R2 - 2 C3 RP + C3^2 P2;
//   Var(f g) - Var(g) = C1 + P2 C2 - [C4 - (2 + C3) C5 - C3 C6 + C3 (2 + C3) P2]
//   with C6 = sum q (f + 1) p = C5 + 2 QP.
// Every term but P2 is proportional to f - 1 or to q f - p, so neither result
// is a small difference of O(1) numbers.  Per-thread sums are fp32, the block
// sums fp64.  The second pass reads the rows again, from L2 where they are
// still resident.
#include "cis_kernels.h"
#include "cis_rowops.cuh"

namespace cis {
namespace {

constexpr int kDiagThreads = 512;
constexpr int kNSums = 9;

// The operator's weight for one candidate j in fp32 (a statistic: no fp64
// decision fallback), from the exponents xp = log2 p_j, xq = log2 q_j, p_j and
// k_j = 2^{xp - xq}; MODE is a compile-time cis_mode_t, so the per-candidate
// loop has no branch on it.
template <int MODE>
__device__ __forceinline__ float elem_weight(float xp, float xq, float p, float k,
                                             const DevParams &P)
{
    if (MODE == CIS_MODE_CIS)
        return fminf(k, fmaf(P.lam_f, fmaxf(1.0f - p, P.kappa_f), 1.0f));
    if (MODE == CIS_MODE_TIS)
        return fminf(k, P.tis_cap_f);
    if (MODE == CIS_MODE_EXACT)
        return fminf(fmaxf(k, P.exact_lo_f), P.exact_hi_f);
    if (MODE == CIS_MODE_BAND)
        return fmaxf(fminf(k, fmaf(P.lam_f, fmaxf(1.0f - p, P.kappa_f), 1.0f)),
                     0.5f * (1.0f + p));
    if (MODE == CIS_MODE_ICEPOP) {  // log k against the band, in log2 units
        const float lk2 = xp - xq;
        return (lk2 < (float)(P.log_icepop_lo * 1.4426950408889634) ||
                lk2 > (float)(P.log_icepop_hi * 1.4426950408889634))
                   ? 0.0f
                   : k;
    }
    if (MODE == CIS_MODE_KPOP) {
        // binary KL both ways with p, q clamped to [1e-8, 1 - 1e-8], in the
        // log domain so that 1 - 1e-8 stays representable
        const float lp = xp * kLn2, lq = xq * kLn2;
        const float lo = -18.420680743952367f;  // log 1e-8
        const float hi = -1e-8f;                // log(1 - 1e-8)
        const float l1p = logf(-expm1f(lp)), l1q = logf(-expm1f(lq));
        const float a = fminf(fmaxf(lp, lo), hi), b = fminf(fmaxf(lq, lo), hi);
        const float a1 = fminf(fmaxf(l1p, lo), hi), b1 = fminf(fmaxf(l1q, lo), hi);
        const float pa = expf(a), qb = expf(b), pa1 = expf(a1), qb1 = expf(b1);
        const float kpq = pa * (a - b) + pa1 * (a1 - b1);
        const float kqp = qb * (b - a) + qb1 * (b1 - a1);
        return fmaxf(kpq, kqp) > (float)P.kpop_phi ? 0.0f : k;
    }
    return 1.0f;  // CIS_MODE_NONE
}

struct DiagShared {
    MaxSum red[kDiagThreads / 32];
    double sums[kDiagThreads / 32][kNSums];
    float lse_p, lse_q;
};

template <typename InT, int MODE>
__global__ void __launch_bounds__(kDiagThreads)
    cis_mismatch_kernel(const InT *zt, const InT *zi, int64_t T, int64_t V, int64_t ld_t,
                        int64_t ld_i, const int32_t *ids, const uint8_t *mask,
                        const DevParams P, float *eps_out, float *logk_out, float *p_out,
                        float *bias2_out, float *dvar_out, int32_t *status)
{
    __shared__ DiagShared sh;
    const int64_t t = blockIdx.x;
    const bool valid = mask == nullptr || mask[t] != 0;
    const int64_t y = ids[t];
    const bool id_ok = y >= 0 && y < V;
    if (!valid || !id_ok) {
        if (threadIdx.x == 0) {
            const float v = valid ? NAN : 0.0f;
            if (valid)
                set_status(status, kStatusBadId);
            eps_out[t] = v;
            if (logk_out) logk_out[t] = v;
            if (p_out) p_out[t] = v;
            if (bias2_out) bias2_out[t] = v;
            if (dvar_out) dvar_out[t] = v;
        }
        return;
    }
    const InT *rt = zt + t * ld_t;
    const InT *ri = zi + t * ld_i;
    // pass 1: each engine's (max, sum) over j != y
    const MaxSum ot = block_ms<kDiagThreads>(row_stats<InT, false, MaxSum, kDiagThreads>(rt, V, y),
                                             sh.red);
    const MaxSum oi = block_ms<kDiagThreads>(row_stats<InT, false, MaxSum, kDiagThreads>(ri, V, y),
                                             sh.red);
    if (threadIdx.x == 0) {
        const float zyt = to_f32(rt[y]), zyi = to_f32(ri[y]);
        const RowScalars st = row_scalars(ot, zyt), si = row_scalars(oi, zyi);
        // eps = logit p - logit q: Lemma 3.1's -delta_y + log sum_{j != y} w_j e^{delta_j}
        // in the normalised gauge, from the log-odds of each engine
        const double dp = ((double)zyt - (double)ot.m) - (double)logf(ot.s);
        const double dq = ((double)zyi - (double)oi.m) - (double)logf(oi.s);
        eps_out[t] = (float)(dp - dq);
        if (logk_out) logk_out[t] = (float)(st.lp64 - si.lp64);
        if (p_out) p_out[t] = expf(st.lp);
        sh.lse_p = st.lse;
        sh.lse_q = si.lse;
    }
    __syncthreads();
    // the exponents in log2 units, x = z log2e - lse log2e (one FMA each);
    // probabilities that flush to 0 add nothing measurable to the sums
    const float op = sh.lse_p * kLog2e, oq = sh.lse_q * kLog2e;
    // pass 2: the sums over every candidate j
    float acc[kNSums] = {0, 0, 0, 0, 0, 0, 0, 0, 0};
    auto add = [&](float a, float b) {
        const float xp = fmaf(a, kLog2e, -op), xq = fmaf(b, kLog2e, -oq);
        const float p = ex2_ftz(xp), q = ex2_ftz(xq);
        const float k = ex2_ftz(xp - xq);
        // a candidate with q = 0 is never drawn: only r = -p counts, so f = 1
        const float f = q > 0.0f ? elem_weight<MODE>(xp, xq, p, k, P) : 1.0f;
        const float fm1 = f - 1.0f;
        const float t1 = q * (fm1 * (f + 1.0f));   // q (f^2 - 1)
        const float t2 = q * fm1;                  // q (f - 1)
        const float r = fmaf(q, f, -p);
        acc[0] = fmaf(p, p, acc[0]);                       // P2
        acc[1] = fmaf(r, r, acc[1]);                       // R2
        acc[2] = fmaf(r, p, acc[2]);                       // RP
        acc[3] = fmaf(t1, fmaf(-2.0f, p, 1.0f), acc[3]);   // C1
        acc[4] += t1;                                      // C2
        acc[5] += t2;                                      // C3
        acc[6] = fmaf(t1, q, acc[6]);                      // C4
        acc[7] = fmaf(t2, p, acc[7]);                      // C5
        acc[8] = fmaf(q, p, acc[8]);                       // QP
    };
    constexpr int EV = 16 / sizeof(InT);
    int64_t j0 = 0;
    if ((reinterpret_cast<uintptr_t>(rt) & 15) == 0 && (reinterpret_cast<uintptr_t>(ri) & 15) == 0) {
        const int64_t nvec = V / EV;
        const uint4 *vt = reinterpret_cast<const uint4 *>(rt);
        const uint4 *vi = reinterpret_cast<const uint4 *>(ri);
        for (int64_t v = threadIdx.x; v < nvec; v += kDiagThreads) {
            float a[EV], b[EV];
            unpack(__ldg(vt + v), a);
            unpack(__ldg(vi + v), b);
#pragma unroll
            for (int e = 0; e < EV; ++e)
                add(a[e], b[e]);
        }
        j0 = nvec * EV;
    }
    for (int64_t j = j0 + threadIdx.x; j < V; j += kDiagThreads)
        add(to_f32(rt[j]), to_f32(ri[j]));
    // block sums in fp64, fixed order
    double d[kNSums];
#pragma unroll
    for (int i = 0; i < kNSums; ++i) {
        double v = (double)acc[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
            v += __shfl_xor_sync(0xffffffffu, v, o);
        d[i] = v;
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0)
#pragma unroll
        for (int i = 0; i < kNSums; ++i)
            sh.sums[wid][i] = d[i];
    __syncthreads();
    if (threadIdx.x == 0) {
        double S[kNSums];
        for (int i = 0; i < kNSums; ++i) {
            S[i] = 0.0;
            for (int w = 0; w < kDiagThreads / 32; ++w)
                S[i] += sh.sums[w][i];
        }
        const double P2 = S[0], R2 = S[1], RP = S[2], C1 = S[3], C2 = S[4], C3 = S[5],
                     C4 = S[6], C5 = S[7], C6 = C5 + 2.0 * S[8];
        const double bias2 = R2 - 2.0 * C3 * RP + C3 * C3 * P2;
        const double dvar = C1 + P2 * C2 - (C4 - (2.0 + C3) * C5 - C3 * C6 + C3 * (2.0 + C3) * P2);
        if (bias2_out) bias2_out[t] = (float)bias2;
        if (dvar_out) dvar_out[t] = (float)dvar;
    }
}


template <typename InT, int MODE>
void launch_mode(const void *zt, const void *zi, int64_t T, int64_t V, int64_t ld_t,
                 int64_t ld_i, const int32_t *ids, const uint8_t *mask, const DevParams &P,
                 float *eps, float *logk, float *p, float *bias2, float *dvar, int32_t *status,
                 cudaStream_t s)
{
    cis_mismatch_kernel<InT, MODE><<<(unsigned)T, kDiagThreads, 0, s>>>(
        static_cast<const InT *>(zt), static_cast<const InT *>(zi), T, V, ld_t, ld_i, ids, mask,
        P, eps, logk, p, bias2, dvar, status);
}

template <typename InT>
void launch_type(const void *zt, const void *zi, int64_t T, int64_t V, int64_t ld_t,
                 int64_t ld_i, const int32_t *ids, const uint8_t *mask, const DevParams &P,
                 float *eps, float *logk, float *p, float *bias2, float *dvar, int32_t *status,
                 cudaStream_t s)
{
#define CIS_DIAG_CASE(M)                                                                          \
    case M:                                                                                      \
        launch_mode<InT, M>(zt, zi, T, V, ld_t, ld_i, ids, mask, P, eps, logk, p, bias2, dvar,    \
                            status, s);                                                          \
        break;
    switch (P.mode) {
        CIS_DIAG_CASE(CIS_MODE_CIS)
        CIS_DIAG_CASE(CIS_MODE_TIS)
        CIS_DIAG_CASE(CIS_MODE_EXACT)
        CIS_DIAG_CASE(CIS_MODE_BAND)
        CIS_DIAG_CASE(CIS_MODE_ICEPOP)
        CIS_DIAG_CASE(CIS_MODE_KPOP)
    default:
        launch_mode<InT, CIS_MODE_NONE>(zt, zi, T, V, ld_t, ld_i, ids, mask, P, eps, logk, p,
                                        bias2, dvar, status, s);
    }
#undef CIS_DIAG_CASE
}

}  // namespace

cudaError_t launch_mismatch(const void *zt, const void *zi, int dtype, int64_t T, int64_t V,
                            int64_t ld_t, int64_t ld_i, const int32_t *ids, const uint8_t *mask,
                            const DevParams &P, float *eps, float *logk, float *p, float *bias2,
                            float *dvar, int32_t *status, cudaStream_t s)
{
    if (T == 0)
        return cudaSuccess;
    if (dtype == CIS_BF16)
        launch_type<__nv_bfloat16>(zt, zi, T, V, ld_t, ld_i, ids, mask, P, eps, logk, p, bias2,
                                   dvar, status, s);
    else
        launch_type<float>(zt, zi, T, V, ld_t, ld_i, ids, mask, P, eps, logk, p, bias2, dvar,
                           status, s);
    return cudaGetLastError();
}

}  // namespace cis

using namespace cis;

extern "C" CIS_API cis_status_t cis_mismatch_diagnostics(
    const void *logits_train, const void *logits_infer, int32_t dtype, int64_t T, int64_t V,
    int64_t ld_train, int64_t ld_infer, const int32_t *ids, const uint8_t *mask,
    const cis_params_t *params, float *eps_out, float *logk_out, float *p_out, float *bias2_out,
    float *dvar_out, int32_t *dev_status, void *stream)
{
    if (T < 0 || T > 0x7fffffffLL || V <= 0 || V > 0x7fffffffLL || ld_train < V ||
        ld_infer < V || (dtype != CIS_F32 && dtype != CIS_BF16))
        return CIS_ERR_INVALID_ARG;
    if (!params_ok(params) || is_seq_mode(params->mode))
        return CIS_ERR_INVALID_ARG;
    if (T == 0)
        return CIS_OK;
    if (logits_train == nullptr || logits_infer == nullptr || ids == nullptr ||
        eps_out == nullptr)
        return CIS_ERR_INVALID_ARG;
    const DevParams P = make_dev_params(*params);
    const cudaError_t e =
        launch_mismatch(logits_train, logits_infer, dtype, T, V, ld_train, ld_infer, ids, mask, P,
                        eps_out, logk_out, p_out, bias2_out, dvar_out, dev_status,
                        (cudaStream_t)stream);
    return e == cudaSuccess ? CIS_OK : CIS_ERR_CUDA;
}
