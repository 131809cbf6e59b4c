// cis_common.cuh -- device helpers shared by the libcis kernels (sm_103a).
//
// Per-token arithmetic of the CIS token pass (arxiv 2609.32444):
//   * the mismatch weight of Algorithm 1 / Eq. 4 (CIS) and Table 8 (TIS,
//     exact ratio, no correction),
//   * the PPO-clipped token objective of Eq. 1 and the scalar c_t that
//     multiplies (softmax - onehot) in the logit gradient,
//   * the row statistics (max / sum of exponentials) the log-softmax needs.
//
// Decisions (truncated or not, PPO clip active or not) are defined in fp64:
// "log k > log cap" with log k = l_w - l_inf evaluated exactly.  The kernels
// evaluate them in fp32 and keep that answer only when it is certain: the
// fp32 operands carry relative errors of a few ulp (expf/expm1f/log1pf/logf
// are accurate to 1-2 ulp, a subtraction to 0.5 ulp), so a gap larger than
// 4e-6 relative cannot change sign in exact arithmetic.  Inside that band the
// comparison is redone in fp64.  The result equals the fp64 decision.
// log p travels as an unevaluated fp32 pair (lp + lp_lo, better than fp32)
// built with error-free sums: fp64 arithmetic is slow on this part (64 cycles
// a dependent operation) and sits on each row's serial path.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "cis.h"

namespace cis {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Hyper-parameters as the kernels use them: fp32 copies for the fast path and
// fp64 values (with logs taken on the host) for the certified fallback.
struct DevParams {
    int32_t mode;
    int32_t agg;
    float lam_f, kappa_f;
    float tis_cap_f, exact_lo_f, exact_hi_f;
    float rho_lo_f, rho_hi_f;  // 1 - c_low, 1 + c_high
    float log_tis_cap_f, log_exact_lo_f, log_exact_hi_f, log_rho_lo_f, log_rho_hi_f;
    double lam, kappa;
    double log_tis_cap, log_exact_lo, log_exact_hi, log_rho_lo, log_rho_hi;
    double log_icepop_lo, log_icepop_hi, kpop_phi;
    double seq_cap, log_seq_cap, log_seq_lo, log_seq_hi;
};

__host__ __device__ __forceinline__ bool is_seq_mode(int32_t mode)
{
    return mode == CIS_MODE_SEQ_TIS || mode == CIS_MODE_SEQ_MIS;
}

// Device status bits (cis_status_t values that can only be seen on the GPU).
constexpr int32_t kStatusTimeout = CIS_ERR_DEVICE_TIMEOUT;
constexpr int32_t kStatusBadId = CIS_ERR_BAD_TOKEN_ID;

// Bounded waits: each mbarrier poll suspends for at most kPollSuspendNs, and a
// wait gives up after kMaxPolls polls (about 2 s) and reports a timeout.
constexpr uint32_t kPollSuspendNs = 1000;
constexpr uint32_t kMaxPolls = 1u << 21;

__device__ __forceinline__ void set_status(int32_t *status, int32_t bits)
{
    if (status)
        atomicOr(status, bits);
}

// bf16 -> fp32 is exact: the bf16 bits are the top half of the binary32.
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

template <typename T> __device__ __forceinline__ float to_f32(T v);
template <> __device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v)
{
    return __bfloat162float(v);
}

// 2^x.  Pass 1 only sums these, so denormal results may flush (.ftz); pass 2
// writes them out, so it keeps subnormal results.
__device__ __forceinline__ float ex2_ftz(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float ex2_full(float x)
{
    float y;
    asm("ex2.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// max with NaN propagation (fmaxf drops a NaN operand).
__device__ __forceinline__ float max_nan(float a, float b)
{
    float r;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
    return r;
}

// Error-free sum (Knuth): a + b = s + e exactly, s = fl(a + b).  Where s is
// not finite the error term is meaningless and is returned as 0.
__device__ __forceinline__ float two_sum(float a, float b, float &e)
{
    const float s = __fadd_rn(a, b);
    const float bv = __fsub_rn(s, a);
    const float er = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bv)), __fsub_rn(b, bv));
    e = isfinite(s) ? er : 0.0f;
    return s;
}

// +1: a > b for certain; -1: a < b for certain (a <= b in the fp64 sense);
// 0: too close to call.  Near a == b the tolerance is 8e-6 relative, which
// covers the operands' combined relative error (at most ~6e-6 where it is
// used).
__device__ __forceinline__ int certain_cmp(float a, float b)
{
    float d = a - b;
    float tol = 4e-6f * (fabsf(a) + fabsf(b)) + 1e-35f;
    if (d > tol)
        return 1;
    if (d < -tol)
        return -1;
    return 0;
}

struct TokenWeight {
    float w;
    float logk;
    uint8_t trunc;
};

// Mismatch weight from log p (training side, the pair lw + lw_lo; lw_lo = 0
// for an fp32 input) and log q (linf, inference side).  Algorithm 1:
// p = exp(lw), k = exp(lw - linf), phi = max(1-p, kappa),
// w = min{k, 1 + lambda*phi}; Table 8 for the other modes.  omp is 1 - p
// where the caller already has it (row_scalars), else negative.
__device__ __forceinline__ TokenWeight token_weight(float lw, float lw_lo, float linf,
                                                    const DevParams &P, float omp = -1.0f)
{
    TokenWeight r;
    float ke;
    const float kh = two_sum(lw, -linf, ke);    // lw - linf = kh + ke exactly
    const float logk = kh + (ke + lw_lo);       // log k, rounded about once
    // the fp64 values, formed only where a decision is taken in fp64
    auto lw64 = [&] { return (double)lw + (double)lw_lo; };
    auto logk64 = [&] { return lw64() - (double)linf; };
    r.logk = logk;
    r.trunc = 0;
    r.w = 1.0f;
    switch (P.mode) {
    case CIS_MODE_CIS: {
        // k > cap compared directly: near the cap, k and cap lie in
        // [1, 1 + lambda], where k's relative error is 2^-24 |log k| (the
        // rounding of log k) plus expf's 2 ulp, at most 6e-6 for any finite
        // fp32 lambda, inside certain_cmp's 4e-6 (k + cap)
        const float om = omp >= 0.0f ? omp : -expm1f(lw);
        const float lam_phi = P.lam_f * fmaxf(om, P.kappa_f);
        const float cap = 1.0f + lam_phi;
        const float k = expf(logk);
        const int s = certain_cmp(k, cap);
        bool tr;
        if (s != 0) {
            tr = s > 0;
        } else {
            const double phi = fmax(-expm1(lw64()), P.kappa);
            tr = logk64() > log1p(P.lam * phi);
        }
        r.trunc = tr;
        r.w = tr ? cap : k;
        break;
    }
    case CIS_MODE_TIS: {
        const int s = certain_cmp(logk, P.log_tis_cap_f);
        const bool tr = s != 0 ? s > 0 : logk64() > P.log_tis_cap;
        r.trunc = tr;
        r.w = tr ? P.tis_cap_f : expf(logk);
        break;
    }
    case CIS_MODE_EXACT: {
        const int sh = certain_cmp(logk, P.log_exact_hi_f);
        const bool hi = sh != 0 ? sh > 0 : logk64() > P.log_exact_hi;
        const int sl = certain_cmp(P.log_exact_lo_f, logk);
        const bool lo = sl != 0 ? sl > 0 : logk64() < P.log_exact_lo;
        r.trunc = hi || lo;
        r.w = hi ? P.exact_hi_f : (lo ? P.exact_lo_f : expf(logk));
        break;
    }
    case CIS_MODE_BAND: {
        // Sec. 4.3: the CIS weight, lifted from below to (1 + p)/2 (the image
        // of e^eps = 1/2); both decisions in fp64
        const double phi = fmax(-expm1(lw64()), P.kappa);
        const double lo = 0.5 * (1.0 + exp(lw64()));
        const bool up = logk64() > log1p(P.lam * phi);
        const bool low = logk64() < log(lo);
        r.trunc = up || low;
        r.w = up ? (float)(1.0 + P.lam * phi) : (low ? (float)lo : expf(logk));
        break;
    }
    case CIS_MODE_ICEPOP: {
        // Table 8: k on [lo, hi] (bounds included), else masked
        const bool out = logk64() < P.log_icepop_lo || logk64() > P.log_icepop_hi;
        r.trunc = out;
        r.w = out ? 0.0f : expf(logk);
        break;
    }
    case CIS_MODE_KPOP: {
        // Table 8 / App. D.5: binary KL both ways in fp64 on probabilities
        // clamped to [1e-8, 1 - 1e-8]; masked when the larger exceeds phi
        const double lo = 1e-8, hi = 1.0 - 1e-8;
        double p = exp(lw64()), q = exp((double)linf);
        p = p < lo ? lo : (p > hi ? hi : p);
        q = q < lo ? lo : (q > hi ? hi : q);
        const double kl_pq = p * log(p / q) + (1.0 - p) * log((1.0 - p) / (1.0 - q));
        const double kl_qp = q * log(q / p) + (1.0 - q) * log((1.0 - q) / (1.0 - p));
        const double m = kl_pq > kl_qp ? kl_pq : kl_qp;
        const bool out = m > P.kpop_phi;
        r.trunc = out;
        r.w = out ? 0.0f : expf(logk);
        break;
    }
    case CIS_MODE_SEQ_TIS:
    case CIS_MODE_SEQ_MIS:
        // the weight is the response's (seq_weight); callers pass it in
        r.w = 0.0f;
        break;
    default:
        break;
    }
    return r;
}

// The weight of every token of a response from log K, the sum of log k over
// its valid tokens (Table 8: Seq-TIS min(K, C), Seq-MIS K 1{K in [lo, hi]}).
__device__ __forceinline__ TokenWeight seq_weight(double logK, const DevParams &P)
{
    TokenWeight r;
    r.logk = (float)logK;
    if (P.mode == CIS_MODE_SEQ_TIS) {
        const bool tr = logK > P.log_seq_cap;
        r.trunc = tr;
        r.w = tr ? (float)P.seq_cap : (float)exp(logK);
    } else {
        const bool out = logK < P.log_seq_lo || logK > P.log_seq_hi;
        r.trunc = out;
        r.w = out ? 0.0f : (float)exp(logK);
    }
    return r;
}

// eps = logit p - logit q (Lemma 3.1), from the two log-probabilities.
__device__ __forceinline__ float token_eps(float lw, float linf)
{
    return (lw - linf) - logf(-expm1f(lw)) + logf(-expm1f(linf));
}

struct TokenLoss {
    float c;      // s w A rho g: multiplies (softmax - onehot) in d loss / d z
    double term;  // -s w min(rho A, clip(rho) A)
};

// Eq. 1 for one token: rho = exp(lp - lp_old) (1 in value without lp_old),
// objective w min(rho A, clip(rho) A); the min takes the unclipped branch on
// ties, so g = 0 only where the clip is strictly active.  log p as the pair
// lp + lp_lo (see token_weight).
__device__ __forceinline__ TokenLoss token_loss(float lp, float lp_lo, bool has_old, float lp_old,
                                                float A, float s, float w, const DevParams &P)
{
    float rho = 1.0f;
    bool g = true;
    if (has_old) {
        float re;
        const float rh = two_sum(lp, -lp_old, re);
        const float lr = rh + (re + lp_lo);
        auto lr64 = [&] { return ((double)lp + (double)lp_lo) - (double)lp_old; };
        rho = expf(lr);
        if (A > 0.0f) {
            const int c = certain_cmp(lr, P.log_rho_hi_f);
            g = c != 0 ? c < 0 : !(lr64() > P.log_rho_hi);
        } else if (A < 0.0f) {
            const int c = certain_cmp(lr, P.log_rho_lo_f);
            g = c != 0 ? c > 0 : !(lr64() < P.log_rho_lo);
        }
    }
    const float rho_c = fminf(fmaxf(rho, P.rho_lo_f), P.rho_hi_f);
    const float obj = g ? rho * A : rho_c * A;
    TokenLoss r;
    r.term = -(double)s * (double)w * (double)obj;
    r.c = g ? s * w * A * rho : 0.0f;
    return r;
}

// ---------------------------------------------------------------------------
// Row statistics over the entries j != y: (m, s) with s = sum e^{z_j - m}.
struct MaxSum {
    float m;
    float s;
};

__device__ __forceinline__ MaxSum ms_combine(MaxSum a, MaxSum b)
{
    const float m = fmaxf(a.m, b.m);
    if (m == -INFINITY)
        return {m, a.s + b.s};  // both empty (their sums are 0 or NaN)
    const float sa = a.m == -INFINITY ? a.s * 0.0f : a.s * ex2_ftz((a.m - m) * kLog2e);
    const float sb = b.m == -INFINITY ? b.s * 0.0f : b.s * ex2_ftz((b.m - m) * kLog2e);
    return {m, sa + sb};
}

__device__ __forceinline__ MaxSum warp_ms(MaxSum v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MaxSum u;
        u.m = __shfl_xor_sync(0xffffffffu, v.m, o);
        u.s = __shfl_xor_sync(0xffffffffu, v.s, o);
        v = ms_combine(v, u);
    }
    return v;
}

// Block-wide (m, s); every thread gets the result.  `sh` needs NT/32 slots.
// kReuse: the slots are used again later, so wait until all have read them.
template <int NT, bool kReuse = true>
__device__ __forceinline__ MaxSum block_ms(MaxSum v, MaxSum *sh)
{
    v = warp_ms(v);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0)
        sh[wid] = v;
    __syncthreads();
    MaxSum r = sh[0];
#pragma unroll
    for (int i = 1; i < NT / 32; ++i)
        r = ms_combine(r, sh[i]);
    if (kReuse)
        __syncthreads();
    return r;
}

// Row statistics with the entropy term: (m, s, u) over a set of entries, with
// s = sum e^{z_j - m} and u = sum e^{z_j - m} (z_j - m).  Moving to a larger
// offset m' scales both by f = e^{m - m'} and shifts u by (m - m') s.
struct MaxSumU {
    float m;
    float s;
    float u;
};

// (m, s) comes from ms_combine itself, so the entropy variants of the kernels
// reduce (m, s) exactly as the others do; u follows the same offsets.
__device__ __forceinline__ MaxSumU msu_combine(MaxSumU a, MaxSumU b)
{
    const MaxSum r = ms_combine(MaxSum{a.m, a.s}, MaxSum{b.m, b.s});
    const float m = r.m;
    if (m == -INFINITY)
        return {m, r.s, a.u + b.u};
    const float ua = a.m == -INFINITY ? a.u * 0.0f
                                      : fmaf(a.m - m, a.s, a.u) * ex2_ftz((a.m - m) * kLog2e);
    const float ub = b.m == -INFINITY ? b.u * 0.0f
                                      : fmaf(b.m - m, b.s, b.u) * ex2_ftz((b.m - m) * kLog2e);
    return {m, r.s, ua + ub};
}

// The pairs (triples) of n CTAs combined at once: the maximum first, then the
// n rescaled sums added in rank order (independent exponentials, one
// dependent step instead of n - 1).  Same empty-set and NaN rules as
// ms_combine / msu_combine.
__device__ __forceinline__ MaxSum combine_flat(const float2 *part, unsigned n)
{
    float M = part[0].x;
    for (unsigned r = 1; r < n; ++r)
        M = fmaxf(M, part[r].x);
    float S = 0.0f;
    for (unsigned r = 0; r < n; ++r) {
        const float2 q = part[r];
        S += (M == -INFINITY || q.x == -INFINITY) ? q.y * (M == -INFINITY ? 1.0f : 0.0f)
                                                   : q.y * ex2_ftz((q.x - M) * kLog2e);
    }
    return {M, S};
}
// Four pairs (the cluster of a 151,936-entry bf16 row), straight-line: two
// 16-byte loads from a 16-byte aligned array, the maximum, then per pair one
// rescaling exponential accumulated by an FMA, in rank order.
__device__ __forceinline__ MaxSum combine4(const float2 *part)
{
    const float4 a = reinterpret_cast<const float4 *>(part)[0];
    const float4 b = reinterpret_cast<const float4 *>(part)[1];
    const float M = fmaxf(fmaxf(a.x, a.z), fmaxf(b.x, b.z));
    if (M == -INFINITY)
        return {M, ((a.y + a.w) + b.y) + b.w};
    // an empty pair (m = -inf) gives ex2(-inf) = 0: s * 0, as in ms_combine
    float S = a.y * ex2_ftz((a.x - M) * kLog2e);
    S = fmaf(a.w, ex2_ftz((a.z - M) * kLog2e), S);
    S = fmaf(b.y, ex2_ftz((b.x - M) * kLog2e), S);
    S = fmaf(b.w, ex2_ftz((b.z - M) * kLog2e), S);
    return {M, S};
}
__device__ __forceinline__ MaxSumU combine_flat(const float4 *part, unsigned n)
{
    float M = part[0].x;
    for (unsigned r = 1; r < n; ++r)
        M = fmaxf(M, part[r].x);
    float S = 0.0f, U = 0.0f;
    for (unsigned r = 0; r < n; ++r) {
        const float4 q = part[r];
        if (M == -INFINITY) {
            S += q.y;
            U += q.z;
        } else if (q.x == -INFINITY) {
            S += q.y * 0.0f;
            U += q.z * 0.0f;
        } else {
            const float f = ex2_ftz((q.x - M) * kLog2e);
            S += q.y * f;
            U += fmaf(q.x - M, q.y, q.z) * f;
        }
    }
    return {M, S, U};
}

__device__ __forceinline__ MaxSumU warp_msu(MaxSumU v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MaxSumU w;
        w.m = __shfl_xor_sync(0xffffffffu, v.m, o);
        w.s = __shfl_xor_sync(0xffffffffu, v.s, o);
        w.u = __shfl_xor_sync(0xffffffffu, v.u, o);
        v = msu_combine(v, w);
    }
    return v;
}

template <int NT, bool kReuse = true>
__device__ __forceinline__ MaxSumU block_msu(MaxSumU v, MaxSumU *sh)
{
    v = warp_msu(v);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0)
        sh[wid] = v;
    __syncthreads();
    MaxSumU r = sh[0];
#pragma unroll
    for (int i = 1; i < NT / 32; ++i)
        r = msu_combine(r, sh[i]);
    if (kReuse)
        __syncthreads();
    return r;
}

// The weight of the common case straight from a row's statistics, without
// logarithms: the CIS, TIS, exact and no-correction operators with the
// current log p as l_w (no l_old, no sequence weight).  From (m', s') over
// j != y and z_y, with t = s' e^{m' - z_y} = (1 - p) / p:
//   p = 1 / (1 + t),   1 - p = t p,   k = p / q = p e^{-l_inf},
// each within ~8 ulp (expf, __fdividef: 2 ulp each), so k and the cap carry
// relative errors near 2e-6, inside certain_cmp's 4e-6 (k + cap).  qinv is
// e^{-l_inf}, formed by the caller ahead of time.  Returns false, deciding
// nothing, where these forms would leave the normal fp32 range
// (|m' - z_y| > 70, l_inf < -70, an empty or non-finite row) or the decision
// is too close to call; the caller then takes the log-domain path
// (row_scalars, token_weight), whose fp64 fallback settles it.
struct DirectWeight {
    float w;
    float omp;  // 1 - p
    float t;    // (1 - p) / p; log p = -log1p(t)
    float E;    // e^{m' - z_y}
    float p;
    uint8_t trunc;
};
__device__ __forceinline__ bool row_weight_direct(MaxSum o, float zy, float linf, float qinv,
                                                  const DevParams &P, DirectWeight &r)
{
    float dl;
    const float dh = two_sum(o.m, -zy, dl);  // m' - z_y = dh + dl exactly
    if (!(fabsf(dh) <= 70.0f) || !(linf >= -70.0f) || !(o.s >= 1.0f) || !(o.s <= 3.0e38f))
        return false;
    const float e = expf(dh);
    r.E = fmaf(e, dl, e);
    const float t = o.s * r.E;
    const float p = __fdividef(1.0f, 1.0f + t);
    const float k = p * qinv;
    r.t = t;
    r.p = p;
    r.omp = t * p;
    r.trunc = 0;
    r.w = 1.0f;
    switch (P.mode) {
    case CIS_MODE_CIS: {
        const float cap = 1.0f + P.lam_f * fmaxf(r.omp, P.kappa_f);
        const int s = certain_cmp(k, cap);
        if (s == 0)
            return false;
        r.trunc = s > 0;
        r.w = s > 0 ? cap : k;
        return true;
    }
    case CIS_MODE_TIS: {
        const int s = certain_cmp(k, P.tis_cap_f);
        if (s == 0)
            return false;
        r.trunc = s > 0;
        r.w = s > 0 ? P.tis_cap_f : k;
        return true;
    }
    case CIS_MODE_EXACT: {
        const int sh = certain_cmp(k, P.exact_hi_f), sl = certain_cmp(P.exact_lo_f, k);
        if (sh == 0 || sl == 0)
            return false;
        r.trunc = sh > 0 || sl > 0;
        r.w = sh > 0 ? P.exact_hi_f : (sl > 0 ? P.exact_lo_f : k);
        return true;
    }
    case CIS_MODE_NONE:
        return true;
    default:
        return false;
    }
}

// Per-row scalars from (m', s') over j != y and z_y.  With the log-odds
//   d = z_y - log sum_{j != y} e^{z_j} = (z_y - m') - log s',
// log p = -softplus(-d) is accurate for p near 0 and near 1 (Sec. 3.3 notes
// that logit p stops being finite when p rounds to 1; d itself stays finite).
// For d <= 0, log p = d - log1p(e^d) can be large in magnitude, so its
// rounding residual is kept too (lp_lo) for the weight; lse - m' is formed
// without cancellation for pass 2.  z_y - m' and the sums with log s' and the
// softplus are error-free fp32 sums (two_sum), not fp64.
struct RowScalars {
    float lp;         // log p of the sampled token (fp32 output)
    float lp_lo;      // log p = lp + lp_lo to better than fp32 (0 for d > 0)
    float lse;        // logsumexp of the row
    float m;          // offset used for the exponent (m' or 0)
    float bias_log2;  // (lse - m) * log2(e), +inf when no other entry is finite
    float omp;        // 1 - p, from the same exponential as the softplus
    __device__ __forceinline__ double lp64() const { return (double)lp + (double)lp_lo; }
};

__device__ __forceinline__ RowScalars row_scalars(MaxSum o, float zy)
{
    RowScalars r;
    if (o.m == -INFINITY && o.s == 0.0f) {
        // every other entry is -inf: p = 1
        r.lp = zy != zy ? zy : 0.0f;
        r.lp_lo = 0.0f;
        r.omp = 0.0f;
        r.lse = zy;
        r.m = 0.0f;
        r.bias_log2 = INFINITY;
        return r;
    }
    float dl, ue;
    const float dh = two_sum(zy, -o.m, dl);          // z_y - m' = dh + dl exactly
    const float ls = logf(o.s);
    const float u = two_sum(dh, -ls, ue);            // dh - ls = u + ue exactly
    const float d = u + (ue + dl);                   // logit p
    float lse_m;                                     // lse - m'
    // 1 - p = sigmoid(-d): e^{-d} / (1 + e^{-d}) for d > 0, 1 / (1 + e^d)
    // otherwise, without the cancellation of 1 - e^{log p}
    if (d > 0.0f) {
        const float e = expf(-d);
        const float t = log1pf(e);                   // softplus(-d) = -log p
        r.omp = __fdividef(e, 1.0f + e);
        r.lp = -t;
        r.lp_lo = 0.0f;
        float ve;
        const float v = two_sum(dh, t, ve);          // (z_y - m') + t
        lse_m = v + (ve + dl);
    } else {
        const float e = expf(d);
        const float t = log1pf(e);                   // softplus(d)
        r.omp = __fdividef(1.0f, 1.0f + e);
        float xe;
        const float x = two_sum(u, -t, xe);          // log p = x + xe + ue + dl
        const float lo = xe + (ue + dl);
        r.lp = x + lo;
        r.lp_lo = isfinite(r.lp) ? lo - (r.lp - x) : 0.0f;
        lse_m = ls + t;
    }
    r.lse = o.m + lse_m;
    r.m = o.m;
    r.bias_log2 = lse_m * kLog2e;
    return r;
}

// Entropy of the row's softmax, H = -sum_j p_j log p_j (the training-side
// entropy the paper logs, App. D), from (m', s', u') over j != y and z_y.
// With p the sampled token's probability and q_j = e^{z_j - m'} / s' the
// distribution over the other entries,
//   H = -p log p - (1 - p) log(1 - p) + (1 - p) H_q,   H_q = log s' - u'/s',
// which has no cancellation when p is close to 0 or to 1; log p and
// log(1 - p) both come from the log-odds d = (z_y - m') - log s'.
__device__ __forceinline__ float row_entropy(MaxSumU o, float zy, float lp)
{
    if (o.m == -INFINITY && o.s == 0.0f)
        return zy != zy ? zy : 0.0f;  // every other entry is -inf: p = 1
    const float ls = logf(o.s);
    float dl, ue;
    const float dh = two_sum(zy, -o.m, dl);
    const float u = two_sum(dh, -ls, ue);
    const float d = u + (ue + dl);  // logit p, as in row_scalars
    // log(1 - p) = -softplus(d)
    const float l1mp = d > 0.0f ? -(d + log1pf(expf(-d))) : -log1pf(expf(d));
    const float p = expf(lp), q = expf(l1mp);
    const float hq = ls - o.u / o.s;
    const float plp = p == 0.0f ? 0.0f : p * lp;      // 0 log 0 = 0
    const float qlq = q == 0.0f ? 0.0f : q * l1mp;
    return -plp - qlq + (q == 0.0f ? 0.0f : q * hq);
}

}  // namespace cis
