// cis_rowwise.cu -- row-streaming kernels of libcis (any row layout).
//
// One CTA per token row.  Pass 1 streams the row once and keeps a running
// (max, sum of exponentials) over the entries j != y_t; the sampled entry is
// left out so that its log-probability comes from the log-odds
//   d = z_y - log sum_{j != y} e^{z_j},   log p = -softplus(-d),
// which stays accurate when p is within an ulp of 1 (Sec. 3.3 notes that the
// logits of p and q stop being finite there; the log-odds form avoids the
// cancellation in 1 - p).  The forward kernel stops there.  The fused kernel
// then forms the weight and the token loss (cis_common.cuh) and streams the
// row a second time -- from L2 when it is still resident -- to write
//   dz_j = c (softmax_j - [j == y]).
// These kernels accept any alignment and row stride; the cluster kernel in
// cis_cluster.cu is the fast path for 16-byte aligned rows.
#include "cis_kernels.h"
#include "cis_rowops.cuh"

namespace cis {
namespace {

constexpr int kRowThreads = 256;

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v)
{
    return __float2bfloat16_rn(v);
}

template <bool kEnt> struct RowShared {
    MaxSum red[kRowThreads / 32];
    float c, m, bias, lp;
};
template <> struct RowShared<true> {
    MaxSumU red[kRowThreads / 32];
    float c, m, bias, lp;
};

template <typename InT, typename OutT, bool kBwd, bool kEnt>
__global__ void __launch_bounds__(kRowThreads) cis_fused_row_kernel(const PassArgs a)
{
    __shared__ RowShared<kEnt> sh;
    const int64_t t = blockIdx.x;
    const bool valid = a.mask == nullptr || a.mask[t] != 0;
    const int64_t y = a.ids[t];
    const bool id_ok = y >= 0 && y < a.V;
    if (!valid || !id_ok) {
        if (kBwd) {
            OutT *orow = reinterpret_cast<OutT *>(a.dz) + t * a.ld_out;
            for (int64_t j = threadIdx.x; j < a.V; j += kRowThreads)
                orow[j] = from_f32<OutT>(0.0f);
        }
        if (threadIdx.x == 0) {
            const float lp = valid ? NAN : 0.0f;
            if (valid)
                set_status(a.status, kStatusBadId);
            if (a.lp_out) a.lp_out[t] = lp;
            if (a.lse_out) a.lse_out[t] = lp;
            if (!kBwd && a.lp64_out) a.lp64_out[t] = lp;
            if (kEnt) a.entropy_out[t] = lp;
            if (kBwd) {
                if (a.w_out) a.w_out[t] = 0.0f;
                if (a.trunc_out) a.trunc_out[t] = 0;
                a.ws_w[t] = 0.0f;
                a.ws_trunc[t] = 0;
                a.ws_logk[t] = 0.0f;
                a.ws_terms[t] = valid ? (double)NAN : 0.0;
            }
        }
        return;
    }
    const InT *row = reinterpret_cast<const InT *>(a.logits) + t * a.ld;
    MaxSum o;
    MaxSumU ou{0.0f, 0.0f, 0.0f};
    if constexpr (kEnt) {
        ou = block_msu<kRowThreads>(row_stats<InT, !kBwd, MaxSumU>(row, a.V, y), sh.red);
        o = MaxSum{ou.m, ou.s};
    } else {
        o = block_ms<kRowThreads>(row_stats<InT, !kBwd>(row, a.V, y), sh.red);
    }
    if (threadIdx.x == 0) {
        const RowScalars rs = row_scalars(o, to_f32(row[y]));
        if (kEnt)
            a.entropy_out[t] = row_entropy(ou, to_f32(row[y]), rs.lp);
        if (a.lp_out) a.lp_out[t] = rs.lp;
        if (a.lse_out) a.lse_out[t] = rs.lse;
        if (!kBwd && a.lp64_out) a.lp64_out[t] = rs.lp64();
        if (kBwd) {
            const bool has_old = a.lp_old != nullptr;
            TokenWeight tw = token_weight(has_old ? a.lp_old[t] : rs.lp,
                                          has_old ? 0.0f : rs.lp_lo, a.lp_inf[t], a.P,
                                          has_old ? -1.0f : rs.omp);
            if (a.w_in) {  // a sequence operator: the response's weight
                tw.w = a.w_in[t];
                tw.trunc = a.trunc_in[t];
            }
            const TokenLoss tl = token_loss(rs.lp, rs.lp_lo, has_old,
                                            has_old ? a.lp_old[t] : 0.0f, a.adv[t], a.scale[t],
                                            tw.w, a.P);
            if (a.w_out) a.w_out[t] = tw.w;
            if (a.trunc_out) a.trunc_out[t] = tw.trunc;
            a.ws_w[t] = tw.w;
            a.ws_trunc[t] = tw.trunc;
            a.ws_logk[t] = tw.logk;
            a.ws_terms[t] = tl.term;
            sh.c = tl.c;
            sh.m = rs.m;
            sh.bias = rs.bias_log2;
            sh.lp = rs.lp;
        }
    }
    if (!kBwd)
        return;
    __syncthreads();
    const float c = sh.c, m = sh.m, bias = sh.bias;
    const float dzy = c * expm1f(sh.lp);  // c (p - 1)
    OutT *orow = reinterpret_cast<OutT *>(a.dz) + t * a.ld_out;
    for (int64_t j = threadIdx.x; j < a.V; j += kRowThreads) {
        const float z = to_f32(row[j]);
        const float v = j == y ? dzy : c * ex2_full(fmaf(z - m, kLog2e, -bias));
        orow[j] = from_f32<OutT>(v);
    }
}

template <typename InT, typename OutT, bool kBwd>
cudaError_t launch_row(const PassArgs &a, cudaStream_t s)
{
    if (a.T == 0)
        return cudaSuccess;
    if (a.entropy_out)
        cis_fused_row_kernel<InT, OutT, kBwd, true><<<(unsigned)a.T, kRowThreads, 0, s>>>(a);
    else
        cis_fused_row_kernel<InT, OutT, kBwd, false><<<(unsigned)a.T, kRowThreads, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_token_logprobs(const PassArgs &a, int dtype, cudaStream_t s)
{
    if (dtype == CIS_BF16)
        return launch_row<__nv_bfloat16, float, false>(a, s);
    return launch_row<float, float, false>(a, s);
}

cudaError_t launch_rowwise_fwd_bwd(const PassArgs &a, int dtype, int out_dtype, cudaStream_t s)
{
    if (dtype == CIS_BF16) {
        if (out_dtype == CIS_BF16)
            return launch_row<__nv_bfloat16, __nv_bfloat16, true>(a, s);
        return launch_row<__nv_bfloat16, float, true>(a, s);
    }
    if (out_dtype == CIS_BF16)
        return launch_row<float, __nv_bfloat16, true>(a, s);
    return launch_row<float, float, true>(a, s);
}

}  // namespace cis
