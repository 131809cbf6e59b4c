// cis_small.cu -- the [T]-sized kernels of libcis.
//
//   cis_scales_kernel   the loss normaliser s_t: 1/n over the n valid tokens
//                   (Algorithm 1) or 1/(G |y_i|) per response (Eq. 1); it
//                   also clears the device status word of the call.
//   cis_weights_kernel  cis_weights: Algorithm 1 / Table 8, one thread per token.
//   cis_reduce_kernel   deterministic sums (one CTA per 256 tokens, then the
//                   last CTA in index order) of the per-token loss terms and the
//                   statistics the paper logs (App. D.1: share of tokens acted
//                   on, largest |log k|; App. D.5: the truncated excess).
#include "cis_kernels.h"

namespace cis {
namespace {

constexpr int kSmallThreads = 1024;
constexpr int kSeqThreads = 256;  // one CTA per response
constexpr int kMaxSeqInShared = 12000;

__device__ __forceinline__ bool is_valid(const uint8_t *mask, int64_t t)
{
    return mask == nullptr || mask[t] != 0;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// The loss normaliser.  global_counts (device {N, G}, or null): the batch's
// counts over every shard, used in place of this call's own.
__global__ void __launch_bounds__(kSmallThreads)
    cis_scales_kernel(const uint8_t *mask, int64_t T, const int32_t *cu, int64_t B, int agg,
                  float *scale, int32_t *status, uint32_t *ticket, const int64_t *global_counts)
{
    __shared__ long long part[kSmallThreads / 32];
    __shared__ int cnt[kMaxSeqInShared];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (threadIdx.x == 0 && status)
        *status = 0;
    if (threadIdx.x == 0 && ticket)  // the reduction at the end of this call counts from 0
        *ticket = 0;
    if (agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN && cu != nullptr) {
        // valid tokens of each response (one warp per response)
        for (int64_t i = wid; i < B; i += kSmallThreads / 32) {
            int64_t lo = cu[i], hi = cu[i + 1];
            lo = lo < 0 ? 0 : (lo > T ? T : lo);
            hi = hi < lo ? lo : (hi > T ? T : hi);
            int c = 0;
            for (int64_t t = lo + lane; t < hi; t += 32)
                c += is_valid(mask, t);
            c = warp_sum(c);
            if (lane == 0)
                cnt[i] = c;
        }
        __syncthreads();
        long long g = 0;
        for (int64_t i = threadIdx.x; i < B; i += kSmallThreads)
            g += cnt[i] > 0;
        g = warp_sum(g);
        if (lane == 0)
            part[wid] = g;
        for (int64_t t = threadIdx.x; t < T; t += kSmallThreads)
            scale[t] = 0.0f;
        __syncthreads();
        long long G = 0;
        for (int i = 0; i < kSmallThreads / 32; ++i)
            G += part[i];
        if (global_counts)
            G = global_counts[1];
        for (int64_t i = wid; i < B; i += kSmallThreads / 32) {
            int64_t lo = cu[i], hi = cu[i + 1];
            lo = lo < 0 ? 0 : (lo > T ? T : lo);
            hi = hi < lo ? lo : (hi > T ? T : hi);
            const int n = cnt[i];
            const float s = n > 0 ? (float)(1.0 / ((double)G * (double)n)) : 0.0f;
            for (int64_t t = lo + lane; t < hi; t += 32)
                scale[t] = is_valid(mask, t) ? s : 0.0f;
        }
        return;
    }
    long long n = 0;
    for (int64_t t = threadIdx.x; t < T; t += kSmallThreads)
        n += is_valid(mask, t);
    n = warp_sum(n);
    if (lane == 0)
        part[wid] = n;
    __syncthreads();
    long long N = 0;
    for (int i = 0; i < kSmallThreads / 32; ++i)
        N += part[i];
    if (global_counts)
        N = global_counts[0];
    const float s = N > 0 ? (float)(1.0 / (double)N) : 0.0f;
    for (int64_t t = threadIdx.x; t < T; t += kSmallThreads)
        scale[t] = is_valid(mask, t) ? s : 0.0f;
}

// This call's {N, G}: valid tokens, and responses with a valid token (one
// warp per response), for the all-reduce of a token-sharded run.
__global__ void __launch_bounds__(kSmallThreads)
    cis_count_kernel(const uint8_t *mask, int64_t T, const int32_t *cu, int64_t B,
                     int64_t *counts)
{
    __shared__ long long part[2][kSmallThreads / 32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    long long n = 0, g = 0;
    for (int64_t t = threadIdx.x; t < T; t += kSmallThreads)
        n += is_valid(mask, t);
    if (cu != nullptr) {
        for (int64_t i = wid; i < B; i += kSmallThreads / 32) {
            int64_t lo = cu[i], hi = cu[i + 1];
            lo = lo < 0 ? 0 : (lo > T ? T : lo);
            hi = hi < lo ? lo : (hi > T ? T : hi);
            int c = 0;
            for (int64_t t = lo + lane; t < hi; t += 32)
                c += is_valid(mask, t);
            c = warp_sum(c);
            if (lane == 0)
                g += c > 0;
        }
    }
    n = warp_sum(n);
    g = warp_sum(g);
    if (lane == 0) {
        part[0][wid] = n;
        part[1][wid] = g;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        long long N = 0, G = 0;
        for (int i = 0; i < kSmallThreads / 32; ++i) {
            N += part[0][i];
            G += part[1][i];
        }
        counts[0] = N;
        counts[1] = G;
    }
}

__global__ void cis_weights_kernel(const float *lp_w, const float *lp_inf, const uint8_t *mask,
                               int64_t T, const DevParams P, float *w_out, uint8_t *trunc_out,
                               float *eps_out)
{
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
         t += (int64_t)gridDim.x * blockDim.x) {
        float w = 0.0f, e = 0.0f;
        uint8_t tr = 0;
        if (is_valid(mask, t)) {
            const float lw = lp_w[t], li = lp_inf[t];
            const TokenWeight tw = token_weight(lw, 0.0f, li, P);
            w = tw.w;
            tr = tw.trunc;
            if (eps_out)
                e = token_eps(lw, li);
        }
        w_out[t] = w;
        if (trunc_out)
            trunc_out[t] = tr;
        if (eps_out)
            eps_out[t] = e;
    }
}

// One CTA per response: the fp64 sum of log k over its valid tokens in a
// fixed order (thread-strided partial sums, then a tree), then the response's
// weight for each of them (seq_weight, Table 8).
__global__ void __launch_bounds__(kSeqThreads)
    cis_seq_weights_kernel(const double *lw64, const float *lw32, const float *lp_inf,
                           const int32_t *ids, int64_t V, const uint8_t *mask,
                           const int32_t *cu, int64_t T, const DevParams P, float *w,
                           uint8_t *trunc)
{
    __shared__ double red[kSeqThreads];
    const int64_t i = blockIdx.x;
    int64_t b = cu[i], e = cu[i + 1];
    b = b < 0 ? 0 : (b > T ? T : b);
    e = e < b ? b : (e > T ? T : e);
    auto used = [&](int64_t t) {
        return is_valid(mask, t) && (ids == nullptr || (ids[t] >= 0 && (int64_t)ids[t] < V));
    };
    double acc = 0.0;
    for (int64_t t = b + threadIdx.x; t < e; t += kSeqThreads)
        if (used(t))
            acc += (lw64 ? lw64[t] : (double)lw32[t]) - (double)lp_inf[t];
    red[threadIdx.x] = acc;
    __syncthreads();
    for (int off = kSeqThreads / 2; off > 0; off >>= 1) {
        if (threadIdx.x < off)
            red[threadIdx.x] += red[threadIdx.x + off];
        __syncthreads();
    }
    const TokenWeight tw = seq_weight(red[0], P);
    for (int64_t t = b + threadIdx.x; t < e; t += kSeqThreads)
        if (used(t)) {
            w[t] = tw.w;
            if (trunc)
                trunc[t] = tw.trunc;
        }
}

struct RedPart {
    double loss, excess, ent;
    long long nvalid, ntrunc;
    float maxlk;
};

__device__ __forceinline__ RedPart red_add(RedPart a, const RedPart &b)
{
    a.loss += b.loss;
    a.excess += b.excess;
    a.ent += b.ent;
    a.nvalid += b.nvalid;
    a.ntrunc += b.ntrunc;
    a.maxlk = fmaxf(a.maxlk, b.maxlk);
    return a;
}

__device__ __forceinline__ RedPart red_shfl(const RedPart &v, int o)
{
    RedPart r;
    r.loss = __shfl_xor_sync(0xffffffffu, v.loss, o);
    r.excess = __shfl_xor_sync(0xffffffffu, v.excess, o);
    r.ent = __shfl_xor_sync(0xffffffffu, v.ent, o);
    r.nvalid = __shfl_xor_sync(0xffffffffu, v.nvalid, o);
    r.ntrunc = __shfl_xor_sync(0xffffffffu, v.ntrunc, o);
    r.maxlk = __shfl_xor_sync(0xffffffffu, v.maxlk, o);
    return r;
}

__device__ __forceinline__ RedPart red_warp(RedPart v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v = red_add(v, red_shfl(v, o));
    return v;
}

// Sums over the tokens in fp64, deterministic and spread over many SMs (fp64
// arithmetic runs at a small fraction of the fp32 rate here, so one CTA
// summing every token was bound by its SM's fp64 pipe).  CTA b takes tokens
// [256 b, 256 b + 256), one per thread, and reduces them in a fixed tree
// (within each warp, then over the warps in order) into parts[b]; the last
// CTA to finish (a ticket, zeroed by the scales kernel at the start of the
// call) adds the parts in index order the same way and writes the results.
__device__ __forceinline__ RedPart block_red(RedPart p, RedPart *sh)
{
    constexpr int kWarps = kRedTokens / 32;
    p = red_warp(p);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0)
        sh[wid] = p;
    __syncthreads();
    RedPart r{0.0, 0.0, 0.0, 0, 0, 0.0f};
    if (wid == 0) {
        r = lane < kWarps ? sh[lane] : r;
        r = red_warp(r);
    }
    __syncthreads();
    return r;  // valid in thread 0
}

__global__ void __launch_bounds__(kRedTokens)
    cis_reduce_kernel(const uint8_t *mask, int64_t T, const double *terms, const float *logk,
                  const float *w, const uint8_t *trunc, const float *entropy,
                  const int32_t *status, RedPart *parts, uint32_t *ticket, cis_stats_t *stats,
                  double *loss_out)
{
    __shared__ RedPart sh[kRedTokens / 32];
    __shared__ bool last;
    RedPart p{0.0, 0.0, 0.0, 0, 0, 0.0f};
    const int64_t t = (int64_t)blockIdx.x * kRedTokens + threadIdx.x;
    if (t < T) {
        p.loss = terms[t];
        if (is_valid(mask, t)) {
            p.nvalid = 1;
            const float lk = logk[t];
            p.maxlk = fabsf(lk);
            if (trunc[t]) {
                p.ntrunc = 1;
                p.excess = exp((double)lk) - (double)w[t];
            }
            if (entropy)
                p.ent = (double)entropy[t];
        }
    }
    p = block_red(p, sh);
    if (threadIdx.x == 0) {
        parts[blockIdx.x] = p;
        __threadfence();
        last = atomicAdd(ticket, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last)
        return;
    __threadfence();
    const volatile RedPart *vp = parts;
    RedPart q{0.0, 0.0, 0.0, 0, 0, 0.0f};
    for (unsigned b = threadIdx.x; b < gridDim.x; b += kRedTokens) {
        RedPart x;
        x.loss = vp[b].loss;
        x.excess = vp[b].excess;
        x.ent = vp[b].ent;
        x.nvalid = vp[b].nvalid;
        x.ntrunc = vp[b].ntrunc;
        x.maxlk = vp[b].maxlk;
        q = red_add(q, x);
    }
    q = block_red(q, sh);
    if (threadIdx.x == 0) {
        if (loss_out)
            *loss_out = q.loss;
        if (stats) {
            stats->loss = q.loss;
            stats->trunc_excess = q.excess;
            stats->n_valid = q.nvalid;
            stats->n_truncated = q.ntrunc;
            stats->max_abs_logk = q.maxlk;
            stats->status = status ? *status : 0;
            stats->entropy_sum = q.ent;
        }
    }
}

}  // namespace

cudaError_t launch_scales(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens, int64_t B,
                          int agg, float *scale, int32_t *status, uint32_t *ticket,
                          cudaStream_t s, const int64_t *global_counts)
{
    if (agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN && B > kMaxSeqInShared)
        return cudaErrorNotSupported;
    cis_scales_kernel<<<1, kSmallThreads, 0, s>>>(mask, T, cu_seqlens, B, agg, scale, status,
                                                  ticket, global_counts);
    return cudaGetLastError();
}

cudaError_t launch_count_valid(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                               int64_t B, int64_t *counts, cudaStream_t s)
{
    if (B > kMaxSeqInShared)
        return cudaErrorNotSupported;
    cis_count_kernel<<<1, kSmallThreads, 0, s>>>(mask, T, cu_seqlens, B, counts);
    return cudaGetLastError();
}

cudaError_t launch_weights(const float *lp_w, const float *lp_inf, const uint8_t *mask,
                           int64_t T, const DevParams &P, float *w_out, uint8_t *trunc_out,
                           float *eps_out, cudaStream_t s)
{
    if (T == 0)
        return cudaSuccess;
    int64_t blocks = (T + 255) / 256;
    if (blocks > 4096)
        blocks = 4096;
    cis_weights_kernel<<<(unsigned)blocks, 256, 0, s>>>(lp_w, lp_inf, mask, T, P, w_out, trunc_out,
                                                    eps_out);
    return cudaGetLastError();
}

cudaError_t launch_reduce(const PassArgs &a, cis_stats_t *stats, double *loss, cudaStream_t s)
{
    if (a.red_parts == nullptr || a.red_ticket == nullptr)
        return cudaErrorInvalidValue;
    static_assert(sizeof(RedPart) <= kRedPartBytes, "a partial sum must fit its slot");
    const int64_t blocks = a.T > 0 ? (a.T + kRedTokens - 1) / kRedTokens : 1;
    cis_reduce_kernel<<<(unsigned)blocks, kRedTokens, 0, s>>>(
        a.mask, a.T, a.ws_terms, a.ws_logk, a.ws_w, a.ws_trunc, a.entropy_out, a.status,
        static_cast<RedPart *>(a.red_parts), a.red_ticket, stats, loss);
    return cudaGetLastError();
}

cudaError_t launch_seq_weights(const double *lw64, const float *lw32, const float *lp_inf,
                               const int32_t *ids, int64_t V, const uint8_t *mask,
                               const int32_t *cu_seqlens, int64_t B, int64_t T,
                               const DevParams &P, float *w, uint8_t *trunc, cudaStream_t s)
{
    if (B <= 0 || T <= 0)
        return cudaSuccess;
    if (B > 0x7fffffffLL)
        return cudaErrorInvalidValue;
    cis_seq_weights_kernel<<<(unsigned)B, kSeqThreads, 0, s>>>(lw64, lw32, lp_inf, ids, V, mask,
                                                                cu_seqlens, T, P, w, trunc);
    return cudaGetLastError();
}

}  // namespace cis

