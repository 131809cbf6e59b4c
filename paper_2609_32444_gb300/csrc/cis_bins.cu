// cis_bins.cu -- confidence-binned counts and sums of per-token values.
//
// The paper reports its statistics by bins of confidence: the sampled tokens
// binned by p_t with E[k_t - f_t] in each bin (Sec. 4.3, Fig. 5b), and
// logarithmic bins of 1 - p_t for the displacement and the log ratio (App.
// A.5).  cis_binned_sums takes any per-token key (p, 1 - p, ...) and up to four
// per-token values (k - f, the diagnostics' bias2 and dvar, ...) and gives
// each bin's count and the fp64 sums of the values; means are sum / count.
//
// Deterministic: CTA c takes token chunks c, c + grid, ... of 256 tokens; per
// chunk, warp w sums bins w, w + 8, ... over the chunk's tokens in a fixed
// order (lane by lane, then a fixed butterfly) into the CTA's running
// partials; the last CTA to finish adds the CTAs' partials in index order.
#include "cis_kernels.h"
#include "cis_nvtx.h"

namespace cis {
namespace {

constexpr int kBinTokens = 256;  // tokens per chunk, one per thread
constexpr int kBinWarps = kBinTokens / 32;
constexpr int kMaxBinCtas = 1024;
constexpr int kMaxBins = CIS_MAX_BINS;
constexpr int kMaxBinValues = CIS_MAX_BIN_VALUES;

struct BinArgs {
    double edges[kMaxBins + 1];
    const float *values[kMaxBinValues];
    int nbins;
};

// The bin of key x: edges[b] <= x < edges[b + 1], the last bin closed on the
// right; -1 for a key outside [edges[0], edges[nbins]] or NaN.
__device__ __forceinline__ int bin_of(float key, const BinArgs &a)
{
    const double x = (double)key;
    if (!(x >= a.edges[0] && x <= a.edges[a.nbins]))
        return -1;
    int lo = 0, hi = a.nbins;  // edges[lo] <= x; the bin is in [lo, hi)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (a.edges[mid] <= x)
            lo = mid;
        else
            hi = mid;
    }
    return lo;
}

__device__ __forceinline__ double warp_sum_d(double v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// NV value arrays.  parts: [grid][nbins][NV + 1] (the count first), the
// ticket zeroed before the launch.
template <int NV>
__global__ void __launch_bounds__(kBinTokens)
    cis_binned_sums_kernel(const float *key, const uint8_t *mask, int64_t T,
                           const __grid_constant__ BinArgs a, double *parts, uint32_t *ticket,
                           int64_t *counts_out, double *sums_out)
{
    constexpr int kF = NV + 1;  // count, then the sums
    __shared__ int sbin[kBinTokens];
    __shared__ float sval[NV > 0 ? NV : 1][kBinTokens];
    __shared__ double sacc[kMaxBins * kF];
    __shared__ bool last;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int k = threadIdx.x; k < a.nbins * kF; k += kBinTokens)
        sacc[k] = 0.0;
    const int64_t nchunks = (T + kBinTokens - 1) / kBinTokens;
    for (int64_t ch = blockIdx.x; ch < nchunks; ch += gridDim.x) {
        const int64_t t = ch * kBinTokens + threadIdx.x;
        int b = -1;
        if (t < T && (mask == nullptr || mask[t] != 0))
            b = bin_of(key[t], a);
        sbin[threadIdx.x] = b;
#pragma unroll
        for (int i = 0; i < NV; ++i)
            sval[i][threadIdx.x] = b >= 0 ? a.values[i][t] : 0.0f;
        __syncthreads();
        for (int bin = warp; bin < a.nbins; bin += kBinWarps) {
            double c = 0.0, s[NV > 0 ? NV : 1];
#pragma unroll
            for (int i = 0; i < NV; ++i)
                s[i] = 0.0;
            for (int j = lane; j < kBinTokens; j += 32) {
                if (sbin[j] == bin) {
                    c += 1.0;
#pragma unroll
                    for (int i = 0; i < NV; ++i)
                        s[i] += (double)sval[i][j];
                }
            }
            c = warp_sum_d(c);
#pragma unroll
            for (int i = 0; i < NV; ++i)
                s[i] = warp_sum_d(s[i]);
            if (lane == 0) {  // this warp owns the bin's accumulators
                sacc[bin * kF] += c;
#pragma unroll
                for (int i = 0; i < NV; ++i)
                    sacc[bin * kF + 1 + i] += s[i];
            }
        }
        __syncthreads();  // the chunk's keys and values are read before the next
    }
    double *mine = parts + (size_t)blockIdx.x * a.nbins * kF;
    for (int k = threadIdx.x; k < a.nbins * kF; k += kBinTokens)
        mine[k] = sacc[k];
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        last = atomicAdd(ticket, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last)
        return;
    __threadfence();
    const volatile double *vp = parts;
    for (int k = threadIdx.x; k < a.nbins * kF; k += kBinTokens) {
        double acc = 0.0;
        for (unsigned c = 0; c < gridDim.x; ++c)
            acc += vp[(size_t)c * a.nbins * kF + k];
        const int bin = k / kF, f = k - bin * kF;
        if (f == 0)
            counts_out[bin] = (int64_t)acc;
        else
            sums_out[(size_t)(f - 1) * a.nbins + bin] = acc;
    }
}

int64_t bin_ctas(int64_t T)
{
    const int64_t n = (T + kBinTokens - 1) / kBinTokens;
    return n < 1 ? 1 : (n > kMaxBinCtas ? kMaxBinCtas : n);
}

size_t bin_parts_bytes(int64_t T, int nbins, int nvalues)
{
    return (size_t)bin_ctas(T) * (size_t)nbins * (size_t)(nvalues + 1) * sizeof(double);
}

}  // namespace
}  // namespace cis

using namespace cis;

extern "C" {

CIS_API cis_status_t cis_binned_sums_workspace_size(int64_t T, int32_t nbins, int32_t nvalues,
                                                    size_t *bytes)
{
    if (bytes == nullptr || T < 0 || nbins < 1 || nbins > kMaxBins || nvalues < 0 ||
        nvalues > kMaxBinValues)
        return CIS_ERR_INVALID_ARG;
    *bytes = (bin_parts_bytes(T, nbins, nvalues) + 255) / 256 * 256 + 256;
    return CIS_OK;
}

CIS_API cis_status_t cis_binned_sums(const float *key, const uint8_t *mask, int64_t T,
                                     const double *edges, int32_t nbins,
                                     const float *const *values, int32_t nvalues,
                                     int64_t *counts_out, double *sums_out, void *workspace,
                                     size_t workspace_bytes, void *stream)
{
    NvtxRange nvtx_range("cis_binned_sums");
    size_t need = 0;
    if (cis_binned_sums_workspace_size(T, nbins, nvalues, &need) != CIS_OK || edges == nullptr ||
        counts_out == nullptr || (nvalues > 0 && (values == nullptr || sums_out == nullptr)) ||
        (T > 0 && key == nullptr) || workspace == nullptr || workspace_bytes < need ||
        (reinterpret_cast<uintptr_t>(workspace) & 255))
        return CIS_ERR_INVALID_ARG;
    BinArgs a = {};
    a.nbins = nbins;
    for (int b = 0; b <= nbins; ++b) {
        a.edges[b] = edges[b];
        if (!(edges[b] == edges[b]) || (b > 0 && !(edges[b] > edges[b - 1])))
            return CIS_ERR_INVALID_ARG;  // NaN, or not strictly ascending
    }
    for (int i = 0; i < nvalues; ++i) {
        if (T > 0 && values[i] == nullptr)
            return CIS_ERR_INVALID_ARG;
        a.values[i] = values[i];
    }
    cudaStream_t s = (cudaStream_t)stream;
    double *parts = static_cast<double *>(workspace);
    uint32_t *ticket = reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(workspace) + need - 256);
    if (cudaMemsetAsync(ticket, 0, sizeof(uint32_t), s) != cudaSuccess)
        return CIS_ERR_CUDA;
    const unsigned grid = (unsigned)bin_ctas(T);
    switch (nvalues) {
    case 0:
        cis_binned_sums_kernel<0><<<grid, kBinTokens, 0, s>>>(key, mask, T, a, parts, ticket,
                                                              counts_out, sums_out);
        break;
    case 1:
        cis_binned_sums_kernel<1><<<grid, kBinTokens, 0, s>>>(key, mask, T, a, parts, ticket,
                                                              counts_out, sums_out);
        break;
    case 2:
        cis_binned_sums_kernel<2><<<grid, kBinTokens, 0, s>>>(key, mask, T, a, parts, ticket,
                                                              counts_out, sums_out);
        break;
    case 3:
        cis_binned_sums_kernel<3><<<grid, kBinTokens, 0, s>>>(key, mask, T, a, parts, ticket,
                                                              counts_out, sums_out);
        break;
    default:
        cis_binned_sums_kernel<4><<<grid, kBinTokens, 0, s>>>(key, mask, T, a, parts, ticket,
                                                              counts_out, sums_out);
        break;
    }
    return cudaGetLastError() == cudaSuccess ? CIS_OK : CIS_ERR_CUDA;
}

}  // extern "C"
