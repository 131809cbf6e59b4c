// cis_rowops.cuh -- row-streaming building blocks shared by the row kernels
// (cis_rowwise.cu) and the mismatch diagnostics (cis_diag.cu): a running
// (max, sum of exponentials) -- optionally with the entropy term -- over the
// entries j != y of one row, read with 16-byte vector loads.
#pragma once

#include "cis_common.cuh"

namespace cis {
namespace {

// Add EV values to a running (m, s), leaving out position `skip` (-1: none).
template <int EV>
__device__ __forceinline__ void ms_update(MaxSum &acc, const float (&z)[EV], int skip)
{
    float lm = -INFINITY;
#pragma unroll
    for (int i = 0; i < EV; ++i)
        lm = max_nan(lm, i == skip ? -INFINITY : z[i]);
    if (lm > acc.m || lm != lm) {
        acc.s = acc.s * ex2_ftz((acc.m - lm) * kLog2e);
        acc.m = lm;
    }
    if (acc.m != -INFINITY) {
        float e[EV];
#pragma unroll
        for (int i = 0; i < EV; ++i)
            e[i] = i == skip ? 0.0f : ex2_ftz((z[i] - acc.m) * kLog2e);
#pragma unroll
        for (int w = 1; w < EV; w <<= 1)
#pragma unroll
            for (int i = 0; i + w < EV; i += 2 * w)
                e[i] += e[i + w];
        acc.s += e[0];
    }
}

// The same for (m, s, u): (m, s) by the update above, so that it is the same
// bit for bit; u = sum e^{z - m} (z - m) follows the offset.
template <int EV>
__device__ __forceinline__ void ms_update(MaxSumU &acc, const float (&z)[EV], int skip)
{
    const float m0 = acc.m, s0 = acc.s;
    MaxSum ms{acc.m, acc.s};
    ms_update<EV>(ms, z, skip);
    float u = acc.u;
    if (!(ms.m == m0)) {  // the offset moved (or became NaN)
        if (m0 == -INFINITY) {
            u = u * 0.0f;
        } else {
            const float d = m0 - ms.m;
            u = fmaf(d, s0, u) * ex2_ftz(d * kLog2e);
        }
    }
    if (ms.m != -INFINITY) {
#pragma unroll
        for (int i = 0; i < EV; ++i) {
            const float d = z[i] - ms.m;
            const float e = i == skip ? 0.0f : ex2_ftz(d * kLog2e);
            u = fmaf(e, fmaxf(d, -1024.0f), u);
        }
    }
    acc.m = ms.m;
    acc.s = ms.s;
    acc.u = u;
}

template <typename InT, bool kStream>
__device__ __forceinline__ uint4 load16(const uint4 *p)
{
    return kStream ? __ldcs(p) : __ldg(p);
}

// Unpack one 16-byte vector into floats.
__device__ __forceinline__ void unpack(uint4 q, float (&z)[8])
{
    z[0] = bf16_lo(q.x); z[1] = bf16_hi(q.x);
    z[2] = bf16_lo(q.y); z[3] = bf16_hi(q.y);
    z[4] = bf16_lo(q.z); z[5] = bf16_hi(q.z);
    z[6] = bf16_lo(q.w); z[7] = bf16_hi(q.w);
}
__device__ __forceinline__ void unpack(uint4 q, float (&z)[4])
{
    z[0] = __uint_as_float(q.x); z[1] = __uint_as_float(q.y);
    z[2] = __uint_as_float(q.z); z[3] = __uint_as_float(q.w);
}

// This thread's (m, s) -- or (m, s, u) -- over entries j != y of one row.
template <typename InT, bool kStream, typename Acc = MaxSum, int NT = 256>
__device__ Acc row_stats(const InT *row, int64_t V, int64_t y)
{
    constexpr int EV = 16 / sizeof(InT);
    Acc acc{};
    acc.m = -INFINITY;
    int64_t j0 = 0;
    if ((reinterpret_cast<uintptr_t>(row) & 15) == 0) {
        const int64_t nvec = V / EV;
        const uint4 *rv = reinterpret_cast<const uint4 *>(row);
        for (int64_t v = threadIdx.x; v < nvec; v += NT) {
            float z[EV];
            unpack(load16<InT, kStream>(rv + v), z);
            const int64_t rel = y - v * EV;
            ms_update<EV>(acc, z, (rel >= 0 && rel < EV) ? (int)rel : -1);
        }
        j0 = nvec * EV;
    }
    for (int64_t j = j0 + threadIdx.x; j < V; j += NT) {
        float z[1] = {to_f32(row[j])};
        ms_update<1>(acc, z, j == y ? 0 : -1);
    }
    return acc;
}

}  // namespace
}  // namespace cis
