// cis_dsmem.cuh -- building blocks of the cluster kernels (sm_100 and later):
// mbarriers with bounded waits, bulk asynchronous copies from global into
// shared memory, stores into a peer CTA's shared memory counted on its
// mbarrier, cluster barriers, and per-thread row reductions over a slab of
// logits held in shared memory.
#pragma once

#include "cis_common.cuh"

namespace cis {
namespace {

constexpr int kMaxCluster = 8;
constexpr int kChunks = 2;  // a slice is copied in this many pieces (1 to 8 measured: 2 is fastest)

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// Several initialisations, then one fence that makes all of them visible to
// the cluster (and to the async proxy).
__device__ __forceinline__ void mbar_init_only(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                         uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// Bounded wait on phase `parity` of an mbarrier: at most max_polls polls,
// each suspending for up to kPollSuspendNs; false if it never completed.
__device__ __forceinline__ bool mbar_wait_n(uint32_t bar, uint32_t parity, uint32_t max_polls)
{
    for (uint32_t i = 0; i < max_polls; ++i) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(bar), "r"(parity), "r"(kPollSuspendNs)
            : "memory");
        if (done)
            return true;
    }
    return false;
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    return mbar_wait_n(bar, parity, kMaxPolls);
}

__device__ __forceinline__ void cluster_arrive_relaxed()
{
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait()
{
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

// 8 consecutive entries from shared memory as floats.
template <typename InT> __device__ __forceinline__ void load8(const uint8_t *sm, int g,
                                                              float (&z)[8]);
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const uint8_t *sm, int g, float (&z)[8])
{
    const uint4 q = reinterpret_cast<const uint4 *>(sm)[g];
    z[0] = bf16_lo(q.x); z[1] = bf16_hi(q.x);
    z[2] = bf16_lo(q.y); z[3] = bf16_hi(q.y);
    z[4] = bf16_lo(q.z); z[5] = bf16_hi(q.z);
    z[6] = bf16_lo(q.w); z[7] = bf16_hi(q.w);
}
template <>
__device__ __forceinline__ void load8<float>(const uint8_t *sm, int g, float (&z)[8])
{
    const uint4 q0 = reinterpret_cast<const uint4 *>(sm)[2 * g];
    const uint4 q1 = reinterpret_cast<const uint4 *>(sm)[2 * g + 1];
    z[0] = __uint_as_float(q0.x); z[1] = __uint_as_float(q0.y);
    z[2] = __uint_as_float(q0.z); z[3] = __uint_as_float(q0.w);
    z[4] = __uint_as_float(q1.x); z[5] = __uint_as_float(q1.y);
    z[6] = __uint_as_float(q1.z); z[7] = __uint_as_float(q1.w);
}

// Overwrite entry j of the slab with -inf.
template <typename InT> __device__ __forceinline__ void poke_neg_inf(uint8_t *sm, int j);
template <> __device__ __forceinline__ void poke_neg_inf<__nv_bfloat16>(uint8_t *sm, int j)
{
    reinterpret_cast<uint16_t *>(sm)[j] = 0xff80u;  // bf16 -inf
}
template <> __device__ __forceinline__ void poke_neg_inf<float>(uint8_t *sm, int j)
{
    reinterpret_cast<float *>(sm)[j] = -INFINITY;
}

// Running maximum over this thread's groups (NaN propagates), fed chunk by
// chunk.  bf16 rows are compared two entries at a time without unpacking.
template <typename InT> struct MaxAcc;
template <> struct MaxAcc<__nv_bfloat16> {
    __nv_bfloat162 a0, a1;
    __device__ __forceinline__ MaxAcc()
    {
        const uint32_t ninf2 = 0xff80ff80u;
        a0 = a1 = *reinterpret_cast<const __nv_bfloat162 *>(&ninf2);
    }
    __device__ __forceinline__ void consume(const uint8_t *sm, int g0, int g1, int step)
    {
        for (int g = g0; g < g1; g += step) {
            const uint4 q = reinterpret_cast<const uint4 *>(sm)[g];
            a0 = __hmax2_nan(a0, *reinterpret_cast<const __nv_bfloat162 *>(&q.x));
            a1 = __hmax2_nan(a1, *reinterpret_cast<const __nv_bfloat162 *>(&q.y));
            a0 = __hmax2_nan(a0, *reinterpret_cast<const __nv_bfloat162 *>(&q.z));
            a1 = __hmax2_nan(a1, *reinterpret_cast<const __nv_bfloat162 *>(&q.w));
        }
    }
    __device__ __forceinline__ float result() const
    {
        const __nv_bfloat162 a = __hmax2_nan(a0, a1);
        return max_nan(__low2float(a), __high2float(a));
    }
};
template <> struct MaxAcc<float> {
    float m = -INFINITY;
    __device__ __forceinline__ void consume(const uint8_t *sm, int g0, int g1, int step)
    {
        for (int g = g0; g < g1; g += step) {
            float z[8];
            load8<float>(sm, g, z);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                m = max_nan(m, z[i]);
        }
    }
    __device__ __forceinline__ float result() const { return m; }
};

// Sum of 2^{z_i log2e - off} over 8 values, added pairwise.
__device__ __forceinline__ float sum8_exp2_off(const float (&z)[8], float off)
{
    float e[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
        e[i] = ex2_ftz(fmaf(z[i], kLog2e, -off));
    return ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
}

// The same, also accumulating u += e_i x_i with x_i = z_i log2e - off (the
// exponent): the entropy term, in log2 units before the offset correction.
// Entries whose exponential flushes to 0 (x_i <= -126) add nothing; x_i is
// clamped so that -inf entries (e_i = 0) give 0, not NaN.
__device__ __forceinline__ float sum8_exp2_off_u(const float (&z)[8], float off, float &u)
{
    float e[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const float x = fmaf(z[i], kLog2e, -off);
        e[i] = ex2_ftz(x);
        u = fmaf(e[i], fmaxf(x, -1024.0f), u);
    }
    return ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
}

__device__ __forceinline__ uint32_t map_rank(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

// Store (m, s) into another CTA's shared memory; its mbarrier counts the bytes.
__device__ __forceinline__ void st_async_pair(uint32_t dst, float m, float s, uint32_t bar)
{
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];"
        ::"r"(dst), "f"(m), "f"(s), "r"(bar)
        : "memory");
}

// Store (m, s, u, 0) into another CTA's shared memory, counted like the pair.
__device__ __forceinline__ void st_async_quad(uint32_t dst, float m, float s, float u,
                                              uint32_t bar)
{
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, "
        "[%5];" ::"r"(dst),
        "f"(m), "f"(s), "f"(u), "f"(0.0f), "r"(bar)
        : "memory");
}

// Bounded wait for data written by other CTAs of the cluster.
__device__ __forceinline__ bool mbar_wait_cluster_n(uint32_t bar, uint32_t parity,
                                                    uint32_t max_polls)
{
    for (uint32_t i = 0; i < max_polls; ++i) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(bar), "r"(parity), "r"(kPollSuspendNs)
            : "memory");
        if (done)
            return true;
    }
    return false;
}
__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity)
{
    return mbar_wait_cluster_n(bar, parity, kMaxPolls);
}

__device__ __forceinline__ void wait_or_flag(uint32_t bar, bool cluster_scope, int32_t *status)
{
    const bool ok = cluster_scope ? mbar_wait_cluster(bar, 0) : mbar_wait(bar, 0);
    if (!ok) {
        if (threadIdx.x == 0)
            set_status(status, kStatusTimeout);
        if (cluster_scope)  // one more bounded chance before the data is used
            mbar_wait_cluster(bar, 0);
        else
            mbar_wait(bar, 0);
    }
}

}  // namespace
}  // namespace cis
