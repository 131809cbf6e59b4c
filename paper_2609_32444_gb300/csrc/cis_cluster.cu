// cis_cluster.cu -- fused forward + backward token pass, fast path (sm_103a).
//
// A bf16 row of the 151,936-entry vocabulary is 303,872 bytes, more than one
// CTA's shared memory.  A cluster of CS CTAs (1 <= CS <= 8) therefore
// splits each row into CS contiguous slices.  Per row:
//   1. each CTA copies its slice from HBM into shared memory with bulk
//      asynchronous copies (cp.async.bulk, two chunks, each completing on its
//      own mbarrier so that pass 1 starts on the first chunk; no multicast);
//   2. pass 1 over shared memory: per thread the exact maximum of its entries
//      (j != y; bf16 pairs compared packed), then the sum of e^{z - max}; a
//      block reduction gives the CTA's pair (m_c, s_c);
//   3. every CTA stores its pair into slot [rank] of every CTA of the cluster
//      (st.async into distributed shared memory, counted on the receiver's
//      mbarrier, so a CTA waits for the data only, not for a cluster barrier);
//      each CTA combines the CS pairs in rank order, so all CTAs hold
//      bit-identical row scalars;
//   4. thread 0 forms log p (log-odds form, cis_common.cuh), the weight
//      (Algorithm 1 / Table 8) and the token loss (Eq. 1);
//   5. pass 2 over shared memory writes dz = c (softmax - onehot) with 16-byte
//      streaming stores.
// HBM traffic is one read of the logits and one write of dz.  Rows are
// independent; several clusters share an SM, so one cluster's copy overlaps
// another's arithmetic.
#include <cooperative_groups.h>
#include <stdlib.h>

#include "cis_dsmem.cuh"
#include "cis_kernels.h"

namespace cg = cooperative_groups;

namespace cis {
namespace {


// 8 results to global memory with streaming (evict-first) 16-byte stores.
template <typename OutT> __device__ __forceinline__ void store8(OutT *dst, const float (&v)[8]);
template <>
__device__ __forceinline__ void store8<__nv_bfloat16>(__nv_bfloat16 *dst, const float (&v)[8])
{
    uint4 q;
    __nv_bfloat162 h;
    h = __floats2bfloat162_rn(v[0], v[1]); q.x = *reinterpret_cast<uint32_t *>(&h);
    h = __floats2bfloat162_rn(v[2], v[3]); q.y = *reinterpret_cast<uint32_t *>(&h);
    h = __floats2bfloat162_rn(v[4], v[5]); q.z = *reinterpret_cast<uint32_t *>(&h);
    h = __floats2bfloat162_rn(v[6], v[7]); q.w = *reinterpret_cast<uint32_t *>(&h);
    __stcs(reinterpret_cast<uint4 *>(dst), q);
}
template <>
__device__ __forceinline__ void store8<float>(float *dst, const float (&v)[8])
{
    __stcs(reinterpret_cast<float4 *>(dst), make_float4(v[0], v[1], v[2], v[3]));
    __stcs(reinterpret_cast<float4 *>(dst) + 1, make_float4(v[4], v[5], v[6], v[7]));
}


// kEnt: the entropy variant exchanges (m, s, u) instead of (m, s).
template <bool kEnt> struct ClusterShared {
    alignas(8) uint64_t bar[kChunks];  // completion of each copy chunk
    alignas(8) uint64_t xbar;          // arrival of the cluster's (m, s) pairs
    alignas(16) float2 part[kMaxCluster];
    MaxSum red[512 / 32];
    float4 row;  // pass 2's multiplier, exponent offset and c (p - 1): one load
};
template <> struct ClusterShared<true> {
    alignas(8) uint64_t bar[kChunks];
    alignas(8) uint64_t xbar;          // arrival of the cluster's (m, s, u) triples
    float4 part[kMaxCluster];
    MaxSumU red[512 / 32];
    float4 row;
};

template <typename InT, typename OutT, int kThreads, bool kEnt>
__global__ void __launch_bounds__(kThreads) cis_fused_cluster_kernel(const PassArgs a, int64_t slice)
{
    extern __shared__ __align__(128) uint8_t dyn_smem[];
    __shared__ ClusterShared<kEnt> sh;
    // the bulk copy needs a 16-byte aligned destination; 128 bytes of slack
    // are allocated so the slab can start on a 128-byte boundary
    uint8_t *slab = dyn_smem + ((128 - (smem_u32(dyn_smem) & 127)) & 127);
    cg::cluster_group cluster = cg::this_cluster();
    const unsigned rank = cluster.block_rank();
    const unsigned cs = cluster.num_blocks();
    const int64_t t = blockIdx.x / cs;
    const int64_t v0 = (int64_t)rank * slice;
    const int64_t n = v0 < a.V ? (a.V - v0 < slice ? a.V - v0 : slice) : 0;  // multiple of 8
    const int ng = (int)(n / 8);
    constexpr int kGroupBytes = 8 * sizeof(InT);
    OutT *orow = reinterpret_cast<OutT *>(a.dz) + t * a.ld_out + v0;

    const bool valid = a.mask == nullptr || a.mask[t] != 0;
    const int64_t y = a.ids[t];
    const bool id_ok = y >= 0 && y < a.V;
    if (!valid || !id_ok) {  // same branch in every CTA of the cluster
        const float zero[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        for (int g = threadIdx.x; g < ng; g += kThreads)
            store8<OutT>(orow + 8 * g, zero);
        if (rank == 0 && threadIdx.x == 0) {
            const float lp = valid ? NAN : 0.0f;
            if (valid)
                set_status(a.status, kStatusBadId);
            if (a.lp_out) a.lp_out[t] = lp;
            if (kEnt) a.entropy_out[t] = lp;
            if (a.w_out) a.w_out[t] = 0.0f;
            if (a.trunc_out) a.trunc_out[t] = 0;
            a.ws_w[t] = 0.0f;
            a.ws_trunc[t] = 0;
            a.ws_logk[t] = 0.0f;
            a.ws_terms[t] = valid ? (double)NAN : 0.0;
        }
        return;
    }

    // Copy the slice in kChunks pieces, each completing on its own mbarrier.
    const int qg = (ng + kChunks - 1) / kChunks;  // groups per chunk
    const uint32_t xbar = smem_u32(&sh.xbar);
    if (threadIdx.x == 0) {
        for (int c = 0; c < kChunks; ++c)
            mbar_init_only(smem_u32(&sh.bar[c]), 1);
        mbar_init_only(xbar, 1);
        mbar_init_fence();
        // the one local arrival on xbar; the peers' stores bring the bytes
        mbar_expect_tx(xbar, (uint32_t)(cs * (kEnt ? sizeof(float4) : sizeof(float2))));
        const uint8_t *src = reinterpret_cast<const uint8_t *>(a.logits) +
                             (t * a.ld + v0) * (int64_t)sizeof(InT);
        for (int c = 0; c < kChunks; ++c) {
            const int g0 = c * qg, g1 = min(ng, g0 + qg);
            if (g0 >= g1)
                break;
            const uint32_t bytes = (uint32_t)((g1 - g0) * kGroupBytes);
            const uint32_t b = smem_u32(&sh.bar[c]);
            mbar_expect_tx(b, bytes);
            bulk_g2s(smem_u32(slab) + g0 * kGroupBytes, src + (int64_t)g0 * kGroupBytes, bytes,
                     b);
        }
    }
    // Arrive now, wait before the first remote store: every CTA of the
    // cluster has started and initialised its barriers by then.
    cluster_arrive_relaxed();

    // Per-token inputs, fetched while the copy is in flight.
    float zy = 0.0f, linf = 0.0f, lold = 0.0f, adv = 0.0f, sc = 0.0f, qinv = 0.0f;
    if (threadIdx.x == 0) {
        zy = to_f32(reinterpret_cast<const InT *>(a.logits)[t * a.ld + y]);
        linf = a.lp_inf[t];
        lold = a.lp_old ? a.lp_old[t] : 0.0f;
        adv = a.adv[t];
        sc = a.scale[t];
        qinv = expf(-linf);  // 1 / q, off the row's serial path
    }
    __syncthreads();  // barriers initialised before anyone polls them

    // The sampled entry takes no part in the sums over j != y: the thread that
    // owns its 8-entry group (the only thread that reads that group in either
    // pass) overwrites it with -inf in shared memory once its chunk has landed.
    const int64_t yl = y - v0;
    const int gy = (yl >= 0 && yl < n) ? (int)(yl >> 3) : -1;
    const int iy = (int)(yl & 7);

    // Pass 1a: exact maximum of this thread's entries, chunk by chunk as the
    // copy lands.
    MaxAcc<InT> macc;
    for (int c = 0; c < kChunks; ++c) {
        const int g0 = c * qg, g1 = min(ng, g0 + qg);
        if (g0 >= g1)
            break;
        wait_or_flag(smem_u32(&sh.bar[c]), false, a.status);
        if (gy >= g0 && gy < g1 && gy % kThreads == (int)threadIdx.x)
            poke_neg_inf<InT>(slab, 8 * gy + iy);
        const int first = g0 + (int)(((unsigned)threadIdx.x + kThreads - (unsigned)(g0 % kThreads)) %
                                     kThreads);
        macc.consume(slab, first, g1, kThreads);
    }
    const float m = macc.result();

    // Pass 1b: sum of e^{z - max} (8 exponentials added pairwise per group).
    // 2^{(z - m) log2e} is formed with one FMA as 2^{z log2e - cm}, cm = fl(m log2e);
    // the rounding residual of cm is exact (an FMA) and is taken out once at
    // the end, so the sum equals the one over (z - m) log2e.
    float s = 0.0f, u = 0.0f;
    if (m != -INFINITY) {
        const float cm = m * kLog2e;
        const float cm_err = fmaf(m, kLog2e, -cm);  // m log2e - cm, exactly
#pragma unroll 2
        for (int g = threadIdx.x; g < ng; g += kThreads) {
            float z[8];
            load8<InT>(slab, g, z);
            if (kEnt)
                s += sum8_exp2_off_u(z, cm, u);
            else
                s += sum8_exp2_off(z, cm);
        }
        const float f = ex2_ftz(-cm_err);
        if (kEnt)  // sum e (z - m) = f ln2 (sum e x - cm_err sum e)
            u = f * kLn2 * fmaf(-cm_err, s, u);
        s *= f;
    }
    // Exchange the CTA pairs (triples): lane r of warp 0 stores this CTA's
    // values into slot [rank] of CTA r, counted on CTA r's xbar.
    if constexpr (kEnt) {
        const MaxSumU mine = block_msu<kThreads, false>(MaxSumU{m, s, u}, sh.red);
        cluster_wait();
        if (threadIdx.x < cs)
            st_async_quad(map_rank(smem_u32(&sh.part[rank]), threadIdx.x), mine.m, mine.s,
                          mine.u, map_rank(xbar, threadIdx.x));
    } else {
        const MaxSum mine = block_ms<kThreads, false>(MaxSum{m, s}, sh.red);
        cluster_wait();
        if (threadIdx.x < cs)
            st_async_pair(map_rank(smem_u32(&sh.part[rank]), threadIdx.x), mine.m, mine.s,
                          map_rank(xbar, threadIdx.x));
    }
    wait_or_flag(xbar, true, a.status);
    // Everything addressed to this CTA has landed; tell the cluster, and wait
    // for the others' word only at exit (so no CTA leaves while stores into
    // its shared memory may be in flight).
    cluster_arrive_relaxed();

    // Thread 0 forms the row's scalars: the serial part of every row, which
    // the other threads wait for, and which shares the SM's issue slots with
    // the other CTAs' streaming loops, so its instruction count sets its
    // length.  In the common case (row_weight_direct) the weight comes from
    // the row's statistics without logarithms, and log p, log k and the fp64
    // loss term are formed after the barrier by rank 0 alone, which stores
    // them.  Otherwise the log-domain path forms everything here.
    MaxSumU ou{0.0f, 0.0f, 0.0f};
    TokenWeight tw{0.0f, 0.0f, 0};
    double term = 0.0;
    float lp = 0.0f, tdir = 0.0f;
    bool direct = false;
    if (threadIdx.x == 0) {
        MaxSum o;
        if constexpr (kEnt) {
            ou = combine_flat(sh.part, cs);
            o = MaxSum{ou.m, ou.s};
        } else {
            o = cs == 4 ? combine4(sh.part) : combine_flat(sh.part, cs);
        }
        const bool has_old = a.lp_old != nullptr;
        float c, omp, bias_log2, scale = 1.0f;
        DirectWeight dw;
        direct = !has_old && a.w_in == nullptr && row_weight_direct(o, zy, linf, qinv, a.P, dw);
        if (direct) {
            tw.w = dw.w;
            tw.trunc = dw.trunc;
            omp = dw.omp;
            tdir = dw.t;
            c = sc * tw.w * adv;  // s w A rho with rho = 1, g = 1 (Eq. 1 without l_old)
            // The softmax's 1 / (s' + e^{z_y - m'}) = e^{m' - z_y} p, in
            // [2^-102, 1] within the closed forms' range, replaces a logarithm:
            // its binary exponent -J goes into the exponent offset (as the
            // integer "bias" J) and its mantissa 2^J / (...) in [1, 2) into
            // the multiplier, so that every product stays a normal number.
            const float inv = dw.E * dw.p;
            const int J = 127 - (int)((__float_as_uint(inv) >> 23) & 0xff);
            bias_log2 = (float)J;
            scale = inv * __int_as_float((127 + J) << 23);
        } else {
            const RowScalars rs = row_scalars(o, zy);
            tw = token_weight(has_old ? lold : rs.lp, has_old ? 0.0f : rs.lp_lo, linf, a.P,
                              has_old ? -1.0f : rs.omp);
            if (a.w_in) {  // a sequence operator: the response's weight
                tw.w = a.w_in[t];
                tw.trunc = a.trunc_in[t];
            }
            const TokenLoss tl = token_loss(rs.lp, rs.lp_lo, has_old, lold, adv, sc, tw.w, a.P);
            term = tl.term;
            lp = rs.lp;
            c = tl.c;
            omp = rs.omp;
            bias_log2 = rs.bias_log2;
        }
        // Pass 2 forms c softmax_j as cs 2^{z_j log2e - B}: with the power-of-two
        // scale K = clamp(ilogb(c) + 25, 0, 127) (below), B = fl(m log2e + bias
        // - K), and the rounding residual of B folded into cs (with the direct
        // path's scale).  The residual is exact: the product's error from an
        // FMA, the two sums' errors from two-sums (fp32 throughout: fp64
        // operations take 64 cycles each here).
        const int kexp = (int)((__float_as_uint(c) >> 23) & 0xff) - 127 + 25;
        const int K = kexp < 0 ? 0 : (kexp > 127 ? 127 : kexp);
        // c 2^-K exactly: two power-of-two factors, each normal for K <= 127,
        // and every product normal (c 2^-K has exponent -25 unless K is 0)
        float cs = c * __int_as_float((127 - K / 2) << 23) *
                   __int_as_float((127 - (K - K / 2)) << 23);
        float B = INFINITY;
        const float m = o.m == -INFINITY ? 0.0f : o.m;  // row_scalars' offset
        if (bias_log2 != INFINITY) {
            const float p = m * kLog2e, pe = fmaf(m, kLog2e, -p);  // p + pe = m log2e
            float qe, se;
            const float q = two_sum(bias_log2, -(float)K, qe);      // q + qe = bias - K
            B = two_sum(p, q, se);                                   // B + se = p + q
            cs *= ex2_ftz(-(se + pe + qe));
        }
        sh.row = make_float4(cs * scale, B, c * (0.0f - omp), 0.0f);  // c (p - 1): +0 if p = 1
    }
    __syncthreads();
    if (threadIdx.x == 0 && rank == 0) {
        if (direct) {  // log p, log k and the loss term, off the serial path
            lp = -log1pf(tdir);  // p = 1 / (1 + t)
            tw.logk = lp - linf;
            term = -(double)sc * (double)tw.w * (double)adv;
        }
        if (a.lp_out) a.lp_out[t] = lp;
        if (a.w_out) a.w_out[t] = tw.w;
        if (a.trunc_out) a.trunc_out[t] = tw.trunc;
        a.ws_w[t] = tw.w;
        a.ws_trunc[t] = tw.trunc;
        a.ws_logk[t] = tw.logk;
        a.ws_terms[t] = term;
        if (kEnt)
            a.entropy_out[t] = row_entropy(ou, zy, lp);
    }

    // Pass 2: dz = c (softmax - onehot) from the slice in shared memory.
    // c softmax_j is formed as (c 2^-K) 2^(x_j + K) with the flushing
    // exponential.  With K = clamp(ilogb(c) + 25, 0, 127): wherever
    // 2^(x_j + K) would be subnormal, |c softmax_j| < 2^-150 rounds to zero in
    // fp32 and bf16 anyway; c 2^-K stays normal and 2^(x_j + K) finite.  The
    // final multiply keeps subnormal products.
    const float4 row = sh.row;
    const float cs2 = row.x, B = row.y, dzy = row.z;
#pragma unroll 2
    for (int g = threadIdx.x; g < ng; g += kThreads) {
        float z[8], v[8];
        load8<InT>(slab, g, z);
#pragma unroll
        for (int i = 0; i < 8; ++i)
            v[i] = cs2 * ex2_ftz(fmaf(z[i], kLog2e, -B));
        if (g == gy) {  // the sampled entry: c (p - 1)
#pragma unroll
            for (int i = 0; i < 8; ++i)
                v[i] = i == iy ? dzy : v[i];
        }
        store8<OutT>(orow + 8 * g, v);
    }
    cluster_wait();
}

// Cluster size and slice (entries, a multiple of 8) for a row of V entries.
struct Plan {
    int cs;
    int64_t slice;
    size_t smem;
    int nt;  // CTA width: 0 for the default (CIS_CLUSTER_THREADS, else 256)
};

int64_t slice_target_bytes()
{
    static int64_t v = [] {
        const char *e = getenv("CIS_SLICE_KB");
        long kb = e ? atol(e) : 80;
        if (kb < 8) kb = 8;
        if (kb > 200) kb = 200;
        return (int64_t)kb * 1024;
    }();
    return v;
}

// Cluster size forced for tuning sweeps (0: chosen from the slice target).
int forced_cluster()
{
    static int v = [] {
        const char *e = getenv("CIS_CLUSTER");
        const int c = e ? atoi(e) : 0;
        return (c >= 1 && c <= kMaxCluster) ? c : 0;
    }();
    return v;
}

// Smallest cluster size whose slices fit the target (any size 1..8).  Rows
// that fit one slice of the default 80 KB target but not one of 40 KB (a
// 32,000-entry bf16 row, for instance) run on two CTAs of 128 threads: at
// T=4096, V=32000 that took 106.6 us per step against 109.7 us for one CTA of
// 256 threads, and 256 threads on the two halves were slower still (122 us).
// Setting CIS_SLICE_KB or CIS_CLUSTER turns the rule off; CIS_CLUSTER_THREADS
// sets the width of its two CTAs.
bool make_plan(int64_t V, int in_bytes, Plan *p)
{
    const int64_t target = slice_target_bytes();
    const int forced = forced_cluster();
    for (int cs = forced ? forced : 1; cs <= kMaxCluster; ++cs) {
        const int64_t per = (V + cs - 1) / cs;
        const int64_t slice = (per + 7) / 8 * 8;
        if (forced || slice * in_bytes <= target || cs == kMaxCluster) {
            if (slice * in_bytes > 200 * 1024)
                return false;
            p->cs = cs;
            p->slice = slice;
            p->smem = (size_t)(slice * in_bytes) + 128;
            p->nt = 0;
            static const bool slice_set = getenv("CIS_SLICE_KB") != nullptr;
            if (!forced && !slice_set && cs == 1 && slice * in_bytes > 40 * 1024) {
                p->cs = 2;
                p->slice = ((V + 1) / 2 + 7) / 8 * 8;
                p->smem = (size_t)(p->slice * in_bytes) + 128;
                p->nt = 128;
            }
            return true;
        }
    }
    return false;
}

// CTA width forced for tuning sweeps (default 256 threads).
int cluster_threads()
{
    static int v = [] {
        const char *e = getenv("CIS_CLUSTER_THREADS");
        const int n = e ? atoi(e) : 256;
        return (n == 512 || n == 384 || n == 128) ? n : 256;
    }();
    return v;
}

template <typename InT, typename OutT, int NT, bool kEnt = false>
cudaError_t launch_cluster_nt(const PassArgs &a, const Plan &p, cudaStream_t s)
{
    auto kern = cis_fused_cluster_kernel<InT, OutT, NT, kEnt>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(a.T * p.cs), 1, 1);
    cfg.blockDim = dim3(NT, 1, 1);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)p.cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a, p.slice);
}

template <typename InT, typename OutT>
cudaError_t launch_cluster_t(const PassArgs &a, const Plan &p, cudaStream_t s)
{
    if (a.entropy_out)  // the entropy variant is built for 256 threads only
        return launch_cluster_nt<InT, OutT, 256, true>(a, p, s);
    static const bool width_set = getenv("CIS_CLUSTER_THREADS") != nullptr;
    switch (p.nt && !width_set ? p.nt : cluster_threads()) {
    case 512: return launch_cluster_nt<InT, OutT, 512>(a, p, s);
    case 384: return launch_cluster_nt<InT, OutT, 384>(a, p, s);
    case 128: return launch_cluster_nt<InT, OutT, 128>(a, p, s);
    default: return launch_cluster_nt<InT, OutT, 256>(a, p, s);
    }
}

}  // namespace

bool cluster_path_applies(const PassArgs &a, int dtype, int out_dtype)
{
    const int ib = dtype == CIS_BF16 ? 2 : 4;
    const int ob = out_dtype == CIS_BF16 ? 2 : 4;
    if (a.V % 8 != 0)
        return false;
    if ((reinterpret_cast<uintptr_t>(a.logits) & 15) || (a.ld * ib) % 16)
        return false;
    if ((reinterpret_cast<uintptr_t>(a.dz) & 15) || (a.ld_out * ob) % 16)
        return false;
    if (a.T * 8 > 0x7fffffffLL)
        return false;
    Plan p;
    return make_plan(a.V, ib, &p);
}

cudaError_t launch_cluster_fwd_bwd(const PassArgs &a, int dtype, int out_dtype, cudaStream_t s)
{
    if (!cluster_path_applies(a, dtype, out_dtype))
        return cudaErrorNotSupported;
    if (a.T == 0)
        return cudaSuccess;
    Plan p;
    make_plan(a.V, dtype == CIS_BF16 ? 2 : 4, &p);
    if (dtype == CIS_BF16) {
        if (out_dtype == CIS_BF16)
            return launch_cluster_t<__nv_bfloat16, __nv_bfloat16>(a, p, s);
        return launch_cluster_t<__nv_bfloat16, float>(a, p, s);
    }
    if (out_dtype == CIS_BF16)
        return launch_cluster_t<float, __nv_bfloat16>(a, p, s);
    return launch_cluster_t<float, float>(a, p, s);
}

}  // namespace cis
