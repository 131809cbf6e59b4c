// cis_diag.cu -- mismatch diagnostics from the two engines' full logits
// (App. A.5; Sec. 4.3, Fig. 5c-d): per position, the log-odds displacement of
// the sampled token, its log ratio and probability, and -- over the whole
// next-token distribution y ~ q -- the squared bias ||E[(f - k) g]||^2 and the
// variance increase of f g over g, with g = e_y - p the gradient of log p_y
// with respect to the logits and f the weight operator.
//
// Per position, two passes over both engines' rows:
//   pass 1: (max, sum) over j != y of each engine's logits, giving log p,
//           log q, their log-odds d_p, d_q, and lse of each;
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
// is a small difference of O(1) numbers.  Per-thread sums are fp32; the
// one-CTA kernel adds the threads' sums in fp64, the streaming kernel adds a
// warp's in fp32 and the warps' in fp64.
//
// Two kernels compute this:
//   - cis_mismatch_stream_kernel (bf16 rows, V a multiple of 8, 16-byte
//     aligned rows): one CTA per SM walking its rows, a producer warp
//     streaming both rows through a shared-memory ring with bulk copies, once
//     per pass (HBM reads each row once: the second copy comes from L2, and
//     pass 1's bytes are prefetched into L2 two slots ahead), an epilogue warp
//     forming each row's outputs while the consumer warps go on; pass 2
//     forms two candidates per instruction with the packed f32x2 FMA, add
//     and multiply;
//   - cis_mismatch_kernel (any row): one CTA per position streaming both rows
//     from global memory with vector loads, twice.
#include <stdlib.h>

#include "cis_dsmem.cuh"
#include "cis_kernels.h"
#include "cis_rowops.cuh"
#include "cis_nvtx.h"

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
        if (logk_out) logk_out[t] = (float)(st.lp64() - si.lp64());
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


// ---------------------------------------------------------------------------
// Streaming kernel.

// The operator's weight for two candidates at once (f32x2 where the
// arithmetic allows it); the same values as elem_weight lane by lane.  Where
// q = 0 the candidate is never drawn and only r = -p counts: every operator
// here but IcePop and KPop gives a finite f there, so q (f - 1) = 0 without a
// test; those two can return k = inf and keep the explicit guard.
template <int MODE>
__device__ __forceinline__ float2 elem_weight2(float2 xp, float2 xq, float2 p, float2 q, float2 k,
                                               const DevParams &P)
{
    const float2 one = make_float2(1.0f, 1.0f);
    if (MODE == CIS_MODE_CIS || MODE == CIS_MODE_BAND) {
        // 1 + lam max(1 - p, kappa) = max((1 + lam) - lam p, 1 + lam kappa) for
        // lam >= 0: one packed FMA and two maxima per pair
        float2 c = __ffma2_rn(p, make_float2(-P.lam_f, -P.lam_f),
                              make_float2(1.0f + P.lam_f, 1.0f + P.lam_f));
        const float lo = fmaf(P.lam_f, P.kappa_f, 1.0f);
        c = make_float2(fmaxf(c.x, lo), fmaxf(c.y, lo));
        float2 f = make_float2(fminf(k.x, c.x), fminf(k.y, c.y));
        if (MODE == CIS_MODE_BAND) {  // lower edge (1 + p) / 2
            const float2 lo = __ffma2_rn(p, make_float2(0.5f, 0.5f), make_float2(0.5f, 0.5f));
            f = make_float2(fmaxf(f.x, lo.x), fmaxf(f.y, lo.y));
        }
        return f;
    }
    if (MODE == CIS_MODE_TIS)
        return make_float2(fminf(k.x, P.tis_cap_f), fminf(k.y, P.tis_cap_f));
    if (MODE == CIS_MODE_EXACT)
        return make_float2(fminf(fmaxf(k.x, P.exact_lo_f), P.exact_hi_f),
                           fminf(fmaxf(k.y, P.exact_lo_f), P.exact_hi_f));
    if (MODE == CIS_MODE_ICEPOP || MODE == CIS_MODE_KPOP)
        return make_float2(q.x > 0.0f ? elem_weight<MODE>(xp.x, xq.x, p.x, k.x, P) : 1.0f,
                           q.y > 0.0f ? elem_weight<MODE>(xp.y, xq.y, p.y, k.y, P) : 1.0f);
    return one;  // CIS_MODE_NONE
}

// Pass 2 for two candidates (zp: training logits, zq: inference logits), with
// nop = -lse_p log2e and noq = -lse_q log2e.  The sums are kept in the signs
// that need no negation:
//   acc = [P2, R2, -RP, D = sum T1 p, -C2, -C3, -C4, -C5, QP]
// with T2 = q (1 - f) = -q (f - 1), T1 = T2 (1 + f) = -q (f^2 - 1) and
// r' = p - q f = -r; then C1 = sum q (f^2 - 1)(1 - 2p) = C2 + 2 D.  T2, T1
// and r' are each one FMA from -f, so each is rounded once, and two
// instructions a pair fewer (3.15 -> 3.05 ms per call at T=16384, V=151936).
template <int MODE>
__device__ __forceinline__ void diag_pair(float2 zp, float2 zq, float2 nop, float2 noq,
                                          const DevParams &P, float2 (&acc)[kNSums])
{
    const float2 l2e = make_float2(kLog2e, kLog2e);
    const float2 m1 = make_float2(-1.0f, -1.0f);
    const float2 xp = __ffma2_rn(zp, l2e, nop), xq = __ffma2_rn(zq, l2e, noq);
    const float2 p = make_float2(ex2_ftz(xp.x), ex2_ftz(xp.y));
    const float2 q = make_float2(ex2_ftz(xq.x), ex2_ftz(xq.y));
    const float2 d = __ffma2_rn(xq, m1, xp);  // xp - xq, rounded once
    const float2 k = make_float2(ex2_ftz(d.x), ex2_ftz(d.y));
    const float2 f = elem_weight2<MODE>(xp, xq, p, q, k, P);
    const float2 nf = __fmul2_rn(f, m1);
    const float2 T2 = __ffma2_rn(q, nf, q);   // q (1 - f)
    const float2 T1 = __ffma2_rn(T2, f, T2);  // T2 (1 + f)
    const float2 r = __ffma2_rn(q, nf, p);    // p - q f
    acc[0] = __ffma2_rn(p, p, acc[0]);
    acc[1] = __ffma2_rn(r, r, acc[1]);
    acc[2] = __ffma2_rn(r, p, acc[2]);
    acc[3] = __ffma2_rn(T1, p, acc[3]);
    acc[4] = __fadd2_rn(T1, acc[4]);
    acc[5] = __fadd2_rn(T2, acc[5]);
    acc[6] = __ffma2_rn(T1, q, acc[6]);
    acc[7] = __ffma2_rn(T2, p, acc[7]);
    acc[8] = __ffma2_rn(q, p, acc[8]);
}

__device__ __forceinline__ float2 bf16_pair(uint32_t w)
{
    return make_float2(bf16_lo(w), bf16_hi(w));
}

// Sum of 2^{z log2e + noff} over one 8-entry bf16 group, into a packed pair.
__device__ __forceinline__ float2 sum8_exp2_pk(uint4 w, float2 noff, float2 acc)
{
    const float2 l2e = make_float2(kLog2e, kLog2e);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    float2 e[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 x = __ffma2_rn(bf16_pair(ws[i]), l2e, noff);
        e[i] = make_float2(ex2_ftz(x.x), ex2_ftz(x.y));
    }
    return __fadd2_rn(acc, __fadd2_rn(__fadd2_rn(e[0], e[1]), __fadd2_rn(e[2], e[3])));
}

struct DiagArgs {
    const __nv_bfloat16 *zt, *zi;
    int64_t T, V, ld_t, ld_i;
    const int32_t *ids;
    const uint8_t *mask;
    DevParams P;
    float *eps, *logk, *p, *bias2, *dvar;
    int32_t *status;
};

// The layout for NW consumer warps (plus a producer and an epilogue warp)
// and CPS CTAs per SM: a ring slot holds four groups per consumer thread of
// each row, as many slots as fit in about 200 KB / CPS of shared memory (3 of
// 64 KB for 16 warps and one CTA).  Each slot costs every warp a wait, an
// arrive and the loop set-up; four groups a thread amortise that (two, three,
// five and six measured slower).
template <int NW, int CPS = 1> struct StreamCfg {
    static constexpr int kConsThreads = NW * 32;
    static constexpr int kThreads = kConsThreads + 64;  // + the producer and epilogue warps
    static constexpr int kSlotGroups = 4 * kConsThreads;  // 8-entry groups of each row per slot
    static constexpr int kSlotBytes = 2 * kSlotGroups * 16;
    static constexpr int kRingFit = (200 * 1024 / CPS) / kSlotBytes;
    static constexpr int kRing = kRingFit < 8 ? kRingFit : 8;
    static constexpr size_t kSmem = (size_t)kRing * kSlotBytes + 128;
};
constexpr int kMaxRing = 8;
constexpr int kPrefetchSlots = 2;  // L2 prefetch distance of pass 1, in slots
constexpr int kMaxConsWarps = 32;

// Per-row buffers are indexed [row parity]: the epilogue warp reads row i's
// while the consumers fill row i + 1's.
struct StreamShared {
    alignas(8) uint64_t full[kMaxRing];   // a slot's two copies have landed
    alignas(8) uint64_t empty[kMaxRing];  // every consumer warp is done with a slot
    alignas(8) uint64_t epi_full[2];      // every consumer warp has written its sums
    alignas(8) uint64_t epi_empty[2];     // the epilogue warp is done with the buffer
    MaxSum red[2][2][kMaxConsWarps];      // [parity][training, inference][warp] (m, s)
    float wsum[2][kMaxConsWarps][kNSums]; // [parity][warp] the pass-2 sums
    float2 rowstat[2][2];                 // [parity][engine] (m', s')
    float zyv[2][2];                      // [parity][engine] the sampled entries
    int aborted;
};

// The consumer warps' own barrier (the producer warp never joins it).
template <int NT> __device__ __forceinline__ void cons_sync()
{
    asm volatile("bar.sync 1, %0;" ::"n"(NT) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Bulk copy whose lines L2 may evict first (their last read).
__device__ __forceinline__ void bulk_g2s_evict_first(uint32_t dst, const void *src, uint32_t bytes,
                                                     uint32_t bar)
{
    asm volatile(
        "{\n\t.reg .b64 pol;\n\t"
        "createpolicy.fractional.L2::evict_first.b64 pol, 1.0;\n\t"
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], pol;\n\t}" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// An L2 prefetch of bytes at src (16-byte aligned, a multiple of 16 bytes).
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// A wait that runs out marks the CTA as aborted (and the status word): every
// later wait then returns at once, so each role finishes its loops without
// waiting again and the consumers still meet at every barrier.  A slot that
// has already landed costs one poll, without a read of the flag (every warp
// waits once per slot: 3.28 -> 3.20 ms per call at V = 151936).
struct StreamAbort {
    volatile int *flag;
    int32_t *status;
    __device__ __forceinline__ bool on() const { return *flag != 0; }
    __device__ __forceinline__ void wait(uint32_t bar, uint32_t parity) const
    {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(bar), "r"(parity)
            : "memory");
        if (done)
            return;
        if (*flag)
            return;
        if (!mbar_wait(bar, parity)) {
            *flag = 1;
            set_status(status, kStatusTimeout);
        }
    }
};

// The sampled entry of a group set to -inf (pass 1 sums over j != y).
__device__ __forceinline__ uint4 drop_entry(uint4 w, int i)
{
    const uint32_t keep = (i & 1) ? 0x0000ffffu : 0xffff0000u;
    const uint32_t ninf = (i & 1) ? 0xff800000u : 0x0000ff80u;
    const int k = i >> 1;
    w.x = k == 0 ? ((w.x & keep) | ninf) : w.x;
    w.y = k == 1 ? ((w.y & keep) | ninf) : w.y;
    w.z = k == 2 ? ((w.z & keep) | ninf) : w.z;
    w.w = k == 3 ? ((w.w & keep) | ninf) : w.w;
    return w;
}

// Running (max, sum) of one row over 8 more entries: the exact maximum of
// the group (bf16 pairs compared packed, NaN propagating); when it rises the
// sum is rescaled; the exponentials are 2^{z log2e - cm} with cm = fl(m log2e),
// the residual m log2e - cm being taken out once per thread at the end.
__device__ __forceinline__ void pass1_update(uint4 w, float &m, float &cm, float2 &s)
{
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&w);
    const __nv_bfloat162 a = __hmax2_nan(__hmax2_nan(h[0], h[1]), __hmax2_nan(h[2], h[3]));
    const float lm = max_nan(__low2float(a), __high2float(a));
    if (lm > m || lm != lm) {
        const float ncm = lm * kLog2e;
        // cm - ncm < 0 once m is finite (the maximum only rises); while the
        // sum is still empty (m = -inf, cm = 0) a very negative first maximum
        // would make 2^{0 - ncm} overflow and 0 x inf = NaN: the clamp keeps
        // the factor finite there (and changes nothing otherwise)
        const float f = ex2_ftz(fminf(cm - ncm, 0.0f));
        s = __fmul2_rn(s, make_float2(f, f));
        m = lm;
        cm = ncm;
    }
    s = sum8_exp2_pk(w, make_float2(-cm, -cm), s);
}

// The same over four groups (32 entries): one maximum for the four, so that
// the compare and the rare rescale come once per 32 entries (3.20 -> 3.15 ms
// per call at T=16384, V=151936).
__device__ __forceinline__ void pass1_update4(const uint4 (&w)[4], float &m, float &cm, float2 &s)
{
    __nv_bfloat162 g[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&w[i]);
        g[i] = __hmax2_nan(__hmax2_nan(h[0], h[1]), __hmax2_nan(h[2], h[3]));
    }
    const __nv_bfloat162 a = __hmax2_nan(__hmax2_nan(g[0], g[1]), __hmax2_nan(g[2], g[3]));
    const float lm = max_nan(__low2float(a), __high2float(a));
    if (lm > m || lm != lm) {  // as in pass1_update
        const float ncm = lm * kLog2e;
        const float f = ex2_ftz(fminf(cm - ncm, 0.0f));
        s = __fmul2_rn(s, make_float2(f, f));
        m = lm;
        cm = ncm;
    }
    const float2 noff = make_float2(-cm, -cm);
#pragma unroll
    for (int i = 0; i < 4; ++i)
        s = sum8_exp2_pk(w[i], noff, s);
}

// CPS CTAs per SM walk rows t = blockIdx.x, blockIdx.x + gridDim.x, ...  Per
// row, a producer thread streams both rows through a ring of kRing shared-
// memory slots twice (bulk copies of sg groups per row per slot): once for
// pass 1 (from HBM) and once for pass 2 (the same bytes again, mostly from L2,
// where pass 1 left them microseconds earlier; these copies mark the lines
// evict-first).  Pass 2 takes the row's slots last-first, so that the bytes
// pass 1 brought in last are read again first.  The consumer warps:
//   pass 1: per thread a running (max, sum) of each row over its groups,
//           the maximum taken once per full slot (four groups); warp
//           combination, then the row's one barrier, after which every warp
//           combines the warps' pairs itself into both rows' lse;
//   pass 2: the nine sums, two candidates per packed instruction; warp sums
//           in fp32, handed to the epilogue warp through a buffer per row
//           parity.
// The epilogue warp adds the warps' sums in fp64 and forms eps, log k, p,
// bias2 and dvar, while the consumers work on the next row: at T=16384,
// V=151936 that took 3.05 -> 3.00 ms per call against warp 0 doing it between
// two more barriers, with bit-identical outputs.
template <int MODE, int NW, int CPS>
__global__ void __launch_bounds__(StreamCfg<NW, CPS>::kThreads, CPS)
    cis_mismatch_stream_kernel(const DiagArgs a, int sg)
{
    using C = StreamCfg<NW, CPS>;
    constexpr int kConsWarps = NW, kConsThreads = C::kConsThreads, kRing = C::kRing;
    constexpr int kSlotGroups = C::kSlotGroups, kSlotBytes = C::kSlotBytes;
    extern __shared__ __align__(128) uint8_t dyn_smem[];
    __shared__ StreamShared sh;
    uint8_t *ring = dyn_smem + ((128 - (smem_u32(dyn_smem) & 127)) & 127);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ng = (int)(a.V / 8);
    const int nst = (ng + sg - 1) / sg;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(smem_u32(&sh.full[i]), 1);
            mbar_init(smem_u32(&sh.empty[i]), kConsWarps);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&sh.epi_full[i]), kConsWarps);
            mbar_init(smem_u32(&sh.epi_empty[i]), 1);
        }
        sh.aborted = 0;
    }
    __syncthreads();
    const StreamAbort ab{&sh.aborted, a.status};

    if (warp == kConsWarps) {  // producer
        if (lane != 0)
            return;
        uint32_t k = 0;
        for (int64_t t = blockIdx.x; t < a.T && !ab.on(); t += gridDim.x) {
            const int64_t y = a.ids[t];
            if ((a.mask != nullptr && a.mask[t] == 0) || y < 0 || y >= a.V)
                continue;
            const uint8_t *rp = reinterpret_cast<const uint8_t *>(a.zt + t * a.ld_t);
            const uint8_t *rq = reinterpret_cast<const uint8_t *>(a.zi + t * a.ld_i);
            // Pass 1's bytes are prefetched into L2 kPrefetchSlots slots ahead
            // of their copies: this row's slot st + kPrefetchSlots with
            // pass-1 slot st, and the first slots of this CTA's next row with
            // the last slots of pass 2.  Pass 1 then copies from L2 instead
            // of waiting on HBM.  At T=16384, V=151936: 3.00 ms per call
            // without, 2.80 ms with 2 slots ahead (10.20 GB read from HBM),
            // 2.79 with 4 (10.32 GB) or 6 (10.97 GB), and 2.83 ms with the
            // whole next row prefetched during pass 2 (15.47 GB: the L2 no
            // longer holds both rows).  With several CTAs per SM more rows
            // are in flight and the prefetch is left out.
            int64_t tn = CPS == 1 ? t + gridDim.x : a.T;
            for (; tn < a.T; tn += gridDim.x) {
                const int64_t yn = a.ids[tn];
                if ((a.mask == nullptr || a.mask[tn] != 0) && yn >= 0 && yn < a.V)
                    break;
            }
            const uint8_t *np =
                tn < a.T ? reinterpret_cast<const uint8_t *>(a.zt + tn * a.ld_t) : nullptr;
            const uint8_t *nq =
                tn < a.T ? reinterpret_cast<const uint8_t *>(a.zi + tn * a.ld_i) : nullptr;
            for (int pass = 0; pass < 2 && !ab.on(); ++pass)
                for (int st = 0; st < nst; ++st, ++k) {
                    const uint32_t s = k % kRing, u = k / kRing;
                    if (u > 0)
                        ab.wait(smem_u32(&sh.empty[s]), (u - 1) & 1);
                    if (ab.on())
                        break;
                    const int g0 = (pass ? nst - 1 - st : st) * sg, n = min(sg, ng - g0);
                    const uint32_t bytes = (uint32_t)n * 16;
                    const uint32_t full = smem_u32(&sh.full[s]);
                    const uint32_t dst = smem_u32(ring + (size_t)s * kSlotBytes);
                    mbar_expect_tx(full, 2 * bytes);
                    if (pass == 0) {
                        bulk_g2s(dst, rp + (int64_t)g0 * 16, bytes, full);
                        bulk_g2s(dst + kSlotGroups * 16, rq + (int64_t)g0 * 16, bytes, full);
                        if (CPS == 1 && st + kPrefetchSlots < nst) {
                            const int gn = (st + kPrefetchSlots) * sg;
                            const uint32_t nb = (uint32_t)min(sg, ng - gn) * 16;
                            bulk_prefetch_l2(rp + (int64_t)gn * 16, nb);
                            bulk_prefetch_l2(rq + (int64_t)gn * 16, nb);
                        }
                    } else {
                        bulk_g2s_evict_first(dst, rp + (int64_t)g0 * 16, bytes, full);
                        bulk_g2s_evict_first(dst + kSlotGroups * 16, rq + (int64_t)g0 * 16, bytes,
                                             full);
                        const int pi = st - (nst - kPrefetchSlots);  // the next row's slot
                        if (np != nullptr && pi >= 0 && pi < nst) {
                            const int gn = pi * sg;
                            const uint32_t nb = (uint32_t)min(sg, ng - gn) * 16;
                            bulk_prefetch_l2(np + (int64_t)gn * 16, nb);
                            bulk_prefetch_l2(nq + (int64_t)gn * 16, nb);
                        }
                    }
                }
        }
        // copies still in flight land before the CTA may exit: the last
        // use of each slot (k counts the uses issued)
        for (uint32_t j = k > (uint32_t)kRing ? k - kRing : 0; j < k; ++j)
            mbar_wait(smem_u32(&sh.full[j % kRing]), (j / kRing) & 1);
        return;
    }

    if (warp == kConsWarps + 1) {  // row epilogue
        uint32_t rr = 0;  // valid rows so far
        for (int64_t t = blockIdx.x; t < a.T && !ab.on(); t += gridDim.x) {
            const int64_t y = a.ids[t];
            if ((a.mask != nullptr && a.mask[t] == 0) || y < 0 || y >= a.V)
                continue;
            const int b = rr & 1;
            ab.wait(smem_u32(&sh.epi_full[b]), (rr >> 1) & 1);
            if (ab.on())
                break;
            // eps, log k and p; lane 16 forms the inference row's scalars
            const int r = lane >> 4;
            const MaxSum o = MaxSum{sh.rowstat[b][r].x, sh.rowstat[b][r].y};
            const float zyr = sh.zyv[b][r];
            const RowScalars rs = row_scalars(o, zyr);
            const double lp64_q = __shfl_sync(0xffffffffu, rs.lp64(), 16);
            const float om_q = __shfl_sync(0xffffffffu, o.m, 16);
            const float os_q = __shfl_sync(0xffffffffu, o.s, 16);
            const float zy_q = __shfl_sync(0xffffffffu, zyr, 16);
            // the nine sums: the warps' fp32 sums added in fp64 in warp order
            double v = 0.0;
            if (lane < kNSums) {
                v = sh.wsum[b][0][lane];
                for (int w = 1; w < kConsWarps; ++w)
                    v += sh.wsum[b][w][lane];
            }
            double S[kNSums];
#pragma unroll
            for (int i = 0; i < kNSums; ++i)
                S[i] = __shfl_sync(0xffffffffu, v, i);
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(smem_u32(&sh.epi_empty[b]));  // the buffer is read
                // eps = logit p - logit q: Lemma 3.1's -delta_y + log sum_{j != y}
                // w_j e^{delta_j} in the normalised gauge, from the log-odds
                const double dp = ((double)zyr - (double)o.m) - (double)logf(o.s);
                const double dq = ((double)zy_q - (double)om_q) - (double)logf(os_q);
                a.eps[t] = (float)(dp - dq);
                if (a.logk) a.logk[t] = (float)(rs.lp64() - lp64_q);
                if (a.p) a.p[t] = expf(rs.lp);
                const double P2 = S[0], R2 = S[1], RP = -S[2], D = S[3], C2 = -S[4], C3 = -S[5],
                             C4 = -S[6], C5 = -S[7], QP = S[8];
                const double C1 = C2 + 2.0 * D, C6 = C5 + 2.0 * QP;
                const double bias2 = R2 - 2.0 * C3 * RP + C3 * C3 * P2;
                const double dvar =
                    C1 + P2 * C2 - (C4 - (2.0 + C3) * C5 - C3 * C6 + C3 * (2.0 + C3) * P2);
                if (a.bias2) a.bias2[t] = (float)bias2;
                if (a.dvar) a.dvar[t] = (float)dvar;
            }
            ++rr;
        }
        return;
    }

    // consumers
    const int ct = threadIdx.x;
    uint32_t k = 0, rr = 0;  // ring slots used; valid rows so far
    for (int64_t t = blockIdx.x; t < a.T; t += gridDim.x) {
        const bool valid = a.mask == nullptr || a.mask[t] != 0;
        const int64_t y = a.ids[t];
        if (!valid || y < 0 || y >= a.V) {
            if (ct == 0) {
                const float v = valid ? NAN : 0.0f;
                if (valid)
                    set_status(a.status, kStatusBadId);
                a.eps[t] = v;
                if (a.logk) a.logk[t] = v;
                if (a.p) a.p[t] = v;
                if (a.bias2) a.bias2[t] = v;
                if (a.dvar) a.dvar[t] = v;
            }
            continue;
        }
        const int b = rr & 1;
        // the sampled entries, read early (used after pass 1): lane 0 the
        // training row's, lane 16 the inference row's
        float zy = 0.0f;
        if ((lane & 15) == 0)
            zy = to_f32(lane == 0 ? a.zt[t * a.ld_t + y] : a.zi[t * a.ld_i + y]);
        const int gy = (int)(y >> 3), iy = (int)(y & 7);

        // pass 1
        float m_p = -INFINITY, m_q = -INFINITY, cm_p = 0.0f, cm_q = 0.0f;
        float2 s_p = make_float2(0.0f, 0.0f), s_q = make_float2(0.0f, 0.0f);
        for (int st = 0; st < nst; ++st, ++k) {
            const uint32_t s = k % kRing;
            ab.wait(smem_u32(&sh.full[s]), (k / kRing) & 1);
            const uint4 *slot = reinterpret_cast<const uint4 *>(ring + (size_t)s * kSlotBytes);
            const int g0 = st * sg, n = min(sg, ng - g0);
            if (n == 4 * kConsThreads) {  // a full slot: four groups a thread
                uint4 u[4], v[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    u[i] = slot[ct + i * kConsThreads];
                    v[i] = slot[kSlotGroups + ct + i * kConsThreads];
                }
                const int rel = gy - g0 - ct;  // the sampled entry's group, if this thread's
                if (rel >= 0 && rel < 4 * kConsThreads && rel % kConsThreads == 0) {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (rel == i * kConsThreads) {
                            u[i] = drop_entry(u[i], iy);
                            v[i] = drop_entry(v[i], iy);
                        }
                }
                pass1_update4(u, m_p, cm_p, s_p);
                pass1_update4(v, m_q, cm_q, s_q);
            } else
#pragma unroll 1
            for (int j = ct; j < n; j += kConsThreads) {
                uint4 u = slot[j], v = slot[kSlotGroups + j];
                if (g0 + j == gy) {
                    u = drop_entry(u, iy);
                    v = drop_entry(v, iy);
                }
                pass1_update(u, m_p, cm_p, s_p);
                pass1_update(v, m_q, cm_q, s_q);
            }
            __syncwarp();
            if (lane == 0)
                mbar_arrive(smem_u32(&sh.empty[s]));
        }
        MaxSum rp{m_p, s_p.x + s_p.y}, rq{m_q, s_q.x + s_q.y};
        if (m_p != -INFINITY)
            rp.s *= ex2_ftz(-fmaf(m_p, kLog2e, -cm_p));
        if (m_q != -INFINITY)
            rq.s *= ex2_ftz(-fmaf(m_q, kLog2e, -cm_q));
        rp = warp_ms(rp);
        rq = warp_ms(rq);
        if (lane == 0) {
            sh.red[b][0][warp] = rp;
            sh.red[b][1][warp] = rq;
        }
        cons_sync<kConsThreads>();
        // Every warp combines the warps' pairs in the same fixed order (lanes
        // 0-15 the training row's, lane l taking warps l, l + 16, ..., 16-31
        // the inference row's, then a tree over the 16 lanes), so that pass 2
        // starts without a second barrier.  sh.red is double-buffered by row
        // parity: a warp rewrites this row's buffer two rows later, after the
        // next row's barrier, which every warp reaches only once it has read
        // this one.
        const int r = lane >> 4;
        MaxSum o = (lane & 15) < kConsWarps ? sh.red[b][r][lane & 15] : MaxSum{-INFINITY, 0.0f};
        for (int w = (lane & 15) + 16; w < kConsWarps; w += 16)
            o = ms_combine(o, sh.red[b][r][w]);
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) {
            MaxSum x;
            x.m = __shfl_xor_sync(0xffffffffu, o.m, off);
            x.s = __shfl_xor_sync(0xffffffffu, o.s, off);
            o = ms_combine(o, x);
        }
        // Pass 2 needs only the two rows' log-sum-exps, from the larger of m'
        // and z_y so that no exponential overflows:
        //   lse = z_y + log1p(s' e^{m' - z_y})   (z_y >= m', also p = 1)
        //   lse = m' + log(s' + e^{z_y - m'})    (otherwise)
        float lse = 0.0f;
        if ((lane & 15) == 0)
            lse = o.s == 0.0f ? zy  // no other finite entry: p = 1
                  : (zy >= o.m ? zy + log1pf(o.s * expf(o.m - zy))
                               : o.m + logf(o.s + expf(zy - o.m)));
        const float op = __shfl_sync(0xffffffffu, lse, 0) * kLog2e;
        const float oq = __shfl_sync(0xffffffffu, lse, 16) * kLog2e;
        if (warp == 0) {
            // the row statistics for the epilogue warp, once it is done with
            // this buffer (two rows ago)
            if (lane == 0)
                ab.wait(smem_u32(&sh.epi_empty[b]), ((rr >> 1) & 1) ^ 1);
            __syncwarp();
            if ((lane & 15) == 0) {
                sh.rowstat[b][r] = make_float2(o.m, o.s);
                sh.zyv[b][r] = zy;
            }
        }

        // pass 2
        float2 acc[kNSums];
#pragma unroll
        for (int i = 0; i < kNSums; ++i)
            acc[i] = make_float2(0.0f, 0.0f);
        const float2 nop = make_float2(-op, -op), noq = make_float2(-oq, -oq);
        for (int st = 0; st < nst; ++st, ++k) {
            const uint32_t s = k % kRing;
            ab.wait(smem_u32(&sh.full[s]), (k / kRing) & 1);
            const uint4 *slot = reinterpret_cast<const uint4 *>(ring + (size_t)s * kSlotBytes);
            const int n = min(sg, ng - (nst - 1 - st) * sg);
#pragma unroll 1
            for (int j = ct; j < n; j += kConsThreads) {
                const uint4 u = slot[j], v = slot[kSlotGroups + j];
                diag_pair<MODE>(bf16_pair(u.x), bf16_pair(v.x), nop, noq, a.P, acc);
                diag_pair<MODE>(bf16_pair(u.y), bf16_pair(v.y), nop, noq, a.P, acc);
                diag_pair<MODE>(bf16_pair(u.z), bf16_pair(v.z), nop, noq, a.P, acc);
                diag_pair<MODE>(bf16_pair(u.w), bf16_pair(v.w), nop, noq, a.P, acc);
            }
            __syncwarp();
            if (lane == 0)
                mbar_arrive(smem_u32(&sh.empty[s]));
        }
        // warp sums in fp32 (fp64 arithmetic is scarce on this part); the
        // epilogue warp adds the warps' in fp64 and forms the outputs while
        // this warp goes on to the next row
        float ws[kNSums];
#pragma unroll
        for (int i = 0; i < kNSums; ++i) {
            float v = acc[i].x + acc[i].y;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1)
                v += __shfl_xor_sync(0xffffffffu, v, o);
            ws[i] = v;
        }
        if (lane == 0) {
            ab.wait(smem_u32(&sh.epi_empty[b]), ((rr >> 1) & 1) ^ 1);
#pragma unroll
            for (int i = 0; i < kNSums; ++i)
                sh.wsum[b][warp][i] = ws[i];
            mbar_arrive(smem_u32(&sh.epi_full[b]));
        }
        ++rr;
    }
}

// Groups per slot (CIS_DIAG_SLOT_GROUPS, read at each call: small values
// make short rows span several slots in tests), and whether the streaming
// kernel applies at all (CIS_DIAG_KERNEL=row selects the one-CTA kernel).
int diag_slot_groups(int max_groups)
{
    const char *e = getenv("CIS_DIAG_SLOT_GROUPS");
    const long v = e ? atol(e) : max_groups;
    return v < 1 ? 1 : (v > max_groups ? max_groups : (int)v);
}

// Consumer warps per CTA (CIS_DIAG_WARPS, for tuning sweeps): 16 (the
// default) or 24 with one CTA per SM, 8 with two, 4 with four; the ring
// shrinks with the CTA.  At V=151936, two CTAs of 8 warps took 2.84 ms and
// four of 4 2.83 ms (without the L2 prefetch, which they leave out) against
// 2.81 for one of 16.  They keep two or four rows in flight per SM (about 185
// MB between a row's two reads at two, more than the L2 holds), and pass 2
// then re-read a third of its bytes from HBM: 13.2 GB of DRAM reads per call
// against 10.0 (an earlier build).  One CTA of 16 warps keeps HBM at one read
// of each row.  24 warps in one CTA (2 slots of 96 KB) were slower than 16 (3
// of 64 KB).
int diag_warps()
{
    const char *e = getenv("CIS_DIAG_WARPS");
    const int v = e ? atoi(e) : 16;
    return (v == 24 || v == 8 || v == 4) ? v : 16;
}

bool diag_stream_applies(const void *zt, const void *zi, int dtype, int64_t V, int64_t ld_t,
                         int64_t ld_i)
{
    if (dtype != CIS_BF16 || V % 8 != 0)
        return false;
    if ((reinterpret_cast<uintptr_t>(zt) & 15) || (reinterpret_cast<uintptr_t>(zi) & 15) ||
        (ld_t * 2) % 16 || (ld_i * 2) % 16)
        return false;
    const char *e = getenv("CIS_DIAG_KERNEL");
    return !(e && e[0] == 'r');
}

template <int MODE, int NW, int CPS>
cudaError_t launch_stream_nw(const DiagArgs &a, cudaStream_t s)
{
    using C = StreamCfg<NW, CPS>;
    auto kern = cis_mismatch_stream_kernel<MODE, NW, CPS>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::kSmem);
    if (e != cudaSuccess)
        return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int64_t slots = (int64_t)CPS * sms;
    const int64_t grid = a.T < slots ? a.T : slots;
    kern<<<(unsigned)grid, C::kThreads, C::kSmem, s>>>(a, diag_slot_groups(C::kSlotGroups));
    return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_stream_mode(const DiagArgs &a, cudaStream_t s)
{
    switch (diag_warps()) {
    case 24: return launch_stream_nw<MODE, 24, 1>(a, s);
    case 8: return launch_stream_nw<MODE, 8, 2>(a, s);
    case 4: return launch_stream_nw<MODE, 4, 4>(a, s);
    default: return launch_stream_nw<MODE, 16, 1>(a, s);
    }
}

// ---------------------------------------------------------------------------
// Dispatch on the operator (a template parameter of both kernels).

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

#define CIS_DIAG_MODES(X)  \
    X(CIS_MODE_CIS)        \
    X(CIS_MODE_TIS)        \
    X(CIS_MODE_EXACT)      \
    X(CIS_MODE_BAND)       \
    X(CIS_MODE_ICEPOP)     \
    X(CIS_MODE_KPOP)

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
        CIS_DIAG_MODES(CIS_DIAG_CASE)
    default:
        launch_mode<InT, CIS_MODE_NONE>(zt, zi, T, V, ld_t, ld_i, ids, mask, P, eps, logk, p,
                                        bias2, dvar, status, s);
    }
#undef CIS_DIAG_CASE
}

cudaError_t launch_stream(const DiagArgs &a, cudaStream_t s)
{
#define CIS_DIAG_SCASE(M) \
    case M: return launch_stream_mode<M>(a, s);
    switch (a.P.mode) {
        CIS_DIAG_MODES(CIS_DIAG_SCASE)
    default: return launch_stream_mode<CIS_MODE_NONE>(a, s);
    }
#undef CIS_DIAG_SCASE
}
#undef CIS_DIAG_MODES

}  // namespace

cudaError_t launch_mismatch(const void *zt, const void *zi, int dtype, int64_t T, int64_t V,
                            int64_t ld_t, int64_t ld_i, const int32_t *ids, const uint8_t *mask,
                            const DevParams &P, float *eps, float *logk, float *p, float *bias2,
                            float *dvar, int32_t *status, cudaStream_t s)
{
    if (T == 0)
        return cudaSuccess;
    if (diag_stream_applies(zt, zi, dtype, V, ld_t, ld_i)) {
        const DiagArgs a{static_cast<const __nv_bfloat16 *>(zt),
                         static_cast<const __nv_bfloat16 *>(zi),
                         T, V, ld_t, ld_i, ids, mask, P, eps, logk, p, bias2, dvar, status};
        return launch_stream(a, s);
    }
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
    NvtxRange nvtx_range("cis_mismatch_diagnostics");
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
