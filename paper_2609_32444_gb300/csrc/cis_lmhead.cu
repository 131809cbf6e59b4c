// cis_lmhead.cu -- the CIS token pass fused with the LM head (sm_103a).
//
// Logits z = H W^T (H: [T, Hd] hidden states, W: [V, Hd] unembedding, bf16)
// are computed tile by tile on the tensor cores (tcgen05.mma, fp32 in TMEM)
// and never written to global memory.  Three passes:
//
//   FWD  z tiles -> for every token, (max, sum of e^{z - max}) over the tile's
//        entries j != y, and z_y; one pair per (vocab tile, token).
//   TOK  per token: combine the pairs, then log p, the weight (Algorithm 1 /
//        Table 8) and the token loss (Eq. 1) with the same device code as the
//        logits entry points; gives lse_t and c_t.
//   DH   per (token tile, 256-column block of Hd): recompute each z tile,
//        form dz = c (softmax - onehot) in bf16 straight into shared memory in
//        the MMA operand layout, and accumulate dH += dz W in TMEM.
//   DW   per (vocab tile, 256-column block of Hd): recompute the transposed
//        z tile W_j H_i^T, form dz^T the same way, accumulate dW += dz^T H.
//
// Every operand is K-major: dH and dW take W^T and H^T, which the call first
// writes into its workspace.  Warp roles per CTA: warp 0 issues TMA loads into
// a 4-stage ring, warp 1 issues tcgen05.mma (one thread) and owns TMEM, warps
// 2..5 are the epilogue (one TMEM lane = one tile row per thread).  All waits
// are bounded; a wait that runs out sets CIS_ERR_DEVICE_TIMEOUT and the CTA
// carries on to its end so that TMEM is always released.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <stdlib.h>
#include <mutex>

#include <cooperative_groups.h>

#include "cis_kernels.h"
#include "cis_tc.cuh"

namespace cg = cooperative_groups;

namespace cis {
namespace lm {

constexpr int kBM = 128;     // tile rows (M)
constexpr int kBN = 128;     // tile columns of z (N)
constexpr int kBK = 64;      // K block: one 128-byte swizzled row of bf16
constexpr int kN2 = 256;     // Hd columns of dH / dW per CTA
constexpr int kStages = 4;
constexpr int kStageBytes = 32768;
constexpr int kThreads = 192;
constexpr int kFwdGroup = 16;  // vocab tiles per FWD CTA

enum Mode { kFwd = 0, kDh = 1, kDw = 2 };

// OR of `pred` over the 128 epilogue threads (named barrier 1), so that the
// four epilogue warps leave their loop together.
__device__ __forceinline__ int __syncthreads_or_epi(int pred)
{
    int r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.s32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, 128, p;\n\tselp.s32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(pred)
        : "memory");
    return r;
}

struct Params {
    int T, V, Hd;
    int nTt, nVt, nK;
    const int32_t *ids;
    const uint8_t *mask;
    const float *lse;    // DH / DW: per token
    const float *cvec;   // DH / DW: per token, 0 where the token has no gradient
    float2 *part;        // FWD: [nVt, T] (max, sum) over j != y
    float *zy;           // FWD: z at the sampled token
    void *out;           // DH: dH [T, ld_out]; DW: dW [V, ld_out]
    int out_bf16;
    int64_t ld_out;
    int32_t *status;
};

struct Barriers {
    uint64_t full[kStages], empty[kStages];
    uint64_t zfull[2], zempty[2];
    uint64_t dzfull, dzempty, accfull;
};

// A wait that runs out marks the CTA (and, through the status word, every
// later CTA) as aborted: the roles then stop waiting and run to the end, so a
// broken pipeline costs one bounded wait per role instead of one per tile.
struct Abort {
    volatile int *local;
    const volatile int32_t *status;
    __device__ __forceinline__ bool on() const
    {
        return *local != 0 || (*status & kStatusTimeout) != 0;
    }
    __device__ __forceinline__ void wait(uint64_t *bar, uint32_t parity, int32_t *st) const
    {
        if (*local)
            return;
        if (!tc::bar_wait(bar, parity)) {
            *local = 1;
            set_status(st, kStatusTimeout);
        }
    }
};

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    cis_lmhead_kernel(const __grid_constant__ CUtensorMap tmA,
                      const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmB2, const Params p)
{
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t *base = dsm + ((1024 - (tc::smem_addr(dsm) & 1023)) & 1023);
    uint8_t *ring = base;                          // kStages x 32 KB
    uint8_t *dzbuf = base + kStages * kStageBytes; // 32 KB: dz tile, 2 K blocks
    __shared__ __align__(8) Barriers bars;
    __shared__ uint32_t tmem_base;
    __shared__ int aborted;
    __shared__ float col_lse[2][kBN], col_c[2][kBN];
    __shared__ int col_y[2][kBN];

    constexpr uint32_t kTmemCols = MODE == kFwd ? 256 : 512;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // tile assignment
    int a_tile, nB, b_first, hblk = 0;
    if (MODE == kFwd) {
        a_tile = blockIdx.x % p.nTt;
        b_first = (blockIdx.x / p.nTt) * kFwdGroup;
        nB = min(kFwdGroup, p.nVt - b_first);
    } else if (MODE == kDh) {
        a_tile = blockIdx.x % p.nTt;
        hblk = blockIdx.x / p.nTt;
        b_first = 0;
        nB = p.nVt;
    } else {
        a_tile = blockIdx.x % p.nVt;
        hblk = blockIdx.x / p.nVt;
        b_first = 0;
        nB = p.nTt;
    }

    if (threadIdx.x == 0) {
        aborted = 0;
        for (int s = 0; s < kStages; ++s) {
            tc::bar_init(&bars.full[s], 1);
            tc::bar_init(&bars.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::bar_init(&bars.zfull[b], 1);
            tc::bar_init(&bars.zempty[b], 128);
        }
        tc::bar_init(&bars.dzfull, 128);
        tc::bar_init(&bars.dzempty, 1);
        tc::bar_init(&bars.accfull, 1);
        tc::bar_init_fence();
    }
    if (warp == 1)
        tc::tmem_alloc(&tmem_base, kTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = tmem_base;
    const uint32_t tmem_acc = tmem + 256;  // DH / DW accumulator, 256 columns
    const Abort ab{&aborted, p.status};

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            auto next = [&]() {
                ab.wait(&bars.empty[stage], phase ^ 1, p.status);
                tc::bar_expect_tx(&bars.full[stage], kStageBytes);
            };
            auto advance = [&]() {
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1;
                }
            };
            auto load_b2 = [&](int jb) {
                for (int kb = 0; kb < 2; ++kb) {
                    next();
                    tc::tma_load_2d(ring + stage * kStageBytes, &tmB2,
                                    (b_first + jb) * kBN + kb * kBK, hblk * kN2,
                                    &bars.full[stage]);
                    advance();
                }
            };
            for (int jb = 0; jb < nB && !ab.on(); ++jb) {
                for (int k = 0; k < p.nK; ++k) {
                    next();
                    uint8_t *st = ring + stage * kStageBytes;
                    tc::tma_load_2d(st, &tmA, k * kBK, a_tile * kBM, &bars.full[stage]);
                    tc::tma_load_2d(st + kStageBytes / 2, &tmB, k * kBK, (b_first + jb) * kBN,
                                    &bars.full[stage]);
                    advance();
                }
                if (MODE != kFwd && jb >= 1)
                    load_b2(jb - 1);
            }
            if (MODE != kFwd && nB >= 1 && !ab.on())
                load_b2(nB - 1);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issue
        if (lane == 0) {
            constexpr uint32_t kIdZ = tc::idesc_bf16(kBM, kBN);
            constexpr uint32_t kId2 = tc::idesc_bf16(kBM, kN2);
            int stage = 0;
            uint32_t phase = 0;
            auto advance = [&]() {
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1;
                }
            };
            for (int jb = 0; jb <= nB && !ab.on(); ++jb) {
                if (jb < nB) {
                    const int zb = jb & 1;
                    ab.wait(&bars.zempty[zb], ((jb >> 1) & 1) ^ 1, p.status);
                    tc::fence_after_sync();
                    const uint32_t dz = tmem + zb * kBN;
                    for (int k = 0; k < p.nK; ++k) {
                        ab.wait(&bars.full[stage], phase, p.status);
                        tc::fence_after_sync();
                        const uint32_t sa = tc::smem_addr(ring + stage * kStageBytes);
                        const uint32_t sb = sa + kStageBytes / 2;
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk)
                            tc::mma_bf16(dz, tc::desc_sw128(sa + kk * 32),
                                         tc::desc_sw128(sb + kk * 32), kIdZ, (k | kk) != 0);
                        tc::mma_commit(&bars.empty[stage]);
                        advance();
                    }
                    tc::mma_commit(&bars.zfull[zb]);
                }
                if (MODE != kFwd && jb >= 1) {
                    // dH (or dW) += dz (tile jb-1, in shared memory) x B2 chunk
                    ab.wait(&bars.dzfull, (jb - 1) & 1, p.status);
                    tc::fence_after_sync();
                    const uint32_t sdz = tc::smem_addr(dzbuf);
                    for (int kb = 0; kb < 2; ++kb) {
                        ab.wait(&bars.full[stage], phase, p.status);
                        tc::fence_after_sync();
                        const uint32_t sb2 = tc::smem_addr(ring + stage * kStageBytes);
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk)
                            tc::mma_bf16(tmem_acc, tc::desc_sw128(sdz + kb * 16384 + kk * 32),
                                         tc::desc_sw128(sb2 + kk * 32), kId2,
                                         (jb - 1) > 0 || kb > 0 || kk > 0);
                        tc::mma_commit(&bars.empty[stage]);
                        advance();
                    }
                    tc::mma_commit(&bars.dzempty);
                }
            }
            if (MODE != kFwd)
                tc::mma_commit(&bars.accfull);
        }
    } else {
        // ---------------------------------------------------------- epilogue
        const int lg = warp & 3;           // TMEM lane group of this warp
        const int r = lg * 32 + lane;      // tile row of this thread
        const uint32_t lane_off = (uint32_t)(lg * 32) << 16;
        const int e = threadIdx.x - 64;    // 0..127
        const int row = (MODE == kDw ? a_tile * kBM : a_tile * kBM) + r;

        // per-row scalars
        int y_r = -1;
        float lse_r = 0.0f, c_r = 0.0f;
        if (MODE != kDw && row < p.T) {
            y_r = p.ids[row];
            if (MODE == kDh) {
                lse_r = p.lse[row];
                c_r = p.cvec[row];
            }
        }
        for (int jb = 0; jb < nB; ++jb) {
            const int zb = jb & 1;
            const int col0 = (b_first + jb) * kBN;
            // every epilogue warp takes the same path (named barrier below)
            const int stop = ab.on();
            if (__syncthreads_or_epi(stop))
                break;
            if (MODE == kDw) {
                // scalars of this token tile's 128 columns
                const int t = col0 + e;
                const bool ok = t < p.T;
                col_lse[zb][e] = ok ? p.lse[t] : 0.0f;
                col_c[zb][e] = ok ? p.cvec[t] : 0.0f;
                col_y[zb][e] = ok ? p.ids[t] : -1;
                asm volatile("bar.sync 1, 128;" ::: "memory");
            }
            ab.wait(&bars.zfull[zb], (jb >> 1) & 1, p.status);
            tc::fence_after_sync();
            const uint32_t zaddr = tmem + lane_off + zb * kBN;
            if (MODE == kFwd) {
                float m = -INFINITY, s = 0.0f, zyv = 0.0f;
                bool got_y = false;
                for (int c0 = 0; c0 < kBN; c0 += 32) {
                    float v[32];
                    tc::tmem_ld32(zaddr + c0, v);
                    const int cbase = col0 + c0;
                    if (y_r >= cbase && y_r < cbase + 32) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (cbase + i == y_r)
                                zyv = v[i];
                        got_y = true;
                    }
                    float cm = -INFINITY;
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int col = cbase + i;
                        v[i] = (col == y_r || col >= p.V) ? -INFINITY : v[i];
                        cm = fmaxf(cm, v[i]);
                    }
                    if (cm > m) {
                        s = m == -INFINITY ? 0.0f : s * ex2_ftz((m - cm) * kLog2e);
                        m = cm;
                    }
                    if (m != -INFINITY) {
                        float acc = 0.0f;
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            acc += ex2_ftz((v[i] - m) * kLog2e);
                        s += acc;
                    }
                }
                tc::fence_before_sync();
                tc::bar_arrive(&bars.zempty[zb]);
                if (row < p.T) {
                    p.part[(int64_t)(b_first + jb) * p.T + row] = make_float2(m, s);
                    if (got_y)
                        p.zy[row] = zyv;
                }
            } else {
                // dz tile (bf16) into shared memory, operand layout; wait until the
                // previous tile's dz has been consumed by its MMA
                ab.wait(&bars.dzempty, (jb & 1) ^ 1, p.status);
                for (int c0 = 0; c0 < kBN; c0 += 32) {
                    float v[32];
                    tc::tmem_ld32(zaddr + c0, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int col = c0 + i;  // column within the tile
                        float d;
                        // tokens with c = 0 (masked, clipped, past T) give 0 without
                        // touching the exponential (their lse is a placeholder)
                        if (MODE == kDh) {
                            const int gcol = col0 + col;  // vocab index
                            d = (gcol < p.V && c_r != 0.0f)
                                    ? c_r * ex2_ftz((v[i] - lse_r) * kLog2e) -
                                          (gcol == y_r ? c_r : 0.0f)
                                    : 0.0f;
                        } else {
                            const float lt = col_lse[zb][col], ct = col_c[zb][col];
                            d = (row < p.V && ct != 0.0f)
                                    ? ct * ex2_ftz((v[i] - lt) * kLog2e) -
                                          (col_y[zb][col] == row ? ct : 0.0f)
                                    : 0.0f;
                        }
                        v[i] = d;
                    }
                    // 32 values = 4 chunks of 8 bf16 in K block c0 / 64
                    uint8_t *blk = dzbuf + (c0 >> 6) * 16384;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 w;
                        __nv_bfloat162 h;
                        h = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
                        w.x = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
                        w.y = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
                        w.z = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
                        w.w = *reinterpret_cast<uint32_t *>(&h);
                        const int chunk = ((c0 & 63) >> 3) + q;
                        *reinterpret_cast<uint4 *>(blk + tc::sw128_offset(r, chunk)) = w;
                    }
                }
                tc::fence_before_sync();
                tc::bar_arrive(&bars.zempty[zb]);
                tc::fence_proxy_async_smem();
                tc::bar_arrive(&bars.dzfull);
            }
        }
        if (MODE != kFwd) {
            // the accumulated dH / dW block: 128 rows x 256 columns
            ab.wait(&bars.accfull, 0, p.status);
            tc::fence_after_sync();
            const int nrows = MODE == kDh ? p.T : p.V;
            for (int c0 = 0; c0 < kN2; c0 += 32) {
                float v[32];
                tc::tmem_ld32(tmem_acc + lane_off + c0, v);
                if (row < nrows) {
                    const int64_t o = (int64_t)row * p.ld_out + (int64_t)hblk * kN2 + c0;
                    if (p.out_bf16) {
                        __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(p.out) + o;
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 w;
                            __nv_bfloat162 h;
                            h = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
                            w.x = *reinterpret_cast<uint32_t *>(&h);
                            h = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
                            w.y = *reinterpret_cast<uint32_t *>(&h);
                            h = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
                            w.z = *reinterpret_cast<uint32_t *>(&h);
                            h = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
                            w.w = *reinterpret_cast<uint32_t *>(&h);
                            reinterpret_cast<uint4 *>(dst)[q] = w;
                        }
                    } else {
                        float4 *dst = reinterpret_cast<float4 *>(reinterpret_cast<float *>(p.out) + o);
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                    }
                }
            }
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------------------
// Gradient passes shared by a cluster: R = Hd / 256 CTAs, CTA r accumulating
// block r (256 columns) of dH (or dW).  Step j of the sweep is vocabulary tile
// j (dW: token tile j).  Its logit tile is computed once, by the CTA that owns
// the step (j mod R), which forms the bf16 dz tile in its own shared memory
// and bulk-copies it into the same mailbox slot (j mod 2) of every other CTA
// of the cluster; each copy is counted on the receiver's mbarrier.  Every CTA
// consumes every step: block r += dz_j x (W^T or H^T)[block r, tile j].  After
// consuming step j a CTA's MMA commit is multicast to the slot-free mbarrier
// of the owner of step j + 2, which reuses the slot.  A CTA computes the logit
// tile of its k-th owned step t_k = r + kR spread over the R steps of the
// period two before it (4 K blocks per step), so no commit waits on a whole
// tile, and the tile is ready R + 1 steps before it is consumed.
//
// Phases.  Copies into slot s of a CTA arrive in step order, each only after
// the CTA has consumed the previous step of that slot, so neither the mailbox
// nor the per-slot slot-free barrier can run a phase ahead of its waiter.
// Teardown.  Each copy is first recorded in the receiver (a remote max of the
// step index), so after a cluster barrier that ends all copying a CTA knows
// whether a copy into it may still be in flight and waits for it (bounded)
// before the second cluster barrier; only then may a CTA leave.
constexpr int kSlotBytes = 32768;

struct CBarriers {
    uint64_t full[kStages], empty[kStages];
    uint64_t zfull[2], zempty[2];
    uint64_t dzfull[2];     // the dz tile of the step in slot s has landed
    uint64_t slot_free[2];  // every CTA has consumed the step that last used slot s
    uint64_t accfull;
};

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    cis_lmhead_grad_kernel(const __grid_constant__ CUtensorMap tmA,
                           const __grid_constant__ CUtensorMap tmB,
                           const __grid_constant__ CUtensorMap tmB2, const Params p)
{
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t *base = dsm + ((1024 - (tc::smem_addr(dsm) & 1023)) & 1023);
    uint8_t *ring = base;                            // kStages x 32 KB
    uint8_t *slots = base + kStages * kStageBytes;   // 2 x 32 KB dz mailboxes
    __shared__ __align__(8) CBarriers bars;
    __shared__ uint32_t tmem_base;
    __shared__ int aborted;
    __shared__ int last_copied[2];  // latest step copied into slot s by its owner
    __shared__ float col_lse[kBN], col_c[kBN];
    __shared__ int col_y[kBN];

    cg::cluster_group cluster = cg::this_cluster();
    const int R = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int a_tile = blockIdx.x / R;
    const int nB = MODE == kDh ? p.nVt : p.nTt;
    const int Q = p.nK / R;  // K blocks of a logit tile issued per step
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        aborted = 0;
        last_copied[0] = last_copied[1] = -1;
        for (int s = 0; s < kStages; ++s) {
            tc::bar_init(&bars.full[s], 1);
            tc::bar_init(&bars.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::bar_init(&bars.zfull[b], 1);
            tc::bar_init(&bars.zempty[b], 128);
            tc::bar_init(&bars.dzfull[b], 1);
            tc::bar_init(&bars.slot_free[b], R);
        }
        tc::bar_init(&bars.accfull, 1);
        tc::bar_init_fence();
    }
    if (warp == 1)
        tc::tmem_alloc(&tmem_base, 512);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    // every CTA of the cluster has initialised its barriers before any remote use
    tc::cluster_arrive();
    tc::cluster_wait();
    const uint32_t tmem = tmem_base;
    const uint32_t tmem_acc = tmem + 256;
    const Abort ab{&aborted, p.status};
    int consumed = 0;  // MMA thread: steps 0 .. consumed-1 are fully issued
    int expected = -1; // MMA thread: latest step whose copy it announced

    // The ring items in the order both the producer and the MMA issuer take
    // them: fn_z(k, kb) for K block kb of owned tile t_k, fn_step(j) before
    // the two B2 items fn_b2(j, 0), fn_b2(j, 1) of step j.
    auto walk = [&](auto &&fn_z, auto &&fn_step, auto &&fn_b2) {
        if (rank < nB)
            for (int kb = 0; kb < p.nK; ++kb)
                fn_z(0, kb);
        if (rank + R < nB)
            for (int kb = 0; kb < (R - rank) * Q; ++kb)
                fn_z(1, kb);
        for (int j = 0; j < nB && !ab.on(); ++j) {
            int k, pi;
            if (j < rank) {
                k = 1;
                pi = j - rank + R;
            } else {
                k = (j - rank) / R + 2;
                pi = (j - rank) % R;
            }
            if (rank + k * R < nB)
                for (int kb = pi * Q; kb < (pi + 1) * Q; ++kb)
                    fn_z(k, kb);
            fn_step(j);
            fn_b2(j, 0);
            fn_b2(j, 1);
        }
    };

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t used = 0, last_phase = 0;  // per stage: loaded, parity of its last load
            auto next = [&]() -> bool {
                if (ab.on())
                    return false;
                ab.wait(&bars.empty[stage], phase ^ 1, p.status);
                if (ab.on())
                    return false;
                tc::bar_expect_tx(&bars.full[stage], kStageBytes);
                used |= 1u << stage;
                last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
                return true;
            };
            auto adv = [&]() {
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1;
                }
            };
            walk(
                [&](int k, int kb) {
                    if (!next())
                        return;
                    uint8_t *st = ring + stage * kStageBytes;
                    tc::tma_load_2d(st, &tmA, kb * kBK, a_tile * kBM, &bars.full[stage]);
                    tc::tma_load_2d(st + kStageBytes / 2, &tmB, kb * kBK, (rank + k * R) * kBN,
                                    &bars.full[stage]);
                    adv();
                },
                [&](int) {},
                [&](int j, int kb2) {
                    if (!next())
                        return;
                    tc::tma_load_2d(ring + stage * kStageBytes, &tmB2, j * kBN + kb2 * kBK,
                                    rank * kN2, &bars.full[stage]);
                    adv();
                });
            // no load may still be landing when the CTA leaves
            for (int s = 0; s < kStages; ++s)
                if (used & (1u << s))
                    tc::bar_wait(&bars.full[s], (last_phase >> s) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t kIdZ = tc::idesc_bf16(kBM, kBN);
            constexpr uint32_t kId2 = tc::idesc_bf16(kBM, kN2);
            int stage = 0;
            uint32_t phase = 0;
            auto adv = [&]() {
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1;
                }
            };
            walk(
                [&](int k, int kb) {
                    if (ab.on())
                        return;
                    const int zb = k & 1;
                    if (kb == 0)  // the buffer's previous tile has been read
                        ab.wait(&bars.zempty[zb], ((k >> 1) & 1) ^ 1, p.status);
                    ab.wait(&bars.full[stage], phase, p.status);
                    if (ab.on())
                        return;
                    tc::fence_after_sync();
                    const uint32_t sa = tc::smem_addr(ring + stage * kStageBytes);
                    const uint32_t sb = sa + kStageBytes / 2;
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk)
                        tc::mma_bf16(tmem + zb * kBN, tc::desc_sw128(sa + kk * 32),
                                     tc::desc_sw128(sb + kk * 32), kIdZ, (kb | kk) != 0);
                    tc::mma_commit(&bars.empty[stage]);
                    adv();
                    if (kb == p.nK - 1)
                        tc::mma_commit(&bars.zfull[zb]);
                },
                [&](int j) {
                    if (ab.on())
                        return;
                    const int s = j & 1;
                    if (j % R != rank) {  // the owner's copy brings the bytes
                        tc::bar_expect_tx(&bars.dzfull[s], kSlotBytes);
                        expected = j;
                    }
                    if (!tc::bar_wait_cluster(&bars.dzfull[s], (j >> 1) & 1)) {
                        aborted = 1;
                        set_status(p.status, kStatusTimeout);
                    }
                },
                [&](int j, int kb2) {
                    if (ab.on())
                        return;
                    ab.wait(&bars.full[stage], phase, p.status);
                    if (ab.on())
                        return;
                    tc::fence_after_sync();
                    const uint32_t sdz = tc::smem_addr(slots + (j & 1) * kSlotBytes);
                    const uint32_t sb2 = tc::smem_addr(ring + stage * kStageBytes);
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk)
                        tc::mma_bf16(tmem_acc, tc::desc_sw128(sdz + kb2 * 16384 + kk * 32),
                                     tc::desc_sw128(sb2 + kk * 32), kId2,
                                     j > 0 || kb2 > 0 || kk > 0);
                    tc::mma_commit(&bars.empty[stage]);
                    adv();
                    if (kb2 == 1) {
                        if (j + 2 < nB)  // slot j & 1 is free here for step j + 2
                            tc::mma_commit_multicast(&bars.slot_free[j & 1],
                                                     (uint16_t)(1u << ((j + 2) % R)));
                        consumed = j + 1;
                    }
                });
            // every MMA of this CTA (and the arrivals committed with them) is
            // done before the epilogue reads the block or the CTA leaves
            tc::mma_commit(&bars.accfull);
            tc::bar_wait(&bars.accfull, 0);
        }
    } else {
        const int lg = warp & 3;
        const int r = lg * 32 + lane;
        const uint32_t lane_off = (uint32_t)(lg * 32) << 16;
        const int e = threadIdx.x - 64;
        const int row = a_tile * kBM + r;  // token (DH) or vocabulary entry (DW)
        int y_r = -1;
        float lse_r = 0.0f, c_r = 0.0f;
        if (MODE == kDh && row < p.T) {
            y_r = p.ids[row];
            lse_r = p.lse[row];
            c_r = p.cvec[row];
        }
        uint32_t nfree = 0;  // per slot (bit s): parity of its next slot-free phase
        for (int k = 0; rank + k * R < nB; ++k) {
            const int t = rank + k * R;  // the owned step
            const int zb = k & 1, s = t & 1;
            if (__syncthreads_or_epi(ab.on()))
                break;
            if (MODE == kDw) {
                const int tt = t * kBN + e;
                const bool ok = tt < p.T;
                col_lse[e] = ok ? p.lse[tt] : 0.0f;
                col_c[e] = ok ? p.cvec[tt] : 0.0f;
                col_y[e] = ok ? p.ids[tt] : -1;
            }
            ab.wait(&bars.zfull[zb], (k >> 1) & 1, p.status);
            tc::fence_after_sync();
            if (t >= 2) {  // slot s still holds step t - 2 somewhere in the cluster
                if (!ab.on() && !tc::bar_wait_cluster(&bars.slot_free[s], (nfree >> s) & 1)) {
                    aborted = 1;
                    set_status(p.status, kStatusTimeout);
                }
                nfree ^= 1u << s;
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");  // column scalars visible
            uint8_t *slot = slots + s * kSlotBytes;
            const int col0 = t * kBN;
            for (int c0 = 0; c0 < kBN; c0 += 32) {
                float v[32];
                tc::tmem_ld32(tmem + lane_off + zb * kBN + c0, v);
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int col = c0 + i;
                    float d;
                    // tokens with c = 0 (masked, clipped, past T) give 0 without
                    // touching the exponential (their lse is a placeholder)
                    if (MODE == kDh) {
                        const int gcol = col0 + col;
                        d = (gcol < p.V && c_r != 0.0f)
                                ? c_r * ex2_ftz((v[i] - lse_r) * kLog2e) -
                                      (gcol == y_r ? c_r : 0.0f)
                                : 0.0f;
                    } else {
                        const float lt = col_lse[col], ct = col_c[col];
                        d = (row < p.V && ct != 0.0f)
                                ? ct * ex2_ftz((v[i] - lt) * kLog2e) -
                                      (col_y[col] == row ? ct : 0.0f)
                                : 0.0f;
                    }
                    v[i] = d;
                }
                uint8_t *blk = slot + (c0 >> 6) * 16384;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint4 w;
                    __nv_bfloat162 h;
                    h = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
                    w.x = *reinterpret_cast<uint32_t *>(&h);
                    h = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
                    w.y = *reinterpret_cast<uint32_t *>(&h);
                    h = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
                    w.z = *reinterpret_cast<uint32_t *>(&h);
                    h = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
                    w.w = *reinterpret_cast<uint32_t *>(&h);
                    *reinterpret_cast<uint4 *>(blk + tc::sw128_offset(r, ((c0 & 63) >> 3) + q)) = w;
                }
            }
            tc::fence_before_sync();
            tc::bar_arrive(&bars.zempty[zb]);
            tc::fence_proxy_async_smem();
            asm volatile("bar.sync 1, 128;" ::: "memory");  // the whole tile is written
            if (e == 0 && !ab.on()) {
                const uint32_t src = tc::smem_addr(slot);
                const uint32_t bar = tc::smem_addr(&bars.dzfull[s]);
                const uint32_t rec = tc::smem_addr(&last_copied[s]);
                for (int q = 0; q < R; ++q)
                    if (q != rank) {
                        tc::red_max_cluster(tc::map_rank(rec, q), t);
                        tc::bulk_s2s(tc::map_rank(src, q), src, kSlotBytes, tc::map_rank(bar, q));
                    }
                tc::bar_arrive(&bars.dzfull[s]);
            }
        }
        // the accumulated block: 128 rows x 256 columns
        ab.wait(&bars.accfull, 0, p.status);
        tc::fence_after_sync();
        const int nrows = MODE == kDh ? p.T : p.V;
        for (int c0 = 0; c0 < kN2; c0 += 32) {
            float v[32];
            tc::tmem_ld32(tmem_acc + lane_off + c0, v);
            if (row < nrows) {
                const int64_t o = (int64_t)row * p.ld_out + (int64_t)rank * kN2 + c0;
                if (p.out_bf16) {
                    __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(p.out) + o;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 w;
                        __nv_bfloat162 h;
                        h = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
                        w.x = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
                        w.y = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
                        w.z = *reinterpret_cast<uint32_t *>(&h);
                        h = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
                        w.w = *reinterpret_cast<uint32_t *>(&h);
                        reinterpret_cast<uint4 *>(dst)[q] = w;
                    }
                } else {
                    float4 *dst =
                        reinterpret_cast<float4 *>(reinterpret_cast<float *>(p.out) + o);
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                }
            }
        }
    }
    // Teardown: after the first cluster barrier no CTA issues another copy;
    // each CTA then waits for any copy recorded into it that it has not seen
    // land, and no CTA leaves before all have done so.
    __syncwarp();
    tc::fence_before_sync();
    tc::cluster_arrive();
    tc::cluster_wait();
    if (warp == 1 && lane == 0) {
        for (int s = 0; s < 2; ++s) {
            const int L = *reinterpret_cast<volatile int *>(&last_copied[s]);
            if (L >= consumed) {  // recorded but not consumed: it may be landing
                if (L != expected)
                    tc::bar_expect_tx(&bars.dzfull[s], kSlotBytes);
                tc::bar_wait_cluster(&bars.dzfull[s], (L >> 1) & 1);
            }
        }
    }
    __syncwarp();
    tc::cluster_arrive();
    tc::cluster_wait();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 512);
    }
}

// Per token: combine the FWD pairs, then log p, weight, loss, c_t (one warp).
__global__ void cis_lmhead_token_kernel(const PassArgs a, const float2 *part, const float *zy,
                                        int nVt, float *lse_out, float *c_out)
{
    const int64_t t = blockIdx.x * (int64_t)(blockDim.x / 32) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (t >= a.T)
        return;
    const bool valid = a.mask == nullptr || a.mask[t] != 0;
    const int64_t y = a.ids[t];
    const bool id_ok = y >= 0 && y < a.V;
    if (!valid || !id_ok) {
        if (lane == 0) {
            if (valid)
                set_status(a.status, kStatusBadId);
            const float lp = valid ? NAN : 0.0f;
            if (a.lp_out) a.lp_out[t] = lp;
            if (a.w_out) a.w_out[t] = 0.0f;
            if (a.trunc_out) a.trunc_out[t] = 0;
            a.ws_w[t] = 0.0f;
            a.ws_trunc[t] = 0;
            a.ws_logk[t] = 0.0f;
            a.ws_terms[t] = valid ? (double)NAN : 0.0;
            lse_out[t] = 0.0f;
            c_out[t] = 0.0f;
        }
        return;
    }
    MaxSum o{-INFINITY, 0.0f};
    for (int j = lane; j < nVt; j += 32) {
        const float2 q = part[(int64_t)j * a.T + t];
        o = ms_combine(o, MaxSum{q.x, q.y});
    }
    o = warp_ms(o);
    if (lane == 0) {
        const RowScalars rs = row_scalars(o, zy[t]);
        const bool has_old = a.lp_old != nullptr;
        const float lold = has_old ? a.lp_old[t] : 0.0f;
        const TokenWeight tw = token_weight(has_old ? (double)lold : rs.lp64, a.lp_inf[t], a.P);
        const TokenLoss tl = token_loss(rs.lp64, has_old, lold, a.adv[t], a.scale[t], tw.w, a.P);
        if (a.lp_out) a.lp_out[t] = rs.lp;
        if (a.w_out) a.w_out[t] = tw.w;
        if (a.trunc_out) a.trunc_out[t] = tw.trunc;
        a.ws_w[t] = tw.w;
        a.ws_trunc[t] = tw.trunc;
        a.ws_logk[t] = tw.logk;
        a.ws_terms[t] = tl.term;
        lse_out[t] = rs.lse;
        c_out[t] = tl.c;
    }
}

// out[c, r] = in[r, c] for a bf16 [rows, cols] matrix (row stride ld_in).
__global__ void cis_lmhead_transpose_kernel(const __nv_bfloat16 *in, int64_t rows, int64_t cols,
                                            int64_t ld_in, __nv_bfloat16 *out, int64_t ld_out)
{
    __shared__ __nv_bfloat16 tile[32][33];
    const int64_t r0 = (int64_t)blockIdx.y * 32, c0 = (int64_t)blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols)
            tile[i][threadIdx.x] = in[r * ld_in + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t c = c0 + i, r = r0 + threadIdx.x;
        if (c < cols && r < rows)
            out[c * ld_out + r] = tile[threadIdx.x][i];
    }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void *f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// 2-D bf16 tensor map: inner extent `inner`, `outer` rows, row stride `ld`
// elements, box {64, box_rows}, 128-byte swizzle, zero fill out of bounds.
bool make_map(CUtensorMap *m, const void *ptr, int64_t inner, int64_t outer, int64_t ld,
              int box_rows)
{
    auto enc = encoder();
    if (!enc)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    cuuint64_t strides[1] = {(cuuint64_t)(ld * 2)};
    cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides,
               box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr size_t kSmemBytes = kStages * kStageBytes + 32768 + 1024;

template <int MODE>
cudaError_t launch_mode(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                        const Params &p, int grid, cudaStream_t s)
{
    auto k = cis_lmhead_kernel<MODE>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    k<<<grid, kThreads, kSmemBytes, s>>>(a, b, b2, p);
    return cudaGetLastError();
}

constexpr size_t kGradSmemBytes = kStages * kStageBytes + 2 * kSlotBytes + 1024;

template <int MODE>
cudaError_t launch_grad(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                        const Params &p, int clusters, int R, cudaStream_t s)
{
    auto k = cis_lmhead_grad_kernel<MODE>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kGradSmemBytes);
    if (e != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(clusters * R), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kGradSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)R;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k, a, b, b2, p);
}

// Use the cluster gradient kernels?  Needs a portable cluster (Hd <= 2048);
// CIS_LMHEAD_RECOMPUTE=1 selects the recompute kernels instead (for comparison).
bool use_cluster_grad(int64_t H)
{
    static int force_recompute = [] {
        const char *e = getenv("CIS_LMHEAD_RECOMPUTE");
        return e ? atoi(e) : 0;
    }();
    return !force_recompute && H / kN2 <= 8;
}

}  // namespace lm

// Workspace of cis_lmhead_fused, after the token-pass layout of ws_layout(T).
struct LmLayout {
    WsLayout base;
    size_t lse, c, zy, part, wt, ht, total;
    int64_t vp, tp;
};

LmLayout lm_layout(int64_t T, int64_t V, int64_t Hd)
{
    auto up = [](size_t x) { return (x + 1023) / 1024 * 1024; };
    LmLayout L;
    L.base = ws_layout(T);
    const int64_t nVt = (V + lm::kBN - 1) / lm::kBN;
    L.vp = (V + 7) / 8 * 8;
    L.tp = (T + 7) / 8 * 8;
    size_t o = up(L.base.total);
    L.lse = o;
    o = up(o + 4 * (size_t)T);
    L.c = o;
    o = up(o + 4 * (size_t)T);
    L.zy = o;
    o = up(o + 4 * (size_t)T);
    L.part = o;
    o = up(o + 8 * (size_t)T * (size_t)nVt);
    L.wt = o;
    o = up(o + 2 * (size_t)Hd * (size_t)L.vp);
    L.ht = o;
    o = up(o + 2 * (size_t)Hd * (size_t)L.tp);
    L.total = o;
    return L;
}

}  // namespace cis

using namespace cis;

extern "C" {

CIS_API cis_status_t cis_lmhead_workspace_size(int64_t T, int64_t V, int64_t H, size_t *bytes)
{
    if (bytes == nullptr || T < 0 || V <= 0 || H <= 0)
        return CIS_ERR_INVALID_ARG;
    *bytes = lm_layout(T, V, H).total;
    return CIS_OK;
}

CIS_API cis_status_t cis_lmhead_fused(const void *hidden, const void *weight, int64_t T,
                                      int64_t H, int64_t V, const int32_t *ids,
                                      const float *lp_infer, const float *lp_old,
                                      const float *adv, const uint8_t *mask,
                                      const int32_t *cu_seqlens, int64_t B,
                                      const cis_params_t *params, void *dhidden, void *dweight,
                                      int32_t grad_dtype, float *lp_out, float *w_out,
                                      uint8_t *trunc_out, cis_stats_t *stats_out,
                                      double *loss_out, void *workspace, size_t workspace_bytes,
                                      void *stream)
{
    if (T < 0 || T > (1LL << 30) || V <= 0 || V > (1LL << 30) || H <= 0)
        return CIS_ERR_INVALID_ARG;
    if (grad_dtype != CIS_F32 && grad_dtype != CIS_BF16)
        return CIS_ERR_INVALID_ARG;
    if (!params_ok(params))
        return CIS_ERR_INVALID_ARG;
    if (params->agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN && (cu_seqlens == nullptr || B < 0))
        return CIS_ERR_INVALID_ARG;
    if (H % lm::kN2 != 0)
        return CIS_ERR_UNSUPPORTED;  // Hd in blocks of 256 (and so of the 64-wide K blocks)
    const LmLayout L = lm_layout(T, V, H);
    if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 1023) ||
        workspace_bytes < L.total)
        return CIS_ERR_INVALID_ARG;
    if (T > 0 && (hidden == nullptr || weight == nullptr || ids == nullptr ||
                  lp_infer == nullptr || adv == nullptr || dhidden == nullptr ||
                  dweight == nullptr))
        return CIS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(hidden) & 15) || (reinterpret_cast<uintptr_t>(weight) & 15) ||
        (reinterpret_cast<uintptr_t>(dhidden) & 15) || (reinterpret_cast<uintptr_t>(dweight) & 15))
        return CIS_ERR_INVALID_ARG;
    const cis_params_t P = *params;
    cudaStream_t s = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    PassArgs a = {};
    a.T = T;
    a.V = V;
    a.ids = ids;
    a.lp_inf = lp_infer;
    a.lp_old = lp_old;
    a.adv = adv;
    a.mask = mask;
    a.scale = reinterpret_cast<float *>(ws + L.base.scale);
    a.lp_out = lp_out;
    a.w_out = w_out;
    a.trunc_out = trunc_out;
    a.ws_w = reinterpret_cast<float *>(ws + L.base.w);
    a.ws_trunc = ws + L.base.trunc;
    a.ws_logk = reinterpret_cast<float *>(ws + L.base.logk);
    a.ws_terms = reinterpret_cast<double *>(ws + L.base.terms);
    a.status = reinterpret_cast<int32_t *>(ws + L.base.status);
    a.P = make_dev_params(P);
    float *lse = reinterpret_cast<float *>(ws + L.lse);
    float *cv = reinterpret_cast<float *>(ws + L.c);
    float *zy = reinterpret_cast<float *>(ws + L.zy);
    float2 *part = reinterpret_cast<float2 *>(ws + L.part);
    __nv_bfloat16 *wt = reinterpret_cast<__nv_bfloat16 *>(ws + L.wt);
    __nv_bfloat16 *ht = reinterpret_cast<__nv_bfloat16 *>(ws + L.ht);

    float *scale = reinterpret_cast<float *>(ws + L.base.scale);
    cudaError_t e = launch_scales(mask, T, cu_seqlens, B, P.agg, scale, a.status, s);
    if (e != cudaSuccess)
        return e == cudaErrorNotSupported ? CIS_ERR_UNSUPPORTED : CIS_ERR_CUDA;
    if (T > 0) {
        const int nTt = (int)((T + lm::kBM - 1) / lm::kBM);
        const int nVt = (int)((V + lm::kBN - 1) / lm::kBN);
        lm::Params p = {};
        p.T = (int)T;
        p.V = (int)V;
        p.Hd = (int)H;
        p.nTt = nTt;
        p.nVt = nVt;
        p.nK = (int)(H / lm::kBK);
        p.ids = ids;
        p.mask = mask;
        p.lse = lse;
        p.cvec = cv;
        p.part = part;
        p.zy = zy;
        p.status = a.status;
        CUtensorMap mH, mW, mWt, mHt;
        if (!lm::make_map(&mH, hidden, H, T, H, lm::kBM) ||
            !lm::make_map(&mW, weight, H, V, H, lm::kBN) ||
            !lm::make_map(&mWt, wt, V, H, L.vp, lm::kN2) ||
            !lm::make_map(&mHt, ht, T, H, L.tp, lm::kN2))
            return CIS_ERR_UNSUPPORTED;
        // FWD
        e = lm::launch_mode<lm::kFwd>(mH, mW, mW, p,
                                      nTt * ((nVt + lm::kFwdGroup - 1) / lm::kFwdGroup), s);
        if (e != cudaSuccess)
            return CIS_ERR_CUDA;
        // per-token scalars
        lm::cis_lmhead_token_kernel<<<(unsigned)((T + 7) / 8), 256, 0, s>>>(a, part, zy, nVt, lse, cv);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return CIS_ERR_CUDA;
        // transposed copies of W and H (K-major operands of dH and dW)
        dim3 tb(32, 8);
        lm::cis_lmhead_transpose_kernel<<<dim3((unsigned)((H + 31) / 32), (unsigned)((V + 31) / 32)),
                                       tb, 0, s>>>(
            static_cast<const __nv_bfloat16 *>(weight), V, H, H, wt, L.vp);
        lm::cis_lmhead_transpose_kernel<<<dim3((unsigned)((H + 31) / 32), (unsigned)((T + 31) / 32)),
                                       tb, 0, s>>>(
            static_cast<const __nv_bfloat16 *>(hidden), T, H, H, ht, L.tp);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return CIS_ERR_CUDA;
        // dH: A = H (token tiles), B = W (vocab tiles), B2 = W^T
        p.out = dhidden;
        p.out_bf16 = grad_dtype == CIS_BF16;
        p.ld_out = H;
        const int R = (int)(H / lm::kN2);
        const bool clustered = lm::use_cluster_grad(H);
        e = clustered ? lm::launch_grad<lm::kDh>(mH, mW, mWt, p, nTt, R, s)
                      : lm::launch_mode<lm::kDh>(mH, mW, mWt, p, nTt * R, s);
        if (e != cudaSuccess)
            return CIS_ERR_CUDA;
        // dW: A = W (vocab tiles), B = H (token tiles), B2 = H^T
        p.out = dweight;
        e = clustered ? lm::launch_grad<lm::kDw>(mW, mH, mHt, p, nVt, R, s)
                      : lm::launch_mode<lm::kDw>(mW, mH, mHt, p, nVt * R, s);
        if (e != cudaSuccess)
            return CIS_ERR_CUDA;
    }
    return launch_reduce(a, stats_out, loss_out, s) == cudaSuccess ? CIS_OK : CIS_ERR_CUDA;
}

}  // extern "C"
