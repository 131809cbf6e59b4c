// cis_lmhead.cu -- the CIS token pass fused with the LM head (sm_103a).
//
// Logits z = H W^T (H: [T, Hd] hidden states, W: [V, Hd] unembedding, bf16)
// are computed tile by tile on the tensor cores (tcgen05.mma, fp32 in TMEM)
// and never written to global memory.  One persistent GEMM kernel, its tile
// epilogue chosen at compile time, serves every pass:
//
//   FWD  z tiles [128 tokens x 256 vocab] -> per token, (max, sum e^{z - max})
//        over the tile's entries j != y, and z_y.
//   TOK  per token: combine the pairs, then log p, the weight (Algorithm 1 /
//        Table 8) and the token loss (Eq. 1) with the same device code as the
//        logits entry points; gives lse_t and c_t.
//   then for each vocabulary chunk [v0, v0 + w):
//   DZ   recompute the chunk's z tiles, form dz = c (softmax - onehot) in bf16
//        and write it as dz [Tp, w];
//   DH   dH (+)= dz W[v0 : v0 + w]   (K = w, fp32 accumulator);
//   DW   dW[v0 : v0 + w] = dz^T H    (K = T);
//   DH and DW of a chunk run as one launch with a balanced schedule.
//
// dz exists one chunk at a time (the chunk width follows the workspace the
// caller gives); z never exists outside TMEM.  Every operand is read where
// it lies: FWD and DZ take H and W K-major; DH takes dz K-major and W
// MN-major (its columns are the output's); DW takes dz and H MN-major (the
// contraction runs over their rows, the tokens).  An MN-major operand tile
// arrives as boxes of 64 MN entries x 64 K rows (128-byte swizzle): the
// canonical MN-major layout of the shared-memory descriptor, with LBO the
// stride between 64-entry MN blocks and SBO the stride between 8-row K
// groups; the instruction descriptor marks it transposed (bits 15, 16).
//
// The GEMM kernel: 128 x 256 tiles, K blocks of 64 (one 128-byte swizzled row
// of bf16), a 4-stage ring of 48 KB (A 16 KB + B 32 KB), two 256-column fp32
// accumulators in TMEM so that the epilogue of one tile overlaps the main loop
// of the next; persistent CTAs take tiles i, i + grid, i + 2 grid, ...  Warp
// roles: warp 0 issues TMA loads, warp 1 issues tcgen05.mma (one thread) and
// owns TMEM, warps 2..9 are the epilogue: two warps per TMEM lane quadrant
// (one tile row per thread), each taking one 128-column half of the tile, so
// that a tile's epilogue fits in the next tile's main loop.  Epilogue stores
// are 32 bytes per thread (one whole sector of its row) where the output is
// 32-byte aligned.  All waits are bounded: a wait that runs out sets
// CIS_ERR_DEVICE_TIMEOUT, and the CTA drains its own loads and MMAs and runs
// to its end, so that TMEM is always released.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <array>
#include <map>
#include <memory>
#include <mutex>
#include <vector>

#include "cis_kernels.h"
#include "cis_tc.cuh"
#include "cis_nvtx.h"

namespace cis {
namespace lm {

constexpr int kBM = 128;                // tile rows (M)
constexpr int kBN = 256;                // tile columns (N)
constexpr int kBK = 64;                 // K block: one 128-byte swizzled row of bf16
constexpr int kStages = 4;
constexpr int kStageA = kBM * kBK * 2;  // 16 KB
constexpr int kStageB = kBN * kBK * 2;  // 32 KB
constexpr int kStageBytes = kStageA + kStageB;
constexpr int kEpiWarps = 8;            // two per TMEM lane quadrant, one per column half
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kHalf = kBN / 2;          // columns per epilogue half
constexpr uint32_t kTmemCols = 2 * kBN;  // two accumulators
constexpr size_t kSmemBytes = (size_t)kStages * kStageBytes + 1024;
constexpr int kMnBox = 64 * kBK * 2;     // one MN-major box: 64 MN entries x 64 K rows, 8 KB
// dz of one chunk takes 2 Tp bytes per vocabulary column; the default chunk
// keeps it within this many bytes.
constexpr int64_t kDefaultChunkBytes = 1ll << 30;

enum Epi { kStats = 0, kDz = 1, kStore = 2, kAccum = 3 };

// OR of `pred` over the epilogue threads (named barrier 1), so that the
// epilogue warps leave their loop together.
__device__ __forceinline__ int __syncthreads_or_epi(int pred)
{
    int r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.s32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\tselp.s32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(pred), "n"(kEpiThreads)
        : "memory");
    return r;
}

// 32-byte global accesses (sm_100 and later): one full sector per thread, so
// that a warp's store into 32 rows writes 32 whole sectors.  The address must
// be 32-byte aligned.
__device__ __forceinline__ void st_v8(void *p, const uint32_t *w)
{
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]),
                 "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}
// The same with the streaming (evict-first) hint.
__device__ __forceinline__ void st_v8_cs(void *p, const uint32_t *w)
{
    asm volatile("st.global.cs.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]),
                 "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}
__device__ __forceinline__ void ld_v8(const void *p, float *r)
{
    asm volatile("ld.global.v8.f32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=f"(r[0]), "=f"(r[1]), "=f"(r[2]), "=f"(r[3]), "=f"(r[4]), "=f"(r[5]),
                   "=f"(r[6]), "=f"(r[7])
                 : "l"(p));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

// One launch of the GEMM kernel: C[M, N] = A[M, K] B[N, K]^T over tiles
// (m, n) of 128 x 256, with TMA coordinates offset by a_row0 / b_row0 along
// M / N and a_k0 / b_k0 along K.  Whether an operand's tensor map runs along
// M / N in its inner dimension (MN-major) rather than along K is a template
// parameter of the kernel (A_MN, B_MN).
struct GemmArgs {
    int nMt, nNt, nK;
    int raster_n;  // 1: tile i -> (m = i % nMt, n = i / nMt); 0: (m = i / nNt, n = i % nNt)
    int a_row0, a_k0, b_row0, b_k0;
    // kStats, kDz: rows are tokens, columns vocabulary entries col0 + n 256 + c
    int T, V, col0;
    const int32_t *ids;
    const float *lse, *cvec;
    float2 *part;     // kStats: [2 nNt, T] (max, sum) over j != y per 128-column half
    float *part_u;    // kStats: [2 nNt, T] sum e^{z - max} (z - max), or null (no entropy)
    float *zy;        // kStats: z at the sampled token
    uint16_t *dz;     // kDz: bf16 [Tp, ld_dz], column = chunk-local vocabulary index
    int64_t ld_dz;
    // kStore, kAccum: rows m 128 + r < rows_valid of out [., ld_out]; out_v8:
    // out is 32-byte aligned (32-byte accesses), else 16-byte ones
    void *out;
    int out_bf16, rows_valid, out_v8;
    int64_t ld_out;
    int32_t *status;
};

struct Barriers {
    uint64_t full[kStages], empty[kStages];
    uint64_t accfull[2], accempty[2];
    uint64_t done;
};

// A wait that runs out marks the CTA (shared flag) and the grid (status word)
// as aborted: the roles then stop waiting and run to the end, so a broken
// pipeline costs one bounded wait per role instead of one per tile.  on()
// reads the shared flag only; the status word (global memory, one L2 round
// trip) is consulted inside waits that are already taking long.
struct Abort {
    volatile int *local;
    int32_t *status;
    __device__ __forceinline__ bool on() const { return *local != 0; }
    // False once the CTA has aborted (now or earlier): the caller stops.  A
    // phase that has already completed returns at the first poll, without
    // reading the flag (the MMA thread waits once per stage, and every
    // instruction of its loop counts).
    __device__ __forceinline__ bool wait(uint64_t *bar, uint32_t parity) const
    {
        if (tc::bar_try(bar, parity))
            return true;
        if (*local)
            return false;
        if (!tc::bar_wait(bar, parity, status)) {
            *local = 1;
            set_status(status, kStatusTimeout);
            return false;
        }
        return true;
    }
};

// Tile order.  raster_n: groups of kGroupN vocabulary tiles, token tiles
// inside a group, so that the tiles in flight at one time (one per SM) share
// about 152 / kGroupN token tiles of A and kGroupN tiles of B in L2;
// otherwise m-major (the nNt column blocks of a row block together).  16 and
// 32 measured 0.5% faster than 8 on the full-size call, 4 slower.
constexpr int kGroupN = 16;
__device__ __forceinline__ void tile_mn(const GemmArgs &g, int i, int &m, int &n)
{
    if (g.raster_n) {
        const int per = kGroupN * g.nMt;
        const int grp = i / per, j = i - grp * per;
        const int n0 = grp * kGroupN;
        const int gw = g.nNt - n0 < kGroupN ? g.nNt - n0 : kGroupN;
        m = j / gw;
        n = n0 + (j - m * gw);
    } else {
        m = i / g.nNt;
        n = i - m * g.nNt;
    }
}
// Work unit u of a launch: a tile, or with MC (2-CTA clusters) a pair of
// tiles in row tiles 2 mp and 2 mp + 1 of one column tile, CTA `rank` of the
// cluster taking row tile 2 mp + rank.  The pair shares its B tile: each CTA
// loads one half of it and multicasts it to both.  With an odd number of row
// tiles the last pair's second tile lies past the rows (m == nMt): its CTA
// still loads and multicasts its half of B, and its A reads as zeros, but its
// epilogue writes nothing.
template <bool MC> __host__ __device__ __forceinline__ int n_units(const GemmArgs &g)
{
    return MC ? ((g.nMt + 1) >> 1) * g.nNt : g.nMt * g.nNt;
}
template <bool MC>
__device__ __forceinline__ void unit_mn(const GemmArgs &g, int u, int rank, int &m, int &n)
{
    if (!MC) {
        tile_mn(g, u, m, n);
        return;
    }
    GemmArgs gp = g;
    gp.nMt = (g.nMt + 1) >> 1;  // the pairs' own grid of (row pair, column) units
    int mp;
    tile_mn(gp, u, mp, n);
    m = 2 * mp + rank;
}

// Where the producer, or the MMA thread, is in the ring of stages.
struct Ring {
    int stage = 0;
    uint32_t phase = 0;
    __device__ __forceinline__ void next()
    {
        if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
        }
    }
};

// The producer's loads for tile (m, n): nK stages.  `used` and `last` record
// per stage whether it was ever loaded and the parity of its last load, for
// the drain before the CTA leaves.  Returns early once the CTA aborted.
template <bool A_MN, bool B_MN, bool MC>
__device__ __forceinline__ void load_tile(const CUtensorMap &tmA, const CUtensorMap &tmB,
                                          const GemmArgs &g, int m, int n, int rank,
                                          uint8_t *ring, Barriers &bars, const Abort &ab,
                                          Ring &p, uint32_t &used, uint32_t &last)
{
    for (int kb = 0; kb < g.nK; ++kb) {
        if (!ab.wait(&bars.empty[p.stage], p.phase ^ 1))
            return;
        uint64_t *full = &bars.full[p.stage];
        tc::bar_expect_tx(full, kStageBytes);
        used |= 1u << p.stage;
        last = (last & ~(1u << p.stage)) | (p.phase << p.stage);
        uint8_t *st = ring + p.stage * kStageBytes;
        const int ka = g.a_k0 + kb * kBK, kbb = g.b_k0 + kb * kBK;
        if (A_MN) {  // MN-major: boxes of 64 rows of M along the inner dimension
#pragma unroll
            for (int i = 0; i < kBM / 64; ++i)
                tc::tma_load_2d(st + i * kMnBox, &tmA, g.a_row0 + m * kBM + 64 * i, ka, full);
        } else {
            tc::tma_load_2d(st, &tmA, ka, g.a_row0 + m * kBM, full);
        }
        if (MC) {  // this CTA's half of B, to both CTAs
            if (B_MN) {
#pragma unroll
                for (int i = 2 * rank; i < 2 * rank + 2; ++i)
                    tc::tma_load_2d_mc(st + kStageA + i * kMnBox, &tmB,
                                       g.b_row0 + n * kBN + 64 * i, kbb, full, 0x3);
            } else {
                tc::tma_load_2d_mc(st + kStageA + rank * (kStageB / 2), &tmB, kbb,
                                   g.b_row0 + n * kBN + rank * (kBN / 2), full, 0x3);
            }
        } else if (B_MN) {
#pragma unroll
            for (int i = 0; i < kBN / 64; ++i)
                tc::tma_load_2d(st + kStageA + i * kMnBox, &tmB, g.b_row0 + n * kBN + 64 * i,
                                kbb, full);
        } else {
            tc::tma_load_2d(st + kStageA, &tmB, kbb, g.b_row0 + n * kBN, full);
        }
        p.next();
    }
}

// The MMAs of one tile into the accumulator at TMEM column d: nK stages of
// four K=16 steps.  Returns early once the CTA aborted.
template <bool A_MN, bool B_MN, bool MC>
__device__ __forceinline__ void mma_tile(const GemmArgs &g, uint32_t d, uint8_t *ring,
                                         Barriers &bars, const Abort &ab, Ring &p)
{
    constexpr uint32_t kId =
        tc::idesc_bf16(kBM, kBN) | ((uint32_t)A_MN << 15) | ((uint32_t)B_MN << 16);
    // a K step of 16: 32 bytes along a K-major row, 16 rows (2 K groups) of an
    // MN-major tile
    constexpr uint32_t a_step = A_MN ? 16 * 128 : 32, b_step = B_MN ? 16 * 128 : 32;
    // Descriptors of stage 0's A and B tiles; a stage, and a K step inside
    // it, only move the start address, which sits in the low bits (address
    // >> 4, below 2^14 for any shared-memory address), so they are added
    // there.
    const uint32_t s0 = tc::smem_addr(ring);
    const uint64_t da0 = A_MN ? tc::desc_sw128_mn(s0, kMnBox) : tc::desc_sw128(s0);
    const uint64_t db0 =
        B_MN ? tc::desc_sw128_mn(s0 + kStageA, kMnBox) : tc::desc_sw128(s0 + kStageA);
    for (int kb = 0; kb < g.nK; ++kb) {
        if (!ab.wait(&bars.full[p.stage], p.phase))
            return;
        tc::fence_after_sync();
        const uint64_t so = (uint64_t)((p.stage * kStageBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
            tc::mma_bf16(d, da0 + so + (kk * a_step >> 4), db0 + so + (kk * b_step >> 4), kId,
                         (kb | kk) != 0);
        if (MC)  // the stage is free in this CTA and in the peer
            tc::mma_commit_mc(&bars.empty[p.stage], 0x3);
        else
            tc::mma_commit(&bars.empty[p.stage]);
        p.next();
    }
}

// The epilogue of one tile for one thread: TMEM lane r (tile row r of row
// tile m), column half `half` of column tile n; taddr addresses the lane's
// first column of the tile's accumulator.
template <int EPI>
__device__ __forceinline__ void epilogue_tile(const GemmArgs &g, uint32_t taddr, int m, int n,
                                              int r, int half)
{
    const int cbeg = half * kHalf;
    if (EPI == kStats) {
        const int row = m * kBM + r;  // token
        const int y_r = row < g.T ? g.ids[row] : -1;
        const bool ent = g.part_u != nullptr;
        float mx = -INFINITY, s = 0.0f, u = 0.0f, zyv = 0.0f;
        bool got_y = false;
        for (int c0 = cbeg; c0 < cbeg + kHalf; c0 += 32) {
            float v[32];
            tc::tmem_ld32(taddr + c0, v);
            const int base = g.col0 + n * kBN + c0;
            if (y_r >= base && y_r < base + 32) {
#pragma unroll
                for (int q = 0; q < 32; ++q)
                    if (base + q == y_r)
                        zyv = v[q];
                got_y = true;
            }
            float cm = -INFINITY;
#pragma unroll
            for (int q = 0; q < 32; ++q) {
                const int col = base + q;
                v[q] = (col == y_r || col >= g.V) ? -INFINITY : v[q];
                cm = fmaxf(cm, v[q]);
            }
            if (cm > mx) {
                if (mx == -INFINITY) {
                    s = 0.0f;
                    u = 0.0f;
                } else {
                    const float d = mx - cm, f = ex2_ftz(d * kLog2e);
                    u = fmaf(d, s, u) * f;
                    s *= f;
                }
                mx = cm;
            }
            if (mx != -INFINITY) {
                float a = 0.0f, au = 0.0f;
                if (ent) {  // the entropy term, e (z - max)
#pragma unroll
                    for (int q = 0; q < 32; ++q) {
                        const float d = v[q] - mx, e = ex2_ftz(d * kLog2e);
                        a += e;
                        au = fmaf(e, fmaxf(d, -1024.0f), au);
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < 32; ++q)
                        a += ex2_ftz((v[q] - mx) * kLog2e);
                }
                s += a;
                u += au;
            }
        }
        if (row < g.T) {  // one (max, sum) per 128-column half
            const int64_t pi = (int64_t)(2 * n + half) * g.T + row;
            g.part[pi] = make_float2(mx, s);
            if (ent)
                g.part_u[pi] = u;
            if (got_y)
                g.zy[row] = zyv;
        }
    } else if (EPI == kDz) {
        const int row = m * kBM + r;  // token; rows up to Tp are allocated
        const bool live = row < g.T;
        // tokens with c = 0 (masked, clipped, past T) give 0 without
        // touching the exponential (their lse is a placeholder)
        const float c_r = live ? g.cvec[row] : 0.0f;
        const float lse_r = live ? g.lse[row] : 0.0f;
        const int y_r = live ? g.ids[row] : -1;
        const int cl0 = n * kBN;  // chunk-local column of the tile
        for (int c0 = cbeg; c0 < cbeg + kHalf; c0 += 32) {
            float v[32];
            tc::tmem_ld32(taddr + c0, v);
            const int gc0 = g.col0 + cl0 + c0;  // vocabulary index of v[0]
            uint32_t w[16];
#pragma unroll
            for (int q = 0; q < 32; q += 2) {
                float d[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int gc = gc0 + q + h;
                    d[h] = (gc < g.V && c_r != 0.0f)
                               ? c_r * ex2_ftz((v[q + h] - lse_r) * kLog2e) -
                                     (gc == y_r ? c_r : 0.0f)
                               : 0.0f;
                }
                w[q >> 1] = pack_bf16x2(d[0], d[1]);
            }
            // 64 bytes of the row in two full-sector stores (read back by
            // the next two launches, DH and DW)
            uint16_t *drow = g.dz + (int64_t)row * g.ld_dz + cl0 + c0;
            st_v8_cs(drow, w);
            st_v8_cs(drow + 16, w + 8);
        }
    } else {
        const int lr = m * kBM + r;  // row of the output block
        const bool live = lr < g.rows_valid;
        const int64_t o = (int64_t)lr * g.ld_out + (int64_t)n * kBN;
        for (int c0 = cbeg; c0 < cbeg + kHalf; c0 += 32) {
            float v[32];
            tc::tmem_ld32(taddr + c0, v);
            if (!live)
                continue;
            if (g.out_bf16) {
                uint32_t w[16];
#pragma unroll
                for (int q = 0; q < 16; ++q)
                    w[q] = pack_bf16x2(v[2 * q], v[2 * q + 1]);
                uint16_t *dst = reinterpret_cast<uint16_t *>(g.out) + o + c0;
                if (g.out_v8) {  // streaming: outputs are not re-read here
                    st_v8_cs(dst, w);
                    st_v8_cs(dst + 16, w + 8);
                } else {
                    uint4 *d4 = reinterpret_cast<uint4 *>(dst);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        __stcs(d4 + q, make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2],
                                                  w[4 * q + 3]));
                }
            } else if (g.out_v8) {
                float *dst = reinterpret_cast<float *>(g.out) + o + c0;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float x[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        x[e] = v[8 * q + e];
                    if (EPI == kAccum) {
                        float old[8];
                        ld_v8(dst + 8 * q, old);
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            x[e] += old[e];
                    }
                    st_v8_cs(dst + 8 * q, reinterpret_cast<const uint32_t *>(x));
                }
            } else {
                float4 *dst = reinterpret_cast<float4 *>(
                    reinterpret_cast<float *>(g.out) + o + c0);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    float4 x = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2],
                                           v[4 * q + 3]);
                    if (EPI == kAccum) {
                        const float4 old = dst[q];
                        x.x += old.x;
                        x.y += old.y;
                        x.z += old.z;
                        x.w += old.w;
                    }
                    __stcs(dst + q, x);
                }
            }
        }
    }
}

// Shared memory of a GEMM CTA besides the ring.
struct GemmShared {
    Barriers bars;
    uint32_t tmem_base;
    int aborted;
};

// Barriers, TMEM and (MC) the cluster, before the roles start.
template <bool MC> __device__ __forceinline__ void gemm_setup(GemmShared &sh, int warp)
{
    if (threadIdx.x == 0) {
        sh.aborted = 0;
        for (int s = 0; s < kStages; ++s) {
            tc::bar_init(&sh.bars.full[s], 1);
            // with MC both CTAs' MMAs release a stage: the peer's multicast
            // writes into this CTA's copy of it
            tc::bar_init(&sh.bars.empty[s], MC ? 2 : 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::bar_init(&sh.bars.accfull[b], 1);
            tc::bar_init(&sh.bars.accempty[b], kEpiThreads);
        }
        tc::bar_init(&sh.bars.done, 1);
        tc::bar_init_fence();
    }
    if (warp == 1)
        tc::tmem_alloc(&sh.tmem_base, kTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    if (MC)
        tc::cluster_sync();  // the peer's barriers exist before anything signals them
    tc::fence_after_sync();
}

// The producer's last step: no load may still be landing when the CTA leaves.
__device__ __forceinline__ void drain_loads(Barriers &bars, uint32_t used, uint32_t last)
{
    for (int s = 0; s < kStages; ++s)
        if (used & (1u << s))
            tc::bar_wait(&bars.full[s], (last >> s) & 1);
}

// The MMA thread's last step: every MMA of this CTA is done before TMEM is
// released.
__device__ __forceinline__ void drain_mmas(Barriers &bars)
{
    tc::mma_commit(&bars.done);
    tc::bar_wait(&bars.done, 0);
}

// Every thread, after its role: TMEM freed once nothing uses it; with MC
// neither CTA leaves while the other may still signal its barriers.
template <bool MC> __device__ __forceinline__ void gemm_teardown(GemmShared &sh, int warp)
{
    __syncwarp();
    tc::fence_before_sync();
    __syncthreads();
    if (MC) {
        tc::cluster_sync();
        // after a wait ran out the peer may have issued one more multicast
        // into a stage this CTA no longer waits for: give it time to land
        if (sh.aborted && threadIdx.x == 0) {
            const long long t0 = clock64();
            while (clock64() - t0 < (1ll << 20)) {
            }
        }
        __syncthreads();
    }
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(sh.tmem_base, kTmemCols);
    }
}

// The epilogue warps' part of one tile: wait for its accumulator, drain it,
// hand it back.  Warps 2..9: TMEM lane quadrant warp % 4 (one tile row per
// thread), column half (warp - 2) / 4 of the 256-column tile.
template <int EPI, bool MC>
__device__ __forceinline__ void epilogue_unit(const GemmArgs &g, int m, int n, int i,
                                              uint32_t tmem, int warp, int lane, Barriers &bars,
                                              const Abort &ab)
{
    const int lg = warp & 3;
    const int half = (warp - 2) >> 2;
    const uint32_t lane_off = (uint32_t)(lg * 32) << 16;
    const int acc = i & 1;
    ab.wait(&bars.accfull[acc], (i >> 1) & 1);
    tc::fence_after_sync();
    // with MC, the padding tile of an odd row count has nothing to write
    if (!(MC && m >= g.nMt))
        epilogue_tile<EPI>(g, tmem + lane_off + acc * kBN, m, n, lg * 32 + lane, half);
    tc::fence_before_sync();
    tc::bar_arrive(&bars.accempty[acc]);
}

// The MMA thread's part of one tile: a free accumulator, the tile's MMAs,
// then the accumulator handed to the epilogue.
template <bool A_MN, bool B_MN, bool MC>
__device__ __forceinline__ void mma_unit(const GemmArgs &g, int i, uint32_t tmem, uint8_t *ring,
                                         Barriers &bars, const Abort &ab, Ring &p)
{
    const int acc = i & 1;
    ab.wait(&bars.accempty[acc], ((i >> 1) & 1) ^ 1);
    tc::fence_after_sync();
    mma_tile<A_MN, B_MN, MC>(g, tmem + acc * kBN, ring, bars, ab, p);
    tc::mma_commit(&bars.accfull[acc]);
}

template <int EPI, bool A_MN, bool B_MN, bool MC>
__global__ void __launch_bounds__(kThreads, 1)
    cis_lmhead_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                           const __grid_constant__ CUtensorMap tmB, const GemmArgs g)
{
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t *ring = dsm + ((1024 - (tc::smem_addr(dsm) & 1023)) & 1023);
    __shared__ __align__(8) GemmShared sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nUnits = n_units<MC>(g);
    const int rank = MC ? (int)tc::cluster_ctarank() : 0;
    const int unit0 = MC ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const int ustep = MC ? (int)(gridDim.x >> 1) : (int)gridDim.x;

    gemm_setup<MC>(sh, warp);
    const uint32_t tmem = sh.tmem_base;
    const Abort ab{&sh.aborted, g.status};

    if (warp == 0) {
        if (lane == 0) {  // producer
            Ring p;
            uint32_t used = 0, last = 0;
            for (int u = unit0; u < nUnits && !ab.on(); u += ustep) {
                int m, n;
                unit_mn<MC>(g, u, rank, m, n);
                load_tile<A_MN, B_MN, MC>(tmA, tmB, g, m, n, rank, ring, sh.bars, ab, p, used,
                                          last);
            }
            drain_loads(sh.bars, used, last);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // MMA issue
            Ring p;
            int i = 0;
            for (int u = unit0; u < nUnits && !ab.on(); u += ustep, ++i)
                mma_unit<A_MN, B_MN, MC>(g, i, tmem, ring, sh.bars, ab, p);
            drain_mmas(sh.bars);
        }
    } else {  // epilogue
        int i = 0;
        for (int u = unit0; u < nUnits; u += ustep, ++i) {
            if (__syncthreads_or_epi(ab.on()))
                break;
            int m, n;
            unit_mn<MC>(g, u, rank, m, n);
            epilogue_unit<EPI, MC>(g, m, n, i, tmem, warp, lane, sh.bars, ab);
        }
    }
    gemm_teardown<MC>(sh, warp);
}

// The dH and dW GEMMs of one vocabulary chunk in one launch.  Launched one
// after the other, each ends in a partial wave: dH has 512 pair units of 512 K
// blocks for 76 clusters (6.7 waves), dW 1024 of 256 (13.5 waves).  Here
// every group (a cluster with MC, else a CTA) works through its own list of
// units from both GEMMs: a greedy schedule made on the host, which hands the
// units out in order (all of dH, then dW) to the group that frees up first, by
// their K blocks.  The lists are kernel parameters.
constexpr int kMaxSchedGroups = 160;
constexpr int kMaxSchedUnits = 4096;
constexpr uint16_t kSchedSecond = 0x8000;  // a unit of the second GEMM
struct DualSched {
    uint16_t off[kMaxSchedGroups + 1];  // group c takes unit[off[c]] .. unit[off[c + 1] - 1]
    uint16_t unit[kMaxSchedUnits];      // unit index, | kSchedSecond for the second GEMM
};

// GEMM 0: dH (+)= dz W_c (A = dz K-major, B = W MN-major, EPI0 = kStore on
// the first chunk, kAccum after); GEMM 1: dW_c = dz^T H (A = dz MN-major,
// B = H MN-major, kStore).
template <int EPI0, bool MC>
__global__ void __launch_bounds__(kThreads, 1)
    cis_lmhead_dual_kernel(const __grid_constant__ CUtensorMap tmA0,
                           const __grid_constant__ CUtensorMap tmB0,
                           const __grid_constant__ CUtensorMap tmA1,
                           const __grid_constant__ CUtensorMap tmB1, const GemmArgs g0,
                           const GemmArgs g1, const __grid_constant__ DualSched sc)
{
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t *ring = dsm + ((1024 - (tc::smem_addr(dsm) & 1023)) & 1023);
    __shared__ __align__(8) GemmShared sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = MC ? (int)tc::cluster_ctarank() : 0;
    const int grp = MC ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const int j0 = sc.off[grp], j1 = sc.off[grp + 1];

    gemm_setup<MC>(sh, warp);
    const uint32_t tmem = sh.tmem_base;
    const Abort ab{&sh.aborted, g0.status};

    if (warp == 0) {
        if (lane == 0) {  // producer
            Ring p;
            uint32_t used = 0, last = 0;
            for (int j = j0; j < j1 && !ab.on(); ++j) {
                const int u = sc.unit[j];
                int m, n;
                if (u & kSchedSecond) {
                    unit_mn<MC>(g1, u & ~kSchedSecond, rank, m, n);
                    load_tile<true, true, MC>(tmA1, tmB1, g1, m, n, rank, ring, sh.bars, ab, p,
                                              used, last);
                } else {
                    unit_mn<MC>(g0, u, rank, m, n);
                    load_tile<false, true, MC>(tmA0, tmB0, g0, m, n, rank, ring, sh.bars, ab, p,
                                               used, last);
                }
            }
            drain_loads(sh.bars, used, last);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // MMA issue
            Ring p;
            for (int j = j0; j < j1 && !ab.on(); ++j) {
                if (sc.unit[j] & kSchedSecond)
                    mma_unit<true, true, MC>(g1, j - j0, tmem, ring, sh.bars, ab, p);
                else
                    mma_unit<false, true, MC>(g0, j - j0, tmem, ring, sh.bars, ab, p);
            }
            drain_mmas(sh.bars);
        }
    } else {  // epilogue
        for (int j = j0; j < j1; ++j) {
            if (__syncthreads_or_epi(ab.on()))
                break;
            const int u = sc.unit[j];
            int m, n;
            if (u & kSchedSecond) {
                unit_mn<MC>(g1, u & ~kSchedSecond, rank, m, n);
                epilogue_unit<kStore, MC>(g1, m, n, j - j0, tmem, warp, lane, sh.bars, ab);
            } else {
                unit_mn<MC>(g0, u, rank, m, n);
                epilogue_unit<EPI0, MC>(g0, m, n, j - j0, tmem, warp, lane, sh.bars, ab);
            }
        }
    }
    gemm_teardown<MC>(sh, warp);
}

// dst[i] = bf16(src[i]) (round to nearest even)
__global__ void cis_lmhead_to_bf16_kernel(const float *src, uint16_t *dst, int64_t n)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = __bfloat16_as_ushort(__float2bfloat16_rn(src[i]));
}

// Per token: combine the FWD pairs, then log p, weight, loss, c_t (one warp).
__global__ void cis_lmhead_token_kernel(const PassArgs a, const float2 *part, const float *part_u,
                                        const float *zy, int nVt, float *lse_out, float *c_out)
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
            if (a.entropy_out) a.entropy_out[t] = lp;
            lse_out[t] = 0.0f;
            c_out[t] = 0.0f;
        }
        return;
    }
    MaxSum o{-INFINITY, 0.0f};
    MaxSumU ou{-INFINITY, 0.0f, 0.0f};
    if (part_u) {
        for (int j = lane; j < nVt; j += 32) {
            const float2 q = part[(int64_t)j * a.T + t];
            ou = msu_combine(ou, MaxSumU{q.x, q.y, part_u[(int64_t)j * a.T + t]});
        }
        ou = warp_msu(ou);
        o = MaxSum{ou.m, ou.s};
    } else {
        for (int j = lane; j < nVt; j += 32) {
            const float2 q = part[(int64_t)j * a.T + t];
            o = ms_combine(o, MaxSum{q.x, q.y});
        }
        o = warp_ms(o);
    }
    if (lane == 0) {
        const RowScalars rs = row_scalars(o, zy[t]);
        if (part_u && a.entropy_out)
            a.entropy_out[t] = row_entropy(ou, zy[t], rs.lp);
        if (is_seq_mode(a.P.mode) && a.w_in == nullptr) {
            // sequence operator, first sweep: log p only (the response's
            // weight needs every token of the response)
            if (a.lp64_out)
                a.lp64_out[t] = rs.lp64();
            return;
        }
        const bool has_old = a.lp_old != nullptr;
        const float lold = has_old ? a.lp_old[t] : 0.0f;
        TokenWeight tw = token_weight(has_old ? lold : rs.lp, has_old ? 0.0f : rs.lp_lo,
                                      a.lp_inf[t], a.P, has_old ? -1.0f : rs.omp);
        if (a.w_in) {
            tw.w = a.w_in[t];
            tw.trunc = a.trunc_in[t];
        }
        const TokenLoss tl =
            token_loss(rs.lp, rs.lp_lo, has_old, lold, a.adv[t], a.scale[t], tw.w, a.P);
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

template <int EPI, bool A_MN = false, bool B_MN = false>
cudaError_t launch_gemm(const CUtensorMap &a, const CUtensorMap &b, const GemmArgs &g,
                        cudaStream_t s)
{
    const int tiles = g.nMt * g.nNt;
    if (tiles <= 0 || g.nK <= 0)
        return cudaSuccess;
    auto k = cis_lmhead_gemm_kernel<EPI, A_MN, B_MN, false>;
    const size_t smem = kSmemBytes;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess)
        return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int grid = tiles < sms ? tiles : sms;
    k<<<grid, kThreads, smem, s>>>(a, b, g);
    return cudaGetLastError();
}

// The same GEMM on 2-CTA clusters that share each B tile (multicast).  `b`
// must be a map whose box is half of B's tile: 128 rows for a K-major B, the
// 64-wide boxes of an MN-major one.
template <int EPI, bool A_MN = false, bool B_MN = false>
cudaError_t launch_gemm_mc(const CUtensorMap &a, const CUtensorMap &b, const GemmArgs &g,
                           cudaStream_t s)
{
    const int units = ((g.nMt + 1) / 2) * g.nNt;
    if (units <= 0 || g.nK <= 0)
        return cudaSuccess;
    auto k = cis_lmhead_gemm_kernel<EPI, A_MN, B_MN, true>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(2);
    int clusters = 0;
    if ((e = cudaOccupancyMaxActiveClusters(&clusters, k, &cfg)) != cudaSuccess)
        return e;
    if (clusters <= 0)
        return cudaErrorNotSupported;
    cfg.gridDim = dim3((unsigned)(2 * (units < clusters ? units : clusters)));
    e = cudaLaunchKernelEx(&cfg, k, a, b, g);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// The groups that run at once: co-resident 2-CTA clusters (MC), else SMs.
template <typename K> cudaError_t resident_groups(K kern, bool mc, int *groups)
{
    int dev = 0, sms = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    if (!mc) {
        *groups = sms;
        return cudaSuccess;
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if ((e = cudaOccupancyMaxActiveClusters(groups, kern, &cfg)) != cudaSuccess)
        return e;
    return *groups > 0 ? cudaSuccess : cudaErrorNotSupported;
}

// The greedy schedule of a dual launch: units n0 of GEMM 0 (c0 K blocks
// each), then n1 of GEMM 1 (c1 each), each to the group whose list ends
// earliest (ties: the lowest group).  The units of one GEMM go out in order,
// so the groups at work at any time hold neighbouring units, which share their
// operands in L2.  False if it does not fit a DualSched.
static bool make_dual_sched(int n0, int c0, int n1, int c1, int groups, DualSched *s)
{
    if (groups < 1 || groups > kMaxSchedGroups || n0 + n1 > kMaxSchedUnits || n0 < 0 ||
        n1 < 0 || n0 >= kSchedSecond || n1 >= kSchedSecond)
        return false;
    std::vector<int64_t> end(groups, 0);
    std::vector<std::vector<uint16_t>> lists(groups);
    for (int j = 0; j < n0 + n1; ++j) {
        int best = 0;
        for (int c = 1; c < groups; ++c)
            if (end[c] < end[best])
                best = c;
        const bool second = j >= n0;
        end[best] += second ? c1 : c0;
        lists[best].push_back(second ? (uint16_t)((j - n0) | kSchedSecond) : (uint16_t)j);
    }
    int k = 0;
    for (int c = 0; c < groups; ++c) {
        s->off[c] = (uint16_t)k;
        for (uint16_t u : lists[c])
            s->unit[k++] = u;
    }
    for (int c = groups; c <= kMaxSchedGroups; ++c)
        s->off[c] = (uint16_t)k;
    return true;
}

// One launch of cis_lmhead_dual_kernel over both GEMMs' units; false (and no
// launch) if the schedule does not fit, so that the caller launches them one
// after the other.  Schedules are kept per shape: a call makes two (full
// chunks, the last chunk).
template <int EPI0, bool MC>
cudaError_t launch_dual(const CUtensorMap &a0, const CUtensorMap &b0, const GemmArgs &g0,
                        const CUtensorMap &a1, const CUtensorMap &b1, const GemmArgs &g1,
                        cudaStream_t s, bool *launched)
{
    *launched = false;
    auto k = cis_lmhead_dual_kernel<EPI0, MC>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    int groups = 0;
    if ((e = resident_groups(k, MC, &groups)) != cudaSuccess)
        return e;
    const int n0 = MC ? n_units<true>(g0) : n_units<false>(g0);
    const int n1 = MC ? n_units<true>(g1) : n_units<false>(g1);
    if (g0.nK <= 0 || g1.nK <= 0 || n0 <= 0 || n1 <= 0)
        return cudaSuccess;
    static std::mutex mu;
    static std::map<std::array<int, 5>, std::unique_ptr<DualSched>> cache;
    std::unique_ptr<DualSched> sc(new DualSched());  // this call's copy
    {
        std::lock_guard<std::mutex> lock(mu);
        const std::array<int, 5> key = {n0, g0.nK, n1, g1.nK, groups};
        auto it = cache.find(key);
        if (it == cache.end()) {
            std::unique_ptr<DualSched> p(new DualSched());
            if (!make_dual_sched(n0, g0.nK, n1, g1.nK, groups, p.get()))
                return cudaSuccess;
            if (cache.size() >= 64)  // a process that sees many shapes keeps the last few
                cache.clear();
            it = cache.emplace(key, std::move(p)).first;
        }
        *sc = *it->second;
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = MC ? 2 : 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(groups * (MC ? 2 : 1)));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = MC ? 1 : 0;
    e = cudaLaunchKernelEx(&cfg, k, a0, b0, a1, b1, g0, g1, *sc);
    if (e == cudaSuccess)
        e = cudaGetLastError();
    *launched = e == cudaSuccess;
    return e;
}

// Whether a chunk's dH and dW run as one launch (CIS_LMHEAD_DUAL=0: one after
// the other; the results are the same either way).
static bool dual_on()
{
    const char *e = getenv("CIS_LMHEAD_DUAL");
    return !(e && e[0] == '0');
}

// Which GEMMs run on 2-CTA multicast clusters: a bit mask over FWD (1), DZ
// (2), DH (4) and DW (8); all by default, CIS_LMHEAD_MC overrides it.  The
// results are bit for bit the same either way: each tile's MMAs and epilogue
// are unchanged, only where half of B comes from differs.
static int mc_mask()
{
    const char *e = getenv("CIS_LMHEAD_MC");
    return e && e[0] ? (int)strtol(e, nullptr, 0) & 15 : 15;
}

}  // namespace lm

// Workspace of cis_lmhead_fused, after the token-pass layout of ws_layout(T),
// for vocabulary chunks of Vc columns (a multiple of 256).
struct LmLayout {
    WsLayout base;
    size_t lse, c, zy, part, part_u, dh, dz, total;
    int64_t Tp, Vc;
};

static int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

LmLayout lm_layout(int64_t T, int64_t V, int64_t Hd, int64_t Vc)
{
    auto up = [](size_t x) { return (x + 1023) / 1024 * 1024; };
    LmLayout L;
    L.base = ws_layout(T);
    const int64_t nVt = (V + lm::kBN - 1) / lm::kBN;
    L.Tp = round_up(T, lm::kBM);
    L.Vc = Vc;
    size_t o = up(L.base.total);
    L.lse = o;
    o = up(o + 4 * (size_t)T);
    L.c = o;
    o = up(o + 4 * (size_t)T);
    L.zy = o;
    o = up(o + 4 * (size_t)T);
    L.part = o;  // one (max, sum) per 128-column half tile
    o = up(o + 8 * (size_t)T * (size_t)(2 * nVt));
    L.part_u = o;
    o = up(o + 4 * (size_t)T * (size_t)(2 * nVt));
    L.dh = o;
    o = up(o + 4 * (size_t)T * (size_t)Hd);
    L.dz = o;
    o = up(o + 2 * (size_t)L.Tp * (size_t)Vc);
    L.total = o;
    return L;
}

// The widest chunk: every vocabulary column at once.
static int64_t max_chunk(int64_t V) { return round_up(V, lm::kBN); }

// The default chunk: dz within kDefaultChunkBytes.
static int64_t default_chunk(int64_t T, int64_t V)
{
    const int64_t Tp = round_up(T, lm::kBM);
    int64_t c = Tp > 0 ? lm::kDefaultChunkBytes / (2 * Tp) / lm::kBN * lm::kBN : max_chunk(V);
    if (c < lm::kBN)
        c = lm::kBN;
    return c < max_chunk(V) ? c : max_chunk(V);
}

// The widest chunk whose layout fits in `bytes`; 0 if not even 256 columns do.
static int64_t chunk_for_bytes(int64_t T, int64_t V, int64_t Hd, size_t bytes)
{
    const size_t fixed = lm_layout(T, V, Hd, 0).total;
    if (bytes < fixed)
        return 0;
    const size_t per = 2 * (size_t)round_up(T, lm::kBM);
    int64_t c = per > 0 ? (int64_t)((bytes - fixed) / per) / lm::kBN * lm::kBN : max_chunk(V);
    if (c > max_chunk(V))
        c = max_chunk(V);
    while (c >= lm::kBN && lm_layout(T, V, Hd, c).total > bytes)
        c -= lm::kBN;
    return c >= lm::kBN ? c : 0;
}

}  // namespace cis

using namespace cis;

extern "C" {

CIS_API cis_status_t cis_lmhead_workspace_size(int64_t T, int64_t V, int64_t H, size_t *bytes)
{
    if (bytes == nullptr || T < 0 || V <= 0 || H <= 0)
        return CIS_ERR_INVALID_ARG;
    *bytes = lm_layout(T, V, H, default_chunk(T, V)).total;
    return CIS_OK;
}

CIS_API cis_status_t cis_lmhead_workspace_size_chunk(int64_t T, int64_t V, int64_t H,
                                                     int64_t chunk, size_t *bytes)
{
    if (bytes == nullptr || T < 0 || V <= 0 || H <= 0 || chunk <= 0 || chunk % lm::kBN != 0)
        return CIS_ERR_INVALID_ARG;
    *bytes = lm_layout(T, V, H, chunk < max_chunk(V) ? chunk : max_chunk(V)).total;
    return CIS_OK;
}

CIS_API cis_status_t cis_lmhead_fused(const void *hidden, const void *weight, int64_t T,
                                      int64_t H, int64_t V, const int32_t *ids,
                                      const float *lp_infer, const float *lp_old,
                                      const float *adv, const uint8_t *mask,
                                      const int32_t *cu_seqlens, int64_t B,
                                      const cis_params_t *params, void *dhidden, void *dweight,
                                      int32_t grad_dtype, float *lp_out, float *w_out,
                                      uint8_t *trunc_out, float *entropy_out,
                                      cis_stats_t *stats_out, double *loss_out, void *workspace,
                                      size_t workspace_bytes, void *stream)
{
    NvtxRange nvtx_range("cis_lmhead_fused");
    if (T < 0 || T > (1LL << 30) || V <= 0 || V > (1LL << 30) || H <= 0 || H > (1LL << 20))
        return CIS_ERR_INVALID_ARG;
    if (grad_dtype != CIS_F32 && grad_dtype != CIS_BF16)
        return CIS_ERR_INVALID_ARG;
    if (!params_ok(params))
        return CIS_ERR_INVALID_ARG;
    if ((params->agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN || is_seq_mode(params->mode)) &&
        (cu_seqlens == nullptr || B < 0))
        return CIS_ERR_INVALID_ARG;
    if (H % lm::kBN != 0)
        return CIS_ERR_UNSUPPORTED;  // Hd in blocks of 256 (and so of the 64-wide K blocks)
    if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 1023))
        return CIS_ERR_INVALID_ARG;
    const int64_t Vc = chunk_for_bytes(T, V, H, workspace_bytes);
    if (Vc == 0)
        return CIS_ERR_INVALID_ARG;  // smaller than the layout for 256-column chunks
    const LmLayout L = lm_layout(T, V, H, Vc);
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
    a.entropy_out = entropy_out;
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
    float *part_u = entropy_out ? reinterpret_cast<float *>(ws + L.part_u) : nullptr;
    uint16_t *dz = reinterpret_cast<uint16_t *>(ws + L.dz);
    float *dh_acc = grad_dtype == CIS_F32 ? static_cast<float *>(dhidden)
                                          : reinterpret_cast<float *>(ws + L.dh);

    float *scale = reinterpret_cast<float *>(ws + L.base.scale);
    a.red_parts = ws + L.base.parts;
    a.red_ticket = reinterpret_cast<uint32_t *>(ws + L.base.ticket);
    cudaError_t e = launch_scales(mask, T, cu_seqlens, B, P.agg, scale, a.status, a.red_ticket, s,
                                  P.global_counts);
    if (e != cudaSuccess)
        return e == cudaErrorNotSupported ? CIS_ERR_UNSUPPORTED : CIS_ERR_CUDA;
    if (T > 0) {
        const int nTt = (int)((T + lm::kBM - 1) / lm::kBM);
        const int nVt = (int)((V + lm::kBN - 1) / lm::kBN);
        const int nHt = (int)(H / lm::kBN);
        // K-major maps of H and W (FWD, DZ) and MN-major ones (boxes of 64
        // rows: W as DH's B operand, H as DW's)
        // (mWh: W in boxes of half a B tile, for the multicast clusters)
        const int mc = lm::mc_mask();
        CUtensorMap mH, mW, mWh, mWmn, mHmn;
        if (!lm::make_map(&mH, hidden, H, T, H, lm::kBM) ||
            !lm::make_map(&mW, weight, H, V, H, lm::kBN) ||
            !lm::make_map(&mWh, weight, H, V, H, lm::kBN / 2) ||
            !lm::make_map(&mWmn, weight, H, V, H, 64) ||
            !lm::make_map(&mHmn, hidden, H, T, H, 64))
            return CIS_ERR_UNSUPPORTED;
        lm::GemmArgs g = {};
        g.T = (int)T;
        g.V = (int)V;
        g.ids = ids;
        g.lse = lse;
        g.cvec = cv;
        g.part = part;
        g.part_u = part_u;
        g.zy = zy;
        g.dz = dz;
        g.ld_dz = Vc;
        g.status = a.status;
        // FWD: z tiles of H W^T, row statistics
        g.nMt = nTt;
        g.nNt = nVt;
        g.nK = (int)(H / lm::kBK);
        g.raster_n = 1;
        if (((mc & 1) ? lm::launch_gemm_mc<lm::kStats>(mH, mWh, g, s)
                      : lm::launch_gemm<lm::kStats>(mH, mW, g, s)) != cudaSuccess)
            return CIS_ERR_CUDA;
        // per-token scalars
        if (is_seq_mode(P.mode)) {
            // sequence operator: log p of every token (fp64, into the terms
            // array, which the second sweep then overwrites), the responses'
            // weights, then the token scalars with those weights
            if (lp_old == nullptr) {
                PassArgs f = a;
                f.lp64_out = a.ws_terms;
                lm::cis_lmhead_token_kernel<<<(unsigned)((T + 7) / 8), 256, 0, s>>>(
                    f, part, part_u, zy, 2 * nVt, lse, cv);
                if ((e = cudaGetLastError()) != cudaSuccess)
                    return CIS_ERR_CUDA;
            }
            if (cudaMemsetAsync(a.ws_w, 0, 4 * (size_t)T, s) != cudaSuccess ||
                cudaMemsetAsync(a.ws_trunc, 0, (size_t)T, s) != cudaSuccess)
                return CIS_ERR_CUDA;
            if (launch_seq_weights(lp_old ? nullptr : a.ws_terms, lp_old, lp_infer, ids, V, mask,
                                   cu_seqlens, B, T, a.P, a.ws_w, a.ws_trunc, s) != cudaSuccess)
                return CIS_ERR_CUDA;
            a.w_in = a.ws_w;
            a.trunc_in = a.ws_trunc;
        }
        lm::cis_lmhead_token_kernel<<<(unsigned)((T + 7) / 8), 256, 0, s>>>(a, part, part_u, zy,
                                                                            2 * nVt, lse, cv);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return CIS_ERR_CUDA;
        for (int64_t v0 = 0; v0 < V; v0 += Vc) {
            const int64_t w = V - v0 < Vc ? V - v0 : Vc;
            // DZ: recompute the chunk's z tiles, write dz
            g.nMt = nTt;
            g.nNt = (int)((w + lm::kBN - 1) / lm::kBN);
            g.nK = (int)(H / lm::kBK);
            g.raster_n = 1;
            g.a_row0 = 0;
            g.a_k0 = 0;
            g.b_row0 = (int)v0;
            g.b_k0 = 0;
            g.col0 = (int)v0;
            if (((mc & 2) ? lm::launch_gemm_mc<lm::kDz>(mH, mWh, g, s)
                          : lm::launch_gemm<lm::kDz>(mH, mW, g, s)) != cudaSuccess)
                return CIS_ERR_CUDA;
            // dz K-major (DH's A: rows are tokens) and MN-major (DW's A: its
            // M runs along dz's columns; rows past T read as zeros)
            CUtensorMap mDz, mDzmn;
            if (!lm::make_map(&mDz, dz, w, L.Tp, Vc, lm::kBM) ||
                !lm::make_map(&mDzmn, dz, w, T, Vc, 64))
                return CIS_ERR_UNSUPPORTED;
            // DH (+)= dz W[chunk]: A = dz [Tp, w] K-major, B = W rows v0 .. v0 + w
            // MN-major (N along Hd, K along the vocabulary)
            lm::GemmArgs gdh = g;
            gdh.nMt = nTt;
            gdh.nNt = nHt;
            gdh.nK = (int)((w + lm::kBK - 1) / lm::kBK);
            gdh.raster_n = 0;
            gdh.a_row0 = 0;
            gdh.a_k0 = 0;
            gdh.b_row0 = 0;
            gdh.b_k0 = (int)v0;
            gdh.out = dh_acc;
            gdh.out_bf16 = 0;
            gdh.out_v8 = (reinterpret_cast<uintptr_t>(dh_acc) & 31) == 0;
            gdh.rows_valid = (int)T;
            gdh.ld_out = H;
            // DW[chunk] = dz^T H: A = dz MN-major (M along the chunk's columns,
            // K along the tokens), B = H MN-major (N along Hd, K along tokens)
            lm::GemmArgs gdw = gdh;
            gdw.nMt = (int)((w + lm::kBM - 1) / lm::kBM);
            gdw.nNt = nHt;
            gdw.nK = (int)((T + lm::kBK - 1) / lm::kBK);
            gdw.raster_n = 0;
            gdw.b_k0 = 0;
            gdw.out = static_cast<uint8_t *>(dweight) +
                      (size_t)v0 * (size_t)H * (grad_dtype == CIS_BF16 ? 2 : 4);
            gdw.out_bf16 = grad_dtype == CIS_BF16;
            gdw.out_v8 = (reinterpret_cast<uintptr_t>(gdw.out) & 31) == 0;
            gdw.rows_valid = (int)w;
            // both in one launch where the schedule fits (and both take the
            // same CTA grouping), else one after the other
            bool done = false;
            if (lm::dual_on() && ((mc & 12) == 12 || (mc & 12) == 0)) {
                const bool pair = (mc & 12) == 12;
                if (v0 == 0)
                    e = pair ? lm::launch_dual<lm::kStore, true>(mDz, mWmn, gdh, mDzmn, mHmn, gdw,
                                                                 s, &done)
                             : lm::launch_dual<lm::kStore, false>(mDz, mWmn, gdh, mDzmn, mHmn,
                                                                  gdw, s, &done);
                else
                    e = pair ? lm::launch_dual<lm::kAccum, true>(mDz, mWmn, gdh, mDzmn, mHmn, gdw,
                                                                 s, &done)
                             : lm::launch_dual<lm::kAccum, false>(mDz, mWmn, gdh, mDzmn, mHmn,
                                                                  gdw, s, &done);
                if (e != cudaSuccess)
                    return CIS_ERR_CUDA;
            }
            if (!done) {
                if (mc & 4)
                    e = v0 == 0 ? lm::launch_gemm_mc<lm::kStore, false, true>(mDz, mWmn, gdh, s)
                                : lm::launch_gemm_mc<lm::kAccum, false, true>(mDz, mWmn, gdh, s);
                else
                    e = v0 == 0 ? lm::launch_gemm<lm::kStore, false, true>(mDz, mWmn, gdh, s)
                                : lm::launch_gemm<lm::kAccum, false, true>(mDz, mWmn, gdh, s);
                if (e != cudaSuccess)
                    return CIS_ERR_CUDA;
                if (((mc & 8) ? lm::launch_gemm_mc<lm::kStore, true, true>(mDzmn, mHmn, gdw, s)
                              : lm::launch_gemm<lm::kStore, true, true>(mDzmn, mHmn, gdw, s)) !=
                    cudaSuccess)
                    return CIS_ERR_CUDA;
            }
        }
        if (grad_dtype == CIS_BF16) {
            lm::cis_lmhead_to_bf16_kernel<<<1184, 256, 0, s>>>(
                dh_acc, static_cast<uint16_t *>(dhidden), T * H);
            if ((e = cudaGetLastError()) != cudaSuccess)
                return CIS_ERR_CUDA;
        }
    }
    return launch_reduce(a, stats_out, loss_out, s) == cudaSuccess ? CIS_OK : CIS_ERR_CUDA;
}

}  // extern "C"
