// cis_kernels.h -- launch interface between the C ABI (cis_api.cu) and the
// kernels.  Internal to libcis.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "cis_common.cuh"

namespace cis {

// Everything one fused token-pass launch needs.  Pointers are device pointers.
struct PassArgs {
    const void *logits;
    int64_t T, V, ld;
    const int32_t *ids;
    const float *lp_inf;   // may be null for the forward-only kernel
    const float *lp_old;   // null: on-policy (rho = 1 in value)
    const float *adv;
    const uint8_t *mask;   // null: every token valid
    const float *scale;    // s_t [T]
    void *dz;              // [T, ld_out] of the output dtype
    int64_t ld_out;
    float *lp_out;         // optional user outputs
    float *lse_out;
    float *w_out;
    uint8_t *trunc_out;
    float *ws_w;           // workspace copies used by the reduction
    uint8_t *ws_trunc;
    float *ws_logk;
    double *ws_terms;
    int32_t *status;
    DevParams P;
    // sequence operators: weights formed beforehand (seq_weight); the pass
    // uses them instead of token_weight's
    const float *w_in;
    const uint8_t *trunc_in;
    double *lp64_out;      // forward-only kernel: log p in fp64 (may be null)
    float *entropy_out;    // per-token entropy of the softmax (may be null)
    void *red_parts;       // the reduction's per-CTA partial sums (workspace)
    uint32_t *red_ticket;  // its completion counter (zeroed by the scales kernel)
};

// Host-side parameter checks and the kernels' copy of the parameters.
bool params_ok(const cis_params_t *p);
DevParams make_dev_params(const cis_params_t &p);

// Workspace layout (offsets in bytes from the 256-byte aligned base).
// status: a 256-byte block (the status word at 0, the reduction's ticket at
// 64); parts: one 64-byte partial sum per 256 tokens.
struct WsLayout {
    size_t status, ticket, scale, terms, logk, w, trunc, parts, total;
};
constexpr int kRedTokens = 256;  // tokens per CTA of the reduction
constexpr int kRedPartBytes = 64;
constexpr size_t ws_round_up(size_t x) { return (x + 255) / 256 * 256; }
constexpr WsLayout ws_layout(int64_t T)
{
    const size_t n = (size_t)(T > 0 ? T : 0);
    WsLayout L{};
    size_t o = 0;
    L.status = o;
    L.ticket = o + 64;
    o += 256;
    L.scale = o;
    o = ws_round_up(o + 4 * n);
    L.terms = o;
    o = ws_round_up(o + 8 * n);
    L.logk = o;
    o = ws_round_up(o + 4 * n);
    L.w = o;
    o = ws_round_up(o + 4 * n);
    L.trunc = o;
    o = ws_round_up(o + n);
    L.parts = o;
    o = ws_round_up(o + (size_t)kRedPartBytes * ((n + kRedTokens - 1) / kRedTokens + (n == 0)));
    L.total = o;
    return L;
}

// Sequence operators: w[t], trunc[t] for the valid tokens of each response
// from the fp64 sum of log k = lw - lp_inf over its valid tokens with an id
// in [0, V) (lw64 if given, else lw32); other tokens are not written.
// Response ranges are clamped to [0, T), so bad offsets cannot reach memory
// outside the T-long arrays.
cudaError_t launch_seq_weights(const double *lw64, const float *lw32, const float *lp_inf,
                               const int32_t *ids, int64_t V, const uint8_t *mask,
                               const int32_t *cu_seqlens, int64_t B, int64_t T,
                               const DevParams &P, float *w, uint8_t *trunc, cudaStream_t s);

// Forward-only: lp (and lse) of the sampled token, one CTA per row.
cudaError_t launch_token_logprobs(const PassArgs &a, int dtype, cudaStream_t s);

// Fused forward + backward, any layout: one CTA per row, second read from L2.
cudaError_t launch_rowwise_fwd_bwd(const PassArgs &a, int dtype, int out_dtype,
                                   cudaStream_t s);

// Fused forward + backward, 16-byte aligned rows: a cluster of CTAs splits
// each row, each CTA keeps its slice in shared memory (one HBM read).
// Returns cudaErrorNotSupported when the shape does not fit the kernel.
cudaError_t launch_cluster_fwd_bwd(const PassArgs &a, int dtype, int out_dtype,
                                   cudaStream_t s);
bool cluster_path_applies(const PassArgs &a, int dtype, int out_dtype);

// Loss scales s_t (and clears the status word).
cudaError_t launch_count_valid(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens,
                               int64_t B, int64_t *counts, cudaStream_t s);
cudaError_t launch_scales(const uint8_t *mask, int64_t T, const int32_t *cu_seqlens, int64_t B,
                          int agg, float *scale, int32_t *status, uint32_t *ticket,
                          cudaStream_t s, const int64_t *global_counts = nullptr);

// Elementwise weights (cis_weights).
cudaError_t launch_weights(const float *lp_w, const float *lp_inf, const uint8_t *mask,
                           int64_t T, const DevParams &P, float *w_out, uint8_t *trunc_out,
                           float *eps_out, cudaStream_t s);

// Deterministic reduction of the per-token terms into the loss and stats.
cudaError_t launch_reduce(const PassArgs &a, cis_stats_t *stats, double *loss,
                          cudaStream_t s);

}  // namespace cis
