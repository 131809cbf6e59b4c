// cis_host.cu -- the fused token pass for callers whose buffers live in host
// memory: logits in, dlogits out, streamed through the GPU in row chunks.
//
// The logits of a batch (4.98 GB for T=16384, V=151936, bf16) and their
// gradient cross the host link once each.  The call splits the rows into
// chunks: host->device copies of the next chunks, the fused kernel on chunk k
// (the caller's stream) and device->host copies of the previous chunks run
// concurrently, ordered by events, with three staging buffers per direction,
// each with its own copy stream (so that several copy engines work at once).  The loss
// normaliser is computed once for the whole batch before the first chunk and
// the loss is reduced once after the last, so the results are those of
// cis_loss_fwd_bwd on the whole batch.
#include <mutex>
#include <vector>

#include "cis_kernels.h"
#include "cis_nvtx.h"

namespace cis {
namespace {

constexpr int kMaxDev = 64;
constexpr int kBufs = 3;  // staging buffers (and copy streams) per direction

// Copy streams per device, created on first use and kept: staging buffer b is
// always filled on h2d[b] and drained on d2h[b].
struct HostStreams {
    cudaStream_t h2d[kBufs] = {}, d2h[kBufs] = {};
};
std::mutex g_mu;
HostStreams g_streams[kMaxDev];

cudaError_t streams_for_device(HostStreams **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev < 0 || dev >= kMaxDev)
        return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> g(g_mu);
    HostStreams &s = g_streams[dev];
    for (int b = 0; b < kBufs; ++b) {
        if (!s.h2d[b] &&
            (e = cudaStreamCreateWithFlags(&s.h2d[b], cudaStreamNonBlocking)) != cudaSuccess)
            return e;
        if (!s.d2h[b] &&
            (e = cudaStreamCreateWithFlags(&s.d2h[b], cudaStreamNonBlocking)) != cudaSuccess)
            return e;
    }
    *out = &s;
    return cudaSuccess;
}

struct HostLayout {
    WsLayout base;
    size_t ids, lpi, lpo, adv, mask, cu, lp, w, tr, ent, stats, loss, in[kBufs], out[kBufs],
        total;
};

HostLayout host_layout(int64_t T, int64_t V, int isz, int osz, int64_t chunk, int64_t B)
{
    auto up = [](size_t x) { return (x + 255) / 256 * 256; };
    const size_t n = (size_t)T;
    HostLayout L;
    L.base = ws_layout(T);
    size_t o = up(L.base.total);
    L.ids = o; o = up(o + 4 * n);
    L.lpi = o; o = up(o + 4 * n);
    L.lpo = o; o = up(o + 4 * n);
    L.adv = o; o = up(o + 4 * n);
    L.mask = o; o = up(o + n);
    L.cu = o; o = up(o + 4 * (size_t)(B + 1));
    L.lp = o; o = up(o + 4 * n);
    L.w = o; o = up(o + 4 * n);
    L.tr = o; o = up(o + n);
    L.ent = o; o = up(o + 4 * n);
    L.stats = o; o = up(o + sizeof(cis_stats_t));
    L.loss = o; o = up(o + 8);
    for (int b = 0; b < kBufs; ++b) {
        L.in[b] = o;
        o = up(o + (size_t)chunk * V * isz);
        L.out[b] = o;
        o = up(o + (size_t)chunk * V * osz);
    }
    L.total = o;
    return L;
}

int dbytes(int32_t dt) { return dt == CIS_BF16 ? 2 : 4; }

}  // namespace
}  // namespace cis

using namespace cis;

extern "C" {

CIS_API cis_status_t cis_loss_host_workspace_size(int64_t T, int64_t V, int32_t dtype,
                                                  int32_t dlogits_dtype, int64_t chunk_tokens,
                                                  int64_t B, size_t *bytes)
{
    if (bytes == nullptr || T < 0 || V <= 0 || chunk_tokens <= 0 || B < 0 ||
        (dtype != CIS_F32 && dtype != CIS_BF16) ||
        (dlogits_dtype != CIS_F32 && dlogits_dtype != CIS_BF16))
        return CIS_ERR_INVALID_ARG;
    *bytes = host_layout(T, V, dbytes(dtype), dbytes(dlogits_dtype), chunk_tokens, B).total;
    return CIS_OK;
}

CIS_API cis_status_t cis_loss_fwd_bwd_host(
    const void *logits, int32_t dtype, int64_t T, int64_t V, const int32_t *ids,
    const float *lp_infer, const float *lp_old, const float *adv, const uint8_t *mask,
    const int32_t *cu_seqlens, int64_t B, const cis_params_t *params, void *dlogits,
    int32_t dlogits_dtype, float *lp_out, float *w_out, uint8_t *trunc_out, float *entropy_out,
    cis_stats_t *stats_out, double *loss_out, int64_t chunk_tokens, void *workspace,
    size_t workspace_bytes, void *stream)
{
    NvtxRange nvtx_range("cis_loss_fwd_bwd_host");
    if (T < 0 || T > 0x7fffffffLL || V <= 0 || chunk_tokens <= 0 ||
        (dtype != CIS_F32 && dtype != CIS_BF16) ||
        (dlogits_dtype != CIS_F32 && dlogits_dtype != CIS_BF16))
        return CIS_ERR_INVALID_ARG;
    if (!params_ok(params))
        return CIS_ERR_INVALID_ARG;
    if ((params->agg == CIS_AGG_SEQ_MEAN_TOKEN_MEAN || is_seq_mode(params->mode)) &&
        (cu_seqlens == nullptr || B < 0))
        return CIS_ERR_INVALID_ARG;
    // a sequence operator's weights need every row's log p before the first
    // chunk's dlogits unless they come from lp_old
    if (is_seq_mode(params->mode) && lp_old == nullptr && T > 0)
        return CIS_ERR_UNSUPPORTED;
    const int isz = dbytes(dtype), osz = dbytes(dlogits_dtype);
    const HostLayout L = host_layout(T, V, isz, osz, chunk_tokens, B < 0 ? 0 : B);
    if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 255) ||
        workspace_bytes < L.total)
        return CIS_ERR_INVALID_ARG;
    if (T > 0 && (logits == nullptr || ids == nullptr || lp_infer == nullptr ||
                  adv == nullptr || dlogits == nullptr))
        return CIS_ERR_INVALID_ARG;
    HostStreams *hs = nullptr;
    if (streams_for_device(&hs) != cudaSuccess)
        return CIS_ERR_CUDA;
    cudaStream_t sc = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    auto dptr = [&](size_t off) { return ws + off; };
    const size_t n = (size_t)T;
    cudaError_t e = cudaSuccess;
#define CIS_TRY(x)                                                                             \
    do {                                                                                       \
        if ((e = (x)) != cudaSuccess)                                                          \
            return CIS_ERR_CUDA;                                                               \
    } while (0)

    // the small per-token inputs, on the compute stream
    CIS_TRY(cudaMemcpyAsync(dptr(L.ids), ids, 4 * n, cudaMemcpyHostToDevice, sc));
    CIS_TRY(cudaMemcpyAsync(dptr(L.lpi), lp_infer, 4 * n, cudaMemcpyHostToDevice, sc));
    CIS_TRY(cudaMemcpyAsync(dptr(L.adv), adv, 4 * n, cudaMemcpyHostToDevice, sc));
    if (lp_old)
        CIS_TRY(cudaMemcpyAsync(dptr(L.lpo), lp_old, 4 * n, cudaMemcpyHostToDevice, sc));
    if (mask)
        CIS_TRY(cudaMemcpyAsync(dptr(L.mask), mask, n, cudaMemcpyHostToDevice, sc));
    if (cu_seqlens)
        CIS_TRY(cudaMemcpyAsync(dptr(L.cu), cu_seqlens, 4 * (size_t)(B + 1),
                                cudaMemcpyHostToDevice, sc));

    PassArgs a = {};
    a.T = T;
    a.V = V;
    a.ld = V;
    a.ld_out = V;
    a.ids = reinterpret_cast<const int32_t *>(dptr(L.ids));
    a.lp_inf = reinterpret_cast<const float *>(dptr(L.lpi));
    a.lp_old = lp_old ? reinterpret_cast<const float *>(dptr(L.lpo)) : nullptr;
    a.adv = reinterpret_cast<const float *>(dptr(L.adv));
    a.mask = mask ? dptr(L.mask) : nullptr;
    float *scale = reinterpret_cast<float *>(dptr(L.base.scale));
    a.scale = scale;
    a.lp_out = reinterpret_cast<float *>(dptr(L.lp));
    a.w_out = reinterpret_cast<float *>(dptr(L.w));
    a.trunc_out = dptr(L.tr);
    a.entropy_out = entropy_out ? reinterpret_cast<float *>(dptr(L.ent)) : nullptr;
    a.ws_w = reinterpret_cast<float *>(dptr(L.base.w));
    a.ws_trunc = dptr(L.base.trunc);
    a.ws_logk = reinterpret_cast<float *>(dptr(L.base.logk));
    a.ws_terms = reinterpret_cast<double *>(dptr(L.base.terms));
    a.status = reinterpret_cast<int32_t *>(dptr(L.base.status));
    a.P = make_dev_params(*params);
    const int32_t *cu_dev = cu_seqlens ? reinterpret_cast<const int32_t *>(dptr(L.cu)) : nullptr;
    a.red_parts = dptr(L.base.parts);
    a.red_ticket = reinterpret_cast<uint32_t *>(dptr(L.base.ticket));
    CIS_TRY(launch_scales(a.mask, T, cu_dev, B, params->agg, scale, a.status, a.red_ticket, sc,
                          params->global_counts));
    if (T > 0 && is_seq_mode(params->mode)) {
        // the responses' weights from lp_old, read by every chunk's pass
        CIS_TRY(cudaMemsetAsync(a.ws_w, 0, 4 * n, sc));
        CIS_TRY(cudaMemsetAsync(a.ws_trunc, 0, n, sc));
        CIS_TRY(launch_seq_weights(nullptr, a.lp_old, a.lp_inf, a.ids, V, a.mask, cu_dev, B, T,
                                   a.P, a.ws_w, a.ws_trunc, sc));
        a.w_in = a.ws_w;
        a.trunc_in = a.ws_trunc;
    }

    const int64_t nchunks = (T + chunk_tokens - 1) / chunk_tokens;
    std::vector<cudaEvent_t> ev;  // per chunk: copied in, computed, copied out
    auto mkev = [&]() {
        cudaEvent_t x;
        e = cudaEventCreateWithFlags(&x, cudaEventDisableTiming);
        if (e == cudaSuccess)
            ev.push_back(x);
        return x;
    };
    cudaEvent_t start = mkev();
    std::vector<cudaEvent_t> e_in(nchunks), e_comp(nchunks), e_out(nchunks);
    for (int64_t k = 0; k < nchunks && e == cudaSuccess; ++k) {
        e_in[k] = mkev();
        e_comp[k] = mkev();
        e_out[k] = mkev();
    }
    cis_status_t st = CIS_OK;
    if (e != cudaSuccess) {
        st = CIS_ERR_CUDA;
    } else {
        // the copy streams start after the small inputs and the normaliser
        cudaEventRecord(start, sc);
        for (int b = 0; b < kBufs; ++b) {
            cudaStreamWaitEvent(hs->h2d[b], start, 0);
            cudaStreamWaitEvent(hs->d2h[b], start, 0);
        }
        for (int64_t k = 0; k < nchunks; ++k) {
            const int b = (int)(k % kBufs);
            const int64_t r0 = k * chunk_tokens;
            const int64_t rows = (T - r0 < chunk_tokens) ? T - r0 : chunk_tokens;
            uint8_t *in = dptr(L.in[b]), *out = dptr(L.out[b]);
            // buffer b was last read by the kernel of chunk k - kBufs
            if (k >= kBufs)
                cudaStreamWaitEvent(hs->h2d[b], e_comp[k - kBufs], 0);
            cudaMemcpyAsync(in, static_cast<const uint8_t *>(logits) + r0 * V * isz,
                            (size_t)rows * V * isz, cudaMemcpyHostToDevice, hs->h2d[b]);
            cudaEventRecord(e_in[k], hs->h2d[b]);
            // the kernel needs its input, and its output buffer drained (k - kBufs)
            cudaStreamWaitEvent(sc, e_in[k], 0);
            if (k >= kBufs)
                cudaStreamWaitEvent(sc, e_out[k - kBufs], 0);
            PassArgs c = a;
            c.logits = in;
            c.T = rows;
            c.ids = a.ids + r0;
            c.lp_inf = a.lp_inf + r0;
            c.lp_old = a.lp_old ? a.lp_old + r0 : nullptr;
            c.adv = a.adv + r0;
            c.mask = a.mask ? a.mask + r0 : nullptr;
            c.scale = a.scale + r0;
            c.dz = out;
            c.lp_out = a.lp_out + r0;
            c.w_out = a.w_out + r0;
            c.trunc_out = a.trunc_out + r0;
            c.entropy_out = a.entropy_out ? a.entropy_out + r0 : nullptr;
            c.ws_w = a.ws_w + r0;
            c.ws_trunc = a.ws_trunc + r0;
            c.ws_logk = a.ws_logk + r0;
            c.ws_terms = a.ws_terms + r0;
            c.w_in = a.w_in ? a.w_in + r0 : nullptr;
            c.trunc_in = a.trunc_in ? a.trunc_in + r0 : nullptr;
            cudaError_t ke = cluster_path_applies(c, dtype, dlogits_dtype)
                                 ? launch_cluster_fwd_bwd(c, dtype, dlogits_dtype, sc)
                                 : launch_rowwise_fwd_bwd(c, dtype, dlogits_dtype, sc);
            if (ke != cudaSuccess) {
                st = CIS_ERR_CUDA;
                break;
            }
            cudaEventRecord(e_comp[k], sc);
            cudaStreamWaitEvent(hs->d2h[b], e_comp[k], 0);
            cudaMemcpyAsync(static_cast<uint8_t *>(dlogits) + r0 * V * osz, out,
                            (size_t)rows * V * osz, cudaMemcpyDeviceToHost, hs->d2h[b]);
            cudaEventRecord(e_out[k], hs->d2h[b]);
        }
        if (st == CIS_OK) {
            cis_stats_t *stats_dev = reinterpret_cast<cis_stats_t *>(dptr(L.stats));
            double *loss_dev = reinterpret_cast<double *>(dptr(L.loss));
            if (launch_reduce(a, stats_dev, loss_dev, sc) != cudaSuccess)
                st = CIS_ERR_CUDA;
            // the caller's stream completes only after every copy out
            for (int64_t k = nchunks - kBufs < 0 ? 0 : nchunks - kBufs; k < nchunks; ++k)
                cudaStreamWaitEvent(sc, e_out[k], 0);
            if (st == CIS_OK && lp_out)
                cudaMemcpyAsync(lp_out, a.lp_out, 4 * n, cudaMemcpyDeviceToHost, sc);
            if (st == CIS_OK && w_out)
                cudaMemcpyAsync(w_out, a.w_out, 4 * n, cudaMemcpyDeviceToHost, sc);
            if (st == CIS_OK && trunc_out)
                cudaMemcpyAsync(trunc_out, a.trunc_out, n, cudaMemcpyDeviceToHost, sc);
            if (st == CIS_OK && entropy_out)
                cudaMemcpyAsync(entropy_out, a.entropy_out, 4 * n, cudaMemcpyDeviceToHost, sc);
            if (st == CIS_OK && stats_out)
                cudaMemcpyAsync(stats_out, stats_dev, sizeof(cis_stats_t),
                                cudaMemcpyDeviceToHost, sc);
            if (st == CIS_OK && loss_out)
                cudaMemcpyAsync(loss_out, loss_dev, 8, cudaMemcpyDeviceToHost, sc);
            if (cudaGetLastError() != cudaSuccess)
                st = CIS_ERR_CUDA;
        }
    }
    for (cudaEvent_t x : ev)
        cudaEventDestroy(x);  // released once the recorded work completes
#undef CIS_TRY
    return st;
}

}  // extern "C"
