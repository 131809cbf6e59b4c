// cis_noalloc.cu -- the fused token pass for callers that cannot allocate.
//
// cis_loss_fwd_bwd needs a few bytes of device scratch per token (the loss
// normaliser, the per-token loss terms and statistics, the status word), which
// its caller allocates and passes in.  Some callers cannot do that: code that
// runs as a plug-in inside a host framework that owns every byte of device
// memory (inference servers and training runtimes that hand out no allocator
// to extensions), or plain C callers with no device allocator of their own.
// For them, cis_loss_fwd_bwd_noalloc takes its scratch from a fixed array in
// the library's static device memory instead.  It calls no allocating routine.
//
// The array is sized for CIS_NOALLOC_MAX_TOKENS tokens.  Every GPU that loads
// the library holds one copy until the process exits.  All calls share it:
// the status word is reset at the start of every call and every other byte is
// written before it is read, but two calls whose GPU work overlaps race.
#include <mutex>

#include "cis_kernels.h"

namespace cis {
namespace {

constexpr int64_t kMaxTokens = CIS_NOALLOC_MAX_TOKENS;

// Bytes ws_layout() asks for at kMaxTokens: a 256-byte status block, then the
// scale (4 B), term (8 B), log k (4 B), weight (4 B) and flag (1 B) arrays,
// each rounded up to 256 bytes, and the reduction's partial sums (64 B per
// 256 tokens).
constexpr size_t kScratchBytes = 256 + 4 * kMaxTokens + 8 * kMaxTokens + 4 * kMaxTokens +
                                 4 * kMaxTokens + 1 * kMaxTokens +
                                 kRedPartBytes * ((kMaxTokens + kRedTokens - 1) / kRedTokens);

// The scratch itself.  In host code this name is only a host-side stand-in:
// its device address is looked up per device with cudaGetSymbolAddress.
static __device__ __align__(256) uint8_t g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_lock;
void *g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device (looked up once per device).
cis_status_t scratch_address(void **out)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return CIS_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return CIS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> guard(g_lock);
    if (g_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr)
            return CIS_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return CIS_OK;
}

}  // namespace
}  // namespace cis

using namespace cis;

extern "C" CIS_API cis_status_t cis_loss_fwd_bwd_noalloc(
    const void *logits, int32_t dtype, int64_t T, int64_t V, int64_t ld, const int32_t *ids,
    const float *lp_infer, const float *lp_old, const float *adv, const uint8_t *mask,
    const int32_t *cu_seqlens, int64_t B, const cis_params_t *params, void *dlogits,
    int32_t dlogits_dtype, int64_t ld_out, float *lp_out, float *w_out, uint8_t *trunc_out,
    float *entropy_out, cis_stats_t *stats_out, double *loss_out, void *stream)
{
    if (T > kMaxTokens)
        return CIS_ERR_UNSUPPORTED;
    if (ws_layout(T < 0 ? 0 : T).total > kScratchBytes)
        return CIS_ERR_UNSUPPORTED;
    void *scratch = nullptr;
    const cis_status_t st = scratch_address(&scratch);
    if (st != CIS_OK)
        return st;
    return cis_loss_fwd_bwd(logits, dtype, T, V, ld, ids, lp_infer, lp_old, adv, mask,
                            cu_seqlens, B, params, dlogits, dlogits_dtype, ld_out, lp_out, w_out,
                            trunc_out, entropy_out, stats_out, loss_out, scratch, kScratchBytes,
                            stream);
}
