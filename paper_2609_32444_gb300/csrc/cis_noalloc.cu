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
#include "cis_kernels.h"
#include "cis_nvtx.h"

namespace cis {
namespace {

constexpr int64_t kMaxTokens = CIS_NOALLOC_MAX_TOKENS;

// Exactly what cis_loss_fwd_bwd asks of a workspace for kMaxTokens tokens.
constexpr size_t kScratchBytes = ws_layout(kMaxTokens).total;
static_assert(kScratchBytes % 256 == 0, "the scratch is a whole number of 256-byte blocks");

// The scratch itself.  In host code this name is only a host-side stand-in:
// its device address is looked up with cudaGetSymbolAddress.
static __device__ __align__(256) uint8_t g_scratch[kScratchBytes];

// Device address of g_scratch in the current context.  Looked up on every
// call, not cached: a cached address would outlive a context that a caller
// tears down (cudaDeviceReset) or swaps for another on the same device, and
// the next call would then write through a dangling pointer.  The lookup is a
// host-side query; it allocates nothing.
cis_status_t scratch_address(void **out)
{
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr)
        return CIS_ERR_CUDA;
    *out = p;
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
    NvtxRange nvtx_range("cis_loss_fwd_bwd_noalloc");
    if (T > kMaxTokens)
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
