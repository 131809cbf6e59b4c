// cis_selftest.cu -- self-test of the bounded waits: every wait in the
// library's kernels polls an mbarrier a bounded number of times, then records
// CIS_ERR_DEVICE_TIMEOUT in a device status word and lets the kernel run to
// its end, so that the context stays usable.  This kernel waits on an
// mbarrier that nothing ever completes, through the same wait helpers with a
// caller-chosen poll limit, and reports the timeout the same way.
#include "cis_dsmem.cuh"
#include "cis_kernels.h"
#include "cis_nvtx.h"

namespace cis {
namespace {

__global__ void cis_selftest_wait_kernel(uint32_t max_polls, int cluster_scope, int32_t *status)
{
    __shared__ alignas(8) uint64_t bar;
    const uint32_t b = smem_u32(&bar);
    if (threadIdx.x == 0)
        mbar_init(b, 1);  // one arrival expected, none ever made
    __syncthreads();
    const bool ok = cluster_scope ? mbar_wait_cluster_n(b, 0, max_polls)
                                  : mbar_wait_n(b, 0, max_polls);
    if (!ok && threadIdx.x == 0)
        set_status(status, kStatusTimeout);
}

}  // namespace
}  // namespace cis

using namespace cis;

extern "C" CIS_API cis_status_t cis_selftest_bounded_wait(uint32_t max_polls, int32_t cluster_scope,
                                                          int32_t *dev_status, void *stream)
{
    NvtxRange nvtx_range("cis_selftest_bounded_wait");
    if (dev_status == nullptr || max_polls == 0 || max_polls > kMaxPolls ||
        (cluster_scope != 0 && cluster_scope != 1))
        return CIS_ERR_INVALID_ARG;
    cis_selftest_wait_kernel<<<1, 64, 0, (cudaStream_t)stream>>>(max_polls, cluster_scope,
                                                                 dev_status);
    return cudaGetLastError() == cudaSuccess ? CIS_OK : CIS_ERR_CUDA;
}
