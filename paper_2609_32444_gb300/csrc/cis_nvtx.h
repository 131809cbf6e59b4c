// cis_nvtx.h -- a named NVTX range around each call of the C ABI, so that a
// profiler's timeline (Nsight Systems, or ncu's NVTX filters) shows which
// library call issued which kernels.  NVTX v3 is header-only: with no tool
// attached, a push or pop is one test of a function pointer.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace cis {

class NvtxRange {
public:
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};

}  // namespace cis
