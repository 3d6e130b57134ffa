// One (dtype, mode) pair of the fast row kernels (sjd_fast.cuh), chosen by
// SJD_FAST_DT (SJD_BF16 or SJD_F32) and SJD_FAST_MODE (kModeVerify,
// kModeStep or kModeFromLogits as integers): the build compiles this file
// once per pair, so that the variants compile in parallel.

#ifndef SJD_FAST_DT
#error "define SJD_FAST_DT and SJD_FAST_MODE"
#endif

#include "sjd_fast.cuh"

namespace sjd {

template cudaError_t fast_launch<SJD_FAST_DT, SJD_FAST_MODE>(const DevParams&, const void*, const void*, bool,
                                                             int32_t*, int32_t*, int32_t*, cudaStream_t);
template cudaError_t fast_raise_smem<SJD_FAST_DT, SJD_FAST_MODE>(int);

}  // namespace sjd
