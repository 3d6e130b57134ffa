// Dispatch of the fast row kernels (sjd_fast.cuh, one translation unit per
// dtype and mode: sjd_fast_part.cu).

#include <mutex>

#include "sjd_internal.h"

namespace sjd {
namespace {

// The limit is a setting of the whole process (per device): contexts of
// different configurations only ever raise it, one at a time.
std::mutex g_fast_smem_mutex;

template <int DT>
cudaError_t launch_t(const DevParams& p, int mode, const void* cond, const void* uncond, bool use_cfg, int32_t* oc,
                     int32_t* on, int32_t* of, cudaStream_t s) {
  switch (mode) {
    case kModeVerify: return fast_launch<DT, kModeVerify>(p, cond, uncond, use_cfg, oc, on, of, s);
    case kModeStep: return fast_launch<DT, kModeStep>(p, cond, uncond, use_cfg, oc, on, of, s);
    default: return fast_launch<DT, kModeFromLogits>(p, cond, uncond, use_cfg, oc, on, of, s);
  }
}

}  // namespace

cudaError_t raise_fast_row_kernel_smem(int bytes) {
  std::lock_guard<std::mutex> lock(g_fast_smem_mutex);
  cudaError_t e = cudaSuccess;
  auto acc = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
  acc(fast_raise_smem<SJD_BF16, kModeVerify>(bytes));
  acc(fast_raise_smem<SJD_BF16, kModeStep>(bytes));
  acc(fast_raise_smem<SJD_BF16, kModeFromLogits>(bytes));
  acc(fast_raise_smem<SJD_F32, kModeVerify>(bytes));
  acc(fast_raise_smem<SJD_F32, kModeStep>(bytes));
  acc(fast_raise_smem<SJD_F32, kModeFromLogits>(bytes));
  return e;
}

cudaError_t launch_fast_row(const DevParams& p, int mode, int dtype, const void* cond, const void* uncond,
                            bool use_cfg, int32_t* oc, int32_t* on, int32_t* of, cudaStream_t s) {
  const cudaError_t e = dtype == SJD_BF16 ? launch_t<SJD_BF16>(p, mode, cond, uncond, use_cfg, oc, on, of, s)
                                           : launch_t<SJD_F32>(p, mode, cond, uncond, use_cfg, oc, on, of, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace sjd
