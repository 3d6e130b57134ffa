// sjd_step_noalloc: the fused Jacobi step for callers that cannot allocate
// device memory. The decode state is a buffer the caller hands in; the
// step's scratch (per-row results, last-CTA tickets, counters) lives in the
// fixed array below, which every GPU that loads the library holds until the
// process exits. Nothing here calls cudaMalloc, cudaFree or any allocating
// library routine.

#include <cstring>
#include <mutex>

#include "sjd_internal.h"

namespace {

// Scratch shared by every call of sjd_step_noalloc (per device).
static __device__ __align__(256) unsigned char g_noalloc_scratch[SJD_NOALLOC_SCRATCH_BYTES];

constexpr size_t kStatusBytes = 256;  // tail of the state buffer: device status word

struct DeviceSetup {
  bool done = false;
  unsigned char* scratch = nullptr;  // device address of g_noalloc_scratch
};

std::mutex g_setup_mutex;
DeviceSetup g_setup[64];

// Device address of the scratch array on the current device (looked up once
// per device, with that device current).
int scratch_address(int dev, unsigned char** out) {
  if (dev < 0 || dev >= 64) return SJD_ERR_ARG;
  DeviceSetup& s = g_setup[dev];
  if (!s.done) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return SJD_ERR_CUDA;
    s.scratch = static_cast<unsigned char*>(p);
    s.done = true;
  }
  *out = s.scratch;
  return SJD_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int sjd_step_noalloc(const sjd_config* cfg, void* state_dev, size_t* state_bytes,
                                int32_t reset, const void* cond_dev, const void* uncond_dev,
                                int32_t* committed_dev, int32_t* n_commit_dev,
                                int32_t* first_rej_dev, void* cuda_stream) {
  if (!cfg || !state_bytes) return SJD_ERR_ARG;
  if (!sjd::check_config(cfg).empty() || cfg->pd_tree) return SJD_ERR_ARG;
  sjd::Layout L;
  sjd::DevParams P{};
  sjd::plan(cfg, &L, &P);
  const size_t need = L.persistent_end + kStatusBytes;
  if (!state_dev) {
    *state_bytes = need;
    return SJD_OK;
  }
  if (*state_bytes < need) return SJD_ERR_CAPACITY;
  if ((reinterpret_cast<uintptr_t>(state_dev) & 255u) != 0) return SJD_ERR_ARG;
  const size_t scratch_need = L.fast_scratch - L.persistent_end;  // the general kernel's scratch
  if (scratch_need > SJD_NOALLOC_SCRATCH_BYTES) return SJD_ERR_CAPACITY;
  if (!cond_dev || (!uncond_dev && cfg->cfg_scale != 1.0f)) return SJD_ERR_ARG;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SJD_ERR_CUDA;
  unsigned char* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    const int rc = scratch_address(dev, &scratch);
    if (rc != SJD_OK) return rc;
    int optin = 0;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
      return SJD_ERR_CUDA;
    if (P.smem_bytes + 2048 > static_cast<uint32_t>(optin)) return SJD_ERR_CAPACITY;
    if (sjd::raise_row_kernel_smem(static_cast<int>(P.smem_bytes)) != cudaSuccess) return SJD_ERR_CUDA;
  }

  // persistent state in the caller's buffer, scratch in the fixed array
  unsigned char* st = static_cast<unsigned char*>(state_dev);
  // scratch offsets of the layout start at persistent_end
  auto sc = [&](size_t off) { return scratch + (off - L.persistent_end); };
  P.q_ids = reinterpret_cast<int32_t*>(st + L.q_ids);
  P.q_prob = reinterpret_cast<float*>(st + L.q_prob);
  P.q_len = reinterpret_cast<int32_t*>(st + L.q_len);
  P.cand = reinterpret_cast<int32_t*>(st + L.cand);
  P.gsize = reinterpret_cast<int32_t*>(st + L.gsize);
  P.win_tok = reinterpret_cast<int32_t*>(st + L.win_tok);
  P.abs_pos = reinterpret_cast<int32_t*>(st + L.abs_pos);
  P.last_tok = reinterpret_cast<int32_t*>(st + L.last_tok);
  P.step_t = reinterpret_cast<uint32_t*>(st + L.step_t);
  P.err = reinterpret_cast<uint32_t*>(st + L.persistent_end);
  P.res_x = reinterpret_cast<int32_t*>(sc(L.res_x));
  P.res_dev = reinterpret_cast<int32_t*>(sc(L.res_dev));
  P.res_alt = reinterpret_cast<int32_t*>(sc(L.res_alt));
  P.res_altn = reinterpret_cast<int32_t*>(sc(L.res_altn));
  P.res_xf = reinterpret_cast<int32_t*>(sc(L.res_xf));
  P.res_altf = reinterpret_cast<int32_t*>(sc(L.res_altf));
  P.res_altfn = reinterpret_cast<int32_t*>(sc(L.res_altfn));
  P.ticket = reinterpret_cast<uint32_t*>(sc(L.ticket));
  P.first_rej = reinterpret_cast<int32_t*>(sc(L.first_rej));
  P.n_commit = reinterpret_cast<int32_t*>(sc(L.n_commit));
  P.committed = reinterpret_cast<int32_t*>(sc(L.committed));
  P.stats = reinterpret_cast<unsigned long long*>(sc(L.stats));

  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaSuccess;
  if (reset) {
    e = cudaMemsetAsync(st, 0, need, s);
    if (e == cudaSuccess) e = sjd::launch_init(P, s);
  }
  // the last-CTA tickets must start at zero; the array keeps the last call's contents
  if (e == cudaSuccess) e = cudaMemsetAsync(P.ticket, 0, static_cast<size_t>(P.B) * 4, s);
  if (e != cudaSuccess) return SJD_ERR_CUDA;

  const size_t esz = cfg->logit_dtype == SJD_BF16 ? 2 : 4;
  const bool use_cfg = uncond_dev != nullptr && cfg->cfg_scale != 1.0f;
  const bool vec = (static_cast<size_t>(cfg->vocab) * esz) % 16 == 0 &&
                   static_cast<size_t>(P.al0 + P.nL) <= static_cast<size_t>(cfg->vocab) &&
                   aligned16(cond_dev) && (!use_cfg || aligned16(uncond_dev));
  e = sjd::launch_row(P, sjd::kModeStep, cfg->logit_dtype, vec, cond_dev, use_cfg ? uncond_dev : nullptr,
                      use_cfg, committed_dev, n_commit_dev, first_rej_dev, s);
  return e == cudaSuccess ? SJD_OK : SJD_ERR_CUDA;
}
