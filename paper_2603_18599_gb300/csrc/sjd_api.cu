// Host side of the C ABI declared in include/sjd.h: configuration checks,
// workspace layout, launches and the decode loop.

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "sjd_internal.h"

using sjd::DevParams;
using sjd::Layout;

struct sjd_ctx {
  sjd_config cfg;
  DevParams P;
  Layout L;
  cudaStream_t stream;
  unsigned char* ws;
  size_t ws_bytes;
  bool pending;          // a verify awaits sjd_draft(SJD_DRAFT_PD)
  int32_t* abs_before;   // [B] device scratch of the decode loop
  bool force_general;    // SJD_KERNEL=general: always use the general row kernel
  bool early_logits;     // sjd_set_early_logits: sjd_step / sjd_verify_step logits precede the previous kernel
  std::string last_error;
  // sjd_step_host with two stages: copies on a stream of their own, each into
  // the stage the step before last read (one stream: splitting the rows over
  // four streams measured slower, 107 against 124 GB/s on GB300)
  static constexpr int kCopyStreams = 1;
  cudaStream_t copy_stream[kCopyStreams] = {};
  cudaEvent_t ev_copied[2][kCopyStreams] = {};      // stage s holds this step's rows
  cudaEvent_t ev_consumed[2] = {nullptr, nullptr};  // the kernel that read stage s is done
  int next_stage = 0;
  ~sjd_ctx() {
    for (int k = 0; k < 2; ++k) {
      for (int i = 0; i < kCopyStreams; ++i)
        if (ev_copied[k][i]) cudaEventDestroy(ev_copied[k][i]);
      if (ev_consumed[k]) cudaEventDestroy(ev_consumed[k]);
    }
    for (int i = 0; i < kCopyStreams; ++i)
      if (copy_stream[i]) cudaStreamDestroy(copy_stream[i]);
  }
};

namespace sjd {

namespace {
size_t up(size_t x, size_t a) { return (x + a - 1) / a * a; }
constexpr size_t kAlign = 256;
}  // namespace

int min_support(const sjd_config* c) {
  const int veff = c->allowed_hi - c->allowed_lo;
  return c->top_k > 0 ? std::min(c->top_k, veff) : veff;
}

// Returns an empty string when the configuration is valid.
std::string check_config(const sjd_config* c) {
  if (!c) return "config is NULL";
  if (c->batch < 1) return "batch must be >= 1";
  if (c->window < 1 || c->window > kMaxWindow) return "window must be in [1, 1024]";
  if (c->vocab < 1) return "vocab must be >= 1";
  if (c->allowed_lo < 0 || c->allowed_hi > c->vocab || c->allowed_lo >= c->allowed_hi)
    return "need 0 <= allowed_lo < allowed_hi <= vocab";
  if (!std::isfinite(c->cfg_scale)) return "cfg_scale must be finite";
  if (!(c->temperature > 0.0f) || !std::isfinite(c->temperature)) return "temperature must be > 0";
  if (c->top_k < 0) return "top_k must be >= 0";
  if (!(c->top_p > 0.0f && c->top_p <= 1.0f)) return "top_p must be in (0, 1]";
  if (c->pd_k < 1 || c->pd_k > kMaxK) return "pd_k must be in [1, 8]";
  if (c->pd_depth < 0) return "pd_depth must be >= 0";
  if (c->adaptive_continuation != 0 && c->adaptive_continuation != 1)
    return "adaptive_continuation must be 0 or 1";
  if (c->logit_dtype != SJD_F32 && c->logit_dtype != SJD_BF16) return "logit_dtype must be SJD_F32 or SJD_BF16";
  if (c->support_cap < min_support(c)) return "support_cap must be >= min(top_k, allowed_hi - allowed_lo)";
  if (c->max_steps < 1) return "max_steps must be >= 1";
  if (c->pd_tree != 0 && c->pd_tree != 1) return "pd_tree must be 0 or 1";
  if (c->pd_tree) {
    if (!c->adaptive_continuation) return "the full tree needs adaptive_continuation = 1";
    if (c->pd_k < 2 || c->pd_depth < 1) return "the full tree needs pd_k >= 2 and pd_depth >= 1";
    long long n = 1;
    for (int d = 0; d < c->pd_depth; ++d) n *= c->pd_k;
    if (n > 256) return "the full tree needs pd_k^pd_depth <= 256";
  }
  return std::string();
}

// Workspace layout and the kernel parameters that do not depend on the
// workspace address.
void plan(const sjd_config* c, Layout* L, DevParams* P) {
  const size_t B = c->batch, W = c->window, S = c->support_cap, K = c->pd_k;
  P->group_of = nullptr;  // the lossless acceptance test unless sjd_set_relaxed_groups
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = up(o + bytes, kAlign);
    return at;
  };
  L->q_ids = take(B * W * S * 4);
  L->q_prob = take(B * W * S * 4);
  L->q_len = take(B * W * 4);
  L->cand = take(B * W * K * 4);
  L->gsize = take(B * W * 4);
  L->win_tok = take(B * W * 4);
  L->abs_pos = take(B * 4);
  L->last_tok = take(B * 4);
  L->step_t = take(B * 4);
  // the full tree: K^d token slots at every depth d = 1..D
  size_t tree_n = 0, kd = 1, X = 0;
  for (int d = 1; c->pd_tree && d <= c->pd_depth; ++d) {
    kd *= K;
    tree_n += kd;
    if (d < c->pd_depth) X += kd - 1;
  }
  const size_t tree_g = c->pd_tree ? kd / K - 1 : 0;
  L->tree_tok = take(B * tree_n * 4);
  L->tree_depth = take(B * 4);
  L->persistent_end = o;
  const size_t Km1 = K > 1 ? K - 1 : 1;
  L->res_x = take(B * W * 4);
  L->res_dev = take(B * W * 4);
  L->res_alt = take(B * W * Km1 * 4);
  L->res_altn = take(B * W * 4);
  L->res_xf = take(B * W * 4);
  L->res_altf = take(B * W * Km1 * 4);
  L->res_altfn = take(B * W * 4);
  L->ticket = take(B * 4);
  L->first_rej = take(B * 4);
  L->n_commit = take(B * 4);
  L->committed = take(B * W * 4);
  L->err = take(4 * 4);
  L->stats = take(kStatsWords * 8);
  L->abs_before = take(B * 4);  // decode-loop scratch
  L->res_node = take(B * X * 4);
  L->res_tree = take(B * W * tree_g * K * 4);
  const size_t tq = c->pd_tree ? B * W * S * 4 : 0;
  L->tq_ids = take(tq);
  L->tq_prob = take(tq);
  L->tq_len = take(c->pd_tree ? B * W * 4 : 0);
  L->fast_scratch = o;
  L->total = o;

  std::memset(P, 0, sizeof(*P));
  P->tree = c->pd_tree;
  P->X = static_cast<int>(X);
  P->rows_b = c->window + static_cast<int>(X);
  P->tree_n = static_cast<int>(tree_n);
  P->tree_g = static_cast<int>(tree_g);
  P->B = c->batch;
  P->W = c->window;
  P->V = c->vocab;
  P->lo = c->allowed_lo;
  P->hi = c->allowed_hi;
  P->veff = c->allowed_hi - c->allowed_lo;
  P->K = c->pd_k;
  P->D = c->pd_depth;
  P->ac = c->adaptive_continuation;
  P->S = c->support_cap;
  P->topk = c->top_k > 0 ? std::min(c->top_k, P->veff) : P->veff;
  P->cfg = c->cfg_scale;
  P->temp = c->temperature;
  P->top_p = c->top_p;
  if (c->top_p < 1.0f) {
    uint32_t bits;
    std::memcpy(&bits, &c->top_p, 4);
    const int ex = static_cast<int>((bits >> 23) & 0xFFu);
    uint32_t m = bits & 0x7FFFFFu;
    if (ex) {
      m |= 0x800000u;
      P->tau_shift = 150 - ex;
    } else {
      P->tau_shift = 149;
    }
    P->tau_mant = m;
  }
  P->seed_lo = static_cast<uint32_t>(c->seed & 0xFFFFFFFFull);
  P->seed_hi = static_cast<uint32_t>(c->seed >> 32);
  P->uniform_q = 1.0f / static_cast<float>(P->veff);  // IEEE division, round to nearest
  const int epv = c->logit_dtype == SJD_BF16 ? 8 : 4;  // elements per 16 bytes
  P->al0 = c->allowed_lo / epv * epv;
  P->nL = static_cast<int>(up(static_cast<size_t>(c->allowed_hi), epv)) - P->al0;
  P->row_stride = c->vocab;
  P->col0 = 0;
  // shared memory of the row kernel
  size_t s = 0;
  auto stake = [&](size_t bytes) {
    const size_t at = s;
    s = up(s + bytes, 16);
    return static_cast<uint32_t>(at);
  };
  P->off_lv = stake(static_cast<size_t>(P->nL) * 4);
  P->off_hist = stake(kBins * 8);
  P->off_qid = stake(S * 4);
  P->off_qpr = stake(S * 4);
  P->off_pid = stake(S * 4);
  P->off_pcum = stake(S * 8);
  P->off_pp = stake(S * 4);
  if (16 * S <= static_cast<size_t>(P->nL) * 4) {
    // the logits are dead once the row is compacted: reuse their space
    P->off_qP = P->off_lv;
    P->off_cur = P->off_lv + static_cast<uint32_t>(up(S * 4, 16));
    P->off_Rw = P->off_cur + static_cast<uint32_t>(up(S * 4, 16));
  } else {
    P->off_qP = stake(S * 4);
    P->off_cur = stake(S * 4);
    P->off_Rw = stake(S * 8);
  }
  P->smem_bytes = static_cast<uint32_t>(s);

  // fast path: one 128-thread CTA per row streaming its allowed range once;
  // shared memory = candidate list (reused for the small kept arrays and the
  // staged draft row) + head buffer + select histogram + index bitmap
  P->fast_ok = 0;
  P->fast_cpt = 0;
  P->fast_ctas = 0;
  const size_t esz = c->logit_dtype == SJD_BF16 ? 2 : 4;
  const bool rows_aligned = (static_cast<size_t>(c->vocab) * esz) % 16 == 0 && P->al0 + P->nL <= c->vocab;
  // candidate list: 3072 entries of 8 bytes in shared memory, continued in
  // the workspace up to min(nL, 16384) entries
  const size_t lcap = std::min<size_t>(static_cast<size_t>(P->nL), 3072);
  const size_t lmax = std::min<size_t>(static_cast<size_t>(P->nL), 16384);
  if (!c->pd_tree && rows_aligned && P->nL <= 65535 && static_cast<size_t>(P->topk) <= lmax) {
    // Two layouts. Narrow (many rows, 7 CTAs per SM): the kept arrays (up to
    // 128 ids) and the staged draft row live over the dead candidate list.
    // Wide (few rows, when at most two waves result): kept arrays and draft
    // row for the whole support S, apart from the list.
    const size_t nwords = static_cast<size_t>((P->nL + 31) / 32);
    auto layout = [&](bool wide, DevParams* Q) -> size_t {
      const size_t kcap = wide ? S : 128;
      size_t f = 0;
      auto ftake = [&](size_t bytes) {
        const size_t at = f;
        f = up(f + bytes, 16);
        return static_cast<uint32_t>(at);
      };
      const size_t small_bytes = up(2 * kcap, 16) + 3 * up(4 * kcap, 16) + 2 * up(8 * kcap, 16);
      // the list (lcap entries) and one spare entry the branch-free append writes to
      const size_t region = wide ? up(8 * (lcap + 1), 16) : std::max(up(8 * (lcap + 1), 16), small_bytes + up(8 * 256, 16));
      const uint32_t r0 = ftake(region);
      Q->f_list_l = r0;
      Q->f_list_i = 0;
      Q->f_region_bytes = static_cast<uint32_t>(region);
      uint32_t o = wide ? ftake(small_bytes + up(8 * S, 16)) : r0;
      const uint32_t o0 = o;
      auto rtake = [&](size_t bytes) {
        const uint32_t at = o;
        o += static_cast<uint32_t>(up(bytes, 16));
        return at;
      };
      Q->f_pidx = rtake(2 * kcap);
      Q->f_pcum = rtake(8 * kcap);
      Q->f_pp = rtake(4 * kcap);
      Q->f_qP = rtake(4 * kcap);
      Q->f_cur = rtake(4 * kcap);
      Q->f_Rw = rtake(8 * kcap);
      Q->f_stage = o;  // the draft row stage: the rest of its area
      const size_t area = wide ? small_bytes + up(8 * S, 16) : region;
      Q->f_qcap = static_cast<int>((area - (o - o0)) / 8);
      Q->f_list_w = ftake(128 * 16);  // head buffer
      Q->f_hist = ftake(std::max<size_t>(static_cast<size_t>(kFastBins) * 8, nwords * 4));  // also word prefix counts
      Q->f_bitmap = ftake(nwords * 4);
      Q->f_smem_bytes = static_cast<uint32_t>(f);
      Q->f_kcap = static_cast<int>(kcap);
      Q->f_kwide = wide ? 1 : 0;
      Q->f_nt = wide ? 512 : 128;  // few rows: one wide CTA per SM, more threads per row
      return f + 1024 + 1536;  // + reserved + static scratch
    };
    int sms = 152, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      sms = 152;
    size_t per_cta = layout(false, P);
    if (S > 128) {
      DevParams Q = *P;
      const size_t per_wide = layout(true, &Q);
      // one 512-thread CTA per SM (its registers allow no second)
      const size_t ctas = per_wide <= 227 * 1024 ? 1 : 0;
      if (ctas >= 1 && B * W <= 2 * static_cast<size_t>(sms) * ctas) {
        *P = Q;
        per_cta = per_wide;
      }
    }
    P->f_lcap = static_cast<int>(lcap);
    const size_t gcap = lmax - lcap;
    P->f_gcap = static_cast<int>(gcap);
    P->f_glist = up(32 * S, 256);
    P->f_row_bytes = P->f_glist + up(8 * gcap, 256);
    if (per_cta <= 227 * 1024) {
      P->fast_ok = 1;
      P->fast_ctas = static_cast<int>(std::min<size_t>(8, (228 * 1024) / per_cta));
    }
  }
  if (P->fast_ok) L->total = L->fast_scratch + B * W * P->f_row_bytes;
}

}  // namespace sjd

namespace {

constexpr size_t kAlign = 256;
constexpr uint32_t kStateMagic = 0x53444A31u;  // "SDJ1"

size_t up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int fail(sjd_ctx* c, int code, const std::string& why) {
  if (c) c->last_error = why;
  return code;
}

void bind(sjd_ctx* c) {
  unsigned char* w = c->ws;
  const Layout& L = c->L;
  DevParams& P = c->P;
  P.q_ids = reinterpret_cast<int32_t*>(w + L.q_ids);
  P.q_prob = reinterpret_cast<float*>(w + L.q_prob);
  P.q_len = reinterpret_cast<int32_t*>(w + L.q_len);
  P.cand = reinterpret_cast<int32_t*>(w + L.cand);
  P.gsize = reinterpret_cast<int32_t*>(w + L.gsize);
  P.win_tok = reinterpret_cast<int32_t*>(w + L.win_tok);
  P.abs_pos = reinterpret_cast<int32_t*>(w + L.abs_pos);
  P.last_tok = reinterpret_cast<int32_t*>(w + L.last_tok);
  P.step_t = reinterpret_cast<uint32_t*>(w + L.step_t);
  P.res_x = reinterpret_cast<int32_t*>(w + L.res_x);
  P.res_dev = reinterpret_cast<int32_t*>(w + L.res_dev);
  P.res_alt = reinterpret_cast<int32_t*>(w + L.res_alt);
  P.res_altn = reinterpret_cast<int32_t*>(w + L.res_altn);
  P.res_xf = reinterpret_cast<int32_t*>(w + L.res_xf);
  P.res_altf = reinterpret_cast<int32_t*>(w + L.res_altf);
  P.res_altfn = reinterpret_cast<int32_t*>(w + L.res_altfn);
  P.ticket = reinterpret_cast<uint32_t*>(w + L.ticket);
  P.first_rej = reinterpret_cast<int32_t*>(w + L.first_rej);
  P.n_commit = reinterpret_cast<int32_t*>(w + L.n_commit);
  P.committed = reinterpret_cast<int32_t*>(w + L.committed);
  P.err = reinterpret_cast<uint32_t*>(w + L.err);
  P.stats = reinterpret_cast<unsigned long long*>(w + L.stats);
  P.tree_tok = reinterpret_cast<int32_t*>(w + L.tree_tok);
  P.tree_depth = reinterpret_cast<int32_t*>(w + L.tree_depth);
  P.res_node = reinterpret_cast<int32_t*>(w + L.res_node);
  P.res_tree = reinterpret_cast<int32_t*>(w + L.res_tree);
  P.tq_ids = reinterpret_cast<int32_t*>(w + L.tq_ids);
  P.tq_prob = reinterpret_cast<float*>(w + L.tq_prob);
  P.tq_len = reinterpret_cast<int32_t*>(w + L.tq_len);
  P.f_scratch = w + L.fast_scratch;
  c->abs_before = reinterpret_cast<int32_t*>(w + L.abs_before);
}

int cuda_fail(sjd_ctx* c, cudaError_t e, const char* what) {
  return fail(c, SJD_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// 128-bit loads are possible when every row starts on a 16-byte boundary.
bool vec_ok(const sjd_ctx* c, const void* a, const void* b) {
  const size_t esz = c->cfg.logit_dtype == SJD_BF16 ? 2 : 4;
  if ((static_cast<size_t>(c->cfg.vocab) * esz) % 16 != 0) return false;
  if (static_cast<size_t>(c->P.al0 + c->P.nL) > static_cast<size_t>(c->cfg.vocab)) return false;
  return aligned16(a) && (b == nullptr || aligned16(b));
}

int launch_rows_p(sjd_ctx* c, const sjd::DevParams& P0, bool vec, int mode, const void* cond, const void* uncond,
                  int32_t* oc, int32_t* on, int32_t* of) {
  const bool use_cfg = uncond != nullptr && c->cfg.cfg_scale != 1.0f;
  sjd::DevParams P = P0;
  if (mode == sjd::kModeFromLogits) {  // draft logits: the window rows only, no tree
    P.tree = 0;
    P.X = 0;
    P.rows_b = P.W;
  }
  cudaError_t e;
  if (vec && P.fast_ok && !c->force_general) {
    e = sjd::launch_fast_row(P, mode, c->cfg.logit_dtype, cond, use_cfg ? uncond : nullptr, use_cfg, oc, on, of,
                             c->stream);
  } else {
    e = sjd::launch_row(P, mode, c->cfg.logit_dtype, vec, cond, use_cfg ? uncond : nullptr, use_cfg, oc, on, of,
                        c->stream);
  }
  return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "row kernel launch");
}

int launch_rows(sjd_ctx* c, int mode, const void* cond, const void* uncond, int32_t* oc,
                int32_t* on, int32_t* of) {
  return launch_rows_p(c, c->P, vec_ok(c, cond, uncond), mode, cond, uncond, oc, on, of);
}

// The caller's logits of sjd_step / sjd_verify_step, with the early-logits
// guarantee when the context has it.
int launch_rows_caller(sjd_ctx* c, int mode, const void* cond, const void* uncond, int32_t* oc,
                       int32_t* on, int32_t* of) {
  sjd::DevParams P = c->P;
  P.early_logits = c->early_logits ? 1 : 0;
  return launch_rows_p(c, P, vec_ok(c, cond, uncond), mode, cond, uncond, oc, on, of);
}

int device_error_code(uint32_t bits) {
  for (int code = 1; code < 32; ++code)
    if (bits & sjd::err_bit(code)) return code;
  return SJD_OK;
}

const char* code_text(int code) {
  switch (code) {
    case SJD_ERR_NONFINITE: return "NaN or +inf logit in the allowed range (or no finite logit)";
    case SJD_ERR_INVALID_DRAFT: return "a draft token has zero draft probability";
    case SJD_ERR_CAPACITY: return "sparse row capacity exceeded";
    case SJD_ERR_BOUNDS: return "an index outside its array (bounds-checked build); the access was clamped";
    case SJD_ERR_TIMEOUT: return "a bounded wait inside a kernel ran out (reserved: no current kernel waits)";
    default: return "device error";
  }
}

}  // namespace

extern "C" {

size_t sjd_workspace_size(const sjd_config* cfg) {
  if (!sjd::check_config(cfg).empty()) return 0;
  Layout L;
  DevParams P{};
  sjd::plan(cfg, &L, &P);
  return L.total;
}

int sjd_init(const sjd_config* cfg, void* workspace_dev, size_t ws_bytes, void* cuda_stream,
             sjd_ctx** out) {
  if (!out) return SJD_ERR_ARG;
  *out = nullptr;
  const std::string why = sjd::check_config(cfg);
  if (!why.empty()) return SJD_ERR_ARG;
  if (!workspace_dev || (reinterpret_cast<uintptr_t>(workspace_dev) % kAlign) != 0) return SJD_ERR_ARG;
  sjd_ctx* c = new (std::nothrow) sjd_ctx();
  if (!c) return SJD_ERR_CAPACITY;
  c->cfg = *cfg;
  sjd::plan(cfg, &c->L, &c->P);
  c->stream = static_cast<cudaStream_t>(cuda_stream);
  c->ws = static_cast<unsigned char*>(workspace_dev);
  c->ws_bytes = ws_bytes;
  c->pending = false;
  if (ws_bytes < c->L.total) {
    delete c;
    return SJD_ERR_CAPACITY;
  }
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) {
    delete c;
    return SJD_ERR_CUDA;
  }
  if (c->P.smem_bytes + 2048 > static_cast<uint32_t>(optin)) {
    delete c;
    return SJD_ERR_CAPACITY;
  }
  bind(c);
  {
    const char* k = std::getenv("SJD_KERNEL");
    c->force_general = k != nullptr && std::strcmp(k, "general") == 0;
  }
  e = sjd::raise_row_kernel_smem_all(static_cast<int>(c->P.smem_bytes));
  if (e == cudaSuccess && c->P.fast_ok) e = sjd::raise_fast_row_kernel_smem(static_cast<int>(c->P.f_smem_bytes));
  if (e == cudaSuccess) e = cudaMemsetAsync(c->ws, 0, c->L.total, c->stream);
  if (e == cudaSuccess) e = sjd::launch_init(c->P, c->stream);
  if (e != cudaSuccess) {
    delete c;
    return SJD_ERR_CUDA;
  }
  *out = c;
  return SJD_OK;
}

int sjd_verify_step(sjd_ctx* c, const void* cond, const void* uncond, int32_t* committed,
                    int32_t* n_commit, int32_t* first_rej) {
  if (!c) return SJD_ERR_ARG;
  if (!cond) return fail(c, SJD_ERR_ARG, "cond logits are NULL");
  if (!uncond && c->cfg.cfg_scale != 1.0f) return fail(c, SJD_ERR_ARG, "uncond logits are NULL but cfg_scale != 1");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending: call sjd_draft(SJD_DRAFT_PD) first");
  if (c->cfg.pd_tree) return fail(c, SJD_ERR_ARG, "with the full tree the step runs fused (sjd_step)");
  const int rc = launch_rows_caller(c, sjd::kModeVerify, cond, uncond, committed, n_commit, first_rej);
  if (rc == SJD_OK) c->pending = true;
  return rc;
}

int sjd_step(sjd_ctx* c, const void* cond, const void* uncond, int32_t* committed,
             int32_t* n_commit, int32_t* first_rej) {
  if (!c) return SJD_ERR_ARG;
  if (!cond) return fail(c, SJD_ERR_ARG, "cond logits are NULL");
  if (!uncond && c->cfg.cfg_scale != 1.0f) return fail(c, SJD_ERR_ARG, "uncond logits are NULL but cfg_scale != 1");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending: call sjd_draft(SJD_DRAFT_PD) first");
  return launch_rows_caller(c, sjd::kModeStep, cond, uncond, committed, n_commit, first_rej);
}

int sjd_set_early_logits(sjd_ctx* c, int32_t enable) {
  if (!c) return SJD_ERR_ARG;
  c->early_logits = enable != 0;
  return SJD_OK;
}

size_t sjd_host_stage_size(const sjd_config* cfg) {
  if (!cfg || !sjd::check_config(cfg).empty()) return 0;
  sjd::Layout L;
  sjd::DevParams P{};
  sjd::plan(cfg, &L, &P);
  const size_t esz = cfg->logit_dtype == SJD_BF16 ? 2 : 4;
  const size_t one = static_cast<size_t>(cfg->batch) * cfg->window * static_cast<size_t>(P.nL) * esz;
  return 4 * up(one, 256);  // two stages of cond + uncond
}

int sjd_step_host(sjd_ctx* c, const void* cond_host, const void* uncond_host, int64_t host_row_pitch,
                  void* stage_dev, size_t stage_bytes, int32_t* committed, int32_t* n_commit, int32_t* first_rej) {
  if (!c) return SJD_ERR_ARG;
  const bool use_cfg = c->cfg.cfg_scale != 1.0f;
  if (!cond_host || !stage_dev) return fail(c, SJD_ERR_ARG, "host logits or stage buffer are NULL");
  if (use_cfg && !uncond_host) return fail(c, SJD_ERR_ARG, "uncond logits are NULL but cfg_scale != 1");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending: call sjd_draft(SJD_DRAFT_PD) first");
  if (c->cfg.pd_tree) return fail(c, SJD_ERR_ARG, "the full tree takes device logits (sjd_step)");
  const size_t esz = c->cfg.logit_dtype == SJD_BF16 ? 2 : 4;
  const size_t rows = static_cast<size_t>(c->cfg.batch) * c->cfg.window;
  const size_t nL = static_cast<size_t>(c->P.nL);
  const size_t one = up(rows * nL * esz, 256);
  if (host_row_pitch < c->cfg.vocab) return fail(c, SJD_ERR_ARG, "host_row_pitch below the vocabulary size");
  if (stage_bytes < 2 * one) return fail(c, SJD_ERR_CAPACITY, "stage buffer below sjd_host_stage_size()");
  if ((reinterpret_cast<uintptr_t>(stage_dev) & 255u) != 0) return fail(c, SJD_ERR_ARG, "stage buffer not 256-byte aligned");
  // The allowed columns [al0, al0 + nL) of every row (clipped to the row)
  // are copied into a stage as compact rows of nL, one 2-D copy per tensor.
  // With two stages (and the stream not being captured), the copies run on
  // the context's copy stream: a step's copy overlaps the kernel of the step
  // before, and waits only for the kernel that read its stage.
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(c->stream, &cap) != cudaSuccess) return cuda_fail(c, cudaGetLastError(), "capture query");
  const bool two = stage_bytes >= 4 * one && cap == cudaStreamCaptureStatusNone;
  if (two && !c->copy_stream[0]) {
    cudaError_t e = cudaSuccess;
    for (int i = 0; i < sjd_ctx::kCopyStreams && e == cudaSuccess; ++i) {
      e = cudaStreamCreateWithFlags(&c->copy_stream[i], cudaStreamNonBlocking);
      for (int k = 0; k < 2 && e == cudaSuccess; ++k)
        e = cudaEventCreateWithFlags(&c->ev_copied[k][i], cudaEventDisableTiming);
    }
    for (int k = 0; k < 2 && e == cudaSuccess; ++k)
      e = cudaEventCreateWithFlags(&c->ev_consumed[k], cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(c, e, "copy stream set-up");
  }
  const int slot = two ? c->next_stage : 0;
  const int nstreams = two ? sjd_ctx::kCopyStreams : 1;
  const size_t width = std::min(nL, static_cast<size_t>(c->cfg.vocab - c->P.al0)) * esz;
  unsigned char* sc = static_cast<unsigned char*>(stage_dev) + static_cast<size_t>(slot) * 2 * one;
  unsigned char* su = sc + one;
  const size_t spitch = static_cast<size_t>(host_row_pitch) * esz;
  cudaError_t e = cudaSuccess;
  for (int i = 0; i < nstreams && e == cudaSuccess; ++i) {
    cudaStream_t cs = two ? c->copy_stream[i] : c->stream;
    const size_t r0 = rows * i / nstreams, r1 = rows * (i + 1) / nstreams;  // this stream's rows
    if (two) e = cudaStreamWaitEvent(cs, c->ev_consumed[slot], 0);
    if (e == cudaSuccess && r1 > r0)
      e = cudaMemcpy2DAsync(sc + r0 * nL * esz, nL * esz,
                            static_cast<const unsigned char*>(cond_host) + (r0 * static_cast<size_t>(host_row_pitch) + c->P.al0) * esz,
                            spitch, width, r1 - r0, cudaMemcpyHostToDevice, cs);
    if (e == cudaSuccess && use_cfg && r1 > r0)
      e = cudaMemcpy2DAsync(su + r0 * nL * esz, nL * esz,
                            static_cast<const unsigned char*>(uncond_host) + (r0 * static_cast<size_t>(host_row_pitch) + c->P.al0) * esz,
                            spitch, width, r1 - r0, cudaMemcpyHostToDevice, cs);
    if (e == cudaSuccess && two) e = cudaEventRecord(c->ev_copied[slot][i], cs);
    if (e == cudaSuccess && two) e = cudaStreamWaitEvent(c->stream, c->ev_copied[slot][i], 0);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "host logits copy");
  sjd::DevParams P = c->P;
  P.row_stride = static_cast<long long>(nL);
  P.col0 = P.al0;
  const int rc = launch_rows_p(c, P, true, sjd::kModeStep, sc, use_cfg ? su : nullptr, committed, n_commit, first_rej);
  if (rc == SJD_OK && two) {
    e = cudaEventRecord(c->ev_consumed[slot], c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "stage event");
    c->next_stage ^= 1;
  }
  return rc;
}

int sjd_draft(sjd_ctx* c, int32_t mode, const void* q_cond, const void* q_uncond) {
  if (!c) return SJD_ERR_ARG;
  cudaError_t e;
  switch (mode) {
    case SJD_DRAFT_PD:
      if (q_cond || q_uncond) return fail(c, SJD_ERR_ARG, "SJD_DRAFT_PD takes no logits");
      if (!c->pending) return fail(c, SJD_ERR_STATE, "SJD_DRAFT_PD needs a pending sjd_verify_step");
      e = sjd::launch_refresh(c->P, c->stream);
      if (e != cudaSuccess) return cuda_fail(c, e, "refresh kernel launch");
      c->pending = false;
      return SJD_OK;
    case SJD_DRAFT_FROM_LOGITS: {
      if (!q_cond) return fail(c, SJD_ERR_ARG, "draft logits are NULL");
      if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending");
      const int rc = launch_rows(c, sjd::kModeFromLogits, q_cond, q_uncond, nullptr, nullptr, nullptr);
      if (rc == SJD_OK && c->cfg.pd_tree) {  // a window drafted afresh carries no tree
        e = cudaMemsetAsync(c->P.tree_depth, 0, static_cast<size_t>(c->cfg.batch) * 4, c->stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "tree reset");
      }
      return rc;
    }
    case SJD_DRAFT_UNIFORM:
      if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending");
      e = sjd::launch_init(c->P, c->stream);
      return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "init kernel launch");
    default:
      return fail(c, SJD_ERR_ARG, "unknown draft mode");
  }
}

int sjd_decode_loop(sjd_ctx* c, sjd_forward_fn forward, void* user, void* cond_buf,
                    void* uncond_buf, int32_t n_tokens, int32_t* grid, int32_t* accept_len,
                    int32_t* n_steps_out) {
  if (!c) return SJD_ERR_ARG;
  if (c->cfg.pd_tree) return fail(c, SJD_ERR_ARG, "the full tree is stepped with sjd_step and sjd_get_tree");
  if (!forward || !cond_buf || !grid || n_tokens < 1)
    return fail(c, SJD_ERR_ARG, "decode loop needs a forward, a cond buffer, a grid and n_tokens >= 1");
  if (!uncond_buf && c->cfg.cfg_scale != 1.0f) return fail(c, SJD_ERR_ARG, "uncond buffer is NULL but cfg_scale != 1");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending");
  const int B = c->cfg.batch;
  std::vector<int32_t> abs_host(B);
  int steps = 0;
  int rc = SJD_OK;
  bool done = false;
  while (true) {
    cudaError_t e = cudaMemcpyAsync(abs_host.data(), c->P.abs_pos, B * 4, cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "decode loop readback");
    done = true;
    int min_pos = n_tokens;
    for (int b = 0; b < B; ++b) {
      done = done && abs_host[b] >= n_tokens;
      min_pos = std::min(min_pos, abs_host[b]);
    }
    if (done || steps >= c->cfg.max_steps) break;
    // A step commits at most W tokens per batch element, so the slowest one
    // cannot finish in fewer than ceil((n_tokens - min_pos) / W) steps: they
    // run without reading the positions back, and the loop takes exactly the
    // steps it would take checking after every step.
    const int W = c->cfg.window;
    const int burst = std::max(1, std::min((n_tokens - min_pos + W - 1) / W, c->cfg.max_steps - steps));
    for (int i = 0; i < burst && rc == SJD_OK; ++i) {
      if (forward(user, c->P.win_tok, c->P.last_tok, c->P.abs_pos, cond_buf, uncond_buf, c->stream) != 0) {
        rc = fail(c, SJD_ERR_CALLBACK, "forward callback failed");
        break;
      }
      e = cudaMemcpyAsync(c->abs_before, c->P.abs_pos, B * 4, cudaMemcpyDeviceToDevice, c->stream);
      if (e != cudaSuccess) return cuda_fail(c, e, "decode loop copy");
      rc = launch_rows(c, sjd::kModeStep, cond_buf, uncond_buf, nullptr, nullptr, nullptr);
      if (rc != SJD_OK) break;
      e = sjd::launch_append(c->P, c->abs_before, n_tokens, grid,
                             accept_len ? accept_len + static_cast<size_t>(steps) * B : nullptr, c->stream);
      if (e != cudaSuccess) return cuda_fail(c, e, "append kernel launch");
      ++steps;
    }
    if (rc != SJD_OK) break;
  }
  if (n_steps_out) *n_steps_out = steps;
  if (rc != SJD_OK) return rc;
  const int dev_rc = sjd_sync(c);
  if (dev_rc != SJD_OK) return dev_rc;
  if (!done) return fail(c, SJD_ERR_STEP_LIMIT, "decode loop reached max_steps");
  return SJD_OK;
}

int sjd_get_window(sjd_ctx* c, int32_t* tokens, int32_t* cands, int32_t* group, int32_t* abs_pos,
                   int32_t* prev) {
  if (!c) return SJD_ERR_ARG;
  if (!tokens) return fail(c, SJD_ERR_ARG, "tokens buffer is NULL");
  const cudaError_t e = sjd::launch_get_window(c->P, tokens, cands, group, abs_pos, prev, c->stream);
  return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "get_window launch");
}

int sjd_get_tree(sjd_ctx* c, int32_t* tokens, int32_t* depth) {
  if (!c) return SJD_ERR_ARG;
  if (!c->cfg.pd_tree) return fail(c, SJD_ERR_ARG, "the configuration has no full tree");
  cudaError_t e = cudaSuccess;
  if (tokens)
    e = cudaMemcpyAsync(tokens, c->P.tree_tok, static_cast<size_t>(c->cfg.batch) * c->P.tree_n * 4,
                        cudaMemcpyDeviceToDevice, c->stream);
  if (e == cudaSuccess && depth)
    e = cudaMemcpyAsync(depth, c->P.tree_depth, static_cast<size_t>(c->cfg.batch) * 4, cudaMemcpyDeviceToDevice,
                        c->stream);
  return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "tree copy");
}

int sjd_get_rows(sjd_ctx* c, int32_t* ids, float* probs, int32_t* len) {
  if (!c) return SJD_ERR_ARG;
  if (!ids || !probs || !len) return fail(c, SJD_ERR_ARG, "row buffers are NULL");
  const cudaError_t e = sjd::launch_get_rows(c->P, ids, probs, len, c->stream);
  return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "get_rows launch");
}

int sjd_get_state(sjd_ctx* c, void* host_blob, size_t* bytes) {
  if (!c || !bytes) return SJD_ERR_ARG;
  const size_t need = 16 + sizeof(sjd_config) + c->L.persistent_end;
  if (!host_blob) {
    *bytes = need;
    return SJD_OK;
  }
  if (*bytes < need) return fail(c, SJD_ERR_ARG, "state buffer too small");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending");
  unsigned char* h = static_cast<unsigned char*>(host_blob);
  const uint32_t hdr[4] = {kStateMagic, static_cast<uint32_t>(sizeof(sjd_config)),
                           static_cast<uint32_t>(c->L.persistent_end & 0xFFFFFFFFu),
                           static_cast<uint32_t>(c->L.persistent_end >> 32)};
  std::memcpy(h, hdr, 16);
  std::memcpy(h + 16, &c->cfg, sizeof(sjd_config));
  cudaError_t e = cudaMemcpyAsync(h + 16 + sizeof(sjd_config), c->ws, c->L.persistent_end,
                                  cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "get_state copy");
  *bytes = need;
  return SJD_OK;
}

int sjd_set_state(sjd_ctx* c, const void* host_blob, size_t bytes) {
  if (!c || !host_blob) return SJD_ERR_ARG;
  const size_t need = 16 + sizeof(sjd_config) + c->L.persistent_end;
  if (bytes != need) return fail(c, SJD_ERR_ARG, "state size mismatch");
  if (c->pending) return fail(c, SJD_ERR_STATE, "a verify is pending");
  const unsigned char* h = static_cast<const unsigned char*>(host_blob);
  uint32_t hdr[4];
  std::memcpy(hdr, h, 16);
  if (hdr[0] != kStateMagic || hdr[1] != sizeof(sjd_config)) return fail(c, SJD_ERR_ARG, "not a state blob");
  if (std::memcmp(h + 16, &c->cfg, sizeof(sjd_config)) != 0)
    return fail(c, SJD_ERR_ARG, "state blob from a different configuration");
  cudaError_t e = cudaMemcpyAsync(c->ws, h + 16 + sizeof(sjd_config), c->L.persistent_end,
                                  cudaMemcpyHostToDevice, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  return e == cudaSuccess ? SJD_OK : cuda_fail(c, e, "set_state copy");
}

int sjd_stats_ex(sjd_ctx* c, uint64_t* out, int32_t n) {
  if (!c || !out || n < 0) return SJD_ERR_ARG;
  uint64_t raw[sjd::kStatsWords];
  cudaError_t e = cudaMemcpyAsync(raw, c->P.stats, sizeof(raw), cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "stats copy");
  uint64_t all[6];
  for (int k = 0; k < 4; ++k) all[k] = raw[k];
  for (int slot = 0; slot < sjd::kStatsSlots; ++slot)
    for (int k = 0; k < 3; ++k) all[k] += raw[sjd::kStatsSpread + 3 * slot + k];
  all[4] = raw[sjd::kStatsPaths];
  all[5] = raw[sjd::kStatsPaths + 1];
  for (int k = 0; k < n && k < 6; ++k) out[k] = all[k];
  return SJD_OK;
}

int sjd_stats(sjd_ctx* c, uint64_t* out4) { return sjd_stats_ex(c, out4, 4); }

int sjd_sync(sjd_ctx* c) {
  if (!c) return SJD_ERR_ARG;
  uint32_t bits = 0;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&bits, c->P.err, 4, cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->P.err, 0, 4, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "sync");
  const int code = device_error_code(bits);
  if (code != SJD_OK) c->last_error = code_text(code);
  return code;
}

int sjd_set_relaxed_groups(sjd_ctx* c, const int32_t* group_of_dev) {
  if (!c) return SJD_ERR_ARG;
  c->P.group_of = group_of_dev;
  return SJD_OK;
}

int sjd_row_path(const sjd_ctx* c) {
  if (!c) return -1;
  return (c->P.fast_ok && !c->force_general) ? 1 : 0;
}

const char* sjd_last_error(const sjd_ctx* c) {
  if (!c) return "no context";
  return c->last_error.c_str();
}

void sjd_destroy(sjd_ctx* c) { delete c; }

}  // extern "C"
