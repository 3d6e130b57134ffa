// Internal definitions shared by the kernels (sjd_kernels.cu) and the host
// API (sjd_api.cu): workspace layout, kernel parameters, launch entry points.
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>

#include <cuda_runtime.h>

#include "sjd.h"

namespace sjd {

constexpr int kThreads = 512;          // threads of the row kernel
constexpr int kWarps = kThreads / 32;
constexpr int kBins = 2048;            // histogram bins of the threshold select
constexpr int kCandMax = 1024;         // candidates resolved by ranking
constexpr int kMaxK = 8;               // largest PD group (K)
constexpr int kMaxWindow = 1024;
constexpr int kFixBits = 47;           // weights are integers in units of 2^-47

// Philox purposes (counter word 3).
enum Purpose : uint32_t { kAccept = 0, kResidual = 1, kPd = 2, kInit = 3, kSynth = 4, kTree = 5 };

// Error bits of the device status word: bit (code - 1) for code = SJD_ERR_*.
__host__ __device__ constexpr uint32_t err_bit(int code) { return 1u << (code - 1); }

// Row-kernel modes.
enum RowMode : int { kModeVerify = 0, kModeStep = 1, kModeFromLogits = 2 };

// Everything a kernel needs, passed by value.
struct DevParams {
  // problem
  int B, W, V, lo, hi, veff, K, D, ac, S, topk;   // topk = effective k (<= veff)
  float cfg, temp, top_p;
  uint32_t tau_mant;  // top_p = tau_mant * 2^-tau_shift (exact), used when top_p < 1
  int tau_shift;
  uint32_t seed_lo, seed_hi;
  float uniform_q;    // fl32(1 / veff)
  // aligned element range held in shared memory: ids [al0, al0 + nL)
  int al0, nL;
  // logit rows in memory: row r starts row_stride elements after row r - 1,
  // and its element for id v is at v - col0 (full rows: vocab and 0)
  long long row_stride;
  int col0;
  // shared-memory layout (byte offsets) of the row kernel
  uint32_t off_lv, off_hist, off_qid, off_qpr, off_pid, off_pcum, off_pp, off_qP, off_cur, off_Rw;
  uint32_t smem_bytes;
  // fast path (sjd_fast.cuh): one streaming CTA per row; shared-memory layout
  // in bytes (0 in fast_ok: the configuration takes the general kernel)
  // the caller guarantees that each step's logits were written before the
  // previous kernel of the stream started: the fast kernel then streams
  // them before that kernel ends and waits only before reading the state
  int early_logits;
  int fast_ok;               // the fast kernel applies to this configuration
  int fast_cpt, fast_ctas;   // (unused by the streaming kernel) ; CTAs per SM
  int f_lcap;                // capacity of the candidate list in shared memory
  int f_gcap;                // capacity of its continuation in the workspace
  int f_qcap, f_kcap;        // draft-row staging and small kept-array capacities
  uint32_t f_region_bytes;   // size of the candidate-list region (reused by the epilogue)
  int f_kwide;               // kept arrays apart from the list (sized for the support S)
  int f_nt;                  // threads per CTA of the fast kernel: 128 (narrow) or 512 (wide)
  size_t f_row_bytes;        // workspace scratch per row: large kept rows, list continuation
  size_t f_glist;            // offset of the list continuation (8 bytes per entry) in it
  unsigned char* f_scratch;  // [B*W] x f_row_bytes
  uint32_t f_stage, f_list_l, f_list_i, f_list_w, f_qP, f_cur, f_Rw, f_pidx, f_pcum, f_pp, f_hist,
      f_bitmap, f_smem_bytes;
  // persistent state (window slot s of batch b holds absolute positions p
  // with p % W == s; row j of the window is slot (abs_pos[b] + j) % W)
  int32_t* q_ids;      // [B][W][S] ascending ids of the stored draft row
  float* q_prob;       // [B][W][S]
  int32_t* q_len;      // [B][W]    -1: uniform on [lo, hi)
  int32_t* cand;       // [B][W][K] candidate group, cand[0] = the draft
  int32_t* gsize;      // [B][W]
  int32_t* win_tok;    // [B][W]    main-path tokens in window order
  int32_t* abs_pos;    // [B]
  int32_t* last_tok;   // [B]
  uint32_t* step_t;    // [B]
  // per-step results
  int32_t* res_x;      // [B][W] verified token x_j^t (per slot)
  int32_t* res_dev;    // [B][W] x_j^t != c_1
  int32_t* res_alt;    // [B][W][K-1] alternates drawn excluding res_x
  int32_t* res_altn;   // [B][W]
  int32_t* res_xf;     // [B][W] vanilla-SJD tail draw (ac = 0)
  int32_t* res_altf;   // [B][W][K-1]
  int32_t* res_altfn;  // [B][W]
  uint32_t* ticket;    // [B] last-CTA-done counters (reset by the last CTA)
  int32_t* first_rej;  // [B] of the last verify
  int32_t* n_commit;   // [B]
  int32_t* committed;  // [B][W] of the last verify
  uint32_t* err;       // status word
  unsigned long long* stats;  // [kStatsWords]
  // relaxed (lossy) acceptance: token group of every vocabulary id, or
  // nullptr for the lossless test (sjd_set_relaxed_groups)
  const int32_t* group_of;
  // full proactive-drafting tree (tree != 0; general row kernel only):
  // every batch element has rows_b = W + X logit rows, the X after its
  // window rows being the nodes off the main path at depths 1..D-1 (node i
  // >= 1 at depth d is row W + sum_{e<d} (K^e - 1) + i - 1)
  int tree, X, rows_b;
  int tree_n;          // token slots per batch element: sum_{d=1..D} K^d (depth d from sum_{e<d} K^e)
  int tree_g;          // extra groups a window row draws for the next tree: K^(D-1) - 1
  int32_t* tree_tok;   // [B][tree_n] tokens of the tree in the window (-1: no such node)
  int32_t* tree_depth; // [B] depth of that tree (0: none)
  int32_t* res_node;   // [B][X] the result token of each node row
  int32_t* res_tree;   // [B][W][tree_g][K] groups drawn by each window row (per slot; -1: none)
  int32_t* tq_ids;     // [B][W][S] the step's P rows, held until every row has read the old ones
  float* tq_prob;      // [B][W][S]
  int32_t* tq_len;     // [B][W]
};

// Counters: [0..3] totals written by the general kernel; the fast kernel
// spreads (rows, draft entries read, target entries written) over
// kStatsSlots slots from kStatsSpread to avoid one hot address.
constexpr int kStatsSpread = 4;
constexpr int kStatsSlots = 32;
// then the fast kernel's fallbacks: rows streamed a second time, rows whose
// top-k cut was taken over the row read again (the candidate list too long)
constexpr int kStatsPaths = kStatsSpread + 3 * kStatsSlots;
constexpr int kStatsWords = kStatsPaths + 2;

struct Layout {
  size_t q_ids, q_prob, q_len, cand, gsize, win_tok, abs_pos, last_tok, step_t, tree_tok, tree_depth;
  size_t persistent_end;
  size_t res_x, res_dev, res_alt, res_altn, res_xf, res_altf, res_altfn, ticket, first_rej,
      n_commit, committed, err, stats, abs_before, res_node, res_tree, tq_ids, tq_prob, tq_len, fast_scratch;
  size_t total;
};

// Launchers (sjd_kernels.cu). All return cudaGetLastError() after launch.
cudaError_t launch_init(const DevParams& p, cudaStream_t s);
cudaError_t launch_row(const DevParams& p, int mode, int dtype, bool vec, const void* cond,
                       const void* uncond, bool use_cfg, int32_t* out_committed,
                       int32_t* out_ncommit, int32_t* out_firstrej, cudaStream_t s);
cudaError_t launch_refresh(const DevParams& p, cudaStream_t s);
cudaError_t launch_get_window(const DevParams& p, int32_t* tokens, int32_t* cands, int32_t* group,
                              int32_t* abs_pos, int32_t* prev, cudaStream_t s);
cudaError_t launch_get_rows(const DevParams& p, int32_t* ids, float* probs, int32_t* len,
                            cudaStream_t s);
cudaError_t launch_append(const DevParams& p, const int32_t* abs_before, int32_t n_tokens,
                          int32_t* grid, int32_t* accept_len_row, cudaStream_t s);
// Raise (never lower) the dynamic shared-memory limit of every general row kernel.
cudaError_t raise_row_kernel_smem_all(int bytes);
// Fast path (sjd_fast.cu, kernels in sjd_fast.cuh): thread count, launch and shared-memory set-up.
constexpr int kFastThreads = 128;
constexpr int kFastBins = 256;
cudaError_t launch_fast_row(const DevParams& p, int mode, int dtype, const void* cond, const void* uncond,
                            bool use_cfg, int32_t* out_committed, int32_t* out_ncommit,
                            int32_t* out_firstrej, cudaStream_t s);
// Raise (never lower) the dynamic shared-memory limit of every fast row kernel.
cudaError_t raise_fast_row_kernel_smem(int bytes);
// One (dtype, mode) variant of the fast row kernels (sjd_fast.cuh, each
// instantiated in its own translation unit, sjd_fast_part.cu).
template <int DT, int MODE>
cudaError_t fast_launch(const DevParams& p, const void* cond, const void* uncond, bool use_cfg, int32_t* oc,
                        int32_t* on, int32_t* of, cudaStream_t s);
template <int DT, int MODE>
cudaError_t fast_raise_smem(int bytes);
// Raise (never lower) the dynamic shared-memory limit of the fused-step kernels.
cudaError_t raise_row_kernel_smem(int bytes);

// Configuration checks and layout (sjd_api.cu). check_config returns an
// empty string when cfg is valid; plan fills the workspace layout and the
// address-independent kernel parameters.
std::string check_config(const sjd_config* cfg);
void plan(const sjd_config* cfg, Layout* L, DevParams* P);

}  // namespace sjd
