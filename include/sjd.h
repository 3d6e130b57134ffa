/*
 * sjd.h -- C ABI of the GB300 SJD-PAC verify-and-draft library (libsjd.so).
 *
 * SJD-PAC (Kang et al., CVPR 2026) decodes an autoregressive VQ-token image
 * model with a Jacobi window of W (the paper's L) draft tokens. One forward
 * pass of the model over the window yields the target distributions P^t; one
 * pass of this library then verifies every window position against its
 * stale draft distribution, continues past the first rejection (adaptive
 * continuation, Sec. 4.2), drafts K alternatives at the D positions after
 * the first rejection (proactive drafting, Sec. 4.1), shifts the window by
 * the number of committed tokens and refills it (Sec. 3.3), and keeps P^t as
 * the next step's draft distributions (Alg. 1, "Return X^t, P^t").
 *
 * Conventions (all entry points):
 *  - Every pointer named *_dev is device memory owned by the caller. The
 *    library never allocates device memory; its whole state lives in the
 *    caller's workspace (sjd_workspace_size / sjd_init).
 *  - Calls are asynchronous on the CUDA stream given to sjd_init, except
 *    sjd_sync, sjd_get_state, sjd_set_state and sjd_decode_loop, which
 *    synchronise that stream.
 *  - Logit tensors are row-major [B][W][V] (vocabulary innermost), fp32 or
 *    bf16 as configured. Only ids in [allowed_lo, allowed_hi) are read.
 *  - The return value reports argument and launch errors at once. Errors
 *    found on the device (non-finite logits, a draft with zero draft
 *    probability) are latched in a device status word and returned by the
 *    next sjd_sync.
 *  - Inputs are never modified. Results are deterministic: the same inputs,
 *    seed and step give bit-identical outputs on every run.
 *
 * Random numbers: uniform u = (2m+1)/2^24, m = r >> 9, where r is one 32-bit
 * word of Philox-4x32-10 (Salmon et al., SC'11) keyed by the seed and
 * addressed by (absolute position, step, batch, purpose).
 */
#ifndef SJD_H
#define SJD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define SJD_OK 0
#define SJD_ERR_ARG 1            /* invalid argument or configuration            */
#define SJD_ERR_CUDA 2           /* a CUDA runtime call or launch failed         */
#define SJD_ERR_CAPACITY 3       /* workspace, sparse-row capacity or shared
                                    memory too small for the configuration      */
#define SJD_ERR_NONFINITE 4      /* NaN or +inf logit in the allowed range, or a
                                    row without any finite logit                */
#define SJD_ERR_STEP_LIMIT 5     /* sjd_decode_loop reached max_steps            */
#define SJD_ERR_INVALID_DRAFT 6  /* a draft token has zero draft probability     */
#define SJD_ERR_CALLBACK 7       /* the forward callback returned non-zero       */
#define SJD_ERR_STATE 8          /* call out of order (see sjd_draft)            */
#define SJD_ERR_TIMEOUT 9        /* reserved for a bounded wait inside a kernel;
                                    no current kernel waits, so it is not
                                    returned                                    */
#define SJD_ERR_BOUNDS 10        /* the bounds-checked build (libsjd_checked.so)
                                    found an index outside its array; the
                                    access was clamped, results are not valid  */

/* Logit element types. */
#define SJD_F32 0
#define SJD_BF16 1

/* sjd_draft modes. */
#define SJD_DRAFT_PD 0           /* proactive drafting + window refill of the
                                    last sjd_verify_step (Alg. 1, drafting)   */
#define SJD_DRAFT_FROM_LOGITS 1  /* set every row's draft distribution from
                                    draft logits and sample its draft from it   */
#define SJD_DRAFT_UNIFORM 2      /* reset every row to a fresh uniform draft     */

/* Problem statement (Sec. 3.3 and 4; paper defaults Sec. 5.1: top-k 2000,
 * temperature 1, CFG weight 3, K = 4, D = 3, L = 64). */
typedef struct {
  int32_t batch;                 /* B: independent images decoded together     */
  int32_t window;                /* W: Jacobi window length (L), 1..1024       */
  int32_t vocab;                 /* V: row length of the logit tensors         */
  int32_t allowed_lo;            /* sampling restricted to ids [lo, hi)        */
  int32_t allowed_hi;            /*   (the image-token range; full: [0, V))    */
  float cfg_scale;               /* s: l = u + s (c - u); 1 disables guidance  */
  float temperature;             /* T > 0: l / T                               */
  int32_t top_k;                 /* k: keep the k largest logits; 0 = off      */
  float top_p;                   /* tau in (0, 1]: nucleus cut; 1 = off        */
  int32_t pd_k;                  /* K: candidates per drafted position, 1..8   */
  int32_t pd_depth;              /* D: drafted positions after a rejection     */
  int32_t adaptive_continuation; /* 1: SJD-PAC (Sec. 4.2); 0: vanilla SJD tail */
  uint64_t seed;                 /* Philox key                                 */
  int32_t logit_dtype;           /* SJD_F32 or SJD_BF16                        */
  int32_t support_cap;           /* S: capacity of a sparse row; must be
                                    >= min(top_k, hi - lo) (hi - lo if top_k=0) */
  int32_t max_steps;             /* bound of sjd_decode_loop                   */
  int32_t pd_tree;               /* 0: proactive drafting on the main path
                                    (K candidates at each of D positions);
                                    1: the full K-ary tree of depth D, whose
                                    nodes off the main path take logit rows of
                                    their own (see sjd_get_tree)               */
} sjd_config;

typedef struct sjd_ctx sjd_ctx;

/* Bytes of device workspace the configuration needs (0: invalid config). */
size_t sjd_workspace_size(const sjd_config* cfg);

/* Validate cfg, lay the state out in the caller's workspace (workspace_dev,
 * ws_bytes >= sjd_workspace_size(cfg), 256-byte aligned) and start a decode:
 * step 0, every window position p = 0..W-1 fresh, with a uniform draft
 * distribution on [lo, hi) and a uniform draft token (Sec. 3.3, "new tokens
 * are initialized"). cuda_stream is a cudaStream_t (NULL: legacy stream).
 * On success *out receives a host-side handle that holds no device memory.
 * Errors: SJD_ERR_ARG (invalid config or NULL pointer), SJD_ERR_CAPACITY
 * (workspace or shared memory too small), SJD_ERR_CUDA. */
int sjd_init(const sjd_config* cfg, void* workspace_dev, size_t ws_bytes,
             void* cuda_stream, sjd_ctx** out);

/* One verification pass of Alg. 1 over every (b, j) row.
 * cond_dev, uncond_dev: [B][W][V] target logits P^t = M(X^{t-1}) for the
 * conditional and unconditional branches (uncond_dev may be NULL only when
 * cfg_scale == 1). Each row's logits are combined with classifier-free
 * guidance, restricted to [lo, hi), divided by T, cut to the top-k (then
 * top-p) set and normalised (Sec. 5.1). Each row's draft group is verified
 * against the row's stored draft distribution: accept x ~ q iff
 * u < min(1, p(x)/q(x)), else resample from max(p - q, 0) (Sec. 3.2); a
 * group of K candidates is verified in order with the adjusted q^(k) and
 * residual p^(k+1) of Thm. 2. Verification continues past the first
 * rejection (Sec. 4.2).
 * Outputs (device, int32): committed_dev [B][W]: the committed tokens of
 * each batch element in positions 0..n_commit-1 (-1 after); n_commit_dev
 * [B]: first_rej + 1, or W when nothing was rejected; first_rej_dev [B]:
 * 0-based first_rej_idx of Alg. 1 (-1: none). Any output pointer may be NULL.
 * Must be followed by sjd_draft(SJD_DRAFT_PD) before the next verify.
 * Errors: SJD_ERR_ARG, SJD_ERR_STATE (a verify is already pending),
 * SJD_ERR_CUDA; device-side errors via sjd_sync. */
int sjd_verify_step(sjd_ctx* ctx, const void* cond_dev, const void* uncond_dev,
                    int32_t* committed_dev, int32_t* n_commit_dev,
                    int32_t* first_rej_dev);

/* Drafting (Alg. 1, Sec. 4.1, Sec. 3.3).
 * SJD_DRAFT_PD: after sjd_verify_step: if a rejection occurred at i, the
 *   window positions i+1..i+D get K candidates each (the verified token
 *   followed by K-1 tokens drawn without replacement from the position's
 *   target distribution); the window is shifted by n_commit, n_commit fresh
 *   uniform positions are appended, every kept position's draft distribution
 *   becomes its P^t row, and the step counter advances. q_cond_dev and
 *   q_uncond_dev must be NULL. SJD_ERR_STATE if no verify is pending.
 * SJD_DRAFT_FROM_LOGITS: every window row's draft distribution is set to the
 *   processed distribution of the draft logits q_cond_dev / q_uncond_dev
 *   ([B][W][V]; q_uncond_dev NULL: no guidance) and its draft token is
 *   sampled from it. SJD_ERR_STATE if a verify is pending.
 * SJD_DRAFT_UNIFORM: every row gets a fresh uniform draft (as in sjd_init)
 *   at the current positions. SJD_ERR_STATE if a verify is pending. */
int sjd_draft(sjd_ctx* ctx, int32_t mode, const void* q_cond_dev,
              const void* q_uncond_dev);

/* sjd_verify_step followed by sjd_draft(SJD_DRAFT_PD), fused into one kernel
 * launch: one whole Jacobi step (Alg. 1) on the device. Same arguments,
 * outputs and errors as sjd_verify_step. */
int sjd_step(sjd_ctx* ctx, const void* cond_dev, const void* uncond_dev,
             int32_t* committed_dev, int32_t* n_commit_dev, int32_t* first_rej_dev);

/* The caller's guarantee for later sjd_step and sjd_verify_step calls on
 * this context (enable != 0; 0 withdraws it, the default): the logits each
 * call passes were completely written before the previous kernel launched
 * on the context's stream started, and stay unchanged until the call's
 * step completes. The step kernel, launched with programmatic dependent
 * launch, then reads the logits while the previous kernel (normally the
 * previous step) still runs, and waits for that kernel only before it
 * reads or writes the decode state, so that consecutive steps on resident
 * logits overlap. Without the guarantee every read waits. A forward that
 * writes the logits just before the step breaks the guarantee: the decode
 * loop never uses it, nor do sjd_step_host and sjd_step_noalloc. Results are
 * the same bits either way. Errors: SJD_ERR_ARG. */
int sjd_set_early_logits(sjd_ctx* ctx, int32_t enable);

/* Bytes of the device staging buffer sjd_step_host pipelines with: two
 * stages, each holding the allowed columns of every window row, cond and
 * uncond (0 if cfg is invalid). Half of it (one stage) also works, without
 * the overlap. */
size_t sjd_host_stage_size(const sjd_config* cfg);

/* sjd_step on logits held in HOST memory. Only the allowed columns of the
 * B*W rows (ids [allowed_lo, allowed_hi), widened to 16-byte boundaries)
 * cross the host link: one 2-D asynchronous copy per tensor (the copy
 * engines; pinned memory for full speed) into a stage of stage_dev, after
 * which the step runs on those compact rows; the result is that of sjd_step
 * on the full rows. With a stage_dev of sjd_host_stage_size() bytes (two
 * stages) the copies run on a copy stream of the context, alternating
 * between the stages: a step's copy overlaps the kernel of the step before
 * it and waits only for the kernel that read its stage (two steps back),
 * while the kernel waits for its copy on the context's stream. With one
 * stage, or while the context's stream is being captured into a graph, the
 * copies run on the context's stream.
 * cond_host / uncond_host: [B][W][host_row_pitch] logits of the context's
 * dtype, row r at r * host_row_pitch, id v at element v; host_row_pitch >=
 * vocab; uncond_host may be NULL when cfg_scale == 1; the caller keeps them
 * unchanged until the step completes. stage_dev: caller-owned device buffer
 * of sjd_host_stage_size() bytes (or at least half of that), 256-byte
 * aligned, used until the step completes and not shared between contexts.
 * Outputs as sjd_step. Errors: SJD_ERR_ARG, SJD_ERR_STATE, SJD_ERR_CAPACITY
 * (stage too small), SJD_ERR_CUDA. This entry point has no counterpart in
 * the paper: it is the host-input form of the step. */
int sjd_step_host(sjd_ctx* ctx, const void* cond_host, const void* uncond_host, int64_t host_row_pitch,
                  void* stage_dev, size_t stage_bytes, int32_t* committed_dev, int32_t* n_commit_dev,
                  int32_t* first_rej_dev);

/* Target model forward used by sjd_decode_loop
 * (the parallel forward of Alg. 1; outside this library).
 * window_dev [B][W]: main-path window tokens (row 0 at abs_pos[b]);
 * prev_dev [B]: token before row 0 (0 before position 0); abs_pos_dev [B].
 * It must write the [B][W][V] logits of both branches to cond_out_dev /
 * uncond_out_dev (the buffers given to sjd_decode_loop) on `stream` and
 * return 0, or non-zero to abort the loop with SJD_ERR_CALLBACK. */
typedef int (*sjd_forward_fn)(void* user, const int32_t* window_dev,
                              const int32_t* prev_dev, const int32_t* abs_pos_dev,
                              void* cond_out_dev, void* uncond_out_dev,
                              void* stream);

/* Decode n_tokens tokens per batch element (Sec. 3.3 loop around Alg. 1):
 * repeat forward + sjd_step until every batch element has n_tokens
 * committed tokens, at most cfg.max_steps steps.
 * cond_buf_dev / uncond_buf_dev: [B][W][V] logit buffers the forward
 * writes (uncond_buf_dev NULL only when cfg_scale == 1).
 * grid_dev [B][n_tokens]: the generated tokens. accept_len_dev
 * [max_steps][B] (may be NULL): tokens appended per step. *n_steps_out:
 * steps taken. The positions are read back (synchronising the stream) only
 * after ceil((n_tokens - min position) / W) steps, the fewest in which the
 * slowest batch element could finish (a step commits at most W tokens), so
 * the loop takes exactly the steps of a check after every step, with few
 * synchronisations. Errors: SJD_ERR_ARG,
 * SJD_ERR_STEP_LIMIT, SJD_ERR_CALLBACK, SJD_ERR_STATE, SJD_ERR_CUDA and the
 * device-side errors. */
int sjd_decode_loop(sjd_ctx* ctx, sjd_forward_fn forward, void* user,
                    void* cond_buf_dev, void* uncond_buf_dev, int32_t n_tokens,
                    int32_t* grid_dev, int32_t* accept_len_dev,
                    int32_t* n_steps_out);

/* Copy the current window to caller buffers (window order, row 0 first).
 * tokens_dev [B][W] main-path tokens; cands_dev [B][W][K] (may be NULL):
 * candidate groups, -1 padded; group_dev [B][W] (may be NULL): group sizes;
 * abs_pos_dev [B] and prev_dev [B] (may be NULL). */
int sjd_get_window(sjd_ctx* ctx, int32_t* tokens_dev, int32_t* cands_dev,
                   int32_t* group_dev, int32_t* abs_pos_dev, int32_t* prev_dev);

/* Copy every window row's stored draft distribution (the last P^t rows),
 * window order: ids_dev [B][W][S], probs_dev [B][W][S] (fp32), len_dev
 * [B][W] (number of entries; -1 = uniform on [lo, hi)). */
int sjd_get_rows(sjd_ctx* ctx, int32_t* ids_dev, float* probs_dev, int32_t* len_dev);

/* Checkpoint / resume of the whole decode state (synchronous). With
 * host_blob NULL, *bytes receives the blob size. sjd_set_state restores a
 * blob taken from a context of the same configuration; a later step then
 * reproduces the original run bit for bit. SJD_ERR_STATE while a verify is
 * pending; SJD_ERR_ARG on size or configuration mismatch. */
int sjd_get_state(sjd_ctx* ctx, void* host_blob, size_t* bytes);
int sjd_set_state(sjd_ctx* ctx, const void* host_blob, size_t bytes);

/* Counters since sjd_init (synchronous): out[0] rows processed, out[1]
 * sparse draft entries read, out[2] sparse target entries written, out[3]
 * steps. */
int sjd_stats(sjd_ctx* ctx, uint64_t* out4);

/* The same counters and, after them, out[4] rows the fast row kernel
 * streamed a second time (its sampled bound of the k-th largest logit
 * excluded too much, or its candidate list overflowed) and out[5] rows
 * whose top-k cut it took over the row read again (more candidates than
 * its list holds). Writes min(n, 6) counters (synchronous). */
int sjd_stats_ex(sjd_ctx* ctx, uint64_t* out, int32_t n);

/* Allocation-free variant of sjd_step.
 *
 * Some callers cannot allocate device memory at all: code that runs inside
 * another framework's memory pool or plugin interface and may only use the
 * buffers it is handed, or code that must not call cudaMalloc because the
 * host program forbids allocation on its decode path. sjd_init needs a
 * workspace that holds both the decode state and the step's scratch; this
 * entry point needs only the decode state, which is a genuine input and
 * output of a Jacobi step (the window X^{t-1} with its draft distributions
 * P^{t-1} in, X^t and P^t out), and keeps its scratch in a fixed array
 * inside the library. The paper has no counterpart of this entry point; it
 * runs the same fused step as sjd_step, with bit-identical results.
 *
 * state_dev: the decode state, device memory owned by the caller, 256-byte
 *   aligned, *state_bytes long. With state_dev NULL the call only stores
 *   the required size in *state_bytes and returns SJD_OK. The last 256
 *   bytes hold the device status word (uint32, bit code-1 set for each
 *   SJD_ERR_* found on the device); the caller reads and clears it.
 * reset: non-zero starts a new decode in state_dev (as sjd_init does)
 *   before the step; zero continues the decode stored there.
 * cond_dev, uncond_dev, committed_dev, n_commit_dev, first_rej_dev and
 *   cuda_stream: as for sjd_step / sjd_init.
 *
 * Scratch: a static device array of SJD_NOALLOC_SCRATCH_BYTES bytes, which
 * every GPU that loads the library holds until the process exits. A step
 * needs 24 + 8 (K - 1) bytes per window row (B*W rows), 16 bytes per batch
 * element and 832 bytes of counters and status, each of its 14 arrays rounded up to
 * 256 bytes; a configuration that needs more than the array holds is
 * rejected with SJD_ERR_CAPACITY (at K = 8, about 52 000 rows fit). The
 * first call on a device keeps that array's device address for the rest of
 * the process: do not call this entry point on a device again after
 * cudaDeviceReset on it. Every call shares
 * that array, which keeps the last call's contents (the call clears what
 * must start at zero), so calls whose work overlaps on the GPU (other
 * streams, other threads, the same device) race and must be serialised by
 * the caller. The first call on each device looks up the array's device
 * address (with that device current); make that first call before any
 * stream capture. Nothing here allocates memory: no cudaMalloc, cudaFree
 * or allocating library routine is called.
 * Errors: SJD_ERR_ARG, SJD_ERR_CAPACITY, SJD_ERR_CUDA. */
#define SJD_NOALLOC_SCRATCH_BYTES (4u << 20)
int sjd_step_noalloc(const sjd_config* cfg, void* state_dev, size_t* state_bytes,
                     int32_t reset, const void* cond_dev, const void* uncond_dev,
                     int32_t* committed_dev, int32_t* n_commit_dev,
                     int32_t* first_rej_dev, void* cuda_stream);

/* The full K-ary proactive-drafting tree (pd_tree = 1; Sec. 4.1): after a
 * first rejection at f, the positions f+1 .. f+D of the next window carry a
 * tree: node i at depth d (window row d-1) has the children iK .. iK+K-1 at
 * depth d+1, each group K draws without replacement from that position's
 * target (group 0 is the main path's: the row's own token and its K-1
 * alternates). The next sjd_step takes [B, W + X, V] logits, X = sum over
 * d = 1..D-1 of (K^d - 1): after the W window rows, node i >= 1 at depth d
 * (0 < d < D) has row W + sum_{e<d} (K^e - 1) + i - 1, the target
 * conditioned on the path to that node (rows of absent nodes are not read).
 * The step walks the tree from the last committed token: each node's
 * children are verified against the node's own target (Thm. 2), the walk
 * moving to the child that carries the result; the committed prefix ends
 * where no child does, or at the last tree position once the path has left
 * the main path. Only sjd_step runs it (the general row kernel);
 * sjd_verify_step, sjd_step_host, sjd_decode_loop and sjd_step_noalloc
 * return SJD_ERR_ARG with the tree.
 * sjd_get_tree copies the tree of the current window: tokens_dev [B][N],
 * N = sum over d = 1..D of K^d, depth d from slot sum_{e<d} K^e, node i of
 * depth d at that slot + i (-1: no such node); depth_dev [B] the tree's
 * depth (0: none). Either pointer may be NULL. Errors: SJD_ERR_ARG (no
 * tree in the configuration), SJD_ERR_CUDA. */
int sjd_get_tree(sjd_ctx* ctx, int32_t* tokens_dev, int32_t* depth_dev);

/* Relaxed acceptance (LOSSY; off by default). The paper's conclusion names
 * pairing its drafting and verification with a relaxed acceptance criterion
 * of the GSD kind as future work, without a formula. This library's reading:
 * token groups (for example, clusters of the VQ codebook's embeddings) are
 * given as group_of_dev[V] (int32, device memory owned by the caller, kept
 * alive and unchanged while the context steps). Candidate c of a row is
 * then accepted iff u < p^(k)(G(c)) / q^(k)(c), where G(c) is the set of
 * ids whose group equals c's and p^(k)(G(c)) is their total probability;
 * residuals and drafting are unchanged. Decodes are then no longer
 * distributed as plain sampling from the model: the output is biased
 * toward drafts whose group the target supports. With every id in a group
 * of its own the test is the lossless one exactly. group_of_dev NULL
 * restores the lossless test. Applies to sjd_verify_step, sjd_step,
 * sjd_step_host and sjd_decode_loop on this context.
 * Errors: SJD_ERR_ARG (ctx NULL). */
int sjd_set_relaxed_groups(sjd_ctx* ctx, const int32_t* group_of_dev);

/* Synchronise the stream, then return and clear the first device-side
 * error (SJD_OK if none). */
int sjd_sync(sjd_ctx* ctx);

/* Which row kernel this context launches for aligned inputs: 1 = the fast
 * register-resident kernel (allowed range of at most 16384 bf16 / 8192 fp32
 * ids whose rows start on 16-byte boundaries, sparse rows small enough for
 * shared memory), 0 = the general kernel. Both give bit-identical results.
 * The environment variable SJD_KERNEL=general, read by sjd_init, forces the
 * general kernel. */
int sjd_row_path(const sjd_ctx* ctx);

/* Text of the last error on this context (never NULL). */
const char* sjd_last_error(const sjd_ctx* ctx);

/* Free the host handle (the workspace stays the caller's). */
void sjd_destroy(sjd_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* SJD_H */
