"""Python binding of libsjd.so (include/sjd.h): argument marshalling only.

Every step of the verify-and-draft path runs in the CUDA library; this
module loads it with ctypes, passes torch tensors' device pointers and the
current CUDA stream, and turns status codes into exceptions. There is no
fallback: if the library is missing or cannot be loaded, import of the
library raises.
"""

import ctypes
import os
from ctypes import POINTER, byref, c_float, c_int32, c_size_t, c_uint64, c_void_p

import torch

# SJD_LIBRARY=checked selects the build with device-side bounds checks
# (libsjd_checked.so; an index outside its array latches SJD_ERR_BOUNDS).
_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build",
                         "libsjd_checked.so" if os.environ.get("SJD_LIBRARY") == "checked" else "libsjd.so")

SJD_OK = 0
SJD_ERR_ARG = 1
SJD_ERR_CUDA = 2
SJD_ERR_CAPACITY = 3
SJD_ERR_NONFINITE = 4
SJD_ERR_STEP_LIMIT = 5
SJD_ERR_INVALID_DRAFT = 6
SJD_ERR_CALLBACK = 7
SJD_ERR_STATE = 8
SJD_ERR_TIMEOUT = 9
SJD_ERR_BOUNDS = 10

SJD_F32 = 0
SJD_BF16 = 1

SJD_DRAFT_PD = 0
SJD_DRAFT_FROM_LOGITS = 1
SJD_DRAFT_UNIFORM = 2

ERROR_NAMES = {
    SJD_ERR_ARG: "SJD_ERR_ARG", SJD_ERR_CUDA: "SJD_ERR_CUDA", SJD_ERR_CAPACITY: "SJD_ERR_CAPACITY",
    SJD_ERR_NONFINITE: "SJD_ERR_NONFINITE", SJD_ERR_STEP_LIMIT: "SJD_ERR_STEP_LIMIT",
    SJD_ERR_INVALID_DRAFT: "SJD_ERR_INVALID_DRAFT", SJD_ERR_CALLBACK: "SJD_ERR_CALLBACK",
    SJD_ERR_STATE: "SJD_ERR_STATE", SJD_ERR_TIMEOUT: "SJD_ERR_TIMEOUT", SJD_ERR_BOUNDS: "SJD_ERR_BOUNDS",
}


class SJDError(RuntimeError):
    def __init__(self, code, msg=""):
        super().__init__("%s (%d): %s" % (ERROR_NAMES.get(code, "?"), code, msg))
        self.code = code


class sjd_config(ctypes.Structure):
    _fields_ = [
        ("batch", c_int32), ("window", c_int32), ("vocab", c_int32),
        ("allowed_lo", c_int32), ("allowed_hi", c_int32),
        ("cfg_scale", c_float), ("temperature", c_float),
        ("top_k", c_int32), ("top_p", c_float),
        ("pd_k", c_int32), ("pd_depth", c_int32), ("adaptive_continuation", c_int32),
        ("seed", c_uint64), ("logit_dtype", c_int32), ("support_cap", c_int32),
        ("max_steps", c_int32), ("pd_tree", c_int32),
    ]


FORWARD_FN = ctypes.CFUNCTYPE(ctypes.c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                              c_void_p, c_void_p)

_lib = None


def lib_path():
    return _LIB_PATH


def load():
    """Load libsjd.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError("libsjd.so not found at %s: build it with __graft_entry__.build()" % _LIB_PATH)
    L = ctypes.CDLL(_LIB_PATH)
    P = c_void_p
    I32P = POINTER(c_int32)
    L.sjd_workspace_size.argtypes = [POINTER(sjd_config)]
    L.sjd_workspace_size.restype = c_size_t
    L.sjd_init.argtypes = [POINTER(sjd_config), P, c_size_t, P, POINTER(c_void_p)]
    L.sjd_init.restype = c_int32
    for name in ("sjd_verify_step", "sjd_step"):
        getattr(L, name).argtypes = [P, P, P, P, P, P]
        getattr(L, name).restype = c_int32
    L.sjd_draft.argtypes = [P, c_int32, P, P]
    L.sjd_draft.restype = c_int32
    L.sjd_decode_loop.argtypes = [P, FORWARD_FN, P, P, P, c_int32, P, P, I32P]
    L.sjd_decode_loop.restype = c_int32
    L.sjd_get_window.argtypes = [P, P, P, P, P, P]
    L.sjd_get_window.restype = c_int32
    L.sjd_get_tree.argtypes = [P, P, P]
    L.sjd_get_tree.restype = c_int32
    L.sjd_get_rows.argtypes = [P, P, P, P]
    L.sjd_get_rows.restype = c_int32
    L.sjd_get_state.argtypes = [P, P, POINTER(c_size_t)]
    L.sjd_get_state.restype = c_int32
    L.sjd_set_state.argtypes = [P, P, c_size_t]
    L.sjd_set_state.restype = c_int32
    L.sjd_stats.argtypes = [P, POINTER(c_uint64)]
    L.sjd_stats.restype = c_int32
    L.sjd_stats_ex.argtypes = [P, POINTER(c_uint64), c_int32]
    L.sjd_stats_ex.restype = c_int32
    L.sjd_sync.argtypes = [P]
    L.sjd_sync.restype = c_int32
    L.sjd_set_relaxed_groups.argtypes = [P, P]
    L.sjd_set_relaxed_groups.restype = c_int32
    L.sjd_row_path.argtypes = [P]
    L.sjd_row_path.restype = c_int32
    L.sjd_last_error.argtypes = [P]
    L.sjd_last_error.restype = ctypes.c_char_p
    L.sjd_destroy.argtypes = [P]
    L.sjd_destroy.restype = None
    L.sjd_step_noalloc.argtypes = [POINTER(sjd_config), P, POINTER(c_size_t), c_int32, P, P, P, P, P, P]
    L.sjd_step_noalloc.restype = c_int32
    L.sjd_set_early_logits.argtypes = [P, c_int32]
    L.sjd_set_early_logits.restype = c_int32
    L.sjd_host_stage_size.argtypes = [POINTER(sjd_config)]
    L.sjd_host_stage_size.restype = c_size_t
    L.sjd_step_host.argtypes = [P, P, P, ctypes.c_int64, P, c_size_t, P, P, P]
    L.sjd_step_host.restype = c_int32
    _lib = L
    return L


def make_config(batch, window, vocab, allowed_lo=0, allowed_hi=None, cfg_scale=3.0, temperature=1.0,
                top_k=2000, top_p=1.0, pd_k=4, pd_depth=3, adaptive_continuation=1, seed=0,
                logit_dtype=SJD_BF16, support_cap=None, max_steps=100000, pd_tree=0):
    hi = vocab if allowed_hi is None else allowed_hi
    veff = hi - allowed_lo
    if support_cap is None:
        support_cap = min(top_k, veff) if top_k > 0 else veff
    return sjd_config(batch, window, vocab, allowed_lo, hi, cfg_scale, temperature, top_k, top_p,
                      pd_k, pd_depth, adaptive_continuation, seed, logit_dtype, support_cap, max_steps, pd_tree)


def tree_rows(cfg):
    """Extra logit rows per batch element with the full tree (nodes off the
    main path at depths 1..D-1)."""
    return sum(cfg.pd_k ** d - 1 for d in range(1, cfg.pd_depth)) if cfg.pd_tree else 0


def tree_slots(cfg):
    """Token slots of the full tree per batch element (depths 1..D)."""
    return sum(cfg.pd_k ** d for d in range(1, cfg.pd_depth + 1)) if cfg.pd_tree else 0


def workspace_size(cfg):
    return int(load().sjd_workspace_size(byref(cfg)))


def _ptr(t):
    return None if t is None else c_void_p(t.data_ptr())


class SJD:
    """One decode context: the workspace (a torch uint8 tensor) and the
    library handle bound to a CUDA stream."""

    def __init__(self, cfg, device="cuda", stream=None):
        self.L = load()
        self.cfg = cfg
        self.device = torch.device(device)
        if self.device.index is None:
            self.device = torch.device(self.device.type, torch.cuda.current_device())
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        size = workspace_size(cfg)
        if size == 0:
            raise SJDError(SJD_ERR_ARG, "invalid configuration")
        self.workspace = torch.empty(size, dtype=torch.uint8, device=self.device)
        self.ctx = c_void_p()
        rc = self.L.sjd_init(byref(cfg), c_void_p(self.workspace.data_ptr()), size,
                             c_void_p(self.stream.cuda_stream), byref(self.ctx))
        if rc != SJD_OK:
            raise SJDError(rc, "sjd_init failed")
        self.logit_dtype = torch.bfloat16 if cfg.logit_dtype == SJD_BF16 else torch.float32
        self._callback = None

    # -- helpers ------------------------------------------------------------
    def _check(self, rc):
        if rc != SJD_OK:
            raise SJDError(rc, self.L.sjd_last_error(self.ctx).decode())

    def _logits(self, t, name, rows=None):
        if t is None:
            return None
        shape = (self.cfg.batch, self.cfg.window if rows is None else rows, self.cfg.vocab)
        if tuple(t.shape) != shape or t.dtype != self.logit_dtype or not t.is_contiguous() \
                or t.device != self.device:
            raise ValueError("%s must be a contiguous %s tensor of shape %s on %s"
                             % (name, self.logit_dtype, shape, self.device))
        return c_void_p(t.data_ptr())

    def _i32(self, *shape):
        return torch.empty(shape, dtype=torch.int32, device=self.device)

    # -- entry points ---------------------------------------------------------
    def verify_step(self, cond, uncond=None, out=None):
        out = out or (self._i32(self.cfg.batch, self.cfg.window), self._i32(self.cfg.batch),
                      self._i32(self.cfg.batch))
        self._check(self.L.sjd_verify_step(self.ctx, self._logits(cond, "cond"), self._logits(uncond, "uncond"),
                                           *[_ptr(o) for o in out]))
        return out

    def step(self, cond, uncond=None, out=None):
        out = out or (self._i32(self.cfg.batch, self.cfg.window), self._i32(self.cfg.batch),
                      self._i32(self.cfg.batch))
        rows = self.cfg.window + tree_rows(self.cfg)   # the tree's node rows follow the window rows
        self._check(self.L.sjd_step(self.ctx, self._logits(cond, "cond", rows), self._logits(uncond, "uncond", rows),
                                    *[_ptr(o) for o in out]))
        return out

    def set_early_logits(self, enable=True):
        """sjd_set_early_logits: the logits of later step / verify_step calls
        were written before the previous kernel on the context's stream
        started (resident inputs, not a forward just before), so that
        consecutive steps overlap."""
        self._check(self.L.sjd_set_early_logits(self.ctx, 1 if enable else 0))

    def host_stage(self):
        """A device staging buffer for step_host (sjd_host_stage_size bytes:
        two stages, so that a step's host copy overlaps the step before)."""
        n = self.L.sjd_host_stage_size(byref(self.cfg))
        if n == 0:
            raise SJDError(SJD_ERR_ARG, "invalid configuration")
        return torch.empty(n, dtype=torch.uint8, device=self.device)

    def step_host(self, cond_host, uncond_host, stage, out=None):
        """sjd_step_host: cond_host / uncond_host are CPU tensors [B, W, V']
        (V' >= V, contiguous; pinned for an asynchronous copy); only the
        allowed columns are copied into `stage` (from host_stage(); a
        tensor of half its size runs without the copy overlap)."""
        for t, nm in ((cond_host, "cond_host"), (uncond_host, "uncond_host")):
            if t is None:
                continue
            if t.device.type != "cpu" or not t.is_contiguous() or t.dim() != 3:
                raise SJDError(SJD_ERR_ARG, "%s must be a contiguous [B, W, V'] CPU tensor" % nm)
            if t.element_size() != (2 if self.cfg.logit_dtype == SJD_BF16 else 4):
                raise SJDError(SJD_ERR_ARG, "%s has the wrong dtype" % nm)
        out = out or (self._i32(self.cfg.batch, self.cfg.window), self._i32(self.cfg.batch),
                      self._i32(self.cfg.batch))
        pitch = cond_host.shape[-1]
        self._check(self.L.sjd_step_host(self.ctx, c_void_p(cond_host.data_ptr()),
                                         c_void_p(uncond_host.data_ptr()) if uncond_host is not None else None,
                                         pitch, c_void_p(stage.data_ptr()), stage.numel(), *[_ptr(o) for o in out]))
        return out

    def step_raw(self, cond, uncond, committed=None, n_commit=None, first_rej=None):
        """sjd_step without checks or allocation (for timing loops)."""
        return self.L.sjd_step(self.ctx, cond, uncond, committed, n_commit, first_rej)

    def draft_pd(self):
        self._check(self.L.sjd_draft(self.ctx, SJD_DRAFT_PD, None, None))

    def draft_from_logits(self, q_cond, q_uncond=None):
        self._check(self.L.sjd_draft(self.ctx, SJD_DRAFT_FROM_LOGITS, self._logits(q_cond, "q_cond"),
                                     self._logits(q_uncond, "q_uncond")))

    def draft_uniform(self):
        self._check(self.L.sjd_draft(self.ctx, SJD_DRAFT_UNIFORM, None, None))

    def decode_loop(self, forward, n_tokens, cond_buf, uncond_buf=None, accept_len=True):
        """forward(window [B,W] int32, prev [B], abs_pos [B], cond_out, uncond_out) fills the
        logit buffers (torch tensors on the device) for the current window."""
        B, W, V = self.cfg.batch, self.cfg.window, self.cfg.vocab
        grid = torch.full((B, n_tokens), -1, dtype=torch.int32, device=self.device)
        acc = self._i32(self.cfg.max_steps, B).zero_() if accept_len else None
        base = self.workspace.data_ptr()
        nbytes = self.workspace.numel()

        def view(ptr, n):
            # the window, previous-token and position arrays live in the workspace
            off = int(ptr) - base
            if off < 0 or off + 4 * n > nbytes:
                raise RuntimeError("forward argument outside the workspace")
            return self.workspace[off:off + 4 * n].view(torch.int32)

        self.callback_error = None

        def cb(user, win, prev, pos, cbuf, ubuf, stream):
            try:
                forward(view(win, B * W).view(B, W), view(prev, B), view(pos, B), cond_buf, uncond_buf)
                return 0
            except Exception as e:  # reported as SJD_ERR_CALLBACK
                self.callback_error = e
                return 1

        self._callback = FORWARD_FN(cb)
        n_steps = c_int32(0)
        rc = self.L.sjd_decode_loop(self.ctx, self._callback, None, self._logits(cond_buf, "cond_buf"),
                                    self._logits(uncond_buf, "uncond_buf"), n_tokens, _ptr(grid), _ptr(acc),
                                    byref(n_steps))
        if rc == SJD_ERR_CALLBACK and self.callback_error is not None:
            raise SJDError(rc, "forward raised %r" % (self.callback_error,)) from self.callback_error
        self._check(rc)
        steps = n_steps.value
        return grid, (acc[:steps] if acc is not None else None), steps

    def get_window(self):
        B, W, K = self.cfg.batch, self.cfg.window, self.cfg.pd_k
        tok, cands, group, pos, prev = (self._i32(B, W), self._i32(B, W, K), self._i32(B, W),
                                        self._i32(B), self._i32(B))
        self._check(self.L.sjd_get_window(self.ctx, *[_ptr(t) for t in (tok, cands, group, pos, prev)]))
        return tok, cands, group, pos, prev

    def get_tree(self):
        """(tokens [B, N], depth [B]) of the current window's full tree."""
        tok = self._i32(self.cfg.batch, max(1, tree_slots(self.cfg)))
        depth = self._i32(self.cfg.batch)
        self._check(self.L.sjd_get_tree(self.ctx, _ptr(tok), _ptr(depth)))
        return tok, depth

    def get_rows(self):
        B, W, S = self.cfg.batch, self.cfg.window, self.cfg.support_cap
        ids = self._i32(B, W, S)
        probs = torch.empty((B, W, S), dtype=torch.float32, device=self.device)
        n = self._i32(B, W)
        self._check(self.L.sjd_get_rows(self.ctx, _ptr(ids), _ptr(probs), _ptr(n)))
        return ids, probs, n

    def get_state(self):
        size = c_size_t(0)
        self._check(self.L.sjd_get_state(self.ctx, None, byref(size)))
        buf = ctypes.create_string_buffer(size.value)
        self._check(self.L.sjd_get_state(self.ctx, buf, byref(size)))
        return buf.raw

    def set_state(self, blob):
        self._check(self.L.sjd_set_state(self.ctx, blob, len(blob)))

    def stats(self):
        """[rows, draft entries read, target entries written, steps, rows
        streamed twice, rows whose top-k cut was taken over the re-read row]."""
        out = (c_uint64 * 6)()
        self._check(self.L.sjd_stats_ex(self.ctx, out, 6))
        return list(out)

    def sync(self):
        """Returns the device-side status code (0 = OK) and clears it."""
        return int(self.L.sjd_sync(self.ctx))

    def set_relaxed_groups(self, group_of):
        """Relaxed (lossy) acceptance with token groups group_of [V] (int32
        on this device; kept by the caller while the context steps), or the
        lossless test again with None."""
        if group_of is not None:
            if group_of.dtype != torch.int32 or group_of.numel() != self.cfg.vocab or \
                    group_of.device != self.device or not group_of.is_contiguous():
                raise ValueError("group_of must be a contiguous int32 tensor of %d entries on %s"
                                 % (self.cfg.vocab, self.device))
        self._groups = group_of
        self._check(self.L.sjd_set_relaxed_groups(self.ctx, _ptr(group_of)))

    def row_path(self):
        """1: the fast register-resident row kernel; 0: the general one."""
        return int(self.L.sjd_row_path(self.ctx))

    def last_error(self):
        return self.L.sjd_last_error(self.ctx).decode()

    def close(self):
        if self.ctx:
            self.L.sjd_destroy(self.ctx)
            self.ctx = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def step_noalloc_state_bytes(cfg):
    """Size of the decode-state buffer sjd_step_noalloc needs."""
    n = c_size_t(0)
    rc = load().sjd_step_noalloc(byref(cfg), None, byref(n), 0, None, None, None, None, None, None)
    if rc != SJD_OK:
        raise SJDError(rc, "invalid configuration")
    return n.value


def step_noalloc(cfg, state, cond, uncond, committed, n_commit, first_rej, reset=False, stream=None):
    """One fused step through sjd_step_noalloc (the state and all outputs are
    caller tensors on one device; the library allocates nothing). The call
    runs with the state's device current: the library finds its scratch
    array and sets its kernel limits on the current device."""
    for t, nm in ((cond, "cond"), (uncond, "uncond"), (committed, "committed"), (n_commit, "n_commit"),
                  (first_rej, "first_rej")):
        if t is not None and t.device != state.device:
            raise ValueError("%s is on %s, the state on %s" % (nm, t.device, state.device))
    with torch.cuda.device(state.device):
        stream = stream if stream is not None else torch.cuda.current_stream(state.device)
        n = c_size_t(state.numel() * state.element_size())
        rc = load().sjd_step_noalloc(byref(cfg), c_void_p(state.data_ptr()), byref(n), 1 if reset else 0,
                                     _ptr(cond), _ptr(uncond), _ptr(committed), _ptr(n_commit), _ptr(first_rej),
                                     c_void_p(stream.cuda_stream))
    if rc != SJD_OK:
        raise SJDError(rc, "sjd_step_noalloc failed")
