"""Seeded synthetic inputs for the verify-and-draft step.

This module only makes inputs: Gaussian logit rows, the small stand-in model
that plays the target model's role for the full-decode workload, and the
bf16 rounding of inputs. It holds none of the decoding method's arithmetic,
and both the CUDA path and the CPU oracle take their inputs from it.

Every row is generated from its own seed tuple (workload seed, step, batch,
row, kind), so any row of any step can be regenerated on its own.

The paper evaluates on MS-COCO / PartiPrompts prompts with Lumina-mGPT and
Emu3 (Sec. 5.1). Neither the models nor the datasets are available here, so
these synthetic logits stand in for the model's per-position outputs. Each
workload below takes its shape, vocabulary, guidance scale, top-k/top-p and
entropy mix from one of five workloads: a single fp32 step (1 x 16 x 8192), a
32 x 32 decode with the stand-in model (V = 8192), an entropy sweep
(8 x 32 x 16384, sigma 1..5), 100 chained steps with dominant rows
(4 x 32 x 32768), and the full-vocabulary stress step (16 x 64 x 65536, an
8192-id allowed range, top-p 0.9).
"""

from dataclasses import dataclass, field

import numpy as np

COND, UNCOND, QNOISE, DOMINANT = 0, 1, 2, 3

# Value written outside the allowed id range in generated rows. It is larger
# than any in-range logit, so a path that reads outside [lo, hi) picks these
# ids and fails parity at once.
OUT_OF_RANGE_POISON = 64.0


def bf16_round(x):
    """Round fp32 values to the nearest bf16 value (ties to even), as fp32."""
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out = np.where(nan, np.float32(np.nan), out)
    return out.astype(np.float32)


def _rng(*key):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(k) for k in key])))


@dataclass
class Workload:
    """One synthetic workload: shapes, sampler parameters and logit recipe."""
    name: str
    batch: int
    window: int
    vocab: int
    lo: int
    hi: int
    dtype: str                   # "f32" or "bf16"
    cfg_scale: float
    temperature: float
    top_k: int
    top_p: float
    seed: int                    # Philox key of the decode and base seed of the inputs
    sigma: float = 3.0           # std of cond/uncond logits
    q_noise: float = 1.0         # std of the noise added to form draft logits
    sigmas_by_batch: tuple = ()  # entropy sweep: per-batch sigma
    dominant_frac: float = 0.0   # fraction of rows given one dominant logit
    dominant_boost: float = 12.0
    steps: int = 1               # chained Jacobi steps
    ramp: float = 0.0            # + ramp * (1 - 2 (id - lo) / V_eff) on cond and uncond (id-ordered trend)
    pd_k: int = 4
    pd_depth: int = 3
    ac: int = 1

    @property
    def rows(self):
        return self.batch * self.window

    @property
    def v_eff(self):
        return self.hi - self.lo

    def sigma_of(self, b):
        return self.sigmas_by_batch[b] if self.sigmas_by_batch else self.sigma

    def scaled(self, **kw):
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


def workloads():
    """The workloads (names are what they are, with their sizes): five
    configurations, and a larger full decode (90 x 90 tokens, V = 32768)."""
    return {
        "b1w16v8192_f32": Workload("b1w16v8192_f32", 1, 16, 8192, 0, 8192, "f32",
                                   3.0, 1.0, 2000, 1.0, seed=0),
        "decode32x32_b1w16v8192_bf16": Workload("decode32x32_b1w16v8192_bf16", 1, 16, 8192, 0, 8192,
                                                "bf16", 3.0, 1.0, 2000, 1.0, seed=0),
        "decode90x90_b1w16v32768_bf16": Workload("decode90x90_b1w16v32768_bf16", 1, 16, 32768, 0, 32768,
                                                 "bf16", 3.0, 1.0, 2000, 1.0, seed=0),
        "b8w32v16384_bf16_sigma1to5": Workload("b8w32v16384_bf16_sigma1to5", 8, 32, 16384, 0, 16384,
                                               "bf16", 4.0, 1.0, 4096, 1.0, seed=1, q_noise=0.5,
                                               sigmas_by_batch=(1, 2, 3, 4, 5, 1, 2, 3)),
        "b4w32v32768_bf16_dominant_chain100": Workload("b4w32v32768_bf16_dominant_chain100", 4, 32, 32768,
                                                       0, 32768, "bf16", 3.0, 1.0, 2000, 1.0, seed=0,
                                                       dominant_frac=0.1, steps=100),
        "b16w64v65536_bf16_mask8192_topp09": Workload("b16w64v65536_bf16_mask8192_topp09", 16, 64, 65536,
                                                      4, 8196, "bf16", 3.0, 1.0, 2000, 0.9, seed=1234,
                                                      steps=50),
    }


def _round(x, dtype):
    return bf16_round(x) if dtype == "bf16" else np.asarray(x, dtype=np.float32)


def dominant_rows(wl, step):
    """Rows (flat b*W+j) of `step` that get one dominant logit, and the ids."""
    if wl.dominant_frac <= 0:
        return {}
    n = int(round(wl.dominant_frac * wl.rows))
    g = _rng(wl.seed, step, DOMINANT)
    rows = g.permutation(wl.rows)[:n]
    ids = g.integers(wl.lo, wl.hi, size=n)
    return {int(r): int(i) for r, i in zip(rows, ids)}


def logits_row(wl, step, b, j, full_width=True):
    """(cond, uncond, q_cond, q_uncond) fp32 rows of length V (or V_eff).

    In-range values: cond, uncond ~ N(0, sigma_b^2); the draft logits add the
    same N(0, q_noise^2) draw to both, so that after guidance the combined
    draft logit is the combined target logit plus that noise. With
    full_width, ids outside [lo, hi) hold OUT_OF_RANGE_POISON.
    """
    sig = wl.sigma_of(b)
    n = wl.v_eff
    c = _rng(wl.seed, step, b, j, COND).standard_normal(n) * sig
    u = _rng(wl.seed, step, b, j, UNCOND).standard_normal(n) * sig
    dom = dominant_rows(wl, step).get(b * wl.window + j)
    if dom is not None:
        c[dom - wl.lo] += wl.dominant_boost
        u[dom - wl.lo] += wl.dominant_boost
    if wl.ramp:
        trend = wl.ramp * (1.0 - 2.0 * np.arange(n) / n)
        c = c + trend
        u = u + trend
    z = _rng(wl.seed, step, b, j, QNOISE).standard_normal(n) * wl.q_noise
    qc, qu = c + z, u + z
    out = []
    for x in (c, u, qc, qu):
        x = _round(x.astype(np.float32), wl.dtype)
        if full_width:
            full = np.full(wl.vocab, OUT_OF_RANGE_POISON, dtype=np.float32)
            full[wl.lo:wl.hi] = x
            x = full
        out.append(x)
    return tuple(out)


def logits_step(wl, step, batches=None):
    """Full [B, W, V] fp32 arrays (cond, uncond, q_cond, q_uncond) of a step."""
    batches = range(wl.batch) if batches is None else batches
    arrs = [np.empty((len(batches), wl.window, wl.vocab), np.float32) for _ in range(4)]
    for bi, b in enumerate(batches):
        for j in range(wl.window):
            for a, x in zip(arrs, logits_row(wl, step, b, j)):
                a[bi, j] = x
    return tuple(arrs)


class StandInModel:
    """Seeded low-rank stand-in for the target model of the full-decode
    workload: cond = E_out . tanh(E_in[prev] + P[pos]), uncond =
    E_out . tanh(E_in[prev]); weights N(0, 0.05^2) from seeds 0/1/2; the
    token before position 0 is id 0; logits rounded to bf16."""

    def __init__(self, vocab=8192, dim=256, n_pos=1024, std=0.05, seeds=(0, 1, 2)):
        self.E_out = _rng(seeds[0]).standard_normal((vocab, dim)) * std
        self.E_in = _rng(seeds[1]).standard_normal((vocab, dim)) * std
        self.P = _rng(seeds[2]).standard_normal((n_pos, dim)) * std
        self.vocab, self.n_pos = vocab, n_pos

    def forward(self, window, prev, abs_pos):
        """window [B][W] main-path tokens, prev [B], abs_pos [B] ->
        (cond, uncond) fp32 [B, W, V] holding bf16 values."""
        B, W = len(window), len(window[0])
        prev_tok = np.empty((B, W), np.int64)
        pos = np.empty((B, W), np.int64)
        for b in range(B):
            for j in range(W):
                prev_tok[b, j] = prev[b] if j == 0 else window[b][j - 1]
                pos[b, j] = min(abs_pos[b] + j, self.n_pos - 1)
        e = self.E_in[prev_tok]
        hc = np.tanh(e + self.P[pos])
        hu = np.tanh(e)
        cond = bf16_round((hc @ self.E_out.T).astype(np.float32))
        uncond = bf16_round((hu @ self.E_out.T).astype(np.float32))
        return cond, uncond
