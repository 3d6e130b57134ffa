"""Philox-4x32-10 counter-based generator for the CPU oracle.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference leg may import this package. The product path
never does.

Written from the published definition of Philox-4x32 (Salmon, Moraes, Dror,
Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11, section 4.2):
each round multiplies counter words 0 and 2 by two fixed odd constants, takes
the 64-bit products apart into high and low halves, and mixes the high halves
with the other two counter words and the round key; the two key words are
bumped by the Weyl constants (golden ratio and sqrt(3)-1, scaled to 32 bits)
between rounds. Ten rounds are used. The paper under study gives no random
source; the uniform draws of the acceptance test (Sec. 3.2, Alg. 1) are
taken from this generator, keyed by the decode seed and addressed by
(absolute position, step, batch, purpose), so that no result depends on
thread mapping or window layout.
"""

MASK32 = 0xFFFFFFFF

# Multipliers and Weyl key increments of Philox-4x32 (SC'11, Table 2 / Sec. 4.2).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85

# Purposes of the uniform draws of one Jacobi step (counter word 3).
ACCEPT = 0     # acceptance test of candidate k (lane k-1), Alg. 1 / Thm. 2
RESIDUAL = 1   # residual resample max(0, p - q) (lane 0), Eq. 1 / Thm. 1
PD = 2         # proactive-drafting alternates c_2..c_K (lane k-1), Sec. 4.1
INIT = 3       # draft of a freshly appended window position (lanes 0,1), Sec. 3.3
SYNTH = 4      # draft sampled from synthetic draft logits (lane 0)
TREE = 5       # full proactive-drafting tree: draw k of group i (lane i*K + k), Sec. 4.1


def philox4x32_10(ctr, key):
    """One Philox-4x32-10 block: 4 counter words and 2 key words -> 4 words."""
    x0, x1, x2, x3 = (int(c) & MASK32 for c in ctr)
    k0, k1 = (int(k) & MASK32 for k in key)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        prod0 = PHILOX_M0 * x0
        prod1 = PHILOX_M1 * x2
        hi0, lo0 = prod0 >> 32, prod0 & MASK32
        hi1, lo1 = prod1 >> 32, prod1 & MASK32
        x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
    return (x0, x1, x2, x3)


def counter(abs_pos, step, batch, purpose, lane):
    """Counter words for a draw; lanes 0..3 share one block, lane 4+ move on."""
    return (abs_pos & MASK32, step & MASK32, batch & MASK32,
            (purpose + 8 * (lane >> 2)) & MASK32)


def raw32(seed, abs_pos, step, batch, purpose, lane):
    """The 32-bit output word `lane` of the draw's Philox block."""
    key = (seed & MASK32, (seed >> 32) & MASK32)
    return philox4x32_10(counter(abs_pos, step, batch, purpose, lane), key)[lane & 3]


def raw64(seed, abs_pos, step, batch, purpose):
    """Lanes 0 and 1 of the draw's block joined as (lane0 << 32) | lane1."""
    key = (seed & MASK32, (seed >> 32) & MASK32)
    r = philox4x32_10(counter(abs_pos, step, batch, purpose, 0), key)
    return (r[0] << 32) | r[1]


def uniform_odd24(r32):
    """Integer 2m+1 with m = r32 >> 9: the uniform is u = (2m+1) / 2^24.

    u lies in [2^-24, 1 - 2^-24], is never 0 or 1, and is exact in fp32.
    """
    return 2 * (int(r32) >> 9) + 1


def uniform(seed, abs_pos, step, batch, purpose, lane):
    """(odd24, u) for one draw; u = odd24 * 2^-24 as a Python float (exact)."""
    o = uniform_odd24(raw32(seed, abs_pos, step, batch, purpose, lane))
    return o, o / float(1 << 24)
