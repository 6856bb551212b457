"""Philox4x32-10 and the draw layout of the verification path (oracle copy).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Philox4x32-10 is the counter-based generator of Salmon, Moraes, Dror and Shaw,
"Parallel random numbers: as easy as 1, 2, 3" (SC'11): ten rounds of two
32x32->64 multiplications with the round keys bumped by Weyl constants.  It is
written here from that publication; the device side has its own copy.

Draw layout (a reading: the paper draws its uniforms implicitly).  For
sequence b, depth j and draw id d the counter is (b, j, d, 0) and the key is
(seed & 0xffffffff, seed >> 32).  The uniform is (word0 >> 8) * 2^-24, an exact
multiple of 2^-24 in [0, 1).  Draw ids:

    0..15   importance-step selection uniforms (stage m of the pairwise
            stages uses id m; plain IS uses id 0)
    16..31  speculative accept uniforms (the canonical scheme uses 16; the
            sequential-rejection baseline's round i uses 16 + i)
    32      residual resample
    33      bonus token after L accepted positions
    34      truncated alphabet: keep the token drawn on Omega_0
    35      truncated alphabet: replacement drawn outside Omega_0
"""
import numpy as np

PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
MASK32 = 0xFFFFFFFF

DRAW_SELECT = 0
DRAW_ACCEPT = 16
DRAW_RESIDUAL = 32
DRAW_BONUS = 33


def _mulhilo(a, b):
    prod = (a * b) & 0xFFFFFFFFFFFFFFFF
    return prod >> 32, prod & MASK32


def philox4x32_10(ctr, key):
    """Return the four 32-bit output words for counter ``ctr`` (4 ints) and
    key ``key`` (2 ints), as plain Python ints."""
    c0, c1, c2, c3 = (int(x) & MASK32 for x in ctr)
    k0, k1 = (int(x) & MASK32 for x in key)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        hi0, lo0 = _mulhilo(PHILOX_M0, c0)
        hi1, lo1 = _mulhilo(PHILOX_M1, c2)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def uniform(seed, b, j, draw):
    """The uniform in [0, 1) for (sequence b, depth j, draw id), as a float
    that is an exact multiple of 2^-24."""
    seed = int(seed)
    w0 = philox4x32_10((b, j, draw, 0), (seed & MASK32, (seed >> 32) & MASK32))[0]
    return float(w0 >> 8) * (2.0 ** -24)


def philox4x32_10_np(c0, c1, c2, c3, k0, k1):
    """Vectorised variant over numpy uint64 arrays holding 32-bit values;
    used by tests that need many draws.  Same arithmetic as ``philox4x32_10``."""
    c0, c1, c2, c3 = (np.asarray(x, dtype=np.uint64) & MASK32 for x in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & MASK32
    k1 = np.asarray(k1, dtype=np.uint64) & MASK32
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & np.uint64(MASK32)
            k1 = (k1 + np.uint64(PHILOX_W1)) & np.uint64(MASK32)
        p0 = m0 * c0
        p1 = m1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK32)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def uniforms_np(seed, b, j, draw):
    """Vectorised ``uniform`` over broadcastable integer arrays b, j, draw."""
    seed = int(seed)
    b, j, draw = np.broadcast_arrays(np.asarray(b, dtype=np.uint64), np.asarray(j, dtype=np.uint64),
                                     np.asarray(draw, dtype=np.uint64))
    zero = np.zeros_like(b)
    w0 = philox4x32_10_np(b, j, draw, zero, np.full_like(b, seed & MASK32),
                          np.full_like(b, (seed >> 32) & MASK32))[0]
    return (w0 >> np.uint64(8)).astype(np.float64) * (2.0 ** -24)
