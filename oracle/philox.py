"""Philox4x32-10 and the random-number conventions of the verification step.

Test infrastructure only (see ``oracle/__init__``).

Generator: Philox4x32 with 10 rounds, as defined in J. K. Salmon, M. A. Moraes,
R. O. Dror, D. E. Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11,
Section 4 (the Philox S-box built from a 32x32->64 multiply, with the Weyl key
schedule).  Key = 64-bit seed split into (lo, hi) words; counter = 4 words.

Conventions (the paper draws eta, w and G from unspecified generators; these
are the readings this repository fixes, identical on both sides):

* coin eta_j of chain b, step j (0-based)  : counter (b, j, STREAM_COIN, 0), word 0
* residual uniform w of chain b            : counter (b, 0, STREAM_USAMPLE, 0), word 0
* Gaussian noise of a stream, element i    : counter (b, i // 4, stream, sub), the
  four words give four normals by Box-Muller on the pairs (w0, w1), (w2, w3)
* uniform from a word x                    : (x + 1/2) * 2^-32, strictly inside (0, 1)
* Box-Muller from (u0, u1)                 : r = sqrt(-2 ln u0),
                                             (r cos 2 pi u1, r sin 2 pi u1)

All arithmetic here is numpy uint64 / float64.
"""
import numpy as np

# Philox4x32 multipliers and Weyl key increments (Salmon et al., SC'11, Sec. 4).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
MASK32 = 0xFFFFFFFF

STREAM_COIN = 0
STREAM_USAMPLE = 1
STREAM_RESID = 2
STREAM_BONUS = 3
STREAM_DRAFT = 4
STREAM_INIT = 5
STREAM_EM = 6


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32-10 on arrays of counters (broadcast); returns 4 uint64 arrays of 32-bit words.

    One round maps (c0, c1, c2, c3) with key (k0, k1) to
    (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0));
    the key is advanced by the Weyl constants between rounds.
    """
    c0, c1, c2, c3 = (np.asarray(v, dtype=np.uint64) & MASK32 for v in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & MASK32
    k1 = np.asarray(k1, dtype=np.uint64) & MASK32
    c0, c1, c2, c3 = np.broadcast_arrays(c0, c1, c2, c3)
    c0, c1, c2, c3 = (v.copy() for v in (c0, c1, c2, c3))
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        p0 = np.uint64(PHILOX_M0) * c0          # < 2^64: both factors < 2^32
        p1 = np.uint64(PHILOX_M1) * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0), lo1, (hi0 ^ c3 ^ k1), lo0
    return c0, c1, c2, c3


def key_of(seed):
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    return seed & MASK32, seed >> 32


def uniform_of(word):
    """(x + 1/2) 2^-32 in float64: exact, strictly inside (0, 1)."""
    return (np.asarray(word, dtype=np.float64) + 0.5) * (2.0 ** -32)


def box_muller(w0, w1):
    u0 = uniform_of(w0)
    u1 = uniform_of(w1)
    r = np.sqrt(-2.0 * np.log(u0))
    return r * np.cos(2.0 * np.pi * u1), r * np.sin(2.0 * np.pi * u1)


def coin_words(seed, b, j):
    """Raw 32-bit word behind the coin eta_j of chain b (arrays broadcast)."""
    k0, k1 = key_of(seed)
    return philox4x32_10(b, j, STREAM_COIN, 0, k0, k1)[0]


def coins(seed, b, L):
    """eta_0..eta_{L-1} of chain b (step index j is 0-based); b may be an array -> b.shape + (L,)."""
    b = np.asarray(b, dtype=np.uint64)
    return uniform_of(coin_words(seed, b[..., None], np.arange(L, dtype=np.uint64)))


def usample_word(seed, b):
    k0, k1 = key_of(seed)
    return philox4x32_10(b, 0, STREAM_USAMPLE, 0, k0, k1)[0]


def usample_uniform(seed, b):
    """Residual uniform w of chain b (array-valued for an array b)."""
    return uniform_of(usample_word(seed, b))


def normals(seed, b, d, stream, sub=0):
    """d standard normals of chain b on the given stream (element i from block i // 4).

    ``b`` may be an array of chains: the result then has shape b.shape + (d,).
    """
    k0, k1 = key_of(seed)
    nblk = (d + 3) // 4
    b = np.asarray(b, dtype=np.uint64)
    w = philox4x32_10(b[..., None], np.arange(nblk, dtype=np.uint64), stream, sub, k0, k1)
    z0, z1 = box_muller(w[0], w[1])
    z2, z3 = box_muller(w[2], w[3])
    z = np.stack([z0, z1, z2, z3], axis=-1)
    return z.reshape(z.shape[:-2] + (4 * nblk,))[..., :d]


def splitmix64(z):
    """One SplitMix64 output for state z (Steele, Lea, Flood, OOPSLA'14)."""
    m = 0xFFFFFFFFFFFFFFFF
    z &= m
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & m
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & m
    return z ^ (z >> 31)


def round_seed(seed, r):
    """Seed of sampler round r: the (r+1)-th SplitMix64 output of a stream started at seed."""
    return splitmix64((int(seed) + (int(r) + 1) * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF)
