"""Oracle: the replica fingerprint of a coefficient arena (test infrastructure only).

The paper runs on one device and has no counterpart.  In a data-parallel ZO
step every rank holds the same coefficients and applies the same update with
the same regenerated Z (MeZO's property, which Section 3 keeps), so the ranks'
arenas stay bit-identical; a fingerprint of each rank's arena, compared across
ranks, detects one that diverged.  The definition this build fixes:

    h = sum over i of mix64(((i << 32) | w_i) + GAMMA)   (mod 2^64)

with w_i the i-th 32-bit word of the arena (little-endian), GAMMA =
0x9E3779B97F4A7C15 and mix64 the output function of SplitMix64 (G. L. Steele,
D. Lea, C. H. Flood, "Fast splittable pseudorandom number generators",
OOPSLA 2014):

    z ^= z >> 30;  z *= 0xBF58476D1CE4E5B9;  z ^= z >> 27;  z *= 0x94D049BB133111EB;  z ^= z >> 31

(all mod 2^64).  Written here in numpy uint64 arithmetic.
"""
import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
M1 = np.uint64(0xBF58476D1CE4E5B9)
M2 = np.uint64(0x94D049BB133111EB)


def mix64(z):
    """SplitMix64's output function on a uint64 array (wrapping products)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * M1
        z = (z ^ (z >> np.uint64(27))) * M2
    return z ^ (z >> np.uint64(31))


def splitmix64(state, n):
    """The first n outputs of SplitMix64 from `state`: state += GAMMA, output mix64(state)."""
    out = []
    s = np.uint64(state)
    for _ in range(n):
        with np.errstate(over="ignore"):
            s = s + GAMMA
        out.append(int(mix64(s)))
    return out


def arena_hash(words):
    """The fingerprint of a 1-D array of 32-bit words (any 4-byte dtype: its bits are used)."""
    w = np.ascontiguousarray(words).reshape(-1).view(np.uint32).astype(np.uint64)
    i = np.arange(w.size, dtype=np.uint64)
    with np.errstate(over="ignore"):
        terms = mix64(((i << np.uint64(32)) | w) + GAMMA)
        return int(np.sum(terms, dtype=np.uint64))
