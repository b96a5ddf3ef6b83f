"""Oracle: the Gaussian perturbation Z of ZO-Act (test infrastructure only).

Section 3 ("ZO-Act") samples, for every adapted layer and every query, a
perturbation Z ~ N(0, I) of the coefficient matrix.  The paper does not name a
generator.  This build draws Z from the counter-based Philox4x32-10 generator
(J. Salmon, M. Moraes, R. Dror, D. Shaw, "Parallel random numbers: as easy as
1, 2, 3", SC'11) so that Z is never stored: it is a pure function of
(seed, layer_id, query, element index) and is regenerated wherever it is used.

Stream layout (the reading this build fixes, shared with the CUDA side only as a
written definition, not as code):

* key     = (seed & 0xffffffff, seed >> 32)
* counter = (e >> 2, layer_id, query & 0xffffffff, query >> 32), where
  e = i * r + j is the row-major index of Z[i, j] in the [d_out, r] matrix
* the Philox call for counter c yields four 32-bit words w0..w3; element e
  takes word (e & 3).
* Box-Muller on word pairs (w0, w1) and (w2, w3): with
  u1 = ((wa >> 8) + 1) * 2^-24  in (0, 1]   and   u2 = (wb >> 8) * 2^-24 in [0, 1),
  R = sqrt(-2 ln u1),  z_a = R cos(2 pi u2),  z_b = R sin(2 pi u2).
  Using the top 24 bits makes u1 and u2 exactly representable in fp32, so the
  fp32 device code and this fp64 code start from identical uniforms.

Everything here is numpy on uint64 (for the 32x32->64 products) and fp64.
"""
import numpy as np

MASK32 = np.uint64(0xFFFFFFFF)
# Philox4x32 round multipliers and Weyl key increments (Salmon et al., SC'11).
PHILOX_M0 = np.uint64(0xD2511F53)
PHILOX_M1 = np.uint64(0xCD9E8D57)
PHILOX_W0 = np.uint64(0x9E3779B9)
PHILOX_W1 = np.uint64(0xBB67AE85)
TWO_POW_M24 = 2.0 ** -24


def philox4x32_10(counter, key):
    """Philox4x32 with 10 rounds.

    counter: integer array [..., 4] (32-bit words c0..c3); key: [..., 2].
    Returns uint64 array [..., 4] holding the four 32-bit output words.

    One round (Salmon et al., Section 4.2):
        (hi0, lo0) = M0 * c0 ; (hi1, lo1) = M1 * c2       (32x32 -> 64 products)
        c <- (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0)
    and the key is bumped by the Weyl constants before every round but the first.
    """
    counter = np.asarray(counter, dtype=np.uint64)
    key = np.asarray(key, dtype=np.uint64)
    c0, c1, c2, c3 = (counter[..., i] & MASK32 for i in range(4))
    k0 = key[..., 0] & MASK32
    k1 = key[..., 1] & MASK32
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        p0 = PHILOX_M0 * c0          # < 2^64: exact in uint64
        p1 = PHILOX_M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return np.stack([c0, c1, c2, c3], axis=-1)


def stream_words(seed, layer_id, query, n_elems):
    """The raw 32-bit word assigned to each element e in [0, n_elems).

    Returns uint64 array [n_elems] (values < 2^32): word (e & 3) of
    Philox(counter=(e >> 2, layer_id, query_lo, query_hi), key=(seed_lo, seed_hi)).
    """
    seed = int(seed)
    query = int(query)
    n_groups = (int(n_elems) + 3) // 4
    g = np.arange(n_groups, dtype=np.uint64)
    ctr = np.empty((n_groups, 4), dtype=np.uint64)
    ctr[:, 0] = g
    ctr[:, 1] = np.uint64(int(layer_id) & 0xFFFFFFFF)
    ctr[:, 2] = np.uint64(query & 0xFFFFFFFF)
    ctr[:, 3] = np.uint64((query >> 32) & 0xFFFFFFFF)
    key = np.array([seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF], dtype=np.uint64)
    words = philox4x32_10(ctr, np.broadcast_to(key, (n_groups, 2)))
    return words.reshape(-1)[: int(n_elems)]


def box_muller(wa, wb):
    """Two standard normals from two 32-bit words (fp64), as defined above."""
    wa = np.asarray(wa, dtype=np.uint64)
    wb = np.asarray(wb, dtype=np.uint64)
    u1 = ((wa >> np.uint64(8)).astype(np.float64) + 1.0) * TWO_POW_M24
    u2 = (wb >> np.uint64(8)).astype(np.float64) * TWO_POW_M24
    rad = np.sqrt(-2.0 * np.log(u1))
    ang = 2.0 * np.pi * u2
    return rad * np.cos(ang), rad * np.sin(ang)


def normals(seed, layer_id, query, n_elems):
    """Z flattened: the standard normal assigned to each element e (fp64)."""
    n_elems = int(n_elems)
    n_pad = (n_elems + 3) // 4 * 4
    w = stream_words(seed, layer_id, query, n_pad).reshape(-1, 4)
    z = np.empty((w.shape[0], 4), dtype=np.float64)
    z[:, 0], z[:, 1] = box_muller(w[:, 0], w[:, 1])
    z[:, 2], z[:, 3] = box_muller(w[:, 2], w[:, 3])
    return z.reshape(-1)[:n_elems]


def perturbation(seed, layer_id, query, d_out, r):
    """Z for one adapted layer as a [d_out, r] fp64 matrix (Section 3, Z ~ N(0, I)).

    Z[i, j] is element e = i * r + j of the (seed, layer_id, query) stream.
    The paper's Z is r x n (its B is r x n); this build stores the transpose,
    [d_out, r], to match the [d_out, d_in] layout of the frozen weight.
    """
    return normals(seed, layer_id, query, int(d_out) * int(r)).reshape(int(d_out), int(r))
