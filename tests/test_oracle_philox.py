"""Pins for the oracle's perturbation generator (CPU only).

Z ~ N(0, I) (Section 3) from Philox4x32-10 + Box-Muller.  Pinned by the
published known-answer vectors, by the stream layout written out by brute force,
by Box-Muller special values, by distribution tests, and by the estimator
moments of Section 4 (E[<g,z> z] = g, E||<g,z> z||^2 = (k+2)||g||^2).
"""
import os

import numpy as np
import pytest
from scipy import stats

from oracle import philox

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            v = [int(t, 16) for t in line.split()]
            rows.append((v[0:4], v[4:6], v[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat_rows())
def test_philox_known_answers(ctr, key, expect):
    out = philox.philox4x32_10(np.array(ctr), np.array(key))
    assert [int(x) for x in out] == expect


def test_stream_layout_brute_force():
    # element e takes word (e & 3) of counter (e >> 2, layer, q_lo, q_hi), key (seed_lo, seed_hi)
    seed, layer, query = 0x0123456789ABCDEF, 17, (5 << 32) | 9
    words = philox.stream_words(seed, layer, query, 37)
    for e in range(37):
        ctr = np.array([e >> 2, layer, query & 0xFFFFFFFF, query >> 32])
        key = np.array([seed & 0xFFFFFFFF, seed >> 32])
        assert int(words[e]) == int(philox.philox4x32_10(ctr, key)[e & 3])


def test_box_muller_special_values():
    # top 24 bits all ones -> u1 = 1 -> radius 0
    za, zb = philox.box_muller(np.array([0xFFFFFFFF]), np.array([0x12345678]))
    assert za[0] == 0.0 and zb[0] == 0.0
    # u2 = 0 -> angle 0 -> (R, 0) with R = sqrt(-2 ln u1)
    wa = np.array([(1 << 31)])           # u1 = (2^23 + 1) 2^-24
    za, zb = philox.box_muller(wa, np.array([0]))
    u1 = ((1 << 23) + 1) * 2.0 ** -24
    assert za[0] == pytest.approx(np.sqrt(-2 * np.log(u1)), rel=1e-15)
    assert zb[0] == 0.0
    # u2 = 1/4 -> angle pi/2 -> (0, R)
    za, zb = philox.box_muller(wa, np.array([1 << 30]))
    assert abs(za[0]) < 1e-15 and zb[0] == pytest.approx(np.sqrt(-2 * np.log(u1)), rel=1e-15)


def test_normals_pair_words():
    w = philox.stream_words(3, 4, 5, 8).reshape(2, 4)
    z = philox.normals(3, 4, 5, 8).reshape(2, 4)
    a, b = philox.box_muller(w[:, 0], w[:, 1])
    c, d = philox.box_muller(w[:, 2], w[:, 3])
    assert np.array_equal(z, np.stack([a, b, c, d], axis=1))


def test_normals_distribution():
    n = 1 << 20
    z = philox.normals(0, 0, 0, n)
    assert abs(z.mean()) < 5.0 / np.sqrt(n)
    assert abs(z.var() - 1.0) < 5.0 * np.sqrt(2.0 / n)
    assert stats.kstest(z, "norm").pvalue > 1e-3
    # fourth moment of N(0,1) is 3
    assert abs(np.mean(z ** 4) - 3.0) < 0.05
    # the two normals of a Box-Muller pair, and neighbouring pairs, are uncorrelated
    zz = z.reshape(-1, 4)
    for i, j in [(0, 1), (0, 2), (1, 3), (2, 3)]:
        assert abs(np.corrcoef(zz[:, i], zz[:, j])[0, 1]) < 5.0 / np.sqrt(zz.shape[0])


def test_streams_are_distinct():
    base = philox.normals(7, 3, 11, 4096)
    for args in [(8, 3, 11), (7, 4, 11), (7, 3, 12), (7 | (1 << 40), 3, 11), (7, 3, 11 | (1 << 33))]:
        other = philox.normals(*args, 4096)
        assert abs(np.corrcoef(base, other)[0, 1]) < 0.1
        assert not np.any(base == other)


def test_perturbation_layout():
    Z = philox.perturbation(1, 2, 3, 5, 3)
    flat = philox.normals(1, 2, 3, 15)
    assert Z.shape == (5, 3)
    assert np.array_equal(Z.reshape(-1), flat)


def test_estimator_moments_section4():
    # Section 4: for z ~ N(0, I_k), a = <g, z> z has E[a] = g and E||a||^2 = (k+2)||g||^2.
    k, N = 48, 40000
    rng = np.random.default_rng(0)
    g = rng.standard_normal(k)
    Zs = np.stack([philox.normals(123, 9, q, k) for q in range(N)])
    a = (Zs @ g)[:, None] * Zs
    mean = a.mean(axis=0)
    # CLT: E||mean - g||^2 = (k+1)||g||^2 / N
    err = np.linalg.norm(mean - g)
    assert err < 3.0 * np.sqrt((k + 1) / N) * np.linalg.norm(g)
    second = np.mean(np.sum(a * a, axis=1))
    assert second == pytest.approx((k + 2) * g @ g, rel=0.05)
