"""Pins for the oracle's replica fingerprint (CPU only).

mix64 is pinned by SplitMix64's published known answers (the generator's first
outputs from state 0); the fingerprint of a one-word arena holding 0 is the
first of them.  The rest follows from the definition's structure: every word is
tagged with its index (moving a word changes the fingerprint), every bit of
every word counts, and the integer sum does not depend on the order the words
are added in.
"""
import os

import numpy as np
import pytest

from oracle import replica

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "splitmix64_kat.txt")


def _kat():
    with open(GOLDEN) as f:
        return [int(ln, 16) for ln in f if ln.strip() and not ln.startswith("#")]


def test_splitmix64_known_answers():
    kat = _kat()
    assert len(kat) == 4
    assert replica.splitmix64(0, 4) == kat


def test_one_zero_word_is_the_first_splitmix64_output():
    assert replica.arena_hash(np.zeros(1, np.uint32)) == _kat()[0]
    assert replica.arena_hash(np.zeros(0, np.uint32)) == 0


def test_every_bit_and_position_counts():
    rng = np.random.default_rng(0)
    w = rng.integers(0, 2 ** 32, size=37, dtype=np.uint64).astype(np.uint32)
    h = replica.arena_hash(w)
    for i in (0, 5, 36):
        for bit in (0, 17, 31):
            v = w.copy()
            v[i] ^= np.uint32(1 << bit)
            assert replica.arena_hash(v) != h
    v = w.copy()
    v[[3, 30]] = v[[30, 3]]                     # two distinct words swapped
    assert w[3] != w[30] and replica.arena_hash(v) != h


def test_sum_of_tagged_words_in_any_order():
    rng = np.random.default_rng(1)
    w = rng.integers(0, 2 ** 32, size=1000, dtype=np.uint64).astype(np.uint32)
    terms = [int(replica.mix64(np.uint64((i << 32) | int(x)) + replica.GAMMA)) for i, x in enumerate(w)]
    order = rng.permutation(len(terms))
    assert sum(terms[k] for k in order) % 2 ** 64 == replica.arena_hash(w)


@pytest.mark.parametrize("dtype", [np.float32, np.int32])
def test_bits_of_four_byte_types(dtype):
    a = np.arange(-5, 6).astype(dtype)
    assert replica.arena_hash(a) == replica.arena_hash(a.view(np.uint32))
    assert replica.arena_hash(np.array([0.0], np.float32)) != replica.arena_hash(np.array([-0.0], np.float32))
