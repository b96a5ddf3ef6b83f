"""Replica support on the GPU (C ABI) against the oracle: the arena fingerprint bit for bit, and the rank
mean of an all-reduced loss vector exactly (IEEE division on both sides)."""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from paper_2607_01125_gb300 import dp
from oracle import replica

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    c.close()


def _u64(t):
    return int(t.item()) & (2 ** 64 - 1)


@pytest.mark.parametrize("n", [0, 1, 3, 4, 5, 1000, (1 << 20) + 3, 22_020_096])
def test_arena_hash_matches_oracle(ctx, n):
    g = torch.Generator(device=DEV).manual_seed(n)
    a = torch.randn(n, device=DEV, generator=g)
    out = torch.full((1,), -1, dtype=torch.int64, device=DEV)
    zo.zoact_arena_hash(ctx, a, out)
    torch.cuda.synchronize()
    assert _u64(out) == replica.arena_hash(a.cpu().numpy())
    if n >= 4:                                      # one bit of one word changes it
        b = a.clone()
        b.view(torch.int32)[n // 2] ^= 1 << 7
        zo.zoact_arena_hash(ctx, b, out)
        torch.cuda.synchronize()
        assert _u64(out) == replica.arena_hash(b.cpu().numpy()) != replica.arena_hash(a.cpu().numpy())


def test_arena_hash_of_16bit_and_offset_views(ctx):
    w = torch.randn(4097, 64, device=DEV).to(torch.bfloat16)       # bytes as 32-bit words
    out = torch.empty(1, dtype=torch.int64, device=DEV)
    zo.zoact_arena_hash(ctx, w, out)
    torch.cuda.synchronize()
    assert _u64(out) == replica.arena_hash(w.cpu().view(torch.int32).numpy())
    c = torch.randn(1003, device=DEV)
    with pytest.raises(zo.ZoactError) as ei:      # 4-byte aligned, not 16: refused before any launch
        zo.zoact_arena_hash(ctx, c[1:], out)
    assert ei.value.status == zo._lib.ZOACT_ERR_INVALID_ARG
    zo.zoact_arena_hash(ctx, c[4:], out)          # 16-byte aligned view
    torch.cuda.synchronize()
    assert _u64(out) == replica.arena_hash(c[4:].cpu().numpy())


@pytest.mark.parametrize("world", [2, 3, 8])
def test_mean_over_ranks_exact(ctx, world):
    v = torch.randn(33, dtype=torch.float64, device=DEV) * 1e3
    ref = v.cpu().numpy() / world
    zo.zoact_mean_over_ranks(ctx, v, world)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(v.cpu().numpy(), ref)


def test_replica_check_single_process(ctx):
    C = torch.randn(1 << 16, device=DEV)
    st, bad = dp.check_replicas([C, C * 0.5], ctx=ctx)
    assert st == zo._lib.ZOACT_OK and bad == []
    fp = dp.replica_fingerprints([C], ctx=ctx)
    assert fp.shape == (1, 1) and (int(fp[0, 0]) & (2 ** 64 - 1)) == replica.arena_hash(C.cpu().numpy())
