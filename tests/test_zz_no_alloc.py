"""The no-allocation pair forward (zoact_pair_forward_noalloc) against the oracle and zoact_pair_forward.

This entry point serves callers that must not allocate device memory (a
framework that owns every device allocation, a loop that cannot take a
synchronising cudaMalloc, a fixed memory budget): it runs without a context and
keeps its projection scratch in a fixed static device array that every call
shares.  Each case runs a larger call first (which leaves a longer projection
and its split-K partials in the array), then two calls in a row of the checked
shape; both must match the CPU oracle's fp64 pair forward element by element
(the pair-forward tests' fp32 accumulation bound, and 1e-4 of the output scale)
and the regular entry point within 1e-4 of the output scale.  A request that
fills the array exactly runs; one row more is refused.
The file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import layers, philox
from synth import normal

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
MAX = zo._lib.NOALLOC_MAX_PROJ_FLOATS


def n64(t):
    return t.detach().double().cpu().numpy()


def _case(d_in, d_out, r, T, shared, dt, seed):
    X = normal(((T if shared else 2 * T), d_in), seed + 1, DEV, dtype=dt)
    W = normal((d_out, d_in), seed + 2, DEV, std=d_in ** -0.5, dtype=dt)
    U = normal((d_in, r), seed + 3, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), seed + 4, DEV, std=0.3)
    return X, W, U, C


def _oracle(X, W, U, C, eps, T, shared, seed, layer_id, query):
    """The fp64 pair forward (Section 3) and the fp32 accumulation bound of each element."""
    d_out, r = W.shape[0], U.shape[1]
    Zm = philox.perturbation(seed, layer_id, query, d_out, r)
    Cn = n64(C).reshape(d_out, r)
    Y = layers.pair_forward(n64(W), n64(U), Cn, Zm, n64(X), eps, T, shared)
    Xn = n64(X)
    if shared:
        Xn = np.concatenate([Xn, Xn])
    absb = np.abs(Xn) @ np.abs(n64(W)).T + np.abs(Xn @ n64(U)) @ (np.abs(Cn) + abs(eps) * np.abs(Zm)).T
    return Y, 8 * np.sqrt(W.shape[1]) * 2.0 ** -24 * absb + 1e-6


def _noalloc(L, X, T, shared, eps, seed, query, d_out):
    Y = torch.full((2 * T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward_noalloc(L, X, T, shared, eps, seed, query, Y)
    return Y


@pytest.mark.parametrize("d_in,d_out,r,T,shared,dt", [
    (1000, 520, 16, 200, False, torch.bfloat16),
    (4096, 1024, 32, 128, True, torch.bfloat16),
    (256, 200, 8, 37, False, torch.float32),
])
def test_noalloc_matches_oracle_and_pair_forward_twice(d_in, d_out, r, T, shared, dt):
    ctx = zo.Context(0)
    eps, seed, query, lid = 0.5, 21, 3, 4
    # a larger call first: it leaves its projection and split-K partials in the shared array
    Xb, Wb, Ub, Cb = _case(d_in, d_out, r, 4 * T, False, dt, 50)
    _noalloc(zo.make_layer(Wb, Ub, Cb, 9), Xb, 4 * T, False, eps, seed, query, d_out)
    X, W, U, C = _case(d_in, d_out, r, T, shared, dt, 5)
    L = zo.make_layer(W, U, C, lid)
    ref = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, ref)
    Yo, bound = _oracle(X, W, U, C, eps, T, shared, seed, lid, query)
    for call in range(2):
        Y = _noalloc(L, X, T, shared, eps, seed, query, d_out)
        torch.cuda.synchronize()
        a, b = n64(Y), n64(ref)
        assert np.isfinite(a).all()
        err = np.abs(a - Yo)
        assert np.all(err <= bound), (call, err.max())
        assert err.max() <= 1e-4 * np.abs(Yo).max(), call
        # the regular entry point: same tolerance (the low-rank term may ride the tensor cores there)
        assert np.abs(a - b).max() <= 1e-4 * np.abs(b).max(), call
    ctx.close()


def test_noalloc_at_the_limit_and_beyond():
    # rows * r == the array's size: no room is left for split-K partials, so the projection runs in one
    # split and P ends where the status slot begins
    d_in, d_out, r = 64, 64, 16
    T = MAX // r
    eps, seed, query, lid = 0.5, 3, 1, 2
    X, W, U, C = _case(d_in, d_out, r, T, True, torch.bfloat16, 70)
    L = zo.make_layer(W, U, C, lid)
    Y = _noalloc(L, X, T, True, eps, seed, query, d_out)
    ctx = zo.Context(0)
    ref = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, True, eps, seed, query, ref)
    torch.cuda.synchronize()
    a, b = n64(Y), n64(ref)
    assert np.isfinite(a).all()
    assert np.abs(a - b).max() <= 1e-4 * np.abs(b).max()
    rows = np.r_[0:64, T - 64:T + 64, 2 * T - 64:2 * T]        # both ends of both signs against the oracle
    Yo, bound = _oracle(X, W, U, C, eps, T, True, seed, lid, query)
    assert np.all(np.abs(a[rows] - Yo[rows]) <= bound[rows])
    ctx.close()
    # one more row is refused before any launch
    X1 = torch.zeros(T + 1, d_in, dtype=torch.bfloat16, device=DEV)
    Y1 = torch.empty(2 * (T + 1), d_out, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(zo.ZoactError) as ei:
        zo.zoact_pair_forward_noalloc(L, X1, T + 1, True, 1e-3, 0, 0, Y1)
    assert ei.value.status == zo._lib.ZOACT_ERR_TOO_LARGE


def test_noalloc_refuses_requests_beyond_its_scratch():
    d_in, d_out, r = 256, 64, 32
    T = MAX // r                                      # 2T rows * r floats > the array
    X = torch.zeros(2 * T, d_in, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(d_out, d_in, dtype=torch.bfloat16, device=DEV)
    U = torch.zeros(d_in, r, device=DEV)
    C = torch.zeros(d_out * r, device=DEV)
    Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(zo.ZoactError) as ei:
        zo.zoact_pair_forward_noalloc(zo.make_layer(W, U, C, 0), X, T, False, 1e-3, 0, 0, Y)
    assert ei.value.status == zo._lib.ZOACT_ERR_TOO_LARGE
