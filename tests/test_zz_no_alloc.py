"""The no-allocation pair forward (zoact_pair_forward_noalloc) matches zoact_pair_forward.

This entry point serves callers that must not allocate device memory (a
framework that owns every device allocation, a loop that cannot take a
synchronising cudaMalloc, a fixed memory budget): it runs without a context and
keeps its projection scratch in a fixed static device array.  Two calls in a
row must agree with the regular entry point within the tolerance the pair
forward tests use; a request larger than the static array is refused.
The file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from synth import normal

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _case(d_in, d_out, r, T, shared, dt, seed):
    X = normal(((T if shared else 2 * T), d_in), seed + 1, DEV, dtype=dt)
    W = normal((d_out, d_in), seed + 2, DEV, std=d_in ** -0.5, dtype=dt)
    U = normal((d_in, r), seed + 3, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), seed + 4, DEV, std=0.3)
    return X, W, U, C


@pytest.mark.parametrize("d_in,d_out,r,T,shared,dt", [
    (1000, 520, 16, 200, False, torch.bfloat16),
    (4096, 1024, 32, 128, True, torch.bfloat16),
    (256, 200, 8, 37, False, torch.float32),
])
def test_noalloc_matches_pair_forward_twice(d_in, d_out, r, T, shared, dt):
    ctx = zo.Context(0)
    X, W, U, C = _case(d_in, d_out, r, T, shared, dt, 5)
    L = zo.make_layer(W, U, C, 4)
    eps, seed, query = 0.5, 21, 3
    ref = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, ref)
    for call in range(2):
        Y = torch.full((2 * T, d_out), float("nan"), dtype=torch.float32, device=DEV)
        zo.zoact_pair_forward_noalloc(L, X, T, shared, eps, seed, query, Y)
        torch.cuda.synchronize()
        a, b = Y.double().cpu().numpy(), ref.double().cpu().numpy()
        # same tolerance as the pair-forward parity tests (fp32 output): 1e-4 of the output scale
        assert np.isfinite(a).all()
        assert np.abs(a - b).max() <= 1e-4 * np.abs(b).max(), call
    ctx.close()


def test_noalloc_refuses_requests_beyond_its_scratch():
    d_in, d_out, r = 256, 64, 32
    T = zo._lib.NOALLOC_MAX_PROJ_FLOATS // r          # 2T rows * r floats > the array
    X = torch.zeros(2 * T, d_in, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(d_out, d_in, dtype=torch.bfloat16, device=DEV)
    U = torch.zeros(d_in, r, device=DEV)
    C = torch.zeros(d_out * r, device=DEV)
    Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(zo.ZoactError) as ei:
        zo.zoact_pair_forward_noalloc(zo.make_layer(W, U, C, 0), X, T, False, 1e-3, 0, 0, Y)
    assert ei.value.status == zo._lib.ZOACT_ERR_TOO_LARGE
