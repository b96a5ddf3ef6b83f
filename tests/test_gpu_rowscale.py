"""Row scales on the GPU (C ABI) against the oracle: RMS normalisations of the stacks applied inside the pair
forwards instead of as separate passes.

rms(x) = x / sqrt(mean(x^2) + eps) is a per-row scale, so the pair forward of rms(x) equals the pair forward of x
(and of its projection) with every output row times 1/s.  The fp32-output cases check that against the oracle's
pair forward of the normalised input within the fp32 accumulation bound; the sums of squares a launch writes are
checked against the squares of its own stored outputs, and zoact_rms_scale against 1/rms of those outputs.
Launches the kernels cannot apply row scales to are refused before anything is launched.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import layers, philox
from synth import normal

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    c.close()


def n64(t):
    return t.detach().double().cpu().numpy()


def _case(d_in, d_out, r, T, seed):
    # rows of very different norms, as a decoder's unnormalised outputs have
    X = normal((2 * T, d_in), seed + 1, DEV) * (0.5 + 3.0 * torch.rand(2 * T, 1, device=DEV,
                                                                      generator=torch.Generator(DEV).manual_seed(seed)))
    X = X.to(torch.bfloat16)
    W = normal((d_out, d_in), seed + 2, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    U = normal((d_in, r), seed + 3, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), seed + 4, DEV, std=0.3)
    return X, W, U, C


def _inv_rms(X, eps=1e-5):
    x = n64(X)
    return 1.0 / np.sqrt(np.mean(x * x, axis=1) + eps)


@pytest.mark.parametrize("d_in,d_out,r,T", [(1024, 520, 16, 200), (4096, 1024, 16, 256), (2048, 776, 32, 300)])
def test_pair_forward_in_scale_matches_oracle_of_normalised_input(ctx, d_in, d_out, r, T):
    eps, seed, query, lid = 0.5, 9, 2, 3
    X, W, U, C = _case(d_in, d_out, r, T, 30)
    inv = torch.from_numpy(_inv_rms(X).astype(np.float32)).to(DEV)
    L = zo.make_layer(W, U, C, lid)
    Y = torch.full((2 * T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward_rs(ctx, L, X, T, False, eps, seed, query, Y, in_scale=inv)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    Xn = n64(X) * n64(inv)[:, None]                  # the normalised input, in fp64 from the same stored scale
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    Cn = n64(C).reshape(d_out, r)
    ref = layers.pair_forward(n64(W), n64(U), Cn, Zm, Xn, eps, T, False)
    absb = np.abs(Xn) @ np.abs(n64(W)).T + np.abs(Xn @ n64(U)) @ (np.abs(Cn) + eps * np.abs(Zm)).T
    err = np.abs(n64(Y) - ref)
    assert np.all(err <= 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 2.0 ** -14 * absb + 1e-6), err.max()


@pytest.mark.parametrize("gated,ydt,T", [(False, torch.bfloat16, 256), (False, torch.float32, 300),
                                         (True, torch.bfloat16, 256), (True, torch.bfloat16, 384)])
def test_sums_of_squares_and_rms_scale(ctx, gated, ydt, T):
    d_in, d_out, r = 1024, 776 if not gated else 768, 16
    eps, seed, query = 0.25, 5, 1
    X, W, U, C = _case(d_in, d_out, r, T, 40)
    inv_in = torch.from_numpy(_inv_rms(X).astype(np.float32)).to(DEV)
    L = zo.make_layer(W, U, C, 0)
    parts = zo.rowscale_parts(d_out)
    ss = torch.full((parts, 2 * T), float("nan"), device=DEV)
    Y = torch.empty(2 * T, d_out, dtype=ydt, device=DEV)
    if gated:
        X2, W2, U2, C2 = _case(d_in, d_out, r, T, 50)
        L2 = zo.make_layer(W2, U2, C2, 1)
        zo.zoact_pair_forward_gated_rs(ctx, L, L2, X, T, False, eps, seed, query, Y, in_scale=inv_in, out_sumsq=ss)
        ref = torch.empty_like(Y)
        Xs = (X.float() * inv_in[:, None]).to(torch.bfloat16)          # the explicitly normalised input
        zo.zoact_pair_forward_gated(ctx, L, L2, Xs, T, False, eps, seed, query, ref)
    else:
        zo.zoact_pair_forward_rs(ctx, L, X, T, False, eps, seed, query, Y, act=zo.ACT_RELU, in_scale=inv_in,
                                 out_sumsq=ss)
        ref = torch.empty_like(Y)
        Xs = (X.float() * inv_in[:, None]).to(torch.bfloat16)
        zo.zoact_pair_forward(ctx, L, Xs, T, False, eps, seed, query, ref, act=zo.ACT_RELU)
    inv = torch.empty(2 * T, device=DEV)
    zo.zoact_rms_scale(ctx, ss, d_out, inv)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    y = n64(Y)
    # the sums of squares of Y's own stored values, per 64-column part
    want = np.stack([np.sum(y[:, 64 * p:64 * p + 64] ** 2, axis=1) for p in range(parts)])
    np.testing.assert_allclose(n64(ss), want, rtol=2e-6, atol=1e-30)
    np.testing.assert_allclose(n64(inv), 1.0 / np.sqrt(np.mean(y * y, axis=1) + 1e-5), rtol=2e-6)
    # against normalising the input first: one rounding of the normalised input apart
    rr = n64(ref)
    assert np.abs(y - rr).max() <= 2e-2 * np.abs(rr).max()
    assert np.mean(np.abs(y - rr)) <= 5e-3 * np.mean(np.abs(rr))


def test_row_scales_refused_where_not_applied(ctx):
    d_in, d_out, r = 512, 256, 16
    X, W, U, C = _case(d_in, d_out, r, 256, 60)
    L = zo.make_layer(W, U, C, 0)
    inv = torch.ones(512, device=DEV)
    Y = torch.empty(512, d_out, dtype=torch.bfloat16, device=DEV)
    n0 = ctx.launch_count()
    for args in [(X[:256], 256, True), (X[:128], 64, False)]:      # shared input; 128 stacked rows
        with pytest.raises(zo.ZoactError) as ei:
            zo.zoact_pair_forward_rs(ctx, L, args[0], args[1], args[2], 0.1, 0, 0, Y[:2 * args[1]], in_scale=inv)
        assert ei.value.status == zo._lib.ZOACT_ERR_UNSUPPORTED
    assert ctx.launch_count() == n0                   # nothing launched
