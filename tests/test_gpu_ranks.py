"""GPU parity at the paper's larger ranks (r up to 256: the Table 3 ablation) against the oracle.

Above 32 ranks the low-rank term always runs on the tensor cores as three bf16 products of 16-bit
splits (stacked rows; a shared input is stacked first), so fp32 outputs carry the fp32 accumulation
bound plus 2^-14 sum_j |P_j| |T_j| (see test_gpu_kernels.py).  The projection groups ranks by 64
(tensor cores) or 32 (fp32 X) per launch; it is checked against the fp64 product with its fp32 bound.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import philox, layers, optim
from synth import normal, quantize_int4_g128
from test_gpu_kernels import _pair_case, _oracle_pair, _bound

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    assert c.device_status() == 0
    c.close()


def np64(t):
    return t.detach().double().cpu().numpy()


@pytest.mark.parametrize("rows,d_in,r,dt,prepared", [(300, 1000, 48, torch.bfloat16, False),
                                                     (1000, 4096, 256, torch.bfloat16, True),
                                                     (129, 512, 100, torch.float16, True),
                                                     (200, 256, 72, torch.float32, False)])
def test_projection_large_rank(ctx, rows, d_in, r, dt, prepared):
    X = normal((rows, d_in), 1, DEV, dtype=dt)
    U = normal((d_in, r), 2, DEV) / np.sqrt(d_in)
    P = torch.empty(rows, r, dtype=torch.float32, device=DEV)
    if prepared:
        utc = torch.empty(zo.zoact_basis_prepared_bytes(d_in, r), dtype=torch.uint8, device=DEV)
        zo.zoact_basis_prepare(ctx, U, zo._lib.TORCH_DT[dt], utc)
        zo.zoact_lowrank_proj_prepared(ctx, X, utc, r, P)
    else:
        zo.zoact_lowrank_proj(ctx, X, U, P)
    torch.cuda.synchronize()
    Xn, Un = np64(X), np64(U)
    ref = Xn @ Un
    bound = 4 * d_in ** 0.5 * 2.0 ** -24 * (np.abs(Xn) @ np.abs(Un)) + 1e-30
    assert np.all(np.abs(np64(P) - ref) <= bound + 1e-6 * np.abs(ref))


@pytest.mark.parametrize("r", [64, 128, 256])
@pytest.mark.parametrize("T,shared", [(256, False), (300, False), (100, False), (200, True)])
def test_pair_forward_large_rank(ctx, r, T, shared):
    d_in, d_out, eps, seed, query, lid = 1024, 392, 0.5, 21, 3, 8
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, torch.bfloat16, eps, 0.3, seed=90)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, lid), X, T, shared, eps, seed, query, Y)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, lid, query, d_out, r)
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= _bound(d_in, absb, lrabs)), err.max()
    assert err.max() <= 1e-4 * np.abs(ref).max()


@pytest.mark.parametrize("T,shared,nb,r", [(256, True, 2, 128), (130, False, 5, 128), (200, True, 2, 32),
                                          (96, True, 5, 24), (150, False, 2, 32)])
def test_gated_and_multi_large_rank(ctx, T, shared, nb, r):
    # r = 17..32 gated on a shared input keeps its +-Z p tables in narrower column chunks
    d_in, d_out, seed, mu = 512, 400, 8, 0.25
    X = normal(((T if shared else nb * T), d_in), 31, DEV, dtype=torch.bfloat16)
    Wg = normal((d_out, d_in), 32, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    Wu = normal((d_out, d_in), 33, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    U = normal((d_in, r), 34, DEV) / np.sqrt(d_in)
    Cg = normal((d_out * r,), 35, DEV, std=0.2)
    Cu = normal((d_out * r,), 36, DEV, std=0.2)
    pts = [(mu, 4), (-mu, 4)] if nb == 2 else [(0.0, 0)] + [(mu, 10 + j) for j in range(nb - 1)]
    H = torch.empty(nb * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_multi_forward_gated(ctx, zo.make_layer(Wg, U, Cg, 0), zo.make_layer(Wu, U, Cu, 1), X, T, shared, pts,
                                 seed, H)
    torch.cuda.synchronize()

    def lin(Wt, Ct, lid):
        Zs = [None if c == 0.0 else philox.perturbation(seed, lid, q, d_out, r) for c, q in pts]
        return layers.multi_forward(np64(Wt), np64(U), np64(Ct).reshape(d_out, r), Zs, [c for c, _ in pts], np64(X),
                                    T, shared)
    ref = layers.silu(lin(Wg, Cg, 0)) * lin(Wu, Cu, 1)
    assert np.abs(np64(H) - ref).max() <= 1e-4 * np.abs(ref).max()


@pytest.mark.parametrize("T,shared", [(37, False), (64, True)])
def test_fp32_pair_large_rank(ctx, T, shared):
    d_in, d_out, r, eps, seed, query, lid = 256, 200, 100, 0.5, 2, 5, 6
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, torch.float32, eps, 0.3, seed=50)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, lid), X, T, shared, eps, seed, query, Y)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, lid, query, d_out, r)
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= _bound(d_in, absb, lrabs)), err.max()


def test_int4_large_rank(ctx):
    d_in, d_out, r, T, eps, seed, query, lid = 1024, 264, 64, 128, 0.5, 4, 2, 9
    Wf = normal((d_out, d_in), 60, DEV, std=0.02)
    packed, scales = quantize_int4_g128(Wf)
    U = normal((d_in, r), 61, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), 62, DEV, std=0.3)
    X = normal((2 * T, d_in), 63, DEV, dtype=torch.bfloat16)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    L = zo.make_layer(packed, U, C, lid, w_scales=scales, wtype=zo.DT_INT4_G128, d_in=d_in)
    zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Y)
    torch.cuda.synchronize()
    Wd = layers.dequant_int4_g128(packed.cpu().numpy(), scales.float().cpu().numpy(), d_in)
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    ref = layers.pair_forward(Wd, np64(U), np64(C).reshape(d_out, r), Zm, np64(X), eps, T, False)
    err = np.abs(np64(Y) - ref)
    assert err.max() <= 2e-3 * np.abs(ref).max()       # bf16 rounding of the dequantised weights dominates


def test_adam_rank_256(ctx):
    specs = [(0, 1000, 256, 3)]
    n = 1000 * 256
    C = normal((n,), 71, DEV, std=0.1)
    m = torch.zeros(n, device=DEV)
    v = torch.zeros(n, device=DEV)
    C0 = np64(C)
    out = torch.tensor([1.0, 0.5, 0.5, -0.4], dtype=torch.float64, device=DEV)
    zo.zoact_adam_step(ctx, C, m, v, specs, out, 1e-3, 0.9, 0.999, 1e-8, 1, 7, 8)
    torch.cuda.synchronize()
    g = optim.zo_gradient(-0.4, philox.perturbation(7, 3, 8, 1000, 256).reshape(-1))
    f32 = lambda x: float(np.float32(x))
    Cr, _, _ = optim.adam_step(C0, 0, 0, g, f32(1e-3), f32(0.9), f32(0.999), f32(1e-8), 1)
    np.testing.assert_allclose(np64(C), Cr, rtol=1e-4, atol=1e-9)


@pytest.mark.parametrize("r,p", [(128, 16), (256, 16), (40, 24)])
def test_basis_large_rank(ctx, r, p):
    # a planted spectrum with a clear gap after r: the device iteration (k = r + p, parallel Jacobi for
    # k > 64) reaches the exact top-r eigenspace of X^T X and its Ritz values
    from oracle import basis
    rng = np.random.default_rng(r)
    n, d = 3072, 1024
    A = rng.standard_normal((n, 300))
    s = np.concatenate([np.linspace(10.0, 6.0, r), 0.3 * np.ones(300 - r)])
    B = np.linalg.qr(rng.standard_normal((d, 300)))[0].T
    Xn = (A * s) @ B + 1e-3 * rng.standard_normal((n, d))
    X = torch.tensor(Xn, dtype=torch.float32, device=DEV).to(torch.bfloat16)
    Xb = np64(X)
    U = torch.empty(d, r, device=DEV)
    ev = torch.empty(r + p, device=DEV)
    zo.zoact_basis_init(ctx, X, r, U, oversample=p, n_iter=8, seed=2, evals_out=ev)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    Ug = np64(U)
    np.testing.assert_allclose(Ug.T @ Ug, np.eye(r), atol=2e-4)
    lam, V = np.linalg.eigh(Xb.T @ Xb)
    order = np.argsort(lam)[::-1]
    assert basis.subspace_overlap(Ug, V[:, order[:r]]) >= 1 - 1e-5
    np.testing.assert_allclose(np64(ev)[:r], lam[order[:r]], rtol=1e-4)
