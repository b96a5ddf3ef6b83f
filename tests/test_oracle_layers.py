"""Pins for the oracle's adapted linear and INT4 dequantisation (CPU only).

Section 3: W_eff = W + V_r B with B = 0 at init reproduces the base layer; the
perturbed pass is Y+ = XW + (X V_r)(B + mu Z); perturbing inside span(V_r) moves
the output by U_r D_r R (X V_r = U_r D_r).
"""
import numpy as np
import pytest
import torch

from oracle import layers, basis
from synth import quantize_int4_g128


def _rand(rng, *shape):
    return rng.standard_normal(shape)


def test_zero_coefficients_reproduce_base_layer_exactly():
    rng = np.random.default_rng(1)
    W, U, X = _rand(rng, 24, 40), _rand(rng, 40, 4), _rand(rng, 10, 40)
    C = np.zeros((24, 4))
    Z = _rand(rng, 24, 4)
    Y = layers.pair_forward(W, U, C, Z, X, 0.0, 5, False)
    assert np.array_equal(Y, X @ W.T)
    Y = layers.pair_forward(W, U, C, Z, X[:5], 0.0, 5, True)
    assert np.array_equal(Y[:5], X[:5] @ W.T) and np.array_equal(Y[5:], X[:5] @ W.T)


def test_pair_forward_brute_force_loops():
    rng = np.random.default_rng(2)
    d_in, d_out, r, T = 7, 5, 3, 4
    W, U, C, Z = _rand(rng, d_out, d_in), _rand(rng, d_in, r), _rand(rng, d_out, r), _rand(rng, d_out, r)
    X = _rand(rng, 2 * T, d_in)
    eps = 0.37
    Y = layers.pair_forward(W, U, C, Z, X, eps, T, False)
    for t in range(2 * T):
        sigma = 1.0 if t < T else -1.0
        for i in range(d_out):
            acc = 0.0
            for k in range(d_in):
                acc += W[i, k] * X[t, k]
            for j in range(r):
                p = 0.0
                for k in range(d_in):
                    p += U[k, j] * X[t, k]
                acc += (C[i, j] + sigma * eps * Z[i, j]) * p
            assert Y[t, i] == pytest.approx(acc, rel=1e-12, abs=1e-12)


def test_pair_difference_is_2eps_Z_p():
    rng = np.random.default_rng(3)
    W, U, C, Z = _rand(rng, 16, 32), _rand(rng, 32, 4), _rand(rng, 16, 4), _rand(rng, 16, 4)
    X = _rand(rng, 6, 32)
    eps = 1e-3
    Y = layers.pair_forward(W, U, C, Z, X, eps, 6, True)
    P = X @ U
    np.testing.assert_allclose(Y[:6] - Y[6:], 2 * eps * P @ Z.T, rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(0.5 * (Y[:6] + Y[6:]), X @ W.T + P @ C.T, rtol=1e-12, atol=1e-12)


def test_perturbation_identity_section3():
    # Delta W = V_r R  =>  Delta Y = X V_r R = U_r D_r R: the perturbed outputs move
    # only along the top-r left singular directions, scaled by the singular values.
    rng = np.random.default_rng(4)
    n, m, r = 50, 20, 3
    X = _rand(rng, n, 6) @ _rand(rng, 6, m) + 0.01 * _rand(rng, n, m)
    V_r, _ = basis.top_r_basis(X, r)
    Ul, s, _ = np.linalg.svd(X, full_matrices=False)
    R = _rand(rng, 7, r)                             # [d_out, r] as stored
    Y = layers.pair_forward(np.zeros((7, m)), V_r, np.zeros((7, r)), R, X, 1.0, n, True)
    dY = Y[:n]
    # columns of X V_r are orthogonal with norms sigma_1..sigma_r
    XV = X @ V_r
    np.testing.assert_allclose(XV.T @ XV, np.diag(s[:r] ** 2), rtol=1e-10, atol=1e-8 * s[0] ** 2)
    # and they span exactly the top-r left singular vectors
    proj = Ul[:, :r] @ (Ul[:, :r].T @ dY)
    np.testing.assert_allclose(proj, dY, atol=1e-9 * np.abs(dY).max())


@pytest.mark.parametrize("d_in", [256, 200, 131])
def test_int4_dequant_brute_force(d_in):
    rng = np.random.default_rng(5)
    d_out = 3
    packed = rng.integers(0, 256, size=(d_out, (d_in + 1) // 2), dtype=np.uint8)
    scales = rng.standard_normal((d_out, (d_in + 127) // 128)).astype(np.float16)
    W = layers.dequant_int4_g128(packed, scales, d_in)
    for i in range(d_out):
        for k in range(d_in):
            byte = int(packed[i, k // 2])
            nib = byte & 0xF if k % 2 == 0 else byte >> 4
            q = nib - 16 if nib >= 8 else nib
            assert W[i, k] == q * float(scales[i, k // 128])


def test_int4_quantizer_round_trip():
    g = torch.Generator().manual_seed(0)
    W = torch.randn(8, 512, generator=g) * 0.02
    W[0, :128] = 0.0                                   # an all-zero group
    packed, scales = quantize_int4_g128(W)
    Wd = layers.dequant_int4_g128(packed.numpy(), scales.float().numpy(), 512)
    s = np.repeat(scales.float().numpy(), 128, axis=1)
    err = np.abs(Wd - W.double().numpy())
    # symmetric rounding: |w - q s| <= s/2 (+ the fp16 rounding of s times |q| <= 8)
    assert np.all(err <= 0.5 * s + 8 * np.abs(s) * 2 ** -10 + 1e-12)
    assert np.all(Wd[0, :128] == 0.0)


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(6)
    x = rng.standard_normal(10000) * np.exp(rng.uniform(-20, 20, 10000))
    ours = layers.round_to_bf16(x)
    ref = torch.from_numpy(x).float().to(torch.bfloat16).double().numpy()
    assert np.array_equal(ours, ref)


def test_glue_special_values():
    assert layers.gelu_erf(np.array([0.0]))[0] == 0.0
    # GELU(x) - GELU(-x) = x
    x = np.linspace(-5, 5, 101)
    np.testing.assert_allclose(layers.gelu_erf(x) - layers.gelu_erf(-x), x, atol=1e-14)
    np.testing.assert_allclose(layers.silu(np.array([0.0, 1e3])), [0.0, 1e3])
    h = np.arange(2 * 8 * 3, dtype=np.float64).reshape(2, 24)
    rep = layers.repeat_kv(h, 2, 4, 12)
    assert rep.shape == (2, 96)
    np.testing.assert_array_equal(rep[:, 0:12], h[:, 0:12])
    np.testing.assert_array_equal(rep[:, 36:48], h[:, 0:12])
    np.testing.assert_array_equal(rep[:, 48:60], h[:, 12:24])
    y = layers.rms_norm(np.array([[3.0, 4.0]]), eps=0.0)
    np.testing.assert_allclose(y, [[3.0 / np.sqrt(12.5), 4.0 / np.sqrt(12.5)]])
