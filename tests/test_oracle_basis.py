"""Pins for the oracle's activation basis, Algorithm 1 (CPU only).

* a hand-written cyclic Jacobi eigensolver agrees with LAPACK (numpy eigh) and
  with matrices of known eigendecomposition;
* top_r_basis has orthonormal columns (U^T U = I, Appendix A assumption),
  satisfies G U = U Lambda_r and agrees with Jacobi on small inputs;
* the least-squares gap of Section 4: min_B ||X V_r B - R||^2 - min ||X dW - R||^2
  equals sum_{i>r} ||u_i^T R||^2;
* subspace iteration reaches the known top-r eigenspace.
"""
import numpy as np
import pytest

from oracle import basis


def _sym(rng, n):
    A = rng.standard_normal((n, n))
    return A + A.T


@pytest.mark.parametrize("n", [2, 5, 12, 24])
def test_jacobi_matches_lapack(n):
    rng = np.random.default_rng(n)
    A = _sym(rng, n)
    ev_j, V_j = basis.jacobi_eigh(A)
    ev_l = np.sort(np.linalg.eigvalsh(A))[::-1]
    np.testing.assert_allclose(ev_j, ev_l, rtol=1e-11, atol=1e-11 * np.abs(ev_l).max())
    np.testing.assert_allclose(V_j.T @ V_j, np.eye(n), atol=1e-12)
    np.testing.assert_allclose(A @ V_j, V_j * ev_j, atol=1e-10 * np.abs(ev_l).max())


def test_jacobi_known_decomposition():
    rng = np.random.default_rng(7)
    Q = np.linalg.qr(rng.standard_normal((10, 10)))[0]
    lam = np.array([9.0, 7.5, 6.0, 4.0, 3.0, 2.0, 1.0, 0.5, -1.0, -3.0])
    A = Q @ np.diag(lam) @ Q.T
    ev, V = basis.jacobi_eigh(A)
    np.testing.assert_allclose(ev, lam, atol=1e-12)
    # each eigenvector equals the known one up to sign
    for j in range(10):
        assert abs(abs(V[:, j] @ Q[:, j]) - 1.0) < 1e-10


def test_top_r_basis_is_top_eigenspace_and_orthonormal():
    rng = np.random.default_rng(8)
    X = rng.standard_normal((60, 5)) @ rng.standard_normal((5, 24)) + 0.05 * rng.standard_normal((60, 24))
    r = 4
    U, evals = basis.top_r_basis(X, r)
    np.testing.assert_allclose(U.T @ U, np.eye(r), atol=1e-12)
    G = X.T @ X
    np.testing.assert_allclose(G @ U, U * evals[:r], atol=1e-9 * evals[0])
    # agrees with the hand-written Jacobi (after the same sign rule)
    ev_j, V_j = basis.jacobi_eigh(G)
    np.testing.assert_allclose(evals, ev_j, rtol=1e-10, atol=1e-10 * evals[0])
    np.testing.assert_allclose(U, basis.canonical_signs(V_j[:, :r]), atol=1e-8)
    # and with the squared singular values of X
    s = np.linalg.svd(X, compute_uv=False)
    np.testing.assert_allclose(evals[:r], s[:r] ** 2, rtol=1e-10)


def test_sign_rule():
    U = np.array([[0.1, -0.5], [-0.9, 0.5], [0.2, 0.1]])
    S = basis.canonical_signs(U)
    np.testing.assert_array_equal(S[:, 0], -U[:, 0])     # largest |.| is -0.9
    np.testing.assert_array_equal(S[:, 1], -U[:, 1])     # tie 0.5 / 0.5: first index wins (-0.5)


def test_least_squares_gap_section4():
    rng = np.random.default_rng(9)
    n, m, r = 80, 16, 3
    X = rng.standard_normal((n, m)) * np.exp(-0.4 * np.arange(m))
    R = rng.standard_normal((n, 5))
    V_r, _ = basis.top_r_basis(X, r)
    full = np.linalg.lstsq(X, R, rcond=None)
    restricted = np.linalg.lstsq(X @ V_r, R, rcond=None)
    f_star = np.sum((X @ full[0] - R) ** 2)
    phi_star = np.sum((X @ V_r @ restricted[0] - R) ** 2)
    Ul, s, _ = np.linalg.svd(X, full_matrices=False)
    gap = sum(np.sum((Ul[:, i] @ R) ** 2) for i in range(r, m))
    assert phi_star - f_star == pytest.approx(gap, rel=1e-8)
    # a wrong basis (the bottom-r directions) gives a larger gap
    _, ev = np.linalg.eigh(X.T @ X)
    bad = np.linalg.lstsq(X @ ev[:, :r], R, rcond=None)
    assert np.sum((X @ ev[:, :r] @ bad[0] - R) ** 2) - f_star > gap * 1.01


def test_subspace_iteration_reaches_known_eigenspace():
    rng = np.random.default_rng(10)
    d, r = 64, 4
    Q = np.linalg.qr(rng.standard_normal((d, d)))[0]
    lam = 1.0 / np.arange(1, d + 1) ** 1.5
    G = Q @ np.diag(lam) @ Q.T
    U, theta = basis.subspace_iteration(G, r, oversample=8, n_iter=12, seed=3)
    exact = basis.canonical_signs(Q[:, :r])
    assert basis.subspace_overlap(U, exact) > 1 - 1e-12
    np.testing.assert_allclose(U, exact, atol=1e-6)
    np.testing.assert_allclose(theta[:r], lam[:r], rtol=1e-10)


def test_overlap_metric_section53():
    I = np.eye(6)
    assert basis.subspace_overlap(I[:, :2], I[:, :2]) == 1.0
    assert basis.subspace_overlap(I[:, :2], I[:, 2:4]) == 0.0
    assert basis.subspace_overlap(I[:, :2], I[:, 1:3]) == 0.5


def test_gradient_energy_pins():
    # Section 5.3 energy capture ||U^T G||^2 / ||G||^2: 1 inside the span, 0 orthogonal to it, the sum of the
    # squared coordinates in between, and 1 for a complete orthonormal basis
    rng = np.random.default_rng(12)
    d, r, n = 40, 6, 9
    Q = np.linalg.qr(rng.standard_normal((d, d)))[0]
    U, Uperp = Q[:, :r], Q[:, r:]
    A = rng.standard_normal((r, n))
    B = rng.standard_normal((d - r, n))
    assert basis.gradient_energy(U, U @ A)[2] == pytest.approx(1.0, abs=1e-13)
    assert basis.gradient_energy(U, Uperp @ B)[2] == pytest.approx(0.0, abs=1e-13)
    G = U @ A + Uperp @ B
    num, den, ratio = basis.gradient_energy(U, G)
    assert num == pytest.approx(np.sum(A ** 2), rel=1e-12)
    assert den == pytest.approx(np.sum(A ** 2) + np.sum(B ** 2), rel=1e-12)
    assert basis.gradient_energy(Q, G)[2] == pytest.approx(1.0, abs=1e-13)
    # overlap of the same pair of subspaces equals the energy of U2 (as a gradient) in U1, divided by r
    U2 = np.linalg.qr(rng.standard_normal((d, r)))[0]
    assert basis.subspace_overlap(U, U2) == pytest.approx(basis.gradient_energy(U, U2)[0] / r, rel=1e-12)
