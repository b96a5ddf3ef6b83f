"""Oracle: the one-shot activation basis, Algorithm 1 (test infrastructure only).

Algorithm 1 (Subspace Initialization) runs one calibration forward pass, takes
the input activation matrix X_l of each linear layer and keeps the top-r right
singular vectors V_{l,r} of X_l, frozen for the rest of training.  Section 3
motivates this from the thin SVD X = U D V^T.

The right singular vectors of X are the eigenvectors of the uncentred Gram
matrix G = X^T X (X^T X = V D^2 V^T), with eigenvalues the squared singular
values, in the same order.  So the exact basis is the definition written out:

    top_r_basis(X, r) = the r eigenvectors of X^T X with the largest eigenvalues.

The paper does not say how the SVD is computed.  The device path reaches the
same subspace by randomised subspace iteration on G followed by Rayleigh-Ritz;
``subspace_iteration`` below writes those steps out in fp64 so a test can
compare the device result with the same iteration, and ``top_r_basis`` gives
the limit.  Readings the paper leaves open (fixed here):

* no centring (the SVD is of X itself, Section 3);
* sign: each column is flipped so that its entry of largest magnitude is
  positive (the lowest index wins a tie);
* columns in descending eigenvalue order.

``jacobi_eigh`` is a plain cyclic Jacobi eigensolver (Golub & Van Loan,
Section 8.5), used to pin ``top_r_basis`` on small matrices.
"""
import numpy as np

from .philox import perturbation


def canonical_signs(U):
    """Flip each column so its largest-|.| entry is positive (lowest index on ties)."""
    U = np.array(U, np.float64, copy=True)
    for j in range(U.shape[1]):
        i = int(np.argmax(np.abs(U[:, j])))       # argmax returns the first maximum
        if U[i, j] < 0:
            U[:, j] = -U[:, j]
    return U


def gram(X):
    """G = X^T X, uncentred, fp64."""
    X = np.asarray(X, np.float64)
    return X.T @ X


def top_r_basis(X, r):
    """Algorithm 1 for one layer: top-r right singular vectors of X as [d_in, r].

    Also returns the eigenvalues of X^T X in descending order (all d_in of them),
    which tests use for the eigengap.
    """
    G = gram(X)
    evals, evecs = np.linalg.eigh(G)          # ascending
    order = np.argsort(evals)[::-1]
    evals = evals[order]
    U = canonical_signs(evecs[:, order[:r]])
    return U, evals


def jacobi_eigh(A, tol=1e-14, max_sweeps=100):
    """Cyclic Jacobi eigendecomposition of a symmetric matrix (fp64).

    Returns (eigenvalues descending, eigenvectors as columns).
    Each rotation in plane (p, q) zeroes A[p, q]:
        theta = (A[q,q] - A[p,p]) / (2 A[p,q]),
        t = sign(theta) / (|theta| + sqrt(theta^2 + 1)),  c = 1/sqrt(1+t^2), s = t c.
    """
    A = np.array(A, np.float64, copy=True)
    n = A.shape[0]
    V = np.eye(n)
    scale = max(np.sqrt(np.sum(A * A)), 1e-300)
    for _ in range(max_sweeps):
        off = np.sqrt(np.sum(A * A) - np.sum(np.diag(A) ** 2))
        if off <= tol * scale:
            break
        for p in range(n - 1):
            for q in range(p + 1, n):
                apq = A[p, q]
                if abs(apq) <= 1e-300:
                    continue
                theta = (A[q, q] - A[p, p]) / (2.0 * apq)
                if abs(theta) > 1e150:                 # theta^2 would overflow: t ~ 1/(2 theta)
                    t = 0.5 / theta
                else:
                    t = (1.0 if theta >= 0 else -1.0) / (abs(theta) + np.sqrt(theta * theta + 1.0))
                c = 1.0 / np.sqrt(1.0 + t * t)
                s = t * c
                # A <- J^T A J with J the rotation in plane (p, q)
                Ap = A[:, p].copy()
                Aq = A[:, q].copy()
                A[:, p] = c * Ap - s * Aq
                A[:, q] = s * Ap + c * Aq
                Ap = A[p, :].copy()
                Aq = A[q, :].copy()
                A[p, :] = c * Ap - s * Aq
                A[q, :] = s * Ap + c * Aq
                Vp = V[:, p].copy()
                Vq = V[:, q].copy()
                V[:, p] = c * Vp - s * Vq
                V[:, q] = s * Vp + c * Vq
    evals = np.diag(A).copy()
    order = np.argsort(evals)[::-1]
    return evals[order], V[:, order]


def basis_sketch(seed, d_in, k):
    """The Gaussian start block Omega [d_in, k] of the subspace iteration.

    Drawn from the same Philox stream definition as Z, with layer_id 0 and
    query 0 of the basis seed: Omega[i, j] is element i * k + j.
    """
    return perturbation(seed, 0, 0, d_in, k)


def subspace_iteration(G, r, oversample, n_iter, seed):
    """Randomised subspace iteration with Rayleigh-Ritz, in fp64.

    k = r + oversample;  Q_0 = orth(Omega);  Q_i = orth(G Q_{i-1}) for i = 1..n_iter;
    S = Q^T G Q;  S = V diag(theta) V^T (theta descending);  U = Q V[:, :r],
    sign-canonicalised.  orth() is a thin QR; the result does not depend on its
    sign convention.
    """
    G = np.asarray(G, np.float64)
    d = G.shape[0]
    k = min(int(r) + int(oversample), d)
    Q, _ = np.linalg.qr(basis_sketch(seed, d, k))
    for _ in range(int(n_iter)):
        Q, _ = np.linalg.qr(G @ Q)
    S = Q.T @ G @ Q
    S = 0.5 * (S + S.T)
    theta, V = np.linalg.eigh(S)
    order = np.argsort(theta)[::-1]
    U = Q @ V[:, order[:r]]
    return canonical_signs(U), theta[order]


def subspace_overlap(U1, U2):
    """||U1^T U2||_F^2 / r, the subspace stability metric of Section 5.3."""
    U1 = np.asarray(U1, np.float64)
    U2 = np.asarray(U2, np.float64)
    return float(np.sum((U1.T @ U2) ** 2) / U1.shape[1])


def gradient_energy(U, G):
    """Gradient-energy capture of Section 5.3: the share of a weight gradient's energy inside the basis,
    ||U^T G||_F^2 / ||G||_F^2, with U [d_in, r] orthonormal and G [d_in, n] (the gradient of W in the
    paper's [d_in, d_out] orientation).  Returns (||U^T G||_F^2, ||G||_F^2, ratio)."""
    U = np.asarray(U, np.float64)
    G = np.asarray(G, np.float64)
    num = float(np.sum((U.T @ G) ** 2))
    den = float(np.sum(G * G))
    return num, den, num / den
