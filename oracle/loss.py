"""Oracle: the loss pair and the projected-gradient scalar (test infrastructure only).

Section 3 estimates the coefficient gradient from losses of perturbed forward
passes; Algorithm 2 forms a = (L+ - L) / mu and accumulates a * Z.  This build
uses the two-sided (central) form of the same estimator,

    a = (L+ - L-) / (2 eps),     g_hat = a * Z,

where L+ and L- are the losses of the forward passes with C + eps Z and
C - eps Z on the same mini-batch.

The loss is the mean over all T * n output elements of (y - t)^2 (MSE to a
target), or of y^2 when there is no target.  D = L+ - L- is formed from its own
definition, (1/Tn) sum (y+ - y-)(y+ + y- - 2t), instead of subtracting two
nearly equal numbers; in exact arithmetic the two agree.

``loss_queries`` is the paper's own form (Algorithm 2): one unperturbed pass
and q forward-perturbed passes, a_j = (L^(j,+) - L) / mu, each difference again
formed from its own definition.
"""
import numpy as np


def loss_pair(Y, T, target, eps):
    """Return (L_plus, L_minus, D, a) in fp64.

    Y: [2T, n] stacked outputs (rows [0, T) for +eps, [T, 2T) for -eps).
    target: [T, n] or None (None means the loss is mean(y^2)).
    """
    Y = np.asarray(Y, np.float64)
    y_plus, y_minus = Y[:T], Y[T:2 * T]
    t = 0.0 if target is None else np.asarray(target, np.float64)
    count = y_plus.size
    L_plus = np.sum((y_plus - t) ** 2) / count
    L_minus = np.sum((y_minus - t) ** 2) / count
    # (y+ - t)^2 - (y- - t)^2 = (y+ - y-)(y+ + y- - 2t)
    D = np.sum((y_plus - y_minus) * (y_plus + y_minus - 2.0 * t)) / count
    a = D / (2.0 * eps)
    return float(L_plus), float(L_minus), float(D), float(a)


def loss_queries(Y, T, n_blocks, target, mu):
    """Losses of a multi-point evaluation and the one-sided estimator scalars (Algorithm 2).

    Y: [n_blocks * T, n]; block 0 is the unperturbed pass (loss L), block j >= 1
    the pass at C + mu Z^(j) (loss L^(j,+)).  Returns (L, a) with
    L = [L_0, ..., L_{n_blocks-1}] and a = [a_1, ..., a_q],
    a_j = (L_j - L_0) / mu, where L_j - L_0 is formed from its own definition
    (1/Tn) sum (y_j - y_0)(y_j + y_0 - 2t) as in loss_pair.
    """
    Y = np.asarray(Y, np.float64)
    assert Y.shape[0] == n_blocks * T
    t = 0.0 if target is None else np.asarray(target, np.float64)
    blocks = [Y[b * T:(b + 1) * T] for b in range(n_blocks)]
    count = blocks[0].size
    L = [float(np.sum((yb - t) ** 2) / count) for yb in blocks]
    y0 = blocks[0]
    a = []
    for j in range(1, n_blocks):
        D = np.sum((blocks[j] - y0) * (blocks[j] + y0 - 2.0 * t)) / count
        a.append(float(D / mu))
    return L, a
