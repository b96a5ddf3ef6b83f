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
