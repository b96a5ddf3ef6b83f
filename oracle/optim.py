"""Oracle: the optimizer step on the coefficients (test infrastructure only).

Section 3 updates B "with a first-order optimizer such as Adam" fed the
estimated gradient g_hat = a * Z; Section 5 states Adam, and the Appendix B
hyperparameter tables fix weight decay 0 and a constant-with-warmup learning
rate (the host passes the step's lr).  The paper is silent on beta, epsilon and
bias correction; this build reads them as the standard bias-corrected Adam
(Kingma & Ba, 2015):

    m <- b1 m + (1 - b1) g
    v <- b2 v + (1 - b2) g^2
    m_hat = m / (1 - b1^t),   v_hat = v / (1 - b2^t)        (t is 1-based)
    C <- C - lr * m_hat / (sqrt(v_hat) + adam_eps)

The SGD variant ("ZO-Act Full SGD", Table 1) is C <- C - lr * g.
"""
import numpy as np


def adam_step(C, m, v, g, lr, beta1, beta2, adam_eps, step):
    """One Adam step in fp64.  Returns new (C, m, v)."""
    C = np.asarray(C, np.float64)
    m = np.asarray(m, np.float64)
    v = np.asarray(v, np.float64)
    g = np.asarray(g, np.float64)
    m_new = beta1 * m + (1.0 - beta1) * g
    v_new = beta2 * v + (1.0 - beta2) * g * g
    m_hat = m_new / (1.0 - beta1 ** step)
    v_hat = v_new / (1.0 - beta2 ** step)
    C_new = C - lr * m_hat / (np.sqrt(v_hat) + adam_eps)
    return C_new, m_new, v_new


def sgd_step(C, g, lr):
    return np.asarray(C, np.float64) - lr * np.asarray(g, np.float64)


def zo_gradient(a, Z):
    """g_hat = a * Z (Section 3 estimator with one query)."""
    return float(a) * np.asarray(Z, np.float64)


def zo_gradient_queries(a, Zs):
    """g_hat = (1/q) sum_j a_j Z^(j)  (Algorithm 2, averaged over q queries)."""
    q = len(a)
    assert q == len(Zs) and q > 0
    g = np.zeros_like(np.asarray(Zs[0], np.float64))
    for aj, Zj in zip(a, Zs):
        g = g + float(aj) * np.asarray(Zj, np.float64)
    return g / q
