"""Pins for the oracle's multi-point evaluation and the paper's one-sided q-query
estimator (Algorithm 2), CPU only.

* The two-sided pair is the block case coefs = (eps, -eps): multi_forward equals
  pair_forward bit for bit; a block with coef 0 is the unperturbed layer.
* For one adapted linear under MSE the loss is quadratic in C, so the forward
  difference has a closed form: (L(C + mu Z) - L(C)) / mu
  = <grad_C L, Z> + (mu / Tn) ||(X U) Z^T||^2, for every mu.
* Through a non-quadratic graph (two layers with GELU) the forward difference
  converges to <grad L, Z> at rate O(mu): halving mu halves the error.
* Averaged over many queries, g_hat = (1/q) sum_j a_j Z^(j) tends to grad_C L
  (E[Z Z^T] = I), within the Monte-Carlo error.
"""
import numpy as np
import pytest
import torch

from oracle import graphs, layers, loss, optim, philox


def _lin(rng, d_in=12, d_out=9, r=3):
    W = rng.standard_normal((d_out, d_in))
    U = np.linalg.qr(rng.standard_normal((d_in, r)))[0]
    C = 0.1 * rng.standard_normal((d_out, r))
    return W, U, C


@pytest.mark.parametrize("shared", [True, False])
def test_pair_is_the_two_block_case(shared):
    rng = np.random.default_rng(3)
    W, U, C = _lin(rng)
    T, eps = 5, 1e-3
    X = rng.standard_normal((T if shared else 2 * T, W.shape[1]))
    Z = philox.perturbation(7, 4, 2, *C.shape)
    ref = layers.pair_forward(W, U, C, Z, X, eps, T, shared)
    got = layers.multi_forward(W, U, C, [Z, Z], [eps, -eps], X, T, shared)
    assert np.array_equal(ref, got)


def test_zero_coefficient_block_is_the_unperturbed_layer():
    rng = np.random.default_rng(4)
    W, U, C = _lin(rng)
    T = 6
    X = rng.standard_normal((T, W.shape[1]))
    Z = philox.perturbation(1, 1, 1, *C.shape)
    Y = layers.multi_forward(W, U, C, [None, Z], [0.0, 0.5], X, T, True)
    np.testing.assert_allclose(Y[:T], X @ (W + C @ U.T).T, rtol=1e-12, atol=1e-12)
    Y0 = layers.multi_forward(W, U, np.zeros_like(C), [None], [0.0], X, T, True)
    assert np.array_equal(Y0, X @ W.T)


@pytest.mark.parametrize("mu", [1e-1, 1e-3])
@pytest.mark.parametrize("shared", [True, False])
def test_forward_difference_closed_form_on_a_quadratic(mu, shared):
    rng = np.random.default_rng(5)
    W, U, C = _lin(rng)
    T, q = 8, 4
    x = rng.standard_normal((T, W.shape[1]))
    tgt = rng.standard_normal((T, W.shape[0]))
    Zs = [philox.perturbation(11, 3, j, *C.shape) for j in range(1, q + 1)]
    X = x if shared else np.concatenate([x] * (q + 1), axis=0)
    Y = layers.multi_forward(W, U, C, [None] + Zs, [0.0] + [mu] * q, X, T, shared)
    L, a = loss.loss_queries(Y, T, q + 1, tgt, mu)
    P = x @ U
    R = x @ W.T + P @ C.T - tgt
    n = W.shape[0]
    grad = 2.0 / (T * n) * R.T @ P
    assert L[0] == pytest.approx(np.mean(R ** 2), rel=1e-13)
    for j, Zj in enumerate(Zs):
        want = float(np.sum(grad * Zj)) + mu / (T * n) * float(np.sum((P @ Zj.T) ** 2))
        assert a[j] == pytest.approx(want, rel=1e-9, abs=1e-12)
        assert L[j + 1] == pytest.approx(np.mean((R + P @ (mu * Zj).T) ** 2), rel=1e-12)


def test_loss_queries_differences_and_mean_square():
    rng = np.random.default_rng(6)
    T, n, nb, mu = 7, 5, 4, 1e-2
    Y = rng.standard_normal((nb * T, n))
    t = rng.standard_normal((T, n))
    L, a = loss.loss_queries(Y, T, nb, t, mu)
    assert len(L) == nb and len(a) == nb - 1
    for b in range(nb):
        assert L[b] == pytest.approx(np.mean((Y[b * T:(b + 1) * T] - t) ** 2), rel=1e-14)
    for j in range(1, nb):
        assert a[j - 1] == pytest.approx((L[j] - L[0]) / mu, rel=1e-10)
    L2, a2 = loss.loss_queries(Y, T, nb, None, mu)
    assert L2 == pytest.approx(loss.loss_queries(Y, T, nb, np.zeros((T, n)), mu)[0])
    assert a2 == pytest.approx(loss.loss_queries(Y, T, nb, np.zeros((T, n)), mu)[1])


def _toy_layers(rng):
    def lay(d_in, d_out, r, lid):
        return dict(W=rng.standard_normal((d_out, d_in)) / np.sqrt(d_in),
                    U=np.linalg.qr(rng.standard_normal((d_in, r)))[0],
                    C=0.2 * rng.standard_normal((d_out, r)), layer_id=lid)
    return [lay(16, 16, 4, 0), lay(16, 16, 4, 1)]


def test_forward_difference_rate_through_gelu_graph():
    rng = np.random.default_rng(7)
    lays = _toy_layers(rng)
    T = 6
    x = rng.standard_normal((T, 16))
    tgt = rng.standard_normal((T, 16))
    Cs = [torch.tensor(l["C"], requires_grad=True) for l in lays]
    h = torch.tensor(x)
    for i, (l, c) in enumerate(zip(lays, Cs)):
        h = h @ torch.tensor(l["W"]).T + (h @ torch.tensor(l["U"])) @ c.T
        if i == 0:
            h = torch.nn.functional.gelu(h)
    torch.mean((h - torch.tensor(tgt)) ** 2).backward()
    seed, query = 9, 3
    dd = sum(float(np.sum(c.grad.numpy() * philox.perturbation(seed, l["layer_id"], query, *l["C"].shape)))
             for c, l in zip(Cs, lays))
    errs = []
    for mu in (2e-2, 1e-2, 5e-3):
        Y = graphs.toy_forward(lays, x, 0.0, seed, 0, store="fp64", blocks=[(0.0, 0), (mu, query)])
        _, a = loss.loss_queries(Y, T, 2, tgt, mu)
        errs.append(abs(a[0] - dd))
    assert errs[0] / errs[1] == pytest.approx(2.0, rel=0.1)
    assert errs[1] / errs[2] == pytest.approx(2.0, rel=0.1)


def test_query_average_tends_to_the_gradient():
    rng = np.random.default_rng(8)
    W, U, C = _lin(rng, d_in=6, d_out=3, r=2)
    T, mu, q = 4, 1e-7, 4000
    x = rng.standard_normal((T, 6))
    tgt = rng.standard_normal((T, 3))
    Zs = [philox.perturbation(21, 0, j, 3, 2) for j in range(1, q + 1)]
    Y = layers.multi_forward(W, U, C, [None] + Zs, [0.0] + [mu] * q, x, T, True)
    _, a = loss.loss_queries(Y, T, q + 1, tgt, mu)
    g_hat = optim.zo_gradient_queries(a, Zs)
    P = x @ U
    grad = 2.0 / (T * 3) * (x @ W.T + P @ C.T - tgt).T @ P
    # each component of g_hat has standard deviation sqrt((|grad|^2 + grad_i^2) / q)
    sd = np.sqrt((np.sum(grad ** 2) + grad ** 2) / q)
    assert np.all(np.abs(g_hat - grad) <= 4.5 * sd)
    # q = 1 is the single-query estimator a Z
    assert np.array_equal(optim.zo_gradient_queries(a[:1], Zs[:1]), optim.zo_gradient(a[0], Zs[0]))
