"""Pins for the oracle's loss pair, estimator scalar and optimizer step (CPU only).

* For one adapted linear under MSE the loss is quadratic in C, so the central
  difference (L+ - L-)/(2 eps) equals the directional derivative <grad_C L, Z>
  exactly, for every eps (the estimator of Section 3 in two-sided form).
* For a non-quadratic graph (two layers with GELU) the error is O(eps^2).
* Adam at t = 1 has the closed form C - lr g / (|g| + eps); ten steps match
  torch.optim.Adam run on the same gradients (a library special case).
"""
import numpy as np
import pytest
import torch

from oracle import layers, loss, optim, philox, graphs


def test_D_matches_difference_and_mean_square():
    rng = np.random.default_rng(0)
    Y = rng.standard_normal((20, 7))
    t = rng.standard_normal((10, 7))
    Lp, Lm, D, a = loss.loss_pair(Y, 10, t, 1e-3)
    assert Lp == pytest.approx(np.mean((Y[:10] - t) ** 2), rel=1e-14)
    assert Lm == pytest.approx(np.mean((Y[10:] - t) ** 2), rel=1e-14)
    assert D == pytest.approx(Lp - Lm, rel=1e-12, abs=1e-15)
    assert a == pytest.approx(D / 2e-3, rel=1e-15)
    assert loss.loss_pair(Y, 10, None, 1e-3) == pytest.approx(loss.loss_pair(Y, 10, np.zeros((10, 7)), 1e-3))


@pytest.mark.parametrize("eps", [1e-1, 1e-3, 1e-6])
def test_quadratic_loss_central_difference_is_exact(eps):
    rng = np.random.default_rng(1)
    d_in, d_out, r, T = 12, 9, 3, 8
    W, U = rng.standard_normal((d_out, d_in)), rng.standard_normal((d_in, r))
    C = 0.1 * rng.standard_normal((d_out, r))
    X = rng.standard_normal((T, d_in))
    tgt = rng.standard_normal((T, d_out))
    Z = philox.perturbation(5, 2, 0, d_out, r)
    Y = layers.pair_forward(W, U, C, Z, X, eps, T, True)
    _, _, _, a = loss.loss_pair(Y, T, tgt, eps)
    # analytic gradient of L(C) = (1/Tn) sum_t ||W x_t + C U^T x_t - t_t||^2
    P = X @ U
    resid = X @ W.T + P @ C.T - tgt
    grad_C = 2.0 / (T * d_out) * resid.T @ P
    assert a == pytest.approx(float(np.sum(grad_C * Z)), rel=1e-9 if eps > 1e-5 else 1e-6)


def _toy_torch_loss(layers_np, x, tgt):
    Cs = [torch.tensor(l["C"], dtype=torch.float64, requires_grad=True) for l in layers_np]
    xt = torch.tensor(x, dtype=torch.float64)
    h = xt
    for i, l in enumerate(layers_np):
        W = torch.tensor(l["W"])
        U = torch.tensor(l["U"])
        h = h @ W.T + (h @ U) @ Cs[i].T
        if i == 0:
            h = torch.nn.functional.gelu(h)              # exact (erf) GELU
    L = torch.mean((h - torch.tensor(tgt)) ** 2)
    L.backward()
    return [c.grad.numpy() for c in Cs]


def test_toy_graph_central_difference_is_second_order():
    rng = np.random.default_rng(2)
    d, r, T = 32, 4, 6
    lay = [dict(W=rng.standard_normal((d, d)) / np.sqrt(d), U=np.linalg.qr(rng.standard_normal((d, r)))[0],
                C=0.3 * rng.standard_normal((d, r)), layer_id=i) for i in range(2)]
    x = rng.standard_normal((T, d))
    tgt = rng.standard_normal((T, d))
    grads = _toy_torch_loss(lay, x, tgt)
    seed, query = 11, 3
    dd = sum(float(np.sum(g * philox.perturbation(seed, l["layer_id"], query, d, r))) for g, l in zip(grads, lay))
    errs = []
    for eps in [4e-2, 2e-2, 1e-2]:
        Y = graphs.toy_forward(lay, x, eps, seed, query, store="fp64")
        _, _, _, a = loss.loss_pair(Y, T, tgt, eps)
        errs.append(abs(a - dd))
    assert errs[0] / errs[1] == pytest.approx(4.0, rel=0.1)
    assert errs[1] / errs[2] == pytest.approx(4.0, rel=0.1)
    assert errs[2] < 1e-3 * abs(dd) + 1e-9


def test_adam_first_step_closed_form():
    rng = np.random.default_rng(3)
    C, g = rng.standard_normal(100), rng.standard_normal(100)
    lr, eps = 1e-4, 1e-8
    C1, m1, v1 = optim.adam_step(C, np.zeros(100), np.zeros(100), g, lr, 0.9, 0.999, eps, 1)
    np.testing.assert_allclose(C1, C - lr * g / (np.abs(g) + eps), rtol=1e-12, atol=1e-18)
    np.testing.assert_allclose(m1, 0.1 * g, rtol=1e-15)
    np.testing.assert_allclose(v1, 0.001 * g * g, rtol=1e-12)


def test_adam_matches_torch_optim_ten_steps():
    rng = np.random.default_rng(4)
    C0 = rng.standard_normal(64)
    grads = [rng.standard_normal(64) for _ in range(10)]
    p = torch.nn.Parameter(torch.tensor(C0, dtype=torch.float64))
    opt = torch.optim.Adam([p], lr=3e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.0)
    C, m, v = C0, np.zeros(64), np.zeros(64)
    for t, g in enumerate(grads, start=1):
        p.grad = torch.tensor(g)
        opt.step()
        C, m, v = optim.adam_step(C, m, v, g, 3e-3, 0.9, 0.999, 1e-8, t)
    np.testing.assert_allclose(C, p.detach().numpy(), rtol=1e-12, atol=1e-15)


def test_sgd_and_gradient():
    Z = np.arange(6.0).reshape(2, 3)
    g = optim.zo_gradient(2.5, Z)
    np.testing.assert_array_equal(g, 2.5 * Z)
    np.testing.assert_array_equal(optim.sgd_step(np.ones((2, 3)), g, 0.1), 1.0 - 0.25 * Z)
