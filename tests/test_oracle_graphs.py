"""Pins for the oracle's synthetic graphs (CPU only).

Each graph's central-difference scalar a = (L+ - L-)/(2 eps) must converge to
the directional derivative <grad L, Z> at rate O(eps^2), with the gradient taken
by torch autograd through the same wiring written independently in torch.  With
eps = 0 both halves of the stacked output coincide.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import graphs, loss, philox


def _layer(rng, d_in, d_out, r, lid):
    return dict(W=rng.standard_normal((d_out, d_in)) / np.sqrt(d_in),
                U=np.linalg.qr(rng.standard_normal((d_in, r)))[0],
                C=0.2 * rng.standard_normal((d_out, r)), layer_id=lid)


def _rms(x):
    return x / torch.sqrt(torch.mean(x * x, dim=-1, keepdim=True) + 1e-5)


def _torch_lin(l, C, x):
    return x @ torch.tensor(l["W"]).T + (x @ torch.tensor(l["U"])) @ C.T


def _check_rate(fwd, torch_loss, lays, x, tgt, seed=5, query=1, eps_list=(2e-2, 1e-2, 5e-3)):
    Cs = [torch.tensor(l["C"], requires_grad=True) for l in lays]
    L = torch_loss(Cs)
    L.backward()
    dd = sum(float(np.sum(c.grad.numpy() * philox.perturbation(seed, l["layer_id"], query, *l["C"].shape)))
             for c, l in zip(Cs, lays))
    errs = []
    for eps in eps_list:
        Y = fwd(eps, seed, query)
        errs.append(abs(loss.loss_pair(Y, x.shape[0], tgt, eps)[3] - dd))
    assert errs[0] / errs[1] == pytest.approx(4.0, rel=0.15)
    assert errs[1] / errs[2] == pytest.approx(4.0, rel=0.15)
    Y0 = fwd(0.0, seed, query)
    T = x.shape[0]
    np.testing.assert_array_equal(Y0[:T], Y0[T:])


def test_llama_mlp_graph():
    rng = np.random.default_rng(0)
    d, f, r, T = 16, 40, 3, 5
    lays = [_layer(rng, d, f, r, 0), _layer(rng, d, f, r, 1), _layer(rng, f, d, r, 2)]
    x = rng.standard_normal((T, d))
    tgt = rng.standard_normal((T, d))

    def tl(Cs):
        xt = torch.tensor(x)
        h = F.silu(_torch_lin(lays[0], Cs[0], xt)) * _torch_lin(lays[1], Cs[1], xt)
        return torch.mean((_torch_lin(lays[2], Cs[2], h) - torch.tensor(tgt)) ** 2)

    _check_rate(lambda e, s, q: graphs.llama_mlp_forward(lays, x, e, s, q, store="fp64"), tl, lays, x, tgt)


@pytest.mark.parametrize("kind", ["llama", "opt"])
def test_stack_graph(kind):
    rng = np.random.default_rng(1)
    d, f, r, T, nl = 16, 24, 2, 4, 2
    kvd = 8 if kind == "llama" else d
    names = ["q", "k", "v", "o", "gate", "up", "down"] if kind == "llama" else ["q", "k", "v", "o", "fc1", "fc2"]
    dims = {"q": (d, d), "k": (d, kvd), "v": (d, kvd), "o": (d, d), "gate": (d, f), "up": (d, f),
            "down": (f, d), "fc1": (d, f), "fc2": (f, d)}
    dls, lays = [], []
    for L in range(nl):
        dl = {}
        for i, nm in enumerate(names):
            dl[nm] = _layer(rng, *dims[nm], r, L * len(names) + i)
            lays.append(dl[nm])
        dls.append(dl)
    x = rng.standard_normal((T, d))

    def tl(Cs):
        it = iter(Cs)
        h = torch.tensor(x)
        for dl in dls:
            c = {nm: next(it) for nm in names}
            a = _rms(h)
            q, k, v = (_torch_lin(dl[n], c[n], a) for n in ("q", "k", "v"))
            if kind == "llama":  # 4 query heads of width 4, 2 kv heads
                k = k.reshape(-1, 2, 1, 4).expand(-1, 2, 2, 4).reshape(-1, d)
                v = v.reshape(-1, 2, 1, 4).expand(-1, 2, 2, 4).reshape(-1, d)
            o = _torch_lin(dl["o"], c["o"], _rms(q + k + v))
            b = _rms(o)
            if kind == "llama":
                m = _rms(F.silu(_torch_lin(dl["gate"], c["gate"], b)) * _torch_lin(dl["up"], c["up"], b))
                h = _torch_lin(dl["down"], c["down"], m)
            else:
                h = _torch_lin(dl["fc2"], c["fc2"], _rms(torch.relu(_torch_lin(dl["fc1"], c["fc1"], b))))
        return torch.mean(h * h)

    fwd = lambda e, s, q: graphs.stack_forward(dls, x, e, s, q, kind, store="fp64",
                                               n_heads=4, n_kv_heads=2, head_dim=4)
    # ReLU is not smooth: keep eps small enough that no pre-activation changes sign
    _check_rate(fwd, tl, lays, x, None, eps_list=(2e-2, 1e-2, 5e-3) if kind == "llama" else (2e-3, 1e-3, 5e-4))


@pytest.mark.parametrize("kind,blocks", [("llama", None), ("opt", None), ("llama", [(0.0, 0), (0.3, 1), (0.3, 2)])])
def test_stack_one_decoder_at_a_time(kind, blocks):
    # a deep stack run decoder by decoder (first=False after the first) gives the same array as one call
    rng = np.random.default_rng(2)
    d, f, r, T, nl = 16, 24, 2, 5, 3
    kvd = 8 if kind == "llama" else d
    names = ["q", "k", "v", "o", "gate", "up", "down"] if kind == "llama" else ["q", "k", "v", "o", "fc1", "fc2"]
    dims = {"q": (d, d), "k": (d, kvd), "v": (d, kvd), "o": (d, d), "gate": (d, f), "up": (d, f),
            "down": (f, d), "fc1": (d, f), "fc2": (f, d)}
    dls = [{nm: _layer(rng, *dims[nm], r, L * len(names) + i) for i, nm in enumerate(names)} for L in range(nl)]
    x = rng.standard_normal((T, d))
    kw = dict(store="bf16", n_heads=4, n_kv_heads=2, head_dim=4, blocks=blocks)
    whole = graphs.stack_forward(dls, x, 0.1, 3, 4, kind, **kw)
    h = graphs.stack_forward(dls[:1], x, 0.1, 3, 4, kind, **kw)
    for dl in dls[1:]:
        h = graphs.stack_forward([dl], h, 0.1, 3, 4, kind, first=False, **kw)
    np.testing.assert_array_equal(h, whole)
    assert whole.shape == ((2 if blocks is None else len(blocks)) * T, d)
