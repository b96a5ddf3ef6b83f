"""Adapted linears that read one input, run as one launch (zoact_pair_forward_group_rs /
zoact_multi_forward_group_rs), and the strided mixer that reads their outputs.

A group's weights sit in one buffer, rows in layer order, and its layers share the basis (Algorithm 1 gives
linears with one input one basis).  Each layer's columns of the grouped output are checked against the oracle's
pair (or multi-point) forward of that layer alone, with its own C and Philox stream, and bit for bit against the
layer's own call when no last-wave tile is split (every element then has the same Z and the same K order).
Requests one launch cannot serve are refused before anything is launched.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import layers, philox
from synth import normal, quantize_int4_g128

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    c.close()


def n64(t):
    return t.detach().double().cpu().numpy()


def _group(d_in, outs, r, dt, seed, int4=False):
    """One weight buffer for all layers (views per layer), one basis, C and a layer id per layer."""
    n = sum(outs)
    Wf = normal((n, d_in), seed, DEV, std=d_in ** -0.5, dtype=torch.float32 if int4 else dt)
    U = (normal((d_in, r), seed + 1, DEV) / np.sqrt(d_in)).contiguous()
    if int4:
        packed, scales = quantize_int4_g128(Wf)
        Wd = layers.dequant_int4_g128(packed.cpu().numpy(), scales.float().cpu().numpy(), d_in)
    else:
        Wd = n64(Wf)
    lay, ora, c = [], [], 0
    for i, d in enumerate(outs):
        C = normal((d * r,), seed + 10 + i, DEV, std=0.3)
        lid = 20 + 3 * i
        if int4:
            L = zo.make_layer(packed[c:c + d], U, C, lid, w_scales=scales[c:c + d], wtype=zo.DT_INT4_G128, d_in=d_in)
        else:
            L = zo.make_layer(Wf[c:c + d], U, C, lid)
        lay.append(L)
        ora.append(dict(W=Wd[c:c + d], C=n64(C).reshape(d, r), lid=lid, off=c, d=d))
        c += d
    return lay, ora, n64(U)


def _check_against_oracle(Y, ora, U, Xn, blocks_of, T, d_in, ydt, seed):
    """Each layer's columns against the oracle's multi-point forward of that layer (blocks (coef, query))."""
    coefs = [c for c, _ in blocks_of]
    out_r = 2.0 ** -8 if ydt == torch.bfloat16 else (2.0 ** -11 if ydt == torch.float16 else 0.0)
    Yg = n64(Y)
    for o in ora:
        d = o["d"]
        Zs = [philox.perturbation(seed, o["lid"], q, d, U.shape[1]) if c != 0.0 else None for c, q in blocks_of]
        ref = layers.multi_forward(o["W"], U, o["C"], Zs, coefs, Xn, T, False)
        zs = [np.abs(z) for z in Zs if z is not None]
        zabs = np.max(np.stack(zs), axis=0) if zs else 0.0
        absl = np.abs(Xn @ U) @ (np.abs(o["C"]) + max(abs(c) for c in coefs) * zabs).T
        absb = np.abs(Xn) @ np.abs(o["W"]).T + absl
        err = np.abs(Yg[:, o["off"]:o["off"] + d] - ref)
        bound = 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 2.0 ** -14 * absl + out_r * np.abs(ref) + 1e-6
        assert np.all(err <= bound), (o["lid"], err.max())


@pytest.mark.parametrize("d_in,outs,r,T,dt,ydt", [
    (1024, (512, 128, 128), 16, 256, torch.bfloat16, torch.float32),   # grouped-query q, k, v shapes
    (640, (264, 40, 48), 8, 300, torch.float16, torch.float16),        # layers straddle tiles; partial M tile
    (2048, (256, 256, 256, 256), 32, 128, torch.bfloat16, torch.bfloat16),   # four layers, rank 32
])
@pytest.mark.parametrize("multi", [False, True])
def test_group_matches_oracle_and_own_calls(ctx, monkeypatch, d_in, outs, r, T, dt, ydt, multi):
    eps, seed, query = 0.5, 13, 3
    lay, ora, U = _group(d_in, outs, r, dt, 60)
    blocks_of = [(0.0, 0), (eps, 7), (eps, 8), (eps, 9)] if multi else [(eps, query), (-eps, query)]
    nb = len(blocks_of)
    X = normal((nb * T, d_in), 61, DEV, dtype=dt)
    inv = (0.5 + torch.rand(nb * T, device=DEV, generator=torch.Generator(DEV).manual_seed(62))).contiguous()
    n = sum(outs)
    monkeypatch.setenv("ZOACT_SPLIT_TAIL", "0")       # whole tiles: the layer's own call is then bit-identical
    Y = torch.full((nb * T, n), float("nan"), dtype=ydt, device=DEV)
    if multi:
        zo.zoact_multi_forward_group_rs(ctx, lay, X, T, blocks_of, seed, Y, in_scale=inv)
    else:
        zo.zoact_pair_forward_group_rs(ctx, lay, X, T, eps, seed, query, Y, in_scale=inv)
    own = []
    for L, o in zip(lay, ora):
        Yi = torch.full((nb * T, o["d"]), float("nan"), dtype=ydt, device=DEV)
        if multi:
            zo.zoact_multi_forward_rs(ctx, L, X, T, False, blocks_of, seed, Yi, in_scale=inv)
        else:
            zo.zoact_pair_forward_rs(ctx, L, X, T, False, eps, seed, query, Yi, in_scale=inv)
        own.append(Yi)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    for Yi, o in zip(own, ora):
        assert torch.equal(Y[:, o["off"]:o["off"] + o["d"]], Yi), o["lid"]
    # the split tail (the default) changes only the order in which a split tile's K pieces are added
    monkeypatch.delenv("ZOACT_SPLIT_TAIL")
    Y2 = torch.full_like(Y, float("nan"))
    if multi:
        zo.zoact_multi_forward_group_rs(ctx, lay, X, T, blocks_of, seed, Y2, in_scale=inv)
    else:
        zo.zoact_pair_forward_group_rs(ctx, lay, X, T, eps, seed, query, Y2, in_scale=inv)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    Xn = n64(X) * n64(inv)[:, None]
    for Yc in (Y, Y2):
        _check_against_oracle(Yc, ora, U, Xn, blocks_of, T, d_in, ydt, seed)


def test_group_int4_expanded(ctx, monkeypatch):
    # INT4 from 1024 stacked rows: the group's packed rows and scale rows, expanded to bf16 as one array
    d_in, outs, r, T = 512, (256, 64, 64), 16, 512
    eps, seed, query = 0.5, 5, 2
    lay, ora, U = _group(d_in, outs, r, None, 70, int4=True)
    X = normal((2 * T, d_in), 71, DEV, dtype=torch.bfloat16)
    monkeypatch.setenv("ZOACT_SPLIT_TAIL", "0")
    Y = torch.full((2 * T, sum(outs)), float("nan"), dtype=torch.bfloat16, device=DEV)
    zo.zoact_pair_forward_group_rs(ctx, lay, X, T, eps, seed, query, Y)
    for L, o in zip(lay, ora):
        Yi = torch.empty(2 * T, o["d"], dtype=torch.bfloat16, device=DEV)
        zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Yi)
        torch.cuda.synchronize()
        assert torch.equal(Y[:, o["off"]:o["off"] + o["d"]], Yi)
    assert ctx.device_status() == 0
    # against the oracle with the dequantised weights (q s rounded once to bf16 in the expansion)
    Yg, Xn = n64(Y), n64(X)
    for o in ora:
        Zm = philox.perturbation(seed, o["lid"], query, o["d"], r)
        ref = layers.pair_forward(o["W"], U, o["C"], Zm, Xn, eps, T, False)
        absw = np.abs(Xn) @ np.abs(o["W"]).T
        absl = np.abs(Xn @ U) @ (np.abs(o["C"]) + eps * np.abs(Zm)).T
        err = np.abs(Yg[:, o["off"]:o["off"] + o["d"]] - ref)
        # weights rounded to bf16 (2^-9), fp32 accumulation, the 16-bit split of the low-rank term, the output
        bound = (2.0 ** -9 * absw + 8 * np.sqrt(d_in) * 2.0 ** -24 * (absw + absl) + 2.0 ** -14 * absl +
                 2.0 ** -8 * np.abs(ref) + 1e-6)
        assert np.all(err <= bound), err.max()


def test_group_one_layer_is_the_layer_call(ctx):
    d_in, r, T = 512, 16, 256
    lay, ora, U = _group(d_in, (384,), r, torch.bfloat16, 80)
    X = normal((2 * T, d_in), 81, DEV, dtype=torch.bfloat16)
    Y1 = torch.empty(2 * T, 384, dtype=torch.bfloat16, device=DEV)
    Y2 = torch.empty_like(Y1)
    zo.zoact_pair_forward_group_rs(ctx, lay, X, T, 0.5, 3, 1, Y1)
    zo.zoact_pair_forward_rs(ctx, lay[0], X, T, False, 0.5, 3, 1, Y2)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0 and torch.equal(Y1, Y2)


def _expect(status, fn):
    with pytest.raises(zo.ZoactError) as e:
        fn()
    assert e.value.status == status


def test_group_refusals_launch_nothing(ctx, monkeypatch):
    d_in, outs, r = 512, (128, 64, 64), 16
    lay, ora, U = _group(d_in, outs, r, torch.bfloat16, 90)
    n = sum(outs)
    torch.cuda.synchronize()
    # fewer than 256 stacked rows: no CTA-pair launch takes the group
    T = 64
    X = normal((2 * T, d_in), 91, DEV, dtype=torch.bfloat16)
    Y = torch.empty(2 * T, n, dtype=torch.bfloat16, device=DEV)
    n0 = ctx.launch_count()
    _expect(zo._lib.ZOACT_ERR_UNSUPPORTED, lambda: zo.zoact_pair_forward_group_rs(ctx, lay, X, T, 0.5, 1, 1, Y))
    # no tokens: nothing to do, nothing launched
    zo.zoact_pair_forward_group_rs(ctx, lay, X[:0], 0, 0.5, 1, 1, Y[:0])
    # the one-CTA kernel or the epilogue low-rank term: no operand tables
    T = 256
    X = normal((2 * T, d_in), 92, DEV, dtype=torch.bfloat16)
    Y = torch.empty(2 * T, n, dtype=torch.bfloat16, device=DEV)
    for var, val in (("ZOACT_PAIR_KERNEL", "1cta"), ("ZOACT_LOWRANK", "epilogue")):
        monkeypatch.setenv(var, val)
        _expect(zo._lib.ZOACT_ERR_UNSUPPORTED, lambda: zo.zoact_pair_forward_group_rs(ctx, lay, X, T, 0.5, 1, 1, Y))
        monkeypatch.delenv(var)
    assert ctx.launch_count() == n0
    # weights that do not follow one another, or another basis: invalid
    W_sep = [normal((d, d_in), 93 + i, DEV, dtype=torch.bfloat16) for i, d in enumerate(outs)]
    Uq = torch.from_numpy(U.astype(np.float32)).to(DEV)
    Cs = [torch.zeros(d * r, device=DEV) for d in outs]
    sep = [zo.make_layer(W, Uq, C, 40 + i) for i, (W, C) in enumerate(zip(W_sep, Cs))]
    _expect(-1, lambda: zo.zoact_pair_forward_group_rs(ctx, sep, X, T, 0.5, 1, 1, Y))
    U2 = Uq.clone()
    other = [lay[0], zo.make_layer(lay[1]._keep[0], U2, lay[1]._keep[2], 41), lay[2]]
    _expect(-1, lambda: zo.zoact_pair_forward_group_rs(ctx, other, X, T, 0.5, 1, 1, Y))
    assert ctx.launch_count() == n0
    with pytest.raises(ValueError):
        zo.zoact_pair_forward_group_rs(ctx, lay * 2, X, T, 0.5, 1, 1, Y)     # above ZOACT_MAX_GROUP
    torch.cuda.synchronize()
    assert ctx.device_status() == 0


@pytest.mark.parametrize("rows,n,n_rep,head_dim,pad,dt", [(300, 512, 4, 128, 0, torch.bfloat16),
                                                          (77, 384, 1, 64, 0, torch.float16),
                                                          (50, 96, 2, 24, 0, torch.float32),
                                                          (33, 64, 2, 8, 1, torch.bfloat16)])   # rows unaligned
def test_mix_rms_strided(ctx, rows, n, n_rep, head_dim, pad, dt):
    # q, k, v as column views of one [rows, n + 2 n / n_rep (+ pad)] buffer (a grouped q/k/v output): the same
    # values as contiguous copies, and the oracle's rms(q + rep(k) + rep(v)) within the output's rounding
    nk = n // n_rep
    buf = normal((rows, n + 2 * nk + pad), 100, DEV, dtype=dt)
    q, k, v = buf[:, :n], buf[:, n:n + nk], buf[:, n + nk:n + 2 * nk]
    Y1 = torch.empty(rows, n, dtype=dt, device=DEV)
    Y2 = torch.empty_like(Y1)
    zo.zoact_mix_rms(ctx, q, k, v, Y1, n_rep, head_dim)
    zo.zoact_mix_rms(ctx, q.contiguous(), k.contiguous(), v.contiguous(), Y2, n_rep, head_dim)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0 and torch.equal(Y1, Y2)
    m = n64(q) + layers.repeat_kv(n64(k), nk // head_dim, n_rep, head_dim) + \
        layers.repeat_kv(n64(v), nk // head_dim, n_rep, head_dim)
    ref = layers.rms_norm(m)
    tol = {torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11, torch.float32: 1e-6}[dt]
    assert np.abs(n64(Y1) - ref).max() <= 2 * tol * np.abs(ref).max() + 1e-6
