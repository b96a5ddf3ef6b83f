"""Edge cases of the GPU path through the C ABI: empty and one-token inputs, the smallest shapes, the
method's degenerate points, argument errors caught on the host, non-finite inputs, and one
maximum-size launch checked on sampled rows.

Degenerate points of the method (Section 3): eps = 0 makes both signs the same forward (y+ = y-
bit for bit); C = 0 and eps = 0 is the frozen layer y = W x; an evaluation block with coefficient 0
is the unperturbed layer.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import philox, layers, loss as oloss
from synth import normal, quantize_int4_g128
from test_gpu_kernels import _pair_case, _oracle_pair, _bound

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    c.device_status()          # tests below leave the status word clean themselves
    c.close()


def np64(t):
    return t.detach().double().cpu().numpy()


def test_empty_inputs_launch_nothing(ctx):
    W = normal((64, 64), 1, DEV, dtype=torch.bfloat16)
    U = normal((64, 8), 2, DEV)
    C = torch.zeros(64 * 8, device=DEV)
    L = zo.make_layer(W, U, C, 0)
    X = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    Y = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    n0 = ctx.launch_count()
    zo.zoact_pair_forward(ctx, L, X, 0, False, 1e-3, 1, 1, Y)
    zo.zoact_multi_forward(ctx, L, X, 0, True, [(0.0, 0), (1e-3, 1)], 1, Y)
    zo.zoact_lowrank_proj(ctx, X, U, torch.empty(0, 8, device=DEV))
    assert ctx.launch_count() == n0


@pytest.mark.parametrize("shared", [False, True])
@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float32])
def test_eps_zero_gives_identical_signs(ctx, shared, dt):
    d_in, d_out, r, T = 256, 136, 8, 77
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, dt, 0.0, 0.3)
    if not shared:
        X[T:] = X[:T]                     # the same tokens in both halves
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 2), X, T, shared, 0.0, 5, 6, Y)
    torch.cuda.synchronize()
    assert torch.equal(Y[:T], Y[T:])


@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float16, torch.float32])
def test_frozen_layer_at_zero_coefficients(ctx, dt):
    # C = 0 and eps = 0: the adapted layer is the frozen W x (Section 3, B = 0 at initialisation)
    d_in, d_out, r, T = 320, 200, 16, 150
    X, W, U, _ = _pair_case(d_in, d_out, r, T, False, dt, 0.0, 0.0)
    C = torch.zeros(d_out * r, device=DEV)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 0), X, T, False, 0.0, 1, 1, Y)
    torch.cuda.synchronize()
    Xn, Wn = np64(X), np64(W)
    ref = Xn @ Wn.T
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= 8 * np.sqrt(d_in) * 2.0 ** -24 * (np.abs(Xn) @ np.abs(Wn).T) + 1e-6)


def test_single_unperturbed_block(ctx):
    d_in, d_out, r, T = 512, 264, 16, 130
    X, W, U, C = _pair_case(d_in, d_out, r, T, True, torch.bfloat16, 0.0, 0.3)
    Y = torch.empty(T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_multi_forward(ctx, zo.make_layer(W, U, C, 0), X, T, True, [(0.0, 0)], 1, Y)
    torch.cuda.synchronize()
    Cn = np64(C).reshape(d_out, r)
    ref = layers.multi_forward(np64(W), np64(U), Cn, [None], [0.0], np64(X), T, True)
    absb = np.abs(np64(X)) @ np.abs(np64(W)).T
    lrabs = np.abs(np64(X) @ np64(U)) @ np.abs(Cn).T
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= _bound(d_in, absb + lrabs, lrabs))


@pytest.mark.parametrize("d_in,d_out,r,T,dt", [(8, 8, 1, 1, torch.bfloat16), (16, 8, 3, 2, torch.float16),
                                               (4, 8, 1, 1, torch.float32), (128, 8, 1, 1, "int4")])
def test_smallest_shapes(ctx, d_in, d_out, r, T, dt):
    eps, seed, query, lid = 0.5, 3, 4, 7
    if dt == "int4":
        Wf = normal((d_out, d_in), 9, DEV, std=0.02)
        packed, scales = quantize_int4_g128(Wf)
        U = normal((d_in, r), 10, DEV) / np.sqrt(d_in)
        C = normal((d_out * r,), 11, DEV, std=0.3)
        X = normal((2 * T, d_in), 12, DEV, dtype=torch.bfloat16)
        L = zo.make_layer(packed, U, C, lid, w_scales=scales, wtype=zo.DT_INT4_G128, d_in=d_in)
        Wn = layers.dequant_int4_g128(packed.cpu().numpy(), scales.float().cpu().numpy(), d_in)
    else:
        X, W, U, C = _pair_case(d_in, d_out, r, T, False, dt, eps, 0.3)
        L = zo.make_layer(W, U, C, lid)
        Wn = np64(W)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Y)
    torch.cuda.synchronize()
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    ref = layers.pair_forward(Wn, np64(U), np64(C).reshape(d_out, r), Zm, np64(X), eps, T, False)
    tol = (2.0 ** -8 if dt == "int4" else 1e-4) * np.abs(ref).max() + 1e-6
    assert np.abs(np64(Y) - ref).max() <= tol


def test_host_side_argument_errors_launch_nothing(ctx):
    W = normal((64, 64), 1, DEV, dtype=torch.bfloat16)
    U = normal((64, 8), 2, DEV)
    C = torch.zeros(64 * 8, device=DEV)
    X = torch.zeros(20, 64, dtype=torch.bfloat16, device=DEV)
    Y = torch.zeros(20, 64, dtype=torch.bfloat16, device=DEV)
    Xmis = X.view(-1)[1:1 + 18 * 64].view(18, 64)    # 2-byte offset: not 16-byte aligned
    n0 = ctx.launch_count()
    bad = [
        lambda: zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 0), Xmis, 9, False, 1e-3, 1, 1, Y[:18]),  # misaligned
        lambda: zo.zoact_pair_forward(ctx, zo.make_layer(W[:60], U, C, 0), X, 10, False, 1e-3, 1, 1, Y),   # d_out % 8
        lambda: zo.zoact_multi_forward(ctx, zo.make_layer(W, U, C, 0), X, 1, False, [(0.0, 0)] * 18, 1, Y),  # 18 blocks
        lambda: zo.zoact_loss_pair(ctx, Y, 10, 0.0, torch.zeros(4, dtype=torch.float64, device=DEV)),        # eps 0
        lambda: zo.zoact_loss_multi(ctx, Y, 10, 1, 1e-3, torch.zeros(1, dtype=torch.float64, device=DEV)),   # 1 block
    ]
    for f in bad:
        with pytest.raises((zo.ZoactError, ValueError)):
            f()
    U300 = normal((64, 300), 3, DEV)
    with pytest.raises(zo.ZoactError) as e:
        zo.zoact_pair_forward(ctx, zo.make_layer(W, U300, torch.zeros(64 * 300, device=DEV), 0), X, 10, False, 1e-3,
                              1, 1, Y)
    assert e.value.status == -2                   # rank above 256: unsupported
    assert ctx.launch_count() == n0


def test_nonfinite_outputs_are_flagged(ctx):
    T, n = 16, 64
    Y = normal((2 * T, n), 5, DEV, dtype=torch.bfloat16)
    Y[3, 7] = float("inf")
    out = torch.zeros(4, dtype=torch.float64, device=DEV)
    zo.zoact_loss_pair(ctx, Y, T, 1e-3, out)
    assert ctx.device_status() == -4
    outm = torch.zeros(3, dtype=torch.float64, device=DEV)
    zo.zoact_loss_multi(ctx, Y, T, 2, 1e-3, outm)
    assert ctx.device_status() == -4
    assert ctx.device_status() == 0               # read and reset


def test_basis_init_nonfinite_calibration_is_flagged(ctx):
    # one NaN in the calibration activations makes G, and so every basis column, non-finite: the
    # sign fix finds no finite entry to orient a column by and the status word says so
    X = normal((300, 256), 31, DEV)
    X[7, 11] = float("nan")
    U = torch.empty(256, 8, device=DEV)
    zo.zoact_basis_init(ctx, X, 8, U)
    torch.cuda.synchronize()
    assert ctx.device_status() == -4
    X[7, 11] = 0.0
    zo.zoact_basis_init(ctx, X, 8, U)            # the context stays usable
    torch.cuda.synchronize()
    assert ctx.device_status() == 0 and torch.isfinite(U).all()


def test_maximum_size_sampled(ctx):
    # 65536 tokens per perturbation through a 4096 -> 4096 layer (131072 stacked rows, 1 GiB per side):
    # every M tile of the CTA-pair kernel, sampled rows against the oracle
    d_in, d_out, r, T, eps, seed, query, lid = 4096, 4096, 16, 65536, 0.5, 2, 3, 4
    X = normal((2 * T, d_in), 20, DEV, dtype=torch.bfloat16)
    W = normal((d_out, d_in), 21, DEV, std=0.02, dtype=torch.bfloat16)
    U = normal((d_in, r), 22, DEV) / 64
    C = normal((d_out * r,), 23, DEV, std=0.1)
    Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, lid), X, T, False, eps, seed, query, Y)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    rows = np.sort(np.random.default_rng(1).choice(2 * T, 64, replace=False))
    idx = torch.as_tensor(rows, device=DEV)
    Xs, Wn, Un = np64(X[idx]), np64(W), np64(U)
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    sig = np.where(rows < T, 1.0, -1.0)[:, None]
    ref = Xs @ Wn.T + (Xs @ Un) @ np64(C).reshape(d_out, r).T + sig * eps * ((Xs @ Un) @ Zm.T)
    got = np64(Y[idx])
    assert np.all(np.abs(got - ref) <= 2.0 ** -7 * np.abs(ref) + 2e-3 * np.abs(ref).max())
    del X, Y
    torch.cuda.empty_cache()


def test_bounded_wait_timeout_is_reported_and_the_context_recovers(ctx):
    # a bounded wait that runs out (a flag that nothing sets, 1 ms) ends with ZOACT_ERR_TIMEOUT in the status
    # word, not a hang or a trap; the hook also leaves the context's tickets part-counted, as a launch that gave up
    # can, and reading the status repairs them: a split-tail pair forward (600 stacked rows x 520 outputs: 9 tiles
    # in 4 pieces) and a loss pair give the same bits before and after
    d_in, d_out, r, T = 1024, 520, 16, 300
    X, W, U, C = _pair_case(d_in, d_out, r, T, False, torch.bfloat16, 0.5, 0.3, seed=60)
    L = zo.make_layer(W, U, C, 2)

    def run():
        Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
        zo.zoact_pair_forward(ctx, L, X, T, False, 0.5, 3, 1, Y)
        out = torch.zeros(4, dtype=torch.float64, device=DEV)
        zo.zoact_loss_pair(ctx, Y, T, 0.5, out)
        torch.cuda.synchronize()
        return Y, out

    Y0, l0 = run()
    assert ctx.device_status() == 0
    with pytest.raises(zo.ZoactError):
        ctx.debug_timeout(0)                     # outside (0, 1e9]: refused on the host
    ctx.debug_timeout(1_000_000)
    assert ctx.device_status() == -5             # ZOACT_ERR_TIMEOUT, read and reset; tickets zeroed
    assert ctx.device_status() == 0
    Y1, l1 = run()
    assert ctx.device_status() == 0
    assert torch.equal(Y0, Y1) and torch.equal(l0, l1)
