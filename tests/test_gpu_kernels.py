"""GPU parity of each libzoact kernel against the CPU oracle, through the C ABI.

Inputs come from synth (seeded); both sides read the same stored values.
Tolerances (written per test):
  * Philox words and index bookkeeping: bit-exact.
  * fp32 normals: |dz| <= 1e-6 (1 + |z|)  (fp32 logf/sqrtf/sincospif vs fp64 libm).
  * fp32 arithmetic paths: <= 1e-4 of the output scale, and a per-element bound
    from the fp32 accumulation error (c * eps32 * sum |terms|).  Where the
    low-rank term runs on the tensor cores as three bf16 products of 16-bit
    splits, it carries at most 2^-15 sum_j |P_j| |T_j| more (the dropped
    P_lo T_lo and the rounding of the lo parts); the bound adds 2^-14 of it.
  * 16-bit outputs: the bf16/fp16 rounding of the output (2^-8 / 2^-11 relative)
    on top of the fp32 bound; the bar is 2e-2 relative.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import philox, layers, loss as oloss, optim, basis, graphs
from synth import normal, lowrank_activations, quantize_int4_g128

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    assert c.device_status() == 0
    c.close()


def np64(t):
    return t.detach().double().cpu().numpy()


# ---------------- Z ----------------
@pytest.mark.parametrize("seed,layer,query,n", [(0, 0, 0, 4096), (0xDEADBEEF12345678, 77, (3 << 32) | 5, 1001),
                                                (1, 2**32 - 1, 2**64 - 1, 13)])
def test_philox_bit_exact_and_normals(ctx, seed, layer, query, n):
    z = torch.empty(n, dtype=torch.float32, device=DEV)
    w = torch.empty(n, dtype=torch.int32, device=DEV)
    zo.zoact_philox_normals(ctx, seed, layer, query, n, z, w)
    torch.cuda.synchronize()
    words = w.cpu().numpy().view(np.uint32).astype(np.uint64)
    assert np.array_equal(words, philox.stream_words(seed, layer, query, n))
    zr = philox.normals(seed, layer, query, n)
    zg = np64(z)
    assert np.all(np.abs(zg - zr) <= 1e-6 * (1.0 + np.abs(zr)))


# ---------------- projection ----------------
@pytest.mark.parametrize("rows,d_in,r,dt", [(300, 1000, 16, torch.bfloat16), (64, 256, 8, torch.float32),
                                            (1000, 4096, 32, torch.float16), (7, 40, 3, torch.bfloat16),
                                            (2048, 14336, 16, torch.bfloat16)])
def test_lowrank_proj(ctx, rows, d_in, r, dt):
    X = normal((rows, d_in), 1, DEV, dtype=dt)
    U = normal((d_in, r), 2, DEV) / np.sqrt(d_in)
    P = torch.empty(rows, r, dtype=torch.float32, device=DEV)
    zo.zoact_lowrank_proj(ctx, X, U, P)
    torch.cuda.synchronize()
    Xn, Un = np64(X), np64(U)
    ref = Xn @ Un
    bound = 4 * d_in ** 0.5 * 2.0 ** -24 * (np.abs(Xn) @ np.abs(Un)) + 1e-30
    assert np.all(np.abs(np64(P) - ref) <= bound + 1e-6 * np.abs(ref))


# ---------------- pair forward ----------------
def _pair_case(d_in, d_out, r, T, shared, dt, eps, c_scale, seed=0):
    X = normal(((T if shared else 2 * T), d_in), seed + 1, DEV, dtype=dt)
    W = normal((d_out, d_in), seed + 2, DEV, std=d_in ** -0.5, dtype=dt)
    U = normal((d_in, r), seed + 3, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), seed + 4, DEV, std=c_scale)
    return X, W, U, C


def _oracle_pair(X, W, U, C, eps, T, shared, seed, layer_id, query, d_out, r):
    Zm = philox.perturbation(seed, layer_id, query, d_out, r)
    Y = layers.pair_forward(np64(W), np64(U), np64(C).reshape(d_out, r), Zm, np64(X), eps, T, shared)
    Xn, Wn, Un = np64(X), np64(W), np64(U)
    if shared:
        Xn = np.concatenate([Xn, Xn])
    lrabs = (np.abs(Xn @ Un)) @ (np.abs(np64(C).reshape(d_out, r)) + abs(eps) * np.abs(Zm)).T
    absb = np.abs(Xn) @ np.abs(Wn).T + lrabs
    return Y, absb, lrabs


def _bound(d_in, absb, lrabs):
    """fp32 accumulation bound plus the 16-bit split of the low-rank term."""
    return 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 2.0 ** -14 * lrabs + 1e-6


@pytest.mark.parametrize("d_in,d_out,r,T,shared,dt", [
    (256, 256, 8, 64, True, torch.float32),
    (256, 200, 8, 37, False, torch.float32),
    (1000, 520, 16, 200, False, torch.bfloat16),     # 4 M tiles (ragged), 3 N tiles (ragged), ragged K
    (1024, 768, 16, 96, True, torch.bfloat16),       # shared input: 1 M tile, both signs written
    (512, 264, 4, 130, False, torch.float16),        # stacked rows cross a tile with both signs
    (4096, 1024, 32, 128, False, torch.bfloat16),    # rank 32: epilogue table in two chunks
    (320, 128, 1, 20, True, torch.bfloat16),         # rank 1
])
def test_pair_forward_fp32_out(ctx, d_in, d_out, r, T, shared, dt):
    # eps = 0.5 and |C| ~ 0.3 make the low-rank term visible at fp32 precision
    eps, seed, query, layer_id = 0.5, 11, 7, 5
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, dt, eps, 0.3)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    L = zo.make_layer(W, U, C, layer_id)
    zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, Y)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, layer_id, query, d_out, r)
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= _bound(d_in, absb, lrabs)), err.max()
    assert err.max() <= 1e-4 * np.abs(ref).max()


@pytest.mark.parametrize("T,shared,lowrank,kernel", [
    (256, False, "auto", "auto"),        # stacked, tiles inside one block: whole low-rank term on the tensor cores
    (256, False, "epilogue", "auto"),    # the same in fp32 epilogue tables
    (200, False, "auto", "auto"),        # stacked, T below the tile height: C p on the tensor cores
    (300, False, "auto", "auto"),        # stacked, tiles across the sign boundary: two K slots by block parity
    (300, True, "auto", "auto"),         # shared input: C p on the tensor cores, +-eps Z p in the epilogue
    (300, True, "epilogue", "auto"),
    (128, False, "auto", "1cta"),        # one-CTA kernel with the whole term on the tensor cores
    (100, False, "auto", "1cta"),
    (200, False, "auto", "1cta"),        # one-CTA tiles across the sign boundary: two K slots
])
@pytest.mark.parametrize("gated", [False, True])
def test_pair_forward_lowrank_modes(ctx, monkeypatch, T, shared, lowrank, kernel, gated):
    # every placement of the low-rank term gives the oracle's output within the fp32 bound
    if lowrank != "auto":
        monkeypatch.setenv("ZOACT_LOWRANK", lowrank)
    if kernel != "auto":
        monkeypatch.setenv("ZOACT_PAIR_KERNEL", kernel)
    d_in, d_out, r, eps, seed, query = 1024, 392, 16, 0.5, 19, 6
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, torch.bfloat16, eps, 0.3, seed=60)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    if gated:
        W2 = normal((d_out, d_in), 70, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
        U2 = normal((d_in, r), 71, DEV) / np.sqrt(d_in)
        C2 = normal((d_out * r,), 72, DEV, std=0.3)
        zo.zoact_pair_forward_gated(ctx, zo.make_layer(W, U, C, 3), zo.make_layer(W2, U2, C2, 4), X, T, shared,
                                    eps, seed, query, Y)
        torch.cuda.synchronize()
        g, _, _ = _oracle_pair(X, W, U, C, eps, T, shared, seed, 3, query, d_out, r)
        u, _, _ = _oracle_pair(X, W2, U2, C2, eps, T, shared, seed, 4, query, d_out, r)
        ref = layers.silu(g) * u
        assert np.abs(np64(Y) - ref).max() <= 1e-4 * np.abs(ref).max()
    else:
        zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 3), X, T, shared, eps, seed, query, Y)
        torch.cuda.synchronize()
        ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, 3, query, d_out, r)
        err = np.abs(np64(Y) - ref)
        assert np.all(err <= _bound(d_in, absb, lrabs)), err.max()
        assert err.max() <= 1e-4 * np.abs(ref).max()


@pytest.mark.parametrize("d_in,d_out,r,T,shared,dt,act", [
    (1000, 520, 16, 200, False, torch.bfloat16, zo.ACT_NONE),
    (1024, 768, 8, 96, True, torch.bfloat16, zo.ACT_RELU),
    (512, 264, 16, 130, False, torch.float16, zo.ACT_GELU),
    (256, 256, 8, 64, True, torch.float32, zo.ACT_GELU),
])
def test_pair_forward_16bit_out_and_acts(ctx, d_in, d_out, r, T, shared, dt, act):
    eps, seed, query, layer_id = 1e-3, 3, 1, 9
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, dt, eps, 0.05)
    Y = torch.empty(2 * T, d_out, dtype=dt, device=DEV)
    L = zo.make_layer(W, U, C, layer_id)
    zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, Y, act=act)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, layer_id, query, d_out, r)
    ref = {zo.ACT_NONE: lambda y: y, zo.ACT_RELU: layers.relu, zo.ACT_GELU: layers.gelu_erf}[act](ref)
    rel = {torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11, torch.float32: 2.0 ** -23}[dt]
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= rel * np.abs(ref) + _bound(d_in, absb, lrabs))
    assert err.max() <= 2e-2 * np.abs(ref).max()


@pytest.mark.parametrize("which", ["down", "gated"])
def test_pair_forward_full_size_sampled(ctx, which):
    # the bench's launches at full size (Llama-3-8B MLP block, T = 2048, r = 16, bf16 out); the oracle
    # computes 96 sampled token rows (from both halves) over every output column
    T, r, eps, seed, query = 2048, 16, 1e-3, 77, 9
    rng = np.random.default_rng(5)
    if which == "down":
        d_in, d_out = 14336, 4096
        X, W, U, C = _pair_case(d_in, d_out, r, T, False, torch.bfloat16, eps, 0.05, seed=20)
        Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
        zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 2), X, T, False, eps, seed, query, Y)
        torch.cuda.synchronize()
        rows = np.sort(rng.choice(2 * T, 96, replace=False))
        Xs, Wn, Un = np64(X)[rows], np64(W), np64(U)
        Zm = philox.perturbation(seed, 2, query, d_out, r)
        sig = np.where(rows < T, 1.0, -1.0)[:, None]
        Cn = np64(C).reshape(d_out, r)
        ref = Xs @ Wn.T + ((Xs @ Un) @ Cn.T) + sig * eps * ((Xs @ Un) @ Zm.T)
        got = np64(Y)[rows]
    else:
        d_in, d_out = 4096, 14336
        X = normal((T, d_in), 31, DEV, dtype=torch.bfloat16)
        Wg = normal((d_out, d_in), 32, DEV, std=0.02, dtype=torch.bfloat16)
        Wu = normal((d_out, d_in), 33, DEV, std=0.02, dtype=torch.bfloat16)
        U = normal((d_in, r), 34, DEV) / np.sqrt(d_in)
        Cg = normal((d_out * r,), 35, DEV, std=0.05)
        Cu = normal((d_out * r,), 36, DEV, std=0.05)
        H = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
        zo.zoact_pair_forward_gated(ctx, zo.make_layer(Wg, U, Cg, 0), zo.make_layer(Wu, U, Cu, 1), X, T, True,
                                    eps, seed, query, H)
        torch.cuda.synchronize()
        tok = np.sort(rng.choice(T, 48, replace=False))
        Xs, Un = np64(X)[tok], np64(U)
        P = Xs @ Un
        out = []
        for sgn in (1.0, -1.0):
            g = Xs @ np64(Wg).T + P @ (np64(Cg).reshape(d_out, r) + sgn * eps * philox.perturbation(seed, 0, query, d_out, r)).T
            u = Xs @ np64(Wu).T + P @ (np64(Cu).reshape(d_out, r) + sgn * eps * philox.perturbation(seed, 1, query, d_out, r)).T
            out.append(layers.silu(g) * u)
        ref = np.concatenate(out)
        got = np.concatenate([np64(H)[tok], np64(H)[T + tok]])
    err = np.abs(got - ref)
    assert err.max() <= 2e-2 * np.abs(ref).max()
    assert np.all(err <= 2.0 ** -7 * np.abs(ref) + 2e-3 * np.abs(ref).max())


def test_pair_difference_isolates_the_perturbation(ctx):
    # y+ - y- = 2 eps Z p exactly in the definition; fp32 output keeps it visible at eps = 1e-3
    d_in, d_out, r, T = 768, 512, 16, 64
    eps, seed, query, lid = 1e-3, 5, 2, 3
    X, W, U, C = _pair_case(d_in, d_out, r, T, True, torch.bfloat16, eps, 0.1)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, lid), X, T, True, eps, seed, query, Y)
    torch.cuda.synchronize()
    Yn = np64(Y)
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    ref = 2 * eps * (np64(X) @ np64(U)) @ Zm.T
    # the accumulator is common to both halves, so the difference carries only epilogue rounding
    assert np.abs((Yn[:T] - Yn[T:]) - ref).max() <= 1e-6 * np.abs(Yn).max()


@pytest.mark.parametrize("T,shared,dt", [(96, True, torch.bfloat16), (70, False, torch.bfloat16),
                                         (300, True, torch.bfloat16), (200, False, torch.float16)])
def test_pair_forward_gated(ctx, T, shared, dt):
    d_in, d_out, r = 512, 400, 16
    eps, seed, query = 0.25, 8, 4
    X = normal(((T if shared else 2 * T), d_in), 21, DEV, dtype=dt)
    Wg = normal((d_out, d_in), 22, DEV, std=d_in ** -0.5, dtype=dt)
    Wu = normal((d_out, d_in), 23, DEV, std=d_in ** -0.5, dtype=dt)
    Ug = normal((d_in, r), 24, DEV) / np.sqrt(d_in)
    Uu = normal((d_in, r), 25, DEV) / np.sqrt(d_in)
    Cg = normal((d_out * r,), 26, DEV, std=0.2)
    Cu = normal((d_out * r,), 27, DEV, std=0.2)
    H = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward_gated(ctx, zo.make_layer(Wg, Ug, Cg, 0), zo.make_layer(Wu, Uu, Cu, 1), X, T, shared,
                                eps, seed, query, H)
    torch.cuda.synchronize()
    g, _, _ = _oracle_pair(X, Wg, Ug, Cg, eps, T, shared, seed, 0, query, d_out, r)
    u, _, _ = _oracle_pair(X, Wu, Uu, Cu, eps, T, shared, seed, 1, query, d_out, r)
    ref = layers.silu(g) * u
    assert np.abs(np64(H) - ref).max() <= 1e-4 * np.abs(ref).max()



# ---------------- split tail of the CTA-pair kernel ----------------
# With 152 SMs (76 CTA pairs), when the last wave of whole tiles leaves half of the pairs or more idle, its tiles
# are each cut into S = 76 / tail-tiles (<= 4) equal K ranges and the last piece of each adds the partials.
# Cases:
# - 600 stacked rows x 520 outputs: 9 tiles, S = 4;
# - 512 x 256: two tiles, S = 4;
# - a gated launch on a shared input with 16-bit staged outputs (the MLP block's gate/up form): 10 tiles, S = 4;
# - 4096 stacked rows x 4096 (the MLP block's down form, K = 1024): three waves of 76 whole tiles, then 28 tail
#   tiles in two pieces.
@pytest.mark.parametrize("d_in,d_out,r,T,shared,gated,ydt", [
    (1024, 520, 16, 300, False, False, torch.float32),
    (1024, 256, 8, 256, False, False, torch.float32),
    (1024, 520, 16, 300, True, True, torch.bfloat16),
    (1024, 4096, 16, 2048, False, False, torch.float32),
])
def test_pair_forward_split_tail(ctx, monkeypatch, d_in, d_out, r, T, shared, gated, ydt):
    eps, seed, query = 0.5, 13, 2
    X, W, U, C = _pair_case(d_in, d_out, r, T, shared, torch.bfloat16, eps, 0.3, seed=40)
    L = zo.make_layer(W, U, C, 3)
    if gated:
        W2 = normal((d_out, d_in), 51, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
        C2 = normal((d_out * r,), 52, DEV, std=0.3)
        L2 = zo.make_layer(W2, U, C2, 4)           # one basis for gate and up, as the MLP block's
    def run():
        Y = torch.empty(2 * T, d_out, dtype=ydt, device=DEV)
        if gated:
            zo.zoact_pair_forward_gated(ctx, L, L2, X, T, shared, eps, seed, query, Y)
        else:
            zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, Y)
        torch.cuda.synchronize()
        assert ctx.device_status() == 0
        return Y
    Y1, Y2 = run(), run()
    assert torch.equal(Y1, Y2)                     # the fixed piece order makes the sum reproducible
    monkeypatch.setenv("ZOACT_SPLIT_TAIL", "0")
    Yw = run()                                     # whole tiles: the same sums in another order
    monkeypatch.delenv("ZOACT_SPLIT_TAIL")
    assert torch.equal(run(), Y1)                  # the tickets were left at zero
    if gated:
        g, _, _ = _oracle_pair(X, W, U, C, eps, T, shared, seed, 3, query, d_out, r)
        u, _, _ = _oracle_pair(X, W2, U, C2, eps, T, shared, seed, 4, query, d_out, r)
        ref = layers.silu(g) * u
        tol = 2.0 ** -7 * np.abs(ref) + 1e-3 * np.abs(ref).max()
        assert np.all(np.abs(np64(Y1) - ref) <= tol)
        # one bf16 step, or the fp32 summation-order difference where SiLU(g) u is near zero
        assert np.all(np.abs(np64(Y1) - np64(Yw)) <= 2.0 ** -7 * np.abs(np64(Yw)) + 1e-4 * np.abs(ref).max())
    else:
        ref, absb, lrabs = _oracle_pair(X, W, U, C, eps, T, shared, seed, 3, query, d_out, r)
        assert np.all(np.abs(np64(Y1) - ref) <= _bound(d_in, absb, lrabs))
        assert np.all(np.abs(np64(Y1) - np64(Yw)) <= 2 * 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 1e-6)


# ---------------- INT4 weights ----------------
def _int4_layer(d_in, d_out, r, seed, lid):
    Wf = normal((d_out, d_in), seed, DEV, std=0.02)
    packed, scales = quantize_int4_g128(Wf)
    U = normal((d_in, r), seed + 1, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), seed + 2, DEV, std=0.3)
    L = zo.make_layer(packed, U, C, lid, w_scales=scales, wtype=zo.DT_INT4_G128, d_in=d_in)
    Wd = layers.dequant_int4_g128(packed.cpu().numpy(), scales.float().cpu().numpy(), d_in)
    return L, Wd, U, C


@pytest.mark.parametrize("d_in,d_out,r,T,shared", [(1024, 520, 16, 200, False), (512, 256, 32, 64, True),
                                                   (4096, 1024, 16, 130, False)])
def test_pair_forward_int4(ctx, d_in, d_out, r, T, shared):
    # the kernel rounds every dequantised weight q * s to bf16 (scale via bf16): |dw| <= 2^-8 |w|
    eps, seed, query, lid = 0.5, 13, 2, 6
    L, Wd, U, C = _int4_layer(d_in, d_out, r, 40, lid)
    X = normal(((T if shared else 2 * T), d_in), 41, DEV, dtype=torch.bfloat16)
    Y = torch.empty(2 * T, d_out, dtype=torch.float32, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, shared, eps, seed, query, Y)
    torch.cuda.synchronize()
    Zm = philox.perturbation(seed, lid, query, d_out, r)
    Xn = np64(X)
    ref = layers.pair_forward(Wd, np64(U), np64(C).reshape(d_out, r), Zm, Xn, eps, T, shared)
    Xs = np.concatenate([Xn, Xn]) if shared else Xn
    absw = np.abs(Xs) @ np.abs(Wd).T
    absl = np.abs(Xs @ np64(U)) @ (np.abs(np64(C).reshape(d_out, r)) + eps * np.abs(Zm)).T
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= 2.0 ** -8 * absw + _bound(d_in, absw + absl, absl)), err.max()
    assert err.max() <= 2e-2 * np.abs(ref).max()


@pytest.mark.parametrize("d_in,d_out,r,T,shared", [(1024, 520, 16, 600, False), (4096, 768, 8, 1100, True)])
def test_pair_forward_int4_staged(ctx, monkeypatch, d_in, d_out, r, T, shared):
    # W first expanded to bf16 (fp32 product q * s, one rounding), then the bf16 kernel: a shared input from
    # 1024 rows, and stacked rows when ZOACT_INT4=staged asks for it
    monkeypatch.setenv("ZOACT_INT4", "staged")
    test_pair_forward_int4(ctx, d_in, d_out, r, T, shared)


@pytest.mark.parametrize("d_in,d_out,r,T,gated,ydt", [
    (1024, 520, 16, 200, False, torch.float32),     # 400 rows: tiles across the sign boundary (two K slots)
    (4096, 1024, 16, 256, False, torch.bfloat16),   # 512 rows: tiles inside one sign, split last wave
    (2048, 776, 32, 600, False, torch.float32),     # ragged N, rank 32
    (1024, 384, 16, 300, True, torch.bfloat16),     # gated (gate rows on the leader, up rows on the peer)
    (4096, 1024, 8, 1024, True, torch.float32),
])
def test_pair_forward_int4_cta_pairs(ctx, monkeypatch, d_in, d_out, r, T, gated, ydt):
    # ZOACT_INT4=kernel, stacked rows from 256: INT4 dequantised by the CTA-pair kernel's own warps, every weight
    # q * s rounded once to bf16 -- the values the expansion to bf16 holds, so the output is bit-identical to the
    # staged path (same MMAs in the same order) and within the rounding of the weights of the fp64 oracle
    eps, seed, query = 0.5, 17, 4
    L, Wd, U, C = _int4_layer(d_in, d_out, r, 70, 3)
    X = normal((2 * T, d_in), 71, DEV, dtype=torch.bfloat16)
    outs = []
    Lu = None
    if gated:
        Lu, Wu, Uu, Cu = _int4_layer(d_in, d_out, r, 80, 4)
    for mode in ("kernel", "staged"):
        monkeypatch.setenv("ZOACT_INT4", mode)
        Y = torch.full((2 * T, d_out), float("nan"), dtype=ydt, device=DEV)
        if gated:
            zo.zoact_pair_forward_gated(ctx, L, Lu, X, T, False, eps, seed, query, Y)
        else:
            zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Y)
        torch.cuda.synchronize()
        assert ctx.device_status() == 0
        outs.append(Y)
    monkeypatch.delenv("ZOACT_INT4")
    assert torch.equal(outs[0], outs[1])
    Xn = np64(X)
    Zm = philox.perturbation(seed, 3, query, d_out, r)
    ref = layers.pair_forward(Wd, np64(U), np64(C).reshape(d_out, r), Zm, Xn, eps, T, False)
    absw = np.abs(Xn) @ np.abs(Wd).T
    absl = np.abs(Xn @ np64(U)) @ (np.abs(np64(C).reshape(d_out, r)) + eps * np.abs(Zm)).T
    if gated:
        u = layers.pair_forward(Wu, np64(Uu), np64(Cu).reshape(d_out, r), philox.perturbation(seed, 4, query, d_out, r),
                                Xn, eps, T, False)
        ref = layers.silu(ref) * u
        assert np.abs(np64(outs[0]) - ref).max() <= 2e-2 * np.abs(ref).max()
        assert np.mean(np.abs(np64(outs[0]) - ref)) <= 5e-3 * np.mean(np.abs(ref))
        return
    # weights rounded to bf16 (2^-9 relative) plus fp32 accumulation, plus the output's own rounding
    out_r = 2.0 ** -8 if ydt == torch.bfloat16 else 0.0
    err = np.abs(np64(outs[0]) - ref)
    assert np.all(err <= 2.0 ** -9 * absw + _bound(d_in, absw + absl, absl) + out_r * np.abs(ref)), err.max()


def test_pair_forward_gated_int4(ctx):
    _gated_int4(ctx, 96)


def test_pair_forward_gated_int4_staged(ctx):
    _gated_int4(ctx, 1024)


def _gated_int4(ctx, T):
    d_in, d_out, r = 1024, 384, 16
    eps, seed, query = 0.25, 3, 5
    Lg, Wg, Ug, Cg = _int4_layer(d_in, d_out, r, 50, 0)
    Lu, Wu, Uu, Cu = _int4_layer(d_in, d_out, r, 60, 1)
    X = normal((T, d_in), 61, DEV, dtype=torch.bfloat16)
    H = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    zo.zoact_pair_forward_gated(ctx, Lg, Lu, X, T, True, eps, seed, query, H)
    torch.cuda.synchronize()
    g = layers.pair_forward(Wg, np64(Ug), np64(Cg).reshape(d_out, r), philox.perturbation(seed, 0, query, d_out, r),
                            np64(X), eps, T, True)
    u = layers.pair_forward(Wu, np64(Uu), np64(Cu).reshape(d_out, r), philox.perturbation(seed, 1, query, d_out, r),
                            np64(X), eps, T, True)
    ref = layers.silu(g) * u
    assert np.abs(np64(H) - ref).max() <= 2e-2 * np.abs(ref).max()
    assert np.mean(np.abs(np64(H) - ref)) <= 5e-3 * np.mean(np.abs(ref))


# ---------------- loss ----------------
@pytest.mark.parametrize("T,n,dt,with_target", [(64, 256, torch.float32, True), (2048, 4096, torch.bfloat16, True),
                                                (33, 7, torch.bfloat16, False), (300, 1000, torch.float16, True)])
def test_loss_pair(ctx, T, n, dt, with_target):
    Y = normal((2 * T, n), 31, DEV, dtype=dt)
    Y[T:] = (Y[:T].float() + 1e-2 * normal((T, n), 32, DEV)).to(dt)   # close pair: D << L
    tgt = normal((T, n), 33, DEV, dtype=dt) if with_target else None
    out = torch.zeros(4, dtype=torch.float64, device=DEV)
    zo.zoact_loss_pair(ctx, Y, T, 1e-3, out, target=tgt)
    torch.cuda.synchronize()
    Lp, Lm, D, a = oloss.loss_pair(np64(Y), T, None if tgt is None else np64(tgt), 1e-3)
    o = out.cpu().numpy()
    assert o[0] == pytest.approx(Lp, rel=1e-5) and o[1] == pytest.approx(Lm, rel=1e-5)
    assert o[2] == pytest.approx(D, rel=1e-4, abs=1e-7 * Lp)
    assert o[3] == pytest.approx(a, rel=1e-4, abs=1e-7 * Lp / 2e-3)
    assert np.sign(o[3]) == np.sign(a)


# ---------------- Adam / SGD ----------------
def test_adam_step_over_blocks(ctx):
    specs = [(0, 256, 8, 0), (2048, 100, 3, 7), (2352, 14336, 16, 2)]     # (offset, d_out, r, layer_id)
    n = 2352 + 14336 * 16
    C = normal((n,), 41, DEV, std=0.1)
    m = normal((n,), 42, DEV, std=0.01)
    v = normal((n,), 43, DEV, std=0.01).abs()
    C0, m0, v0 = np64(C), np64(m), np64(v)
    out = torch.tensor([1.0, 0.5, 0.5, 0.73], dtype=torch.float64, device=DEV)
    seed, query, step, lr = 99, 12, 3, 1e-3
    zo.zoact_adam_step(ctx, C, m, v, specs, out, lr, 0.9, 0.999, 1e-8, step, seed, query)
    torch.cuda.synchronize()
    Cr, mr, vr = C0.copy(), m0.copy(), v0.copy()
    # the ABI carries lr, betas and eps as fp32: the oracle reads those stored values
    f32 = lambda x: float(np.float32(x))
    for off, d_out, r, lid in specs:
        sl = slice(off, off + d_out * r)
        g = optim.zo_gradient(0.73, philox.perturbation(seed, lid, query, d_out, r).reshape(-1))
        Cr[sl], mr[sl], vr[sl] = optim.adam_step(C0[sl], m0[sl], v0[sl], g, f32(lr), f32(0.9), f32(0.999),
                                                 f32(1e-8), step)
    np.testing.assert_allclose(np64(m), mr, rtol=1e-5, atol=1e-7)
    np.testing.assert_allclose(np64(v), vr, rtol=1e-5, atol=1e-9)
    np.testing.assert_allclose(np64(C), Cr, rtol=1e-4, atol=1e-6 * lr)
    # elements between blocks (2348 .. 2351) are untouched
    np.testing.assert_array_equal(np64(C)[2348:2352], C0[2348:2352])
    np.testing.assert_array_equal(np64(m)[2348:2352], m0[2348:2352])


def test_sgd_and_nonfinite_guard(ctx):
    specs = [(0, 64, 4, 5)]
    C = normal((256,), 51, DEV)
    C0 = np64(C)
    out = torch.tensor([0, 0, 0, -2.0], dtype=torch.float64, device=DEV)
    zo.zoact_sgd_step(ctx, C, specs, out, 0.01, 3, 4)
    torch.cuda.synchronize()
    ref = optim.sgd_step(C0, optim.zo_gradient(-2.0, philox.perturbation(3, 5, 4, 64, 4).reshape(-1)),
                         float(np.float32(0.01)))
    np.testing.assert_allclose(np64(C), ref, rtol=1e-6, atol=1e-7)
    # a NaN estimator leaves C alone and raises the device status
    before = C.clone()
    out[3] = float("nan")
    zo.zoact_sgd_step(ctx, C, specs, out, 0.01, 3, 5)
    assert ctx.device_status(reset=True) == zo._lib.ZOACT_ERR_NONFINITE
    assert torch.equal(C, before)


# ---------------- glue ----------------
@pytest.mark.parametrize("n,dt", [(4096, torch.bfloat16), (5120, torch.float16), (14336, torch.bfloat16),
                                  (20480, torch.float16), (100, torch.bfloat16), (256, torch.float32)])
def test_rms_norm_widths(ctx, n, dt):
    rows = 19
    X = normal((rows, n), 65, DEV, dtype=dt)
    Y = torch.empty_like(X)
    zo.zoact_rms_norm(ctx, X, Y)
    torch.cuda.synchronize()
    ref = layers.rms_norm(np64(X))
    rel = {torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11, torch.float32: 2.0 ** -22}[dt]
    assert np.all(np.abs(np64(Y) - ref) <= rel * np.abs(ref) + 1e-5)


def test_rms_norm_and_mix(ctx):
    rows, n = 37, 4096
    X = normal((rows, n), 61, DEV, dtype=torch.bfloat16)
    Y = torch.empty_like(X)
    zo.zoact_rms_norm(ctx, X, Y)
    q = normal((rows, n), 62, DEV, dtype=torch.bfloat16)
    k = normal((rows, 1024), 63, DEV, dtype=torch.bfloat16)
    v = normal((rows, 1024), 64, DEV, dtype=torch.bfloat16)
    M = torch.empty_like(q)
    zo.zoact_mix_rms(ctx, q, k, v, M, 4, 128)
    torch.cuda.synchronize()
    ref = layers.rms_norm(np64(X))
    assert np.all(np.abs(np64(Y) - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5)
    mix = np64(q) + layers.repeat_kv(np64(k), 8, 4, 128) + layers.repeat_kv(np64(v), 8, 4, 128)
    ref = layers.rms_norm(mix)
    assert np.all(np.abs(np64(M) - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5)


# ---------------- basis ----------------
def test_basis_fp32_matches_oracle_iteration_and_eigenspace(ctx):
    n, d, r, p, iters, seed = 512, 256, 8, 8, 8, 17
    X, _ = lowrank_activations(n, d, 16, 0.1, 71, DEV, dtype=torch.float32, unit_rms=False, noise_is_energy=False)
    U = torch.empty(d, r, dtype=torch.float32, device=DEV)
    ev = torch.empty(r + p, dtype=torch.float32, device=DEV)
    zo.zoact_basis_init(ctx, X, r, U, oversample=p, n_iter=iters, seed=seed, evals_out=ev)
    torch.cuda.synchronize()
    Xn = np64(X)
    Ui, theta = basis.subspace_iteration(basis.gram(Xn), r, p, iters, seed)
    Ue, evals = basis.top_r_basis(Xn, r)
    Ug = np64(U)
    np.testing.assert_allclose(Ug.T @ Ug, np.eye(r), atol=1e-5)
    assert basis.subspace_overlap(Ug, Ue) >= 1 - 1e-6
    np.testing.assert_allclose(Ug, Ui, atol=1e-4)
    np.testing.assert_allclose(np64(ev)[:r], evals[:r], rtol=1e-4)


def test_basis_bf16_tensor_core_gram(ctx):
    n, d, r = 1000, 1024, 16
    X, _ = lowrank_activations(n, d, 32, 0.05, 72, DEV, dtype=torch.bfloat16)
    U = torch.empty(d, r, dtype=torch.float32, device=DEV)
    zo.zoact_basis_init(ctx, X, r, U, oversample=16, n_iter=10, seed=1)
    torch.cuda.synchronize()
    Ue, evals = basis.top_r_basis(np64(X), r)
    gap = (evals[r - 1] - evals[r]) / evals[0]
    ov = basis.subspace_overlap(np64(U), Ue)
    # Davis-Kahan: sin(theta) <~ ||E|| / gap, with E the fp32 Gram error (~1e-6 relative)
    assert ov >= 1 - (1e-5 / gap) ** 2 - 1e-6, (ov, gap)


def test_kernel_timing(ctx):
    # the timing facility records one event pair per tensor-core pair-forward kernel and nothing else
    d_in, d_out, r, T = 512, 264, 16, 130
    X, W, U, C = _pair_case(d_in, d_out, r, T, False, torch.bfloat16, 1e-3, 0.1)
    Y = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    L = zo.make_layer(W, U, C, 1)
    ctx.kernel_timing(True)
    for q in range(3):
        zo.zoact_pair_forward(ctx, L, X, T, False, 1e-3, 1, q, Y)
    ms, n = ctx.kernel_time()
    ctx.kernel_timing(False)
    assert n == 3 and ms > 0.0
    zo.zoact_pair_forward(ctx, L, X, T, False, 1e-3, 1, 0, Y)
    assert ctx.kernel_time() == (0.0, 0)


@pytest.mark.parametrize("gated", [False, True])
@pytest.mark.parametrize("T,d_out,r,dt", [(300, 264, 16, torch.bfloat16), (640, 392, 32, torch.float16),
                                          (257, 136, 4, torch.bfloat16), (512, 520, 8, torch.bfloat16)])
def test_shared_pair_16bit_staged(ctx, gated, T, d_out, r, dt):
    # the two signs on a shared input with 16-bit outputs (CTA pairs): both signs go through shared-memory
    # staging and bulk stores -- rows past T (a partial second M tile) and columns past d_out (a partial last
    # 16-column chunk) must be dropped, the other sign's rows untouched
    d_in, eps, seed, query = 512, 0.5, 23, 7
    X, W, U, C = _pair_case(d_in, d_out, r, T, True, dt, eps, 0.3, seed=90)
    Y = torch.full((2 * T + 8, d_out), 7.0, dtype=dt, device=DEV)         # 8 guard rows after the output
    Yv = Y[:2 * T]
    if gated:
        W2 = normal((d_out, d_in), 95, DEV, std=d_in ** -0.5, dtype=dt)
        U2 = normal((d_in, r), 96, DEV) / np.sqrt(d_in)
        C2 = normal((d_out * r,), 97, DEV, std=0.3)
        zo.zoact_pair_forward_gated(ctx, zo.make_layer(W, U, C, 3), zo.make_layer(W2, U2, C2, 4), X, T, True,
                                    eps, seed, query, Yv)
        torch.cuda.synchronize()
        g, _, _ = _oracle_pair(X, W, U, C, eps, T, True, seed, 3, query, d_out, r)
        u, _, _ = _oracle_pair(X, W2, U2, C2, eps, T, True, seed, 4, query, d_out, r)
        ref = layers.silu(g) * u
    else:
        zo.zoact_pair_forward(ctx, zo.make_layer(W, U, C, 3), X, T, True, eps, seed, query, Yv)
        torch.cuda.synchronize()
        ref, _, _ = _oracle_pair(X, W, U, C, eps, T, True, seed, 3, query, d_out, r)
    assert ctx.device_status() == 0
    rel = {torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11}[dt]
    err = np.abs(np64(Yv) - ref)
    assert np.all(err <= rel * np.abs(ref) + 2e-3 * np.abs(ref).max()), err.max()
    assert torch.all(Y[2 * T:] == 7.0)                                   # nothing written past the output


@pytest.mark.parametrize("d_in,d_out,T,r,dt,act,with_target", [
    (1024, 520, 256, 16, torch.bfloat16, zo.ACT_NONE, True),     # ragged last 16-column chunk of d_out
    (2048, 1024, 512, 16, torch.bfloat16, zo.ACT_NONE, False),   # mean of squares
    (1024, 264, 256, 8, torch.float16, zo.ACT_GELU, True),
    (512, 768, 768, 4, torch.bfloat16, zo.ACT_RELU, True),
])
def test_pair_forward_loss_fused(ctx, d_in, d_out, T, r, dt, act, with_target):
    # the loss pair fused into the pair forward equals the pair forward (rounded output) followed by the loss
    # kernel, and the oracle's loss of the oracle's rounded output
    eps, seed, query, lid = 1e-3, 13, 4, 6
    X, W, U, C = _pair_case(d_in, d_out, r, T, False, dt, eps, 0.05, seed=110)
    tgt = normal((T, d_out), 120, DEV, dtype=dt) if with_target else None
    L = zo.make_layer(W, U, C, lid)
    out = torch.zeros(4, dtype=torch.float64, device=DEV)
    zo.zoact_pair_forward_loss(ctx, L, X, T, eps, seed, query, zo.TORCH_DT[dt], out, target=tgt, act=act)
    Y = torch.empty(2 * T, d_out, dtype=dt, device=DEV)
    zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Y, act=act)
    ref = torch.zeros(4, dtype=torch.float64, device=DEV)
    zo.zoact_loss_pair(ctx, Y, T, eps, ref, target=tgt)
    torch.cuda.synchronize()
    assert ctx.device_status() == 0
    o, rf = out.cpu().numpy(), ref.cpu().numpy()
    # the exact (fp64) losses of the same rounded outputs Y. A compensated fp32 sum of n terms per thread
    # is off by about n u^2 S (u = 2^-24: ~1e-11 for the few hundred to thousand terms a thread adds here),
    # so even D = L+ - L- as a difference of the two sums is accurate; the loss kernel forms D directly
    Yd = Y.double()
    td = tgt.double() if with_target else torch.zeros(T, d_out, dtype=torch.float64, device=DEV)
    Lp_x = ((Yd[:T] - td) ** 2).mean().item()
    Lm_x = ((Yd[T:] - td) ** 2).mean().item()
    D_x = ((Yd[:T] - Yd[T:]) * (Yd[:T] + Yd[T:] - 2 * td)).mean().item()
    assert abs(o[0] - Lp_x) <= 1e-10 * Lp_x and abs(o[1] - Lm_x) <= 1e-10 * Lm_x, (o, Lp_x, Lm_x)
    assert abs(o[2] - D_x) <= 1e-10 * max(Lp_x, Lm_x), (o[2], D_x)
    eps32 = float(np.float32(eps))                   # eps crosses the ABI as a float
    assert abs(o[3] - D_x / (2 * eps32)) <= 1e-10 * max(Lp_x, Lm_x) / (2 * eps32)
    assert np.allclose(o[:2], rf[:2], rtol=1e-7, atol=0), (o, rf)
    assert abs(rf[2] - D_x) <= 1e-7 * max(Lp_x, Lm_x), (rf[2], D_x)
    # the oracle: its own output, rounded to the output type, then its loss pair
    yo, _, _ = _oracle_pair(X, W, U, C, eps, T, False, seed, lid, query, d_out, r)
    yo = {zo.ACT_NONE: lambda y: y, zo.ACT_RELU: layers.relu, zo.ACT_GELU: layers.gelu_erf}[act](yo)
    yo = torch.from_numpy(yo).to(dt).double().numpy()
    Lp, Lm, D, a = oloss.loss_pair(yo, T, np64(tgt) if with_target else None, eps)
    assert abs(o[0] - Lp) <= 1e-3 * Lp and abs(o[1] - Lm) <= 1e-3 * Lm


def test_pair_forward_loss_refusals(ctx):
    # launches that cannot fuse are refused before any pair-forward launch (the caller falls back)
    d_in, d_out, r, eps = 512, 256, 8, 1e-3
    X, W, U, C = _pair_case(d_in, d_out, r, 300, False, torch.bfloat16, eps, 0.05)
    L = zo.make_layer(W, U, C, 1)
    P = torch.zeros(600, r, device=DEV)
    out = torch.zeros(4, dtype=torch.float64, device=DEV)
    n0 = ctx.launch_count()
    for T, ydt in [(300, zo.DT_BF16), (256, zo.DT_FP32)]:
        with pytest.raises(zo.ZoactError) as e:
            zo.zoact_pair_forward_loss(ctx, L, X[:2 * T], T, eps, 1, 1, ydt, out, P=P[:2 * T])
        assert e.value.status == -2
    assert ctx.launch_count() == n0
