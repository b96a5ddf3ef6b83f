"""GPU parity of the multi-point path (Algorithm 2 in the paper's one-sided form)
against the oracle, through the C ABI.

The forward evaluates each adapted linear at n_blocks coefficient points in
one launch; block b of the stacked output is C + coef_b Z(query_b).  Cases
cover T below, at and above the 128/256-row tiles (tiles whose rows span two,
three or four blocks), shared and stacked inputs, gated gate/up pairs, INT4 and
fp32 weights, and the two-sided pair written as blocks.  Tolerances follow
test_gpu_kernels.py: fp32 outputs within the fp32 accumulation bound and 1e-4 of
the output scale; 16-bit outputs within their rounding on top of it (bar 2e-2).
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from paper_2607_01125_gb300.model import AdaptedLinear, ZOStep, coefficient_offsets
from oracle import philox, layers, loss as oloss, optim, graphs
from synth import normal, lowrank_activations, quantize_int4_g128, workload, tensor_seed, random_orthonormal

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
f32 = lambda v: float(np.float32(v))


@pytest.fixture(scope="module")
def ctx():
    c = zo.Context(0)
    yield c
    assert c.device_status() == 0
    c.close()


def np64(t):
    return t.detach().double().cpu().numpy()


def _points(nb, mu, q0=3, two_sided=False):
    if two_sided:
        return [(mu, q0), (-mu, q0)]
    return [(0.0, 0)] + [(mu, q0 + j) for j in range(nb - 1)]


def _oracle(Wn, Un, Cn, Xn, points, T, shared, seed, lid):
    d_out, r = Cn.shape
    Zs = [None if c == 0.0 else philox.perturbation(seed, lid, q, d_out, r) for c, q in points]
    Y = layers.multi_forward(Wn, Un, Cn, Zs, [c for c, _ in points], Xn, T, shared)
    nb = len(points)
    Xs = np.concatenate([Xn] * nb) if shared else Xn
    Zabs = np.concatenate([np.zeros_like(Cn) if z is None else abs(c) * np.abs(z)
                           for z, (c, _) in zip(Zs, points)])
    # per-row |C| + |c_b Z_b| for the accumulation bound
    absb = np.abs(Xs) @ np.abs(Wn).T
    lr_abs = np.concatenate([np.abs(Xs[b * T:(b + 1) * T] @ Un) @ (np.abs(Cn) + Zabs[b * d_out:(b + 1) * d_out]).T
                             for b in range(nb)])
    return Y, absb + lr_abs, lr_abs


@pytest.mark.parametrize("d_in,d_out,r,T,nb,shared,dt", [
    (1024, 520, 16, 200, 9, False, torch.bfloat16),   # 1800 rows: CTA-pair tiles whose halves span 2 blocks
    (512, 264, 16, 50, 9, False, torch.bfloat16),     # T < 128: a tile half spans up to 4 blocks (two passes)
    (768, 512, 16, 300, 9, True, torch.bfloat16),     # shared: 9 outputs per accumulator row, 5 passes
    (512, 264, 8, 40, 3, False, torch.float16),       # 120 rows: one-CTA tiles
    (1024, 520, 16, 256, 9, False, torch.bfloat16),   # tiles inside one block: whole term on the tensor cores
    (1024, 520, 16, 300, 9, False, torch.bfloat16),   # tiles across two blocks: two K slots by block parity
    (4096, 1024, 32, 160, 5, False, torch.bfloat16),  # rank 32: two table chunks per tile
    (256, 200, 8, 37, 4, False, torch.float32),       # fp32 weights: CUDA-core kernel
    (256, 256, 8, 64, 6, True, torch.float32),
])
def test_multi_forward_fp32_out(ctx, d_in, d_out, r, T, nb, shared, dt):
    seed, lid, mu = 17, 4, 0.5
    X = normal(((T if shared else nb * T), d_in), 1, DEV, dtype=dt)
    W = normal((d_out, d_in), 2, DEV, std=d_in ** -0.5, dtype=dt)
    U = normal((d_in, r), 3, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), 4, DEV, std=0.3)
    Y = torch.empty(nb * T, d_out, dtype=torch.float32, device=DEV)
    pts = _points(nb, mu)
    zo.zoact_multi_forward(ctx, zo.make_layer(W, U, C, lid), X, T, shared, pts, seed, Y)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle(np64(W), np64(U), np64(C).reshape(d_out, r), np64(X), pts, T, shared, seed, lid)
    err = np.abs(np64(Y) - ref)
    # fp32 accumulation, plus the 16-bit split of the low-rank term where it runs on the tensor cores
    assert np.all(err <= 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 2.0 ** -14 * lrabs + 1e-6), err.max()
    assert err.max() <= 1e-4 * np.abs(ref).max()


def test_two_sided_blocks_equal_the_pair_forward(ctx):
    # the pair forward is the two-block case: the same kernels, bit for bit
    d_in, d_out, r, T, seed, lid, eps, query = 1024, 520, 16, 200, 9, 2, 1e-3, 5
    X = normal((2 * T, d_in), 5, DEV, dtype=torch.bfloat16)
    W = normal((d_out, d_in), 6, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    U = normal((d_in, r), 7, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), 8, DEV, std=0.05)
    L = zo.make_layer(W, U, C, lid)
    Y1 = torch.empty(2 * T, d_out, dtype=torch.bfloat16, device=DEV)
    Y2 = torch.empty_like(Y1)
    zo.zoact_pair_forward(ctx, L, X, T, False, eps, seed, query, Y1)
    zo.zoact_multi_forward(ctx, L, X, T, False, [(eps, query), (-eps, query)], seed, Y2)
    torch.cuda.synchronize()
    assert torch.equal(Y1, Y2)


@pytest.mark.parametrize("T,nb,shared", [(96, 5, True), (70, 5, False), (300, 3, True), (150, 9, False),
                                         (256, 5, False)])
def test_multi_forward_gated(ctx, T, nb, shared):
    d_in, d_out, r, seed, mu = 512, 400, 16, 8, 0.25
    X = normal(((T if shared else nb * T), d_in), 21, DEV, dtype=torch.bfloat16)
    Wg = normal((d_out, d_in), 22, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    Wu = normal((d_out, d_in), 23, DEV, std=d_in ** -0.5, dtype=torch.bfloat16)
    Ug = normal((d_in, r), 24, DEV) / np.sqrt(d_in)
    Uu = normal((d_in, r), 25, DEV) / np.sqrt(d_in)
    Cg = normal((d_out * r,), 26, DEV, std=0.2)
    Cu = normal((d_out * r,), 27, DEV, std=0.2)
    H = torch.empty(nb * T, d_out, dtype=torch.float32, device=DEV)
    pts = _points(nb, mu)
    zo.zoact_multi_forward_gated(ctx, zo.make_layer(Wg, Ug, Cg, 0), zo.make_layer(Wu, Uu, Cu, 1), X, T, shared,
                                 pts, seed, H)
    torch.cuda.synchronize()
    g, _, _ = _oracle(np64(Wg), np64(Ug), np64(Cg).reshape(d_out, r), np64(X), pts, T, shared, seed, 0)
    u, _, _ = _oracle(np64(Wu), np64(Uu), np64(Cu).reshape(d_out, r), np64(X), pts, T, shared, seed, 1)
    ref = layers.silu(g) * u
    assert np.abs(np64(H) - ref).max() <= 1e-4 * np.abs(ref).max()


@pytest.mark.parametrize("T,nb,shared", [(64, 5, False), (120, 9, True)])
def test_multi_forward_int4(ctx, T, nb, shared):
    d_in, d_out, r, seed, lid, mu = 1024, 520, 16, 13, 6, 0.5
    Wf = normal((d_out, d_in), 40, DEV, std=0.02)
    packed, scales = quantize_int4_g128(Wf)
    U = normal((d_in, r), 41, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), 42, DEV, std=0.3)
    L = zo.make_layer(packed, U, C, lid, w_scales=scales, wtype=zo.DT_INT4_G128, d_in=d_in)
    Wd = layers.dequant_int4_g128(packed.cpu().numpy(), scales.float().cpu().numpy(), d_in)
    X = normal(((T if shared else nb * T), d_in), 43, DEV, dtype=torch.bfloat16)
    Y = torch.empty(nb * T, d_out, dtype=torch.float32, device=DEV)
    pts = _points(nb, mu)
    zo.zoact_multi_forward(ctx, L, X, T, shared, pts, seed, Y)
    torch.cuda.synchronize()
    ref, absb, lrabs = _oracle(Wd, np64(U), np64(C).reshape(d_out, r), np64(X), pts, T, shared, seed, lid)
    err = np.abs(np64(Y) - ref)
    assert np.all(err <= 2.0 ** -8 * absb + 8 * np.sqrt(d_in) * 2.0 ** -24 * absb + 2.0 ** -14 * lrabs + 1e-6), err.max()


def test_multi_forward_full_size_sampled(ctx):
    # the Llama down projection with 9 blocks of T = 2048 (18432 rows), sampled rows of every block
    d_in, d_out, r, T, nb, seed, lid, mu = 14336, 4096, 16, 2048, 9, 77, 2, 1e-3
    X = normal((nb * T, d_in), 50, DEV, dtype=torch.bfloat16)
    W = normal((d_out, d_in), 51, DEV, std=0.02, dtype=torch.bfloat16)
    U = normal((d_in, r), 52, DEV) / np.sqrt(d_in)
    C = normal((d_out * r,), 53, DEV, std=0.05)
    Y = torch.empty(nb * T, d_out, dtype=torch.bfloat16, device=DEV)
    pts = _points(nb, mu, q0=11)
    zo.zoact_multi_forward(ctx, zo.make_layer(W, U, C, lid), X, T, False, pts, seed, Y)
    torch.cuda.synchronize()
    rng = np.random.default_rng(3)
    rows = np.sort(rng.choice(nb * T, 90, replace=False))
    Xs, Wn, Un, Cn = np64(X[torch.as_tensor(rows, device=DEV)]), np64(W), np64(U), np64(C).reshape(d_out, r)
    ref = np.empty((len(rows), d_out))
    for i, row in enumerate(rows):
        c, q = pts[row // T]
        Cb = Cn if c == 0.0 else Cn + c * philox.perturbation(seed, lid, q, d_out, r)
        ref[i] = Xs[i] @ Wn.T + (Xs[i] @ Un) @ Cb.T
    got = np64(Y[torch.as_tensor(rows, device=DEV)])
    err = np.abs(got - ref)
    assert err.max() <= 2e-2 * np.abs(ref).max()
    assert np.all(err <= 2.0 ** -7 * np.abs(ref) + 2e-3 * np.abs(ref).max())


# ---------------- losses and the q-query update ----------------
@pytest.mark.parametrize("T,n,nb,dt,with_target", [(64, 256, 3, torch.float32, True),
                                                   (2048, 4096, 9, torch.bfloat16, True),
                                                   (33, 7, 5, torch.bfloat16, False),
                                                   (300, 1000, 17, torch.float16, True)])
def test_loss_multi(ctx, T, n, nb, dt, with_target):
    y0 = normal((T, n), 61, DEV)
    Y = torch.cat([y0] + [y0 + 1e-2 * normal((T, n), 62 + j, DEV) for j in range(nb - 1)]).to(dt)
    tgt = normal((T, n), 80, DEV, dtype=dt) if with_target else None
    out = torch.zeros(2 * nb - 1, dtype=torch.float64, device=DEV)
    mu = 1e-3
    zo.zoact_loss_multi(ctx, Y, T, nb, mu, out, target=tgt)
    torch.cuda.synchronize()
    Yn = np64(Y)
    L, a = oloss.loss_queries(Yn, T, nb, None if tgt is None else np64(tgt), mu)
    o = out.cpu().numpy()
    np.testing.assert_allclose(o[:nb], L, rtol=1e-5)
    # a_j: fp32 sums of 8 products per vector into fp64
    t = 0.0 if tgt is None else np64(tgt)
    for j in range(1, nb):
        scale = np.mean(np.abs((Yn[j * T:(j + 1) * T] - Yn[:T]) * (Yn[j * T:(j + 1) * T] + Yn[:T] - 2 * t))) / mu
        assert abs(o[nb + j - 1] - a[j - 1]) <= 1e-4 * abs(a[j - 1]) + 1e-6 * scale


@pytest.mark.parametrize("q", [1, 8, 16])
def test_adam_and_sgd_multi(ctx, q):
    specs = [(0, 256, 8, 0), (2048, 100, 3, 7), (2352, 4096, 16, 2)]
    n = 2352 + 4096 * 16
    seed, step, lr = 99, 3, 1e-3
    queries = [1000 + 17 * j for j in range(q)]
    a_host = np.random.default_rng(q).standard_normal(q)
    a = torch.tensor(a_host, dtype=torch.float64, device=DEV)
    C = normal((n,), 41, DEV, std=0.1)
    m = normal((n,), 42, DEV, std=0.01)
    v = normal((n,), 43, DEV, std=0.01).abs()
    C0, m0, v0 = np64(C), np64(m), np64(v)
    zo.zoact_adam_step_multi(ctx, C, m, v, specs, a, queries, lr, 0.9, 0.999, 1e-8, step, seed)
    Cs = C0.copy()
    Cs_t = torch.tensor(Cs, dtype=torch.float32, device=DEV)
    zo.zoact_sgd_step_multi(ctx, Cs_t, specs, a, queries, lr, seed)
    torch.cuda.synchronize()
    Cr, mr, vr, Csr = C0.copy(), m0.copy(), v0.copy(), C0.copy()
    for off, d_out, r, lid in specs:
        sl = slice(off, off + d_out * r)
        g = optim.zo_gradient_queries(a_host, [philox.perturbation(seed, lid, qq, d_out, r).reshape(-1)
                                               for qq in queries])
        Cr[sl], mr[sl], vr[sl] = optim.adam_step(C0[sl], m0[sl], v0[sl], g, f32(lr), f32(0.9), f32(0.999),
                                                 f32(1e-8), step)
        Csr[sl] = optim.sgd_step(C0[sl], g, f32(lr))
    np.testing.assert_allclose(np64(m), mr, rtol=1e-5, atol=1e-7)
    np.testing.assert_allclose(np64(v), vr, rtol=1e-5, atol=1e-9)
    np.testing.assert_allclose(np64(C), Cr, rtol=1e-4, atol=1e-6 * lr)
    np.testing.assert_allclose(np64(Cs_t), Csr, rtol=1e-6, atol=1e-7 * lr)
    np.testing.assert_array_equal(np64(C)[2348:2352], C0[2348:2352])


def test_multi_update_nonfinite_guard(ctx):
    specs = [(0, 64, 4, 5)]
    C = normal((256,), 51, DEV)
    C0 = C.clone()
    a = torch.tensor([0.5, float("nan"), 1.0], dtype=torch.float64, device=DEV)
    zo.zoact_sgd_step_multi(ctx, C, specs, a, [1, 2, 3], 0.01, 3)
    torch.cuda.synchronize()
    assert ctx.device_status() == -4          # ZOACT_ERR_NONFINITE (read and reset)
    assert torch.equal(C, C0)


# ---------------- whole one-sided steps ----------------
def _basis(w, s, bases):
    """A random orthonormal basis per layer input: a decoder's q, k and v read one input and share one basis (as
    Algorithm 1 gives them), so the stack's pair forwards may run them as one launch."""
    name = s.name
    if name.endswith(".k") or name.endswith(".v"):
        name = name[:-2] + ".q"
    if name not in bases:
        bases[name] = random_orthonormal(s.d_in, w.r, tensor_seed(w, "U", name), DEV)
    return bases[name]


def _build(w, n_queries, c_std=0.05):
    dt = {"bf16": torch.bfloat16, "fp16": torch.float16, "fp32": torch.float32}[w.act_dtype]
    specs = w.linears()
    offs = coefficient_offsets(specs, w.r)
    lins, ora, bases = [], {}, {}
    for s, off in zip(specs, offs):
        U = _basis(w, s, bases)
        W = normal((s.d_out, s.d_in), tensor_seed(w, "W", s.name), DEV, std=w.weight_std, dtype=dt)
        lins.append(AdaptedLinear(s.name, W, U, s.layer_id, off, w.r))
    step = ZOStep(zo.Context(0), w.kind, lins, w.T, w.act_dtype, eps=w.eps, lr=w.lr, n_queries=n_queries)
    step.C.copy_(normal(tuple(step.C.shape), tensor_seed(w, "C0"), DEV, std=c_std))
    for l in lins:
        ora[l.name] = dict(W=np64(l.W), U=np64(l.U), C=np64(step.C[l.offset:l.offset + l.d_out * w.r]).reshape(
            l.d_out, w.r), layer_id=l.layer_id)
    return step, ora


def test_toy_one_sided_steps():
    # fp32 toy graph, q = 4: outputs to 1e-4, a_j to 1e-3, C after two Adam steps to 1e-2 lr
    w = workload("toy_fp32")
    q = 4
    step, ora = _build(w, q)
    x, _ = lowrank_activations(w.T, 256, 16, 0.1, tensor_seed(w, "x"), DEV, dtype=torch.float32, unit_rms=False,
                               noise_is_energy=False)
    tgt = normal((w.T, 256), tensor_seed(w, "t"), DEV)
    lay = [ora["l1"], ora["l2"]]
    m = {k: np.zeros_like(v["C"]) for k, v in ora.items()}
    v = {k: np.zeros_like(v["C"]) for k, v in ora.items()}
    for t in (1, 2):
        seed, query = 5, t
        Y = step.forward(x, seed, query).clone()
        out = step.loss(Y, tgt).clone()
        step.update(t, seed, query)
        torch.cuda.synchronize()
        blocks = [(0.0, 0)] + [(w.eps, qq) for qq in step.query_ids(query)]
        Yo = graphs.toy_forward(lay, np64(x), 0.0, seed, 0, store="fp32", blocks=blocks)
        L, a = oloss.loss_queries(Yo, w.T, q + 1, np64(tgt), w.eps)
        assert np.abs(np64(Y) - Yo).max() <= 1e-4 * np.abs(Yo).max()
        o = out.cpu().numpy()
        np.testing.assert_allclose(o[:q + 1], L, rtol=1e-5)
        np.testing.assert_allclose(o[q + 1:], a, rtol=1e-3, atol=1e-3 * np.abs(a).max())
        for name, l in ora.items():
            g = optim.zo_gradient_queries(a, [philox.perturbation(seed, l["layer_id"], qq, *l["C"].shape)
                                              for qq in step.query_ids(query)])
            l["C"], m[name], v[name] = optim.adam_step(l["C"], m[name], v[name], g, f32(w.lr), f32(w.beta1),
                                                       f32(w.beta2), f32(w.adam_eps), t)
            lin = step.by_name[name]
            Cg = np64(step.C[lin.offset:lin.offset + lin.d_out * w.r]).reshape(l["C"].shape)
            assert np.abs(Cg - l["C"]).max() <= 1e-2 * w.lr
    assert step.ctx.device_status() == 0
    step.ctx.close()


@pytest.mark.parametrize("name,n_dec,T,q", [("llama_mlp_bf16", None, 256, 8), ("llama_stack_bf16", 1, 64, 4),
                                            ("llama_stack_bf16", 2, 64, 4)])
def test_bf16_one_sided_step(name, n_dec, T, q):
    # 16-bit graphs: every block's output and every L_b within 2e-2 (the a_j of a bf16 graph at mu = 1e-3 are
    # below the outputs' rounding and are not compared).  The stacks' 5 x 64 stacked rows run the RMS
    # normalisations as row scales (the second decoder's q, k, v take its unnormalised input)
    w = workload(name, T=T) if n_dec is None else workload(name, T=T, n_decoder=n_dec)
    step, ora = _build(w, q, c_std=0.01)
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV)
    tgt = normal((w.T, w.d_model), tensor_seed(w, "t"), DEV, dtype=torch.bfloat16) if w.kind == "llama_mlp" else None
    seed, query = 23, 2
    Y = step.forward(x, seed, query).clone()
    out = step.loss(Y, tgt).clone()
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0
    blocks = [(0.0, 0)] + [(w.eps, qq) for qq in step.query_ids(query)]
    if w.kind == "llama_mlp":
        Yo = graphs.llama_mlp_forward([ora["gate"], ora["up"], ora["down"]], np64(x), 0.0, seed, 0, store="bf16",
                                      blocks=blocks)
    else:
        names = ["q", "k", "v", "o", "gate", "up", "down"]
        Yo = graphs.stack_forward([{nm: ora[f"{L}.{nm}"] for nm in names} for L in range(w.n_decoder)], np64(x), 0.0,
                                  seed, 0, "llama", store="bf16", blocks=blocks)
    L, _ = oloss.loss_queries(Yo, w.T, q + 1, None if tgt is None else np64(tgt), w.eps)
    Yg = np64(Y)
    assert np.abs(Yg - Yo).max() <= 2e-2 * np.abs(Yo).max()
    assert np.mean(np.abs(Yg - Yo)) <= 1e-2 * np.mean(np.abs(Yo))
    np.testing.assert_allclose(out.cpu().numpy()[:q + 1], L, rtol=2e-2)
    step.ctx.close()


@pytest.mark.parametrize("gated", [False, True])
@pytest.mark.parametrize("T,nb,d_out,r,dt", [(300, 9, 264, 16, torch.bfloat16), (257, 3, 136, 8, torch.float16),
                                             (512, 5, 520, 4, torch.bfloat16), (300, 2, 264, 16, torch.bfloat16)])
def test_multi_shared_16bit_staged(ctx, gated, T, nb, d_out, r, dt):
    # evaluation blocks on a shared input with 16-bit outputs (CTA pairs, one basis for gate and up): four rows
    # per thread, outputs staged and written per block through a 3-D store map that drops rows past T (the
    # partial last M tile) and columns past d_out -- no block may spill into the next, nothing past the output
    d_in, seed, mu = 512, 8, 0.25
    pts = _points(nb, mu) if nb > 2 else [(mu, 3), (mu, 4)]          # nb = 2: two queries, not a +/- pair
    X = normal((T, d_in), 41, DEV, dtype=dt)
    Wg = normal((d_out, d_in), 42, DEV, std=d_in ** -0.5, dtype=dt)
    U = normal((d_in, r), 44, DEV) / np.sqrt(d_in)
    Cg = normal((d_out * r,), 46, DEV, std=0.2)
    Y = torch.full((nb * T + 8, d_out), 7.0, dtype=dt, device=DEV)
    Yv = Y[:nb * T]
    if gated:
        Wu = normal((d_out, d_in), 43, DEV, std=d_in ** -0.5, dtype=dt)
        Cu = normal((d_out * r,), 47, DEV, std=0.2)
        zo.zoact_multi_forward_gated(ctx, zo.make_layer(Wg, U, Cg, 0), zo.make_layer(Wu, U, Cu, 1), X, T, True,
                                     pts, seed, Yv)
        torch.cuda.synchronize()
        g, _, _ = _oracle(np64(Wg), np64(U), np64(Cg).reshape(d_out, r), np64(X), pts, T, True, seed, 0)
        u, _, _ = _oracle(np64(Wu), np64(U), np64(Cu).reshape(d_out, r), np64(X), pts, T, True, seed, 1)
        ref = layers.silu(g) * u
    else:
        zo.zoact_multi_forward(ctx, zo.make_layer(Wg, U, Cg, 0), X, T, True, pts, seed, Yv)
        torch.cuda.synchronize()
        ref, _, _ = _oracle(np64(Wg), np64(U), np64(Cg).reshape(d_out, r), np64(X), pts, T, True, seed, 0)
    assert ctx.device_status() == 0
    rel = {torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11}[dt]
    err = np.abs(np64(Yv) - ref)
    assert np.all(err <= rel * np.abs(ref) + 2e-3 * np.abs(ref).max()), err.max()
    assert torch.all(Y[nb * T:] == 7.0)
