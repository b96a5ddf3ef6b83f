"""Whole ZO steps on the GPU (C ABI, model.py) against the oracle's graphs.

Each test draws one set of inputs (synth), runs one ZO step through libzoact --
pair forwards with glue, loss pair, Adam -- and the same step in the fp64
oracle (with bf16/fp16 rounding mirrored where activations are stored).  Bases
are inputs here (random orthonormal U from synth) so the step is tested on its
own; the device basis is tested in test_gpu_kernels.py and below at full width.

Tolerances (the parity bar): 16-bit outputs and L+- within 2e-2 relative; the
estimator scalar a within 2e-2 relative (its sign agreeing) whenever
|L+ - L-| exceeds 2e-2 max(L+, L-).  The 16-bit step tests are built so that
it does: the coefficients are drawn as C = 0.3 Z(seed, layer, query) plus
noise and eps = 0.05, which moves every layer's output along its own
perturbation at first order (on the last linear D = L+ - L- ~ 4 eps 0.3
mean((Z p)^2), about a tenth of L), and each test asserts that bound before
comparing a.  (With eps = 1e-3 and C independent of Z, L+ - L- sits below the
bf16 resolution of the outputs and a is each side's rounding noise.)  Adam
step 1 is then checked on all three arenas: m = (1 - beta1) a Z and
v = (1 - beta2) (a Z)^2 carry |a| (2e-2 and 4e-2 relative), C - lr g/(|g| + eps)
its sign (2e-2 lr).  The fp32 toy graph checks outputs to 1e-4 and a to 1e-3
over two steps.
"""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from paper_2607_01125_gb300.model import AdaptedLinear, ZOStep, coefficient_offsets
from oracle import basis, graphs, loss as oloss, optim, philox
from synth import workload, normal, lowrank_activations, random_orthonormal, tensor_seed, quantize_int4_g128
from oracle import layers as olayers

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
f32 = lambda v: float(np.float32(v))
C_ALIGN = 0.3


def n64(t):
    return t.detach().cpu().double().numpy()


def _basis(w, s, bases):
    """A random orthonormal basis per layer input: a decoder's q, k and v read one input and share one basis (as
    Algorithm 1 gives them), so the stack's pair forwards may run them as one launch."""
    name = s.name
    if name.endswith(".k") or name.endswith(".v"):
        name = name[:-2] + ".q"
    if name not in bases:
        bases[name] = random_orthonormal(s.d_in, w.r, tensor_seed(w, "U", name), DEV)
    return bases[name]


def _build(w, c_std=0.01, align=None, n_queries=None):
    """Weights and bases of workload w on the device, its ZOStep, and a function that gives the oracle's
    fp64 copy of one layer (W, U, C, layer_id) on demand, so that deep stacks never hold every layer's
    fp64 weights at once.

    The coefficients are drawn on the host: N(0, c_std^2), plus C_ALIGN Z(seed, layer, query) from the
    oracle's generator when align = (seed, query).
    """
    dt = {"bf16": torch.bfloat16, "fp16": torch.float16, "fp32": torch.float32}[w.act_dtype]
    specs = w.linears()
    offs = coefficient_offsets(specs, w.r)
    lins, bases = [], {}
    for s, off in zip(specs, offs):
        U = _basis(w, s, bases)
        if w.wtype == "int4_g128":
            Wf = normal((s.d_out, s.d_in), tensor_seed(w, "W", s.name), DEV, std=w.weight_std)
            packed, scales = quantize_int4_g128(Wf)
            del Wf
            lins.append(AdaptedLinear(s.name, packed, U, s.layer_id, off, w.r, w_scales=scales,
                                      wtype=zo.DT_INT4_G128, d_in=s.d_in))
        else:
            W = normal((s.d_out, s.d_in), tensor_seed(w, "W", s.name), DEV, std=w.weight_std, dtype=dt)
            lins.append(AdaptedLinear(s.name, W, U, s.layer_id, off, w.r))
    step = ZOStep(zo.Context(0), w.kind, lins, w.T, w.act_dtype, eps=w.eps, lr=w.lr, n_queries=n_queries)
    C = normal(tuple(step.C.shape), tensor_seed(w, "C0"), "cpu", std=c_std).double().numpy()
    if align is not None:
        for l in lins:
            C[l.offset:l.offset + l.d_out * w.r] += C_ALIGN * philox.perturbation(
                align[0], l.layer_id, align[1], l.d_out, w.r).reshape(-1)
    step.C.copy_(torch.from_numpy(C.astype(np.float32)))
    C_stored = n64(step.C)

    def oracle_layer(name, weights=True):
        l = step.by_name[name]
        d = dict(C=C_stored[l.offset:l.offset + l.d_out * w.r].reshape(l.d_out, w.r), layer_id=l.layer_id)
        if weights:
            d["U"] = n64(l.U)
            if w.wtype == "int4_g128":
                d["W"] = olayers.dequant_int4_g128(l.W.cpu().numpy(), l.w_scales.float().cpu().numpy(), l.d_in)
            else:
                d["W"] = n64(l.W)
        return d

    return step, oracle_layer


def _stack_names(kind):
    return ["q", "k", "v", "o", "gate", "up", "down"] if kind == "llama" else ["q", "k", "v", "o", "fc1", "fc2"]


def _check_step(step, oracle_layer, Y, out, Yo, tgt_o, w, seed, query):
    """Outputs, losses, a, and Adam step 1 (from m = v = 0) of every layer against the oracle."""
    Lp, Lm, D, a = oloss.loss_pair(Yo, w.T, tgt_o, w.eps)
    Yg = n64(Y)
    err_max = float(np.abs(Yg - Yo).max() / np.abs(Yo).max())
    err_mean = float(np.mean(np.abs(Yg - Yo)) / np.mean(np.abs(Yo)))
    assert err_max <= 2e-2, ("max |dY| / max |Y|", err_max)
    # a systematic error shows in the mean long before the max: bf16 rounding noise through a chain of
    # stored activations stays well below 1e-2 of the mean magnitude
    assert err_mean <= 1e-2, ("mean |dY| / mean |Y|", err_mean)
    o = out.cpu().numpy()
    assert abs(o[0] - Lp) <= 2e-2 * Lp and abs(o[1] - Lm) <= 2e-2 * Lm, (o[:2], Lp, Lm)
    # the inputs are built so that the bound applies: a is compared, never skipped
    assert abs(Lp - Lm) > 2e-2 * max(Lp, Lm), ("the test's inputs must make L+ - L- resolvable", Lp, Lm)
    assert np.sign(o[3]) == np.sign(a), (o[3], a)
    assert abs(o[3] - a) <= 2e-2 * abs(a), (o[3], a)
    assert abs(o[2] - D) <= 2e-2 * abs(D), (o[2], D)
    b1, b2, lr, ae = f32(w.beta1), f32(w.beta2), f32(w.lr), f32(w.adam_eps)
    n_checked = 0
    for lin in step.linears:
        l = oracle_layer(lin.name, weights=False)
        sl = slice(lin.offset, lin.offset + lin.d_out * w.r)
        Zl = philox.perturbation(seed, l["layer_id"], query, *l["C"].shape)
        g = optim.zo_gradient(a, Zl)
        Cn, mn, vn = optim.adam_step(l["C"], 0, 0, g, lr, b1, b2, ae, 1)
        Cg, mg, vg = (n64(t[sl]).reshape(l["C"].shape) for t in (step.C, step.m, step.v))
        # a within 2e-2, and the device's normals within 1e-6 (1 + |z|) of the oracle's (fp32 Box-Muller)
        dz = 1e-6 * (1.0 + np.abs(Zl))
        bad = np.abs(mg - mn) > 2e-2 * np.abs(mn) + (1 - b1) * 1.02 * abs(a) * dz
        assert not bad.any(), (lin.name, mg[bad][:4], mn[bad][:4], Zl[bad][:4], o[3], a)
        assert np.all(np.abs(vg - vn) <= 4.1e-2 * np.abs(vn) + (1 - b2) * 1.05 * a * a * (2 * np.abs(Zl) + dz) * dz), \
            lin.name
        # where |g| is within ~1e3 adam_eps the step-1 update depends on |a| itself, and where |z| < 1e-4 the
        # normals' absolute tolerance may flip its sign: those elements are bounded through m, v above
        big = (np.abs(g) > 1e3 * w.adam_eps) & (np.abs(Zl) > 1e-4)
        assert np.abs(Cg - Cn)[big].max() <= 2e-2 * w.lr, (lin.name, o[3], a)
        n_checked += 1
    assert n_checked == len(step.linears)


def _run_step(step, x, tgt, seed, query):
    Y = step.forward(x, seed, query).clone()
    out = step.loss(Y, tgt).clone()
    step.update(1, seed, query)
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0
    return Y, out


def test_llama_mlp_step_full_width():
    # gate/up on the shared input (CTA-pair kernel, epilogue Z tables), down on 512 stacked rows
    seed, query = 17, 1
    w = workload("llama_mlp_bf16", T=256, eps=0.05)
    step, ol = _build(w, align=(seed, query))
    x, _ = lowrank_activations(w.T, 4096, 64, 0.05, tensor_seed(w, "x"), DEV)
    tgt = normal((w.T, 4096), tensor_seed(w, "t"), DEV, dtype=torch.bfloat16)
    Y, out = _run_step(step, x, tgt, seed, query)
    lay = [ol("gate"), ol("up"), ol("down")]
    Yo = graphs.llama_mlp_forward(lay, n64(x), w.eps, seed, query, store="bf16")
    _check_step(step, ol, Y, out, Yo, n64(tgt), w, seed, query)
    step.ctx.close()


@pytest.mark.parametrize("n_queries", [None, 8])
def test_bench_mlp_forward_sampled(n_queries):
    # the bench's MLP-block forward exactly as timed (T = 2048, eps = 1e-3: gate/up on the shared input with the
    # mirrored two-sign or nine-block epilogues, down on the stacked rows), checked on 16 sampled token rows of
    # every evaluation block; every op acts on each row on its own
    w = workload("llama_mlp_bf16")
    assert w.T == 2048
    step, ol = _build(w, n_queries=n_queries)
    x, _ = lowrank_activations(w.T, 4096, 64, 0.05, tensor_seed(w, "x"), DEV)
    seed, query = 41, 3
    if n_queries is None:
        blocks, nb = None, 2
    else:
        blocks = [(0.0, 0)] + [(w.eps, qq) for qq in step.query_ids(query)]
        nb = len(blocks)
    Y = step.forward(x, seed, query)
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0
    tok = np.sort(np.random.default_rng(7).choice(w.T, 16, replace=False))
    rows = np.concatenate([b * w.T + tok for b in range(nb)])
    Yo = graphs.llama_mlp_forward([ol("gate"), ol("up"), ol("down")], n64(x)[tok], w.eps, seed, query, store="bf16",
                                  blocks=blocks)
    _check_outputs(n64(Y)[rows], Yo, "MLP block")
    step.ctx.close()


@pytest.mark.parametrize("name,n_dec,T", [
    ("llama_stack_bf16", 2, 64), ("opt_stack_fp16", 2, 48), ("llama_stack_int4", 1, 64),   # one-CTA kernel
    # 512 stacked rows: the CTA-pair kernel (whole low-rank term on the MMA, split last wave) in the graph, the
    # second decoder's q, k and v as one launch
    ("llama_stack_bf16", 2, 256), ("opt_stack_fp16", 2, 256),
    # 1024 stacked rows: INT4 weights expanded once per call (the second decoder's q, k, v as one array), then the
    # bf16 CTA-pair kernel
    ("llama_stack_int4", 2, 512)])
def test_stack_step(name, n_dec, T):
    w = workload(name, T=T, n_decoder=n_dec, eps=0.05)
    _stack_step_per_decoder(w, 23, 2)


def _check_outputs(Yg, Yo, what):
    err_max = float(np.abs(Yg - Yo).max() / np.abs(Yo).max())
    err_mean = float(np.mean(np.abs(Yg - Yo)) / np.mean(np.abs(Yo)))
    assert err_max <= 2e-2 and err_mean <= 1e-2, (what, err_max, err_mean)


def _stack_step_per_decoder(w, seed, query):
    """One ZO step of stack w on the device, checked decoder by decoder.
    The synthetic stack is chaotic: a relative difference of 1e-3 in a decoder's input grows about 1.45x per
    decoder (measured on the oracle alone, with C = 0 as with C = 0.3 Z), so two correct implementations that
    round a stored activation differently drift apart along the chain (two INT4 decoders at 1024 stacked rows:
    0.74% and 0.77% mean error per decoder, 1.39% through both), and after ~20 decoders their final outputs are
    not comparable element by element.  Each decoder is therefore checked on identical inputs: the oracle is fed
    the GPU's stored input to that decoder, and its output is compared with the GPU's input to the next decoder
    (the step's output after the last).  L+-, D, a and Adam step 1 of all layers are then checked against the
    oracle's last decoder on the GPU's input to it."""
    step, ol = _build(w, align=(seed, query))
    dt = torch.bfloat16 if w.act_dtype == "bf16" else torch.float16
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV, dtype=dt)
    ins = []
    step.on_decoder = lambda L, h: ins.append(h.clone())
    Y, out = _run_step(step, x, None, seed, query)
    assert len(ins) == w.n_decoder and ins[0].shape == (w.T, w.d_model)
    outs = ins[1:] + [Y]
    for L in range(w.n_decoder):
        dl = {nm: ol(f"{L}.{nm}") for nm in _stack_names(w.kind)}
        assert outs[L].shape == (2 * w.T, w.d_model)
        Yo = graphs.stack_forward([dl], n64(ins[L]), w.eps, seed, query, w.kind, store=w.act_dtype,
                                  first=(L == 0))
        _check_outputs(n64(outs[L]), Yo, f"decoder {L}")
    _check_step(step, ol, Y, out, Yo, None, w, seed, query)
    step.ctx.close()


@pytest.mark.parametrize("name", ["llama_stack_bf16", "opt_stack_fp16", "llama_stack_int4"])
def test_stack_step_full_depth(name):
    # Every decoder of the configuration (32 or 40) at full width on 16 tokens per perturbation: layer ids, the
    # shared-input rule of the first decoder and the buffer rotation over the whole chain, each decoder checked
    # on the GPU's stored input to it
    w = workload(name, T=16, eps=0.05)
    assert w.n_decoder in (32, 40)
    _stack_step_per_decoder(w, 29, 3)


@pytest.mark.parametrize("name,n_queries", [("llama_stack_bf16", None), ("opt_stack_fp16", None),
                                            ("llama_stack_int4", None), ("llama_stack_bf16", 8)])
def test_stack_full_size_sampled(name, n_queries):
    # the bench's launches of a stack at full size (T = 4096: 8192 stacked rows for the two-sided pair, 9 x 4096
    # for the one-sided estimator with q = 8; row-scaled normalisations, L2-sized M-groups, split tails, the second
    # decoder's q, k and v as one launch, INT4 expanded per call, eps = 1e-3) on two decoders.  Every op of a
    # decoder acts on each token row on its own, so the oracle runs each decoder on 24 sampled token rows of the
    # GPU's stored input to it (the same rows of every evaluation block) and checks those rows of its output
    w = workload(name, n_decoder=2)
    assert w.T == 4096
    step, ol = _build(w, n_queries=n_queries)
    dt = torch.bfloat16 if w.act_dtype == "bf16" else torch.float16
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV, dtype=dt)
    ins = []
    step.on_decoder = lambda L, h: ins.append(h.clone())
    seed, query = 31, 4
    Y = step.forward(x, seed, query)
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0
    if n_queries is None:
        blocks = None
        nb = 2
    else:
        blocks = [(0.0, 0)] + [(w.eps, qq) for qq in step.query_ids(query)]
        nb = len(blocks)
    tok = np.sort(np.random.default_rng(3).choice(w.T, 24, replace=False))
    rows = np.concatenate([b * w.T + tok for b in range(nb)])
    outs = [ins[1], Y]
    for L in range(2):
        dl = {nm: ol(f"{L}.{nm}") for nm in _stack_names(w.kind)}
        h_in = n64(ins[L])[tok if L == 0 else rows]
        Yo = graphs.stack_forward([dl], h_in, w.eps, seed, query, w.kind, store=w.act_dtype, first=(L == 0),
                                  blocks=blocks)
        _check_outputs(n64(outs[L])[rows], Yo, f"decoder {L}")
    step.ctx.close()


@pytest.mark.parametrize("name,n_queries,r", [("llama_stack_bf16", None, None), ("opt_stack_fp16", None, None),
                                              ("llama_stack_int4", None, None), ("llama_stack_bf16", 8, None),
                                              ("llama_stack_int4", None, 32), ("llama_stack_bf16", None, 256)])
def test_bench_step_every_decoder_sampled(name, n_queries, r):
    # the bench's forward of each stack exactly as timed -- all 32 (Llama, INT4) or 40 (OPT) decoders, T = 4096
    # (8192 stacked rows), eps = 1e-3, row scales, L2-sized M-groups, split tails, q/k/v as one launch, INT4
    # expanded per call -- with every decoder checked on 8 sampled token rows (both signs) of the GPU's stored
    # input to it (every op of a decoder acts on each row on its own); with n_queries the one-sided estimator's
    # q + 1 evaluation blocks (9 x 4096 rows); with r the rank ablation's bench lines (INT4 at the paper's r = 32,
    # the stack at r = 256)
    w = workload(name) if r is None else workload(name, r=r)
    assert w.T == 4096 and w.n_decoder in (32, 40)
    step, ol = _build(w, n_queries=n_queries)
    dt = torch.bfloat16 if w.act_dtype == "bf16" else torch.float16
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV, dtype=dt)
    tok = np.sort(np.random.default_rng(5).choice(w.T, 8, replace=False))
    seed, query = 37, 6
    if n_queries is None:
        blocks, nb = None, 2
    else:
        blocks = [(0.0, 0)] + [(w.eps, qq) for qq in step.query_ids(query)]
        nb = len(blocks)
    rows = np.concatenate([b * w.T + tok for b in range(nb)])
    ins = []
    step.on_decoder = lambda L, h: ins.append(n64(h[torch.from_numpy(tok if L == 0 else rows).to(DEV)]))
    Y = step.forward(x, seed, query)
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0 and len(ins) == w.n_decoder
    outs = ins[1:] + [n64(Y[torch.from_numpy(rows).to(DEV)])]
    for L in range(w.n_decoder):
        dl = {nm: ol(f"{L}.{nm}") for nm in _stack_names(w.kind)}
        Yo = graphs.stack_forward([dl], ins[L], w.eps, seed, query, w.kind, store=w.act_dtype, first=(L == 0),
                                  blocks=blocks)
        _check_outputs(outs[L], Yo, f"decoder {L}")
    step.ctx.close()


def test_toy_two_steps():
    w = workload("toy_fp32")
    step, ol = _build(w, c_std=0.05)
    ora = {nm: ol(nm) for nm in ("l1", "l2")}
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
        Yo = graphs.toy_forward(lay, n64(x), w.eps, seed, query, store="fp32")
        Lp, Lm, D, a = oloss.loss_pair(Yo, w.T, n64(tgt), w.eps)
        assert np.abs(n64(Y) - Yo).max() <= 1e-4 * np.abs(Yo).max()
        o = out.cpu().numpy()
        assert abs(o[3] - a) <= 1e-3 * abs(a)
        for l in lay:
            name = [k for k, vv in ora.items() if vv is l][0]
            g = optim.zo_gradient(a, philox.perturbation(seed, l["layer_id"], query, *l["C"].shape))
            l["C"], m[name], v[name] = optim.adam_step(l["C"], m[name], v[name], g, f32(w.lr), f32(w.beta1),
                                                       f32(w.beta2), f32(w.adam_eps), t)
        for name, l in ora.items():
            lin = step.by_name[name]
            Cg = n64(step.C[lin.offset:lin.offset + lin.d_out * w.r]).reshape(l["C"].shape)
            assert np.abs(Cg - l["C"]).max() <= 1e-2 * w.lr
    step.ctx.close()


def test_basis_full_width():
    # d_in = 14336 (the Llama down projection) with 2048 calibration tokens, as the bench uses.
    # (1) the device iteration equals the oracle's fp64 run of the same iteration (same Omega, n_iter = 8);
    # (2) run to convergence (n_iter = 60) it spans the exact top-16 eigenspace (scipy eigsh on X^T X).
    from scipy.sparse.linalg import LinearOperator, eigsh
    ctx = zo.Context(0)
    n, d, r, p = 2048, 14336, 16, 16
    X, _ = lowrank_activations(n, d, 64, 0.05, 91, DEV)
    Xn = n64(X)
    G = Xn.T @ Xn
    for n_iter in (8, 60):
        U = torch.empty(d, r, device=DEV)
        ev = torch.empty(r + p, device=DEV)
        zo.zoact_basis_init(ctx, X, r, U, oversample=p, n_iter=n_iter, seed=3, evals_out=ev)
        torch.cuda.synchronize()
        assert ctx.device_status() == 0
        Ug = n64(U)
        np.testing.assert_allclose(Ug.T @ Ug, np.eye(r), atol=1e-4)
        if n_iter == 8:
            Ui, theta = basis.subspace_iteration(G, r, p, n_iter, 3)
            assert basis.subspace_overlap(Ug, Ui) >= 1 - 1e-6
            np.testing.assert_allclose(n64(ev)[:r], theta[:r], rtol=1e-4)
        else:
            op = LinearOperator((d, d), matvec=lambda v: Xn.T @ (Xn @ v), dtype=np.float64)
            lam, V = eigsh(op, k=r + 1, which="LA", tol=1e-10)
            order = np.argsort(lam)[::-1]
            lam, V = lam[order], V[:, order]
            assert basis.subspace_overlap(Ug, V[:, :r]) >= 1 - 1e-4
            np.testing.assert_allclose(n64(ev)[:r], lam[:r], rtol=1e-4)
    ctx.close()


@pytest.mark.parametrize("name,n_dec,T", [("llama_stack_bf16", 2, 300), ("llama_stack_int4", 1, 64),
                                          ("llama_mlp_bf16", 1, 256)])
def test_dependent_launch_bit_identical(name, n_dec, T, monkeypatch):
    # programmatic dependent launch only lets a kernel's blocks start early and wait in the kernel for the
    # previous one: three whole steps (forward, loss, Adam) must match the fully serialised stream bit for bit
    w = workload(name, T=T, n_decoder=n_dec)
    step, _ = _build(w)
    dt = torch.bfloat16 if w.act_dtype == "bf16" else torch.float16
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV, dtype=dt)
    tgt = normal((w.T, w.d_model), tensor_seed(w, "t"), DEV, dtype=dt) if w.kind == "llama_mlp" else None
    C0 = step.C.clone()
    monkeypatch.setenv("ZOACT_PDL", "0")
    serial = zo.Context(0)
    runs = []
    for ctx in (step.ctx, serial):
        step.ctx = ctx
        step.C.copy_(C0); step.m.zero_(); step.v.zero_()
        outs = []
        for t in range(1, 4):
            Y = step.forward(x, 5, t)
            outs.append((Y.clone(), step.loss(Y, tgt).clone()))
            step.update(t, 5, t)
        torch.cuda.synchronize()
        assert ctx.device_status() == 0
        runs.append((outs, step.C.clone(), step.m.clone(), step.v.clone()))
    (o1, C1, m1, v1), (o2, C2, m2, v2) = runs
    for (Ya, la), (Yb, lb) in zip(o1, o2):
        assert torch.equal(Ya, Yb) and torch.equal(la, lb)
    assert torch.equal(C1, C2) and torch.equal(m1, m2) and torch.equal(v1, v2)
    serial.close()


def test_run_from_host_matches_device_steps():
    # the end-to-end path (pinned host inputs copied on a side stream, loss vectors read back there) runs the
    # same steps as device-resident inputs: losses and coefficients bit for bit
    from paper_2607_01125_gb300.model import run_from_host
    w = workload("llama_mlp_bf16", T=256)
    step, _ = _build(w)
    n = 4
    xs = [lowrank_activations(w.T, 4096, 64, 0.05, tensor_seed(w, "x", i), DEV)[0] for i in range(n)]
    tgts = [normal((w.T, 4096), tensor_seed(w, "t", i), DEV, dtype=torch.bfloat16) for i in range(n)]
    C0 = step.C.clone()
    ref = []
    for i in range(n):
        Y = step.forward(xs[i], 5, i + 1)
        ref.append(step.loss(Y, tgts[i]).clone())
        step.update(i + 1, 5, i + 1)
    torch.cuda.synchronize()
    C_ref = step.C.clone()
    step.C.copy_(C0); step.m.zero_(); step.v.zero_()
    batches = [(xs[i].cpu().pin_memory(), tgts[i].cpu().pin_memory()) for i in range(n)]
    outs = [torch.empty(ref[0].numel(), dtype=torch.float64).pin_memory() for _ in range(n)]

    def sf(dev, i):
        Y = step.forward(dev[0], 5, i + 1)
        out = step.loss(Y, dev[1])
        step.update(i + 1, 5, i + 1)
        return out

    run_from_host(batches, sf, outs)
    torch.cuda.synchronize()
    for i in range(n):
        assert torch.equal(outs[i], ref[i].cpu()), i
    assert torch.equal(step.C, C_ref)
    assert step.ctx.device_status() == 0
    fixed = torch.zeros(ref[0].numel(), dtype=torch.float64, device=DEV)
    with pytest.raises(ValueError):
        run_from_host(batches, lambda dev, i: fixed, outs)
    torch.cuda.synchronize()
    step.ctx.close()


@pytest.mark.parametrize("name,n_dec,T", [("llama_mlp_bf16", 1, 256), ("llama_stack_bf16", 1, 256)])
def test_forward_loss_matches_forward_then_loss(name, n_dec, T):
    # ZOStep.forward_loss (last linear and loss pair fused) against forward() then loss(): the same losses
    # up to summation order, and the same Adam update of C up to that
    w = workload(name, T=T, n_decoder=n_dec)
    step, _ = _build(w)
    step.fuse_loss = True
    # the fused loss pair takes a normalised input; the stack's row scales would feed the reference's last linear
    # an unnormalised one (one rounding apart), so both runs here normalise explicitly
    step.row_scales = False
    dt = torch.bfloat16
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x"), DEV, dtype=dt)
    tgt = normal((w.T, w.d_model), tensor_seed(w, "t"), DEV, dtype=dt) if w.kind == "llama_mlp" else None
    C0 = step.C.clone()
    n0 = step.ctx.launch_count()
    fused = step.forward_loss(x, tgt, 3, 1).clone()
    n_fused = step.ctx.launch_count() - n0
    step.update(1, 3, 1)
    C1 = step.C.clone()
    step.C.copy_(C0); step.m.zero_(); step.v.zero_()
    n0 = step.ctx.launch_count()
    Y = step.forward(x, 3, 1)
    ref = step.loss(Y, tgt).clone()
    n_ref = step.ctx.launch_count() - n0
    step.update(1, 3, 1)
    torch.cuda.synchronize()
    assert step.ctx.device_status() == 0
    assert n_fused == n_ref - 1                      # the loss kernel is gone
    f, r = fused.cpu().numpy(), ref.cpu().numpy()
    # both against the exact (fp64) losses of the same rounded output
    Yd = Y.double()
    td = tgt.double() if tgt is not None else torch.zeros_like(Yd[:w.T])
    Lp_x, Lm_x = ((Yd[:w.T] - td) ** 2).mean().item(), ((Yd[w.T:] - td) ** 2).mean().item()
    D_x = ((Yd[:w.T] - Yd[w.T:]) * (Yd[:w.T] + Yd[w.T:] - 2 * td)).mean().item()
    assert abs(f[0] - Lp_x) <= 1e-10 * Lp_x and abs(f[1] - Lm_x) <= 1e-10 * Lm_x
    assert abs(f[2] - D_x) <= 1e-10 * max(Lp_x, Lm_x)
    assert np.allclose(r[:2], [Lp_x, Lm_x], rtol=1e-7) and abs(r[2] - D_x) <= 1e-7 * max(Lp_x, Lm_x)
    assert torch.allclose(step.C, C1, rtol=1e-4, atol=1e-9)
    step.ctx.close()
