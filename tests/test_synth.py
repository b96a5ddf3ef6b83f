"""The seeded input generators and workload descriptions that every test and the bench draw from: each
generator's documented structure (seeded determinism, the low-rank and decaying spectra, unit RMS per
token, orthonormal bases) and the workloads' layer shapes and FLOP counts."""
import numpy as np
import torch

from synth import (normal, lowrank_activations, decaying_spectrum_activations, random_orthonormal, workload,
                   tensor_seed)


def test_normal_is_seeded_scaled_and_cast():
    a = normal((64, 32), 7)
    assert torch.equal(a, normal((64, 32), 7))
    assert not torch.equal(a, normal((64, 32), 8))
    b = normal((64, 32), 7, std=0.25)
    assert torch.allclose(b, 0.25 * a)
    c = normal((64, 32), 7, dtype=torch.bfloat16)
    assert c.dtype == torch.bfloat16 and torch.equal(c, a.to(torch.bfloat16))
    big = normal((200_000,), 3)
    assert abs(big.mean().item()) < 0.01 and abs(big.std().item() - 1.0) < 0.01


def test_lowrank_activations_without_noise_have_the_stated_rank_and_unit_rms():
    x, B = lowrank_activations(512, 256, 12, 0.0, 5, dtype=torch.float32)
    assert B.shape == (12, 256)
    rms = x.pow(2).mean(dim=1).sqrt()
    assert torch.allclose(rms, torch.ones_like(rms), atol=1e-5)
    s = torch.linalg.svdvals(x.double())
    assert s[11] > 1e-3 * s[0] and s[12] < 1e-6 * s[0]          # rank 12 up to the fp32 arithmetic
    # rows lie in B's row space
    P = B.double().T @ torch.linalg.pinv(B.double().T)
    assert (x.double() @ P - x.double()).norm() < 1e-5 * x.double().norm()


def test_lowrank_activations_share_a_given_basis_and_mix_noise_by_energy():
    _, B = lowrank_activations(64, 128, 8, 0.0, 1, dtype=torch.float32)
    y, B2 = lowrank_activations(256, 128, 8, 0.0, 2, dtype=torch.float32, basis=B)
    assert B2 is B
    P = B.double().T @ torch.linalg.pinv(B.double().T)
    assert (y.double() @ P - y.double()).norm() < 1e-5 * y.double().norm()
    # noise = 0.25 of the energy: a quarter of the (pre-normalisation) variance outside the signal subspace
    z, Bz = lowrank_activations(4096, 256, 8, 0.25, 3, dtype=torch.float32, unit_rms=False)
    Pz = Bz.double().T @ torch.linalg.pinv(Bz.double().T)
    out = z.double() - z.double() @ Pz
    frac_out = out.pow(2).mean().item() / z.double().pow(2).mean().item()
    assert abs(frac_out - 0.25 * (256 - 8) / 256) < 0.01


def test_decaying_spectrum_is_rank_r_and_decays():
    # the signal's singular values fall as 1/i; the per-token RMS scaling flattens them somewhat (tokens led by
    # the first direction shrink most), so the test asks for a strictly falling spectrum between 1/i and 1/sqrt(i)
    x = decaying_spectrum_activations(8192, 256, 8, 0.0, 4, dtype=torch.float32)
    s = torch.linalg.svdvals(x.double()).numpy()
    ratios = s[:8] / s[0]
    i = np.arange(1, 9)
    assert np.all(np.diff(ratios) < 0)
    assert np.all(ratios[1:] > 1.0 / i[1:]) and np.all(ratios[1:] < 1.0 / np.sqrt(i[1:]))
    assert s[8] < 1e-6 * s[0]


def test_random_orthonormal():
    Q = random_orthonormal(300, 17, 9)
    assert Q.shape == (300, 17)
    assert torch.allclose(Q.double().T @ Q.double(), torch.eye(17, dtype=torch.float64), atol=1e-6)
    assert torch.equal(Q, random_orthonormal(300, 17, 9))


def test_workload_shapes_follow_the_models():
    mlp = workload("llama_mlp_bf16")
    assert [(l.name, l.d_in, l.d_out) for l in mlp.linears()] == [("gate", 4096, 14336), ("up", 4096, 14336),
                                                                   ("down", 14336, 4096)]
    # gate/up share the input (T rows), down sees both signs (2T rows): 2 x 2 T 4096 14336 + 2 x 2T 14336 4096
    T = mlp.T
    assert mlp.gemm_flops() == 2 * (2 * T * 4096 * 14336) + 2 * (2 * T) * 14336 * 4096
    st = workload("llama_stack_bf16")
    lin = st.linears()
    assert len(lin) == 224 and len({l.layer_id for l in lin}) == 224
    assert (lin[1].d_in, lin[1].d_out) == (4096, 1024)            # grouped-query k: 8 KV heads of 128
    assert workload("llama_stack_int4").wtype == "int4_g128"
    opt = workload("opt_stack_fp16")
    assert len(opt.linears()) == 240 and opt.r == 32 and opt.d_model == 5120
    assert (opt.linears()[4].d_in, opt.linears()[4].d_out) == (5120, 20480)
    small = workload("llama_stack_bf16", n_decoder=2, T=256)
    assert len(small.linears()) == 14 and small.T == 256 and small.r == 16


def test_tensor_seeds_are_stable_and_distinct():
    w = workload("llama_mlp_bf16")
    a = tensor_seed(w, "x")
    assert a == tensor_seed(w, "x") and 0 <= a < 2 ** 63
    seeds = {tensor_seed(w, n) for n in ("x", "t", "W", "U", "C", "0.q", "0.k", "1.q")}
    assert len(seeds) == 8
    assert tensor_seed(w, "a", "b") != tensor_seed(w, "ab")          # the path separator counts
    assert tensor_seed(workload("llama_mlp_bf16", seed=1), "x") != a
