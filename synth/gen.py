"""Seeded tensor generators (torch, on any device).

Each generator takes an explicit integer seed and a device, uses its own
torch.Generator, and returns a tensor in the requested storage dtype.  The same
seed on the same device type always gives the same tensor; CPU and CUDA
generators give different streams, so a test draws its inputs once and hands
the same stored values to both sides.
"""
import math

import torch

__all__ = ["normal", "lowrank_activations", "decaying_spectrum_activations",
           "quantize_int4_g128", "random_orthonormal", "DTYPES"]

DTYPES = {"bf16": torch.bfloat16, "fp16": torch.float16, "fp32": torch.float32}


def _gen(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return g


def normal(shape, seed, device="cpu", std=1.0, dtype=torch.float32):
    """N(0, std^2) samples of the given shape, drawn in fp32 then cast to dtype."""
    g = _gen(seed, device)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(dtype)


def lowrank_activations(n_tok, d, rank, noise, seed, device="cpu", dtype=torch.bfloat16,
                        basis=None, unit_rms=True, noise_is_energy=True):
    """Tokens x = signal + noise with a rank-`rank` Gaussian signal.

    signal = A B with A ~ N(0,1)^{n_tok x rank} and B ~ N(0, 1/rank)^{rank x d}, so
    every signal entry has unit variance.  `basis` (a B drawn earlier) lets
    calibration and training tokens share one signal subspace.
    noise_is_energy=True: x = sqrt(1-noise) signal + sqrt(noise) N(0,1)  (noise is
    the fraction of the energy);  False: x = signal + noise * N(0,1).
    unit_rms: rescale every token to unit root-mean-square.
    Returns (x in dtype, B fp32).
    """
    g = _gen(seed, device)
    if basis is None:
        basis = torch.randn(rank, d, generator=g, device=device) / math.sqrt(rank)
    A = torch.randn(n_tok, rank, generator=g, device=device)
    x = A @ basis
    nz = torch.randn(n_tok, d, generator=g, device=device)
    if noise_is_energy:
        x = math.sqrt(1.0 - noise) * x + math.sqrt(noise) * nz
    else:
        x = x + noise * nz
    if unit_rms:
        x = x / x.pow(2).mean(dim=1, keepdim=True).sqrt().clamp_min(1e-12)
    return x.to(dtype), basis


def decaying_spectrum_activations(n_tok, d, rank, noise, seed, device="cpu", dtype=torch.float16):
    """Tokens with a rank-`rank` signal whose singular values decay as i^-1, plus isotropic noise.

    x = A diag(1/i) B + noise * N(0,1), A ~ N(0,1)^{n_tok x rank},
    B = orthonormal rows (QR of a Gaussian), then unit RMS per token (which
    flattens the 1/i decay somewhat: tokens led by the first direction shrink most).
    """
    g = _gen(seed, device)
    B = torch.linalg.qr(torch.randn(d, rank, generator=g, device=device))[0].T.contiguous()  # [rank, d]
    s = 1.0 / torch.arange(1, rank + 1, device=device, dtype=torch.float32)
    A = torch.randn(n_tok, rank, generator=g, device=device) * s * math.sqrt(d)
    x = A @ B + noise * torch.randn(n_tok, d, generator=g, device=device)
    x = x / x.pow(2).mean(dim=1, keepdim=True).sqrt().clamp_min(1e-12)
    return x.to(dtype)


def quantize_int4_g128(W):
    """Symmetric INT4 with groups of 128 along d_in and fp16 group scales.

    s = fp16(absmax(group) / 7);  q = clamp(round_half_even(w / s), -8, 7);
    packed byte k/2 of a row holds element k in its low nibble (even k) or high
    nibble (odd k), as 4-bit two's complement.  A group of zeros gets s = 0, q = 0.
    W: [d_out, d_in] float tensor with d_in % 128 == 0.
    Returns (packed uint8 [d_out, d_in/2], scales fp16 [d_out, d_in/128]).
    """
    d_out, d_in = W.shape
    assert d_in % 128 == 0
    Wf = W.float().reshape(d_out, d_in // 128, 128)
    s = (Wf.abs().amax(dim=2) / 7.0).to(torch.float16)
    sf = s.float().unsqueeze(2)
    q = torch.where(sf > 0, torch.round(Wf / torch.where(sf > 0, sf, torch.ones_like(sf))),
                    torch.zeros_like(Wf))
    q = q.clamp(-8, 7).to(torch.int32).reshape(d_out, d_in)
    nib = (q & 0xF).to(torch.uint8)
    packed = nib[:, 0::2] | (nib[:, 1::2] << 4)
    return packed.contiguous(), s.contiguous()


def random_orthonormal(d, r, seed, device="cpu"):
    """A [d, r] matrix with orthonormal columns (QR of a Gaussian)."""
    g = _gen(seed, device)
    q = torch.linalg.qr(torch.randn(d, r, generator=g, device=device, dtype=torch.float64))[0]
    return q.float().contiguous()
