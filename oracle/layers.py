"""Oracle: the adapted linear layer and its perturbed pair forward (test infrastructure only).

Section 3 ("ZO-Act") parameterises the update of a frozen weight W as
Delta W = V_r B, so the effective weight is W_eff = W + V_r B with B = 0 at
initialisation, and the forward-perturbed pass is

    Y+ = X W + (X V_r)(B + mu Z).

The paper uses row vectors (Y = X W, W in R^{m x n}).  This build stores the
nn.Linear layout: W is [d_out, d_in], the basis U (the paper's V_r) is
[d_in, r], the coefficients C (the transpose of the paper's B) are [d_out, r]
and Z is [d_out, r].  For one token x (a column) the same pass reads

    y(sigma) = W x + (C + sigma * eps * Z)(U^T x),   sigma in {+1, -1}.

The two-sided estimator evaluates sigma = +1 and sigma = -1 on the same batch;
the outputs are stacked along the token axis: rows [0, T) hold sigma = +1 and
rows [T, 2T) hold sigma = -1.

All arithmetic is fp64 on values read exactly from their stored precision.
"""
import numpy as np
import torch
from scipy.special import erf


def pair_forward(W, U, C, Z, X, eps, T, input_shared):
    """Stacked perturbed forward of one adapted linear (Section 3).

    W [d_out, d_in], U [d_in, r], C [d_out, r], Z [d_out, r]: fp64 arrays.
    X: [2T, d_in] stacked input (rows [0, T) see +eps Z, rows [T, 2T) see -eps Z),
       or [T, d_in] when input_shared (both halves see the same x).
    Returns Y [2T, d_out] fp64.
    """
    W = np.asarray(W, np.float64)
    U = np.asarray(U, np.float64)
    C = np.asarray(C, np.float64)
    Z = np.asarray(Z, np.float64)
    X = np.asarray(X, np.float64)
    if input_shared:
        assert X.shape[0] == T
        X_plus, X_minus = X, X
    else:
        assert X.shape[0] == 2 * T
        X_plus, X_minus = X[:T], X[T:]
    # y = W x + (C +- eps Z)(U^T x), written per half as in Section 3.
    Y_plus = X_plus @ W.T + (X_plus @ U) @ (C + eps * Z).T
    Y_minus = X_minus @ W.T + (X_minus @ U) @ (C - eps * Z).T
    return np.concatenate([Y_plus, Y_minus], axis=0)


def multi_forward(W, U, C, Zs, coefs, X, T, input_shared):
    """Forward of one adapted linear at several coefficient points, stacked by blocks.

    Algorithm 2 evaluates the loss at W_eff = W + V_r B (the unperturbed pass)
    and at W + V_r (B + mu Z^(j)) for j = 1..q (Section 3).  Block b of the
    stacked output is the layer evaluated at C + coefs[b] * Zs[b]:

        Y_b = X_b W^T + (X_b U)(C + coefs[b] Z_b)^T

    Zs[b] may be None where coefs[b] == 0 (no perturbation is drawn there).
    X: [n_blocks * T, d_in] (block b in rows [bT, (b+1)T)), or [T, d_in] when
    input_shared (every block sees the same x).  Returns Y [n_blocks * T, d_out].
    The two-sided pair is the case coefs = (eps, -eps) with the same Z twice.
    """
    W = np.asarray(W, np.float64)
    U = np.asarray(U, np.float64)
    C = np.asarray(C, np.float64)
    X = np.asarray(X, np.float64)
    nb = len(coefs)
    assert len(Zs) == nb
    assert X.shape[0] == (T if input_shared else nb * T)
    out = []
    for b in range(nb):
        Xb = X if input_shared else X[b * T:(b + 1) * T]
        if coefs[b] == 0.0:
            Cb = C
        else:
            Cb = C + coefs[b] * np.asarray(Zs[b], np.float64)
        out.append(Xb @ W.T + (Xb @ U) @ Cb.T)
    return np.concatenate(out, axis=0)


def dequant_int4_g128(packed, scales, d_in):
    """Frozen INT4 weight -> fp64, group size 128 along d_in (test infrastructure only).

    The paper fine-tunes an INT4 Llama-3-8B whose weights stay frozen (Section 5,
    "Llama-3-8B-w4"); it does not state the storage format.  This build reads:
    packed [d_out, d_in/2] uint8, element k of a row in byte k/2, low nibble for
    even k and high nibble for odd k, each nibble a 4-bit two's complement
    integer q in [-8, 7]; scales [d_out, d_in/128] (fp16 values); w = q * s.
    """
    # plain torch CPU element-wise ops (multi-threaded): a full Llama-3-8B stack has 7e9 weights
    pk = torch.from_numpy(np.ascontiguousarray(packed, dtype=np.uint8))
    d_out = pk.shape[0]
    # byte k/2 -> (low nibble, high nibble) = elements (k, k + 1)
    q = torch.stack([pk & 0x0F, pk >> 4], dim=-1).reshape(d_out, -1)[:, :d_in].to(torch.int8)
    q = torch.where(q >= 8, q - 16, q)                    # two's complement nibble
    n_groups = (d_in + 127) // 128
    w = torch.zeros(d_out, n_groups * 128, dtype=torch.float64)
    w[:, :d_in] = q
    s = torch.from_numpy(np.asarray(scales, dtype=np.float64))[:, :n_groups]
    w.view(d_out, n_groups, 128).mul_(s[:, :, None])      # every element of group g times s[g]
    return w[:, :d_in].numpy()


# ---- glue ops of the synthetic graphs (exact definitions, fp64) ----

def gelu_erf(x):
    """Exact GELU: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    x = np.asarray(x, np.float64)
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def relu(x):
    return np.maximum(np.asarray(x, np.float64), 0.0)


def silu(x):
    x = np.asarray(x, np.float64)
    return x / (1.0 + np.exp(-x))


def rms_norm(x, eps=1e-5):
    """Per-row RMS normalisation without a gain: x / sqrt(mean(x^2) + eps)."""
    x = np.asarray(x, np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def repeat_kv(x, n_kv_heads, n_rep, head_dim):
    """Grouped-query repeat: each kv head of width head_dim serves n_rep query heads."""
    x = np.asarray(x, np.float64)
    rows = x.shape[0]
    x = x.reshape(rows, n_kv_heads, 1, head_dim)
    x = np.broadcast_to(x, (rows, n_kv_heads, n_rep, head_dim))
    return x.reshape(rows, n_kv_heads * n_rep * head_dim)


def round_to_bf16(x):
    """Round fp64 values to the nearest bf16 (ties to even) via fp32, as stored.

    Used to mirror where an activation is stored at bf16 between layers.
    """
    f = np.asarray(x, np.float64).astype(np.float32)
    b = f.view(np.uint32).astype(np.uint64)
    lsb = (b >> np.uint64(16)) & np.uint64(1)
    b = (b + np.uint64(0x7FFF) + lsb) >> np.uint64(16) << np.uint64(16)
    out = (b & np.uint64(0xFFFFFFFF)).astype(np.uint32).view(np.float32)
    nan = np.isnan(f)
    out = np.where(nan, f, out)
    return out.astype(np.float64)


def round_to_fp16(x):
    """Round fp64 values to fp16 as stored (numpy's IEEE half, ties to even)."""
    return np.asarray(x, np.float64).astype(np.float16).astype(np.float64)


def round_to_fp32(x):
    return np.asarray(x, np.float64).astype(np.float32).astype(np.float64)


STORE_ROUNDING = {"bf16": round_to_bf16, "fp16": round_to_fp16, "fp32": round_to_fp32,
                  "fp64": lambda x: np.asarray(x, np.float64)}
