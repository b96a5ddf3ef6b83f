"""Oracle: synthetic model graphs that chain adapted linears (test infrastructure only).

The paper adapts every linear layer of Llama-3-8B / OPT-13B except embeddings
and heads (Appendix B) and evaluates L+ and L- with all layers perturbed at once
(Algorithm 2).  No model weights or datasets are available here, so the
workloads are synthetic graphs with the paper's layer shapes.  Each graph
returns the stacked final output Y [2T, n] of the perturbed forward passes:
rows [0, T) with every layer at C + eps Z, rows [T, 2T) at C - eps Z.

A layer is a dict with fp64 arrays W [d_out, d_in], U [d_in, r], C [d_out, r]
and an int layer_id.  Z for the layer is regenerated from (seed, layer_id, query).

With ``blocks`` (a list of (coef, query) pairs) a graph is evaluated at several
coefficient points instead: block b of the output has every layer at
C + coef_b Z(seed, layer_id, query_b) -- Algorithm 2's unperturbed pass
(coef 0) followed by its q forward-perturbed passes (coef mu).  The default
(None) is the two-sided pair [(eps, query), (-eps, query)].

``store`` rounds a tensor to the precision the activations are kept in between
ops ("bf16", "fp16", "fp32", or "fp64" for no rounding); it is applied to the
output of every linear and every glue op.

Graph wiring (the reading this build fixes for configurations the paper does
not define as code):

* toy:        h = GELU(L1 x) ; y = L2 h
* llama_mlp:  y = Down(silu(Gate x) * Up x)
* llama/opt stack, per decoder layer, input h:
      a = RMS(h) ; q, k, v = Q a, K a, V a
      o = O RMS(q + rep(k) + rep(v))      (rep: grouped-query head repeat; identity for OPT)
      b = RMS(o)
      llama: h' = Down RMS(silu(Gate b) * Up b)
      opt:   h' = FC2 RMS(ReLU(FC1 b))
  RMS has no gain and eps 1e-5.  The first layer's q/k/v see the same input for
  both signs (the graph input is not perturbed).
"""
import numpy as np

from .layers import (pair_forward, multi_forward, gelu_erf, relu, silu, rms_norm, repeat_kv,
                     STORE_ROUNDING)
from .philox import perturbation


def layer_forward(layer, X, eps, seed, query, T, input_shared, blocks=None):
    d_out, r = layer["W"].shape[0], layer["U"].shape[1]
    if blocks is None:
        Z = perturbation(seed, layer["layer_id"], query, d_out, r)
        return pair_forward(layer["W"], layer["U"], layer["C"], Z, X, eps, T, input_shared)
    Zs = [None if c == 0.0 else perturbation(seed, layer["layer_id"], qb, d_out, r) for c, qb in blocks]
    return multi_forward(layer["W"], layer["U"], layer["C"], Zs, [c for c, _ in blocks], X, T, input_shared)


def toy_forward(layers, x, eps, seed, query, store="fp32", blocks=None):
    """Two 256->256 adapted linears with exact GELU between them."""
    rnd = STORE_ROUNDING[store]
    T = x.shape[0]
    h = rnd(gelu_erf(layer_forward(layers[0], x, eps, seed, query, T, True, blocks)))
    return rnd(layer_forward(layers[1], h, eps, seed, query, T, False, blocks))


def llama_mlp_forward(layers, x, eps, seed, query, store="bf16", blocks=None):
    """SiLU-gated MLP block: layers = (gate, up, down); gate/up share the input x."""
    rnd = STORE_ROUNDING[store]
    T = x.shape[0]
    g = layer_forward(layers[0], x, eps, seed, query, T, True, blocks)
    u = layer_forward(layers[1], x, eps, seed, query, T, True, blocks)
    h = rnd(silu(g) * u)
    return rnd(layer_forward(layers[2], h, eps, seed, query, T, False, blocks))


def stack_forward(decoder_layers, x, eps, seed, query, kind, store="bf16",
                  n_heads=32, n_kv_heads=8, head_dim=128, blocks=None, first=True):
    """Linear stack of the llama / opt kind.  decoder_layers: list of dicts of layers.

    llama dict keys: q k v o gate up down;  opt dict keys: q k v o fc1 fc2.

    first=True: x [T, d] is the graph input, the same for every evaluation
    point.  first=False continues a stack from a later decoder: x is the stacked
    output [n_points * T, d] of the decoders before it (so a deep stack can be
    run one decoder at a time, with one decoder's weights in memory).
    """
    rnd = STORE_ROUNDING[store]
    n_points = 2 if blocks is None else len(blocks)
    T = x.shape[0] if first else x.shape[0] // n_points
    h = np.asarray(x, np.float64)
    shared = first
    for dl in decoder_layers:
        a = rnd(rms_norm(h))
        q = rnd(layer_forward(dl["q"], a, eps, seed, query, T, shared, blocks))
        k = rnd(layer_forward(dl["k"], a, eps, seed, query, T, shared, blocks))
        v = rnd(layer_forward(dl["v"], a, eps, seed, query, T, shared, blocks))
        shared = False
        if kind == "llama":
            n_rep = n_heads // n_kv_heads
            mix = q + repeat_kv(k, n_kv_heads, n_rep, head_dim) + repeat_kv(v, n_kv_heads, n_rep, head_dim)
        else:
            mix = q + k + v
        o = rnd(layer_forward(dl["o"], rnd(rms_norm(mix)), eps, seed, query, T, False, blocks))
        b = rnd(rms_norm(o))
        if kind == "llama":
            g = layer_forward(dl["gate"], b, eps, seed, query, T, False, blocks)
            u = layer_forward(dl["up"], b, eps, seed, query, T, False, blocks)
            m = rnd(rms_norm(rnd(silu(g) * u)))
            h = rnd(layer_forward(dl["down"], m, eps, seed, query, T, False, blocks))
        else:
            f = rnd(relu(layer_forward(dl["fc1"], b, eps, seed, query, T, False, blocks)))
            h = rnd(layer_forward(dl["fc2"], rnd(rms_norm(f)), eps, seed, query, T, False, blocks))
    return h
