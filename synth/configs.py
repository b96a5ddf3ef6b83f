"""Workload descriptions: layer shapes, token counts, ranks and per-tensor seeds.

Five workloads, named by what they are:

* ``toy_fp32``        2 x (256 -> 256) with exact GELU between, r = 8, T = 64,
                      512 calibration tokens, fp32 everywhere.
* ``llama_mlp_bf16``  Llama-3-8B MLP block: gate/up 4096 -> 14336 (shared
                      input), down 14336 -> 4096, SiLU gate, r = 16, T = 2048.
* ``llama_stack_bf16`` 32 decoder layers x {q, k, v, o, gate, up, down} = 224
                      adapted linears, r = 16, T = 16 x 256 = 4096.
* ``llama_stack_int4`` the same stack with frozen W in symmetric INT4, g = 128.
* ``opt_stack_fp16``  40 x {q, k, v, o, fc1, fc2} = 240 adapted linears with
                      ReLU after fc1, r = 32, T = 4096, 4096 calibration tokens.

``n_decoder`` / ``T`` can be reduced for parity runs; the widths stay.
"""
from dataclasses import dataclass, field, replace

__all__ = ["LinearSpec", "Workload", "WORKLOADS", "workload", "tensor_seed"]


@dataclass(frozen=True)
class LinearSpec:
    name: str          # e.g. "3.gate"
    d_in: int
    d_out: int
    layer_id: int      # Philox stream id of this layer's Z


@dataclass(frozen=True)
class Workload:
    name: str
    kind: str          # "toy" | "llama_mlp" | "llama" | "opt"
    act_dtype: str     # activation / weight storage: "fp32" | "bf16" | "fp16"
    wtype: str         # "fp32" | "bf16" | "fp16" | "int4_g128"
    T: int             # tokens per perturbation
    r: int
    eps: float = 1e-3
    n_cal: int = 512
    n_decoder: int = 1
    seed: int = 0
    lr: float = 1e-4
    beta1: float = 0.9
    beta2: float = 0.999
    adam_eps: float = 1e-8
    weight_std: float = 0.02
    extra: dict = field(default_factory=dict, compare=False, hash=False)

    def linears(self):
        """All adapted linears in forward order with their layer ids."""
        out = []
        if self.kind == "toy":
            out = [LinearSpec("l1", 256, 256, 0), LinearSpec("l2", 256, 256, 1)]
        elif self.kind == "llama_mlp":
            out = [LinearSpec("gate", 4096, 14336, 0), LinearSpec("up", 4096, 14336, 1),
                   LinearSpec("down", 14336, 4096, 2)]
        elif self.kind == "llama":
            shapes = [("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
                      ("gate", 4096, 14336), ("up", 4096, 14336), ("down", 14336, 4096)]
            for L in range(self.n_decoder):
                for i, (nm, di, do) in enumerate(shapes):
                    out.append(LinearSpec(f"{L}.{nm}", di, do, 7 * L + i))
        elif self.kind == "opt":
            shapes = [("q", 5120, 5120), ("k", 5120, 5120), ("v", 5120, 5120), ("o", 5120, 5120),
                      ("fc1", 5120, 20480), ("fc2", 20480, 5120)]
            for L in range(self.n_decoder):
                for i, (nm, di, do) in enumerate(shapes):
                    out.append(LinearSpec(f"{L}.{nm}", di, do, 6 * L + i))
        else:
            raise ValueError(self.kind)
        return out

    @property
    def d_model(self):
        return {"toy": 256, "llama_mlp": 4096, "llama": 4096, "opt": 5120}[self.kind]

    def n_coeffs(self):
        return sum(l.d_out * self.r for l in self.linears())

    def gemm_flops(self):
        """Algorithmic flops of the pair forwards of one ZO step (2 M K N per linear;
        layers whose input is shared between the signs run their product once on T rows)."""
        total = 0
        for spec in self.linears():
            shared = self.input_shared(spec)
            rows = self.T if shared else 2 * self.T
            total += 2 * rows * spec.d_in * spec.d_out
        return total

    def input_shared(self, spec):
        """True where both signs feed the same input to the layer."""
        if self.kind == "toy":
            return spec.name == "l1"
        if self.kind == "llama_mlp":
            return spec.name in ("gate", "up")
        return spec.name in ("0.q", "0.k", "0.v")


WORKLOADS = {
    "toy_fp32": Workload("toy_fp32", "toy", "fp32", "fp32", T=64, r=8, n_cal=512,
                         weight_std=1.0 / 16.0, lr=1e-4),
    "llama_mlp_bf16": Workload("llama_mlp_bf16", "llama_mlp", "bf16", "bf16", T=2048, r=16,
                               n_cal=2048),
    "llama_stack_bf16": Workload("llama_stack_bf16", "llama", "bf16", "bf16", T=4096, r=16,
                                 n_cal=512, n_decoder=32),
    "llama_stack_int4": Workload("llama_stack_int4", "llama", "bf16", "int4_g128", T=4096, r=16,
                                 n_cal=512, n_decoder=32),
    "opt_stack_fp16": Workload("opt_stack_fp16", "opt", "fp16", "fp16", T=4096, r=32,
                               n_cal=4096, n_decoder=40),
}


def workload(name, **overrides):
    return replace(WORKLOADS[name], **overrides)


def tensor_seed(w, *parts):
    """Deterministic per-tensor seed from the workload seed and a name path."""
    h = (int(w.seed) * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
    for p in parts:
        for ch in str(p):
            h = ((h ^ ord(ch)) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
        h = ((h ^ 0x2F) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF
