"""bench.py's output contract, checked on the host: the reference arm (the fp64 oracle on the host cores)
prints one JSON line with every key the contract names, a warm-up below three steps is refused, and the
product arm stops with an error when no GPU is present instead of falling back to the CPU."""
import json
import os
import subprocess
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench(*args, timeout=240):
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, capture_output=True,
                          text=True, timeout=timeout)


def test_reference_arm_prints_one_contract_line():
    p = _bench("--impl", "reference", "--steps", "1", "--warmup", "3", "--ref-tokens", "8")
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 3
    assert d["value"] > 0 and d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["config"]["workload"] == "llama_stack_bf16" and d["config"]["adapted_linears"] == 224
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["unit"] == d["unit"] and cb["cores"] >= 1
    assert cb["sample"] and cb["extrapolated"] is True and "32 decoders" in cb["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
    # tokens/s from the (extrapolated) step time: two perturbations of 8 tokens are one ZO step's evaluated
    # tokens, 8 its tokens
    assert d["value"] == pytest.approx(8 / (d["ms_per_step"] * 1e-3), rel=1e-6)


def test_short_warmup_is_refused():
    p = _bench("--impl", "reference", "--steps", "1", "--warmup", "1", timeout=120)
    assert p.returncode != 0 and "warmup" in p.stderr


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_product_arm_fails_without_a_gpu():
    p = _bench("--steps", "1", "--warmup", "3", "--no-cpu-baseline", timeout=180)
    assert p.returncode != 0
    assert not [ln for ln in p.stdout.splitlines() if ln.strip().startswith("{")]   # no bench line
