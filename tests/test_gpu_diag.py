"""GPU parity of the Section 5.3 subspace diagnostics against the oracle (through the C ABI).

fp32 products accumulated over at most a few thousand rows per split, squared and summed in fp64:
relative error well below 1e-5 of ||M||^2 on these sizes; the test bar is 1e-5 relative."""
import numpy as np
import pytest
import torch

import paper_2607_01125_gb300 as zo
from oracle import basis
from synth import normal, random_orthonormal

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


@pytest.mark.parametrize("d,ra,rb", [(4096, 16, 16), (14336, 16, 16), (1000, 256, 256), (777, 5, 33)])
def test_subspace_overlap(ctx, d, ra, rb):
    Ua = random_orthonormal(d, ra, 3, DEV)
    # U_b shares half of U_a's directions
    Ub = random_orthonormal(d, rb, 4, DEV)
    k = min(ra, rb) // 2
    if k > 0:
        Ub[:, :k] = Ua[:, :k]
        Ub = torch.linalg.qr(Ub)[0].contiguous()
    out = torch.zeros(3, dtype=torch.float64, device=DEV)
    zo.zoact_subspace_overlap(ctx, Ua, Ub, out)
    torch.cuda.synchronize()
    ref = basis.subspace_overlap(np64(Ua), np64(Ub))
    assert out[2].item() == pytest.approx(ref, rel=1e-5, abs=1e-7)
    # the metric's fixed points: the same subspace gives 1
    zo.zoact_subspace_overlap(ctx, Ua, Ua, out)
    torch.cuda.synchronize()
    assert out[2].item() == pytest.approx(1.0, abs=1e-5)


@pytest.mark.parametrize("d,n,r,dt", [(4096, 14336, 16, torch.bfloat16), (1024, 3000, 1, torch.float32),
                                      (2048, 1000, 200, torch.float16), (333, 65, 7, torch.float32)])
def test_gradient_energy(ctx, d, n, r, dt):
    U = random_orthonormal(d, r, 5, DEV)
    # a gradient with a planted component in span(U) plus noise
    G = (U @ normal((r, n), 6, DEV) * 3.0 + normal((d, n), 7, DEV)).to(dt)
    out = torch.zeros(3, dtype=torch.float64, device=DEV)
    zo.zoact_gradient_energy(ctx, U, G, out)
    torch.cuda.synchronize()
    num, den, ratio = basis.gradient_energy(np64(U), np64(G))
    o = out.cpu().numpy()
    assert o[0] == pytest.approx(num, rel=1e-5)
    assert o[1] == pytest.approx(den, rel=1e-5)
    assert o[2] == pytest.approx(ratio, rel=1e-5)
