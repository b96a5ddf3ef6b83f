"""Host-side logic of the model and the binding that needs no GPU: the weight colocation that lets a decoder's
q, k and v run as one launch, and the argument checks that refuse malformed grouped and strided calls before any
library call is made."""
import pytest
import torch

import paper_2607_01125_gb300 as zo
from paper_2607_01125_gb300.model import AdaptedLinear, colocate_weights


def _lin(name, d_out, d_in, seed, int4=False):
    g = torch.Generator().manual_seed(seed)
    U = torch.randn(d_in, 4, generator=g)
    if int4:
        W = torch.randint(0, 256, (d_out, d_in // 2), dtype=torch.uint8, generator=g)
        S = torch.rand(d_out, d_in // 128, generator=g).to(torch.float16)
        return AdaptedLinear(name, W, U, seed, 0, 4, w_scales=S, wtype=zo.DT_INT4_G128, d_in=d_in)
    return AdaptedLinear(name, torch.randn(d_out, d_in, generator=g).to(torch.bfloat16), U, seed, 0, 4)


def _contiguous(ls):
    base, rows = ls[0].W, 0
    for l in ls:
        if l.W.data_ptr() != base.data_ptr() + rows * base.stride(0) * base.element_size():
            return False
        if l.w_scales is not None and l.w_scales.data_ptr() != (ls[0].w_scales.data_ptr() + rows *
                                                                ls[0].w_scales.stride(0) *
                                                                ls[0].w_scales.element_size()):
            return False
        rows += l.d_out
    return True


@pytest.mark.parametrize("int4", [False, True])
def test_colocate_weights_keeps_values_and_is_idempotent(int4):
    ls = [_lin("0.q", 64, 256, 1, int4), _lin("0.k", 16, 256, 2, int4), _lin("0.v", 16, 256, 3, int4)]
    before = [(l.W.clone(), None if l.w_scales is None else l.w_scales.clone()) for l in ls]
    assert not _contiguous(ls)
    colocate_weights([ls])
    assert _contiguous(ls)
    for l, (w, s) in zip(ls, before):
        assert l.W.is_contiguous() and torch.equal(l.W, w)
        if s is not None:
            assert l.w_scales.is_contiguous() and torch.equal(l.w_scales, s)
    ptrs = [l.W.data_ptr() for l in ls]
    colocate_weights([ls])                         # already laid out: left alone
    assert [l.W.data_ptr() for l in ls] == ptrs


def test_colocate_weights_leaves_single_layers_alone():
    ls = [_lin("0.o", 32, 128, 4)]
    p = ls[0].W.data_ptr()
    colocate_weights([ls])
    assert ls[0].W.data_ptr() == p


def test_group_binding_refuses_layer_counts_outside_the_range():
    # the binding refuses before it touches the library or a context
    lay = zo.make_layer(torch.zeros(8, 16, dtype=torch.bfloat16), torch.zeros(16, 4), torch.zeros(32), 0)
    X = torch.zeros(2, 16, dtype=torch.bfloat16)
    Y = torch.zeros(2, 8, dtype=torch.bfloat16)
    for n in (0, zo.MAX_GROUP + 1):
        with pytest.raises(ValueError):
            zo.zoact_pair_forward_group_rs(None, [lay] * n, X, 1, 0.5, 1, 1, Y)


def test_strided_mixer_refuses_views_it_cannot_express():
    buf = torch.zeros(4, 96, dtype=torch.bfloat16)
    Y = torch.zeros(4, 32, dtype=torch.bfloat16)
    q = buf[:, :32]
    k = buf[:, 32:48]
    v_other = torch.zeros(4, 40, dtype=torch.bfloat16)[:, :16]       # another row stride than k
    with pytest.raises(ValueError):
        zo.zoact_mix_rms(None, q, k, v_other, Y, 2, 8)
    with pytest.raises(ValueError):
        zo.zoact_mix_rms(None, buf[:, ::3], k, buf[:, 48:64], Y, 2, 8)   # columns not unit-stride
