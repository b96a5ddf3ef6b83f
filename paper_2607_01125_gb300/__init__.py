"""GB300-native hot path of one ZO-Act step (arXiv 2607.01125).

The compute lives in libzoact.so (hand-written CUDA for sm_103a behind the C ABI
of include/zoact.h).  This package holds its ctypes binding (``_lib``), the
in-tree build (``build``) and ``model``, which chains the C-ABI calls into the
ZO steps of the synthetic workloads.  PyTorch provides device memory and
streams only.
"""
from ._lib import (  # noqa: F401
    Context, ZoactError, make_layer, load, status_string,
    zoact_philox_normals, zoact_lowrank_proj, zoact_pair_forward, zoact_pair_forward_gated,
    zoact_pair_forward_noalloc, zoact_pair_forward_loss,
    zoact_loss_pair, zoact_adam_step, zoact_sgd_step, zoact_basis_init, zoact_rms_norm, zoact_mix_rms,
    zoact_multi_forward, zoact_multi_forward_gated, zoact_loss_multi, zoact_adam_step_multi, zoact_sgd_step_multi,
    eval_blocks, one_sided_blocks, MAX_EVAL_BLOCKS,
    zoact_basis_prepared_bytes, zoact_basis_prepare, zoact_lowrank_proj_prepared,
    zoact_subspace_overlap, zoact_gradient_energy, zoact_mean_over_ranks, zoact_arena_hash,
    zoact_pair_forward_rs, zoact_pair_forward_gated_rs, zoact_rms_scale, rowscale_parts,
    zoact_multi_forward_rs, zoact_multi_forward_gated_rs, zoact_pair_forward_group_rs, zoact_multi_forward_group_rs,
    MAX_GROUP,
    DT_FP32, DT_BF16, DT_FP16, DT_INT4_G128, ACT_NONE, ACT_RELU, ACT_GELU, EXPORTS, LIB_PATH, TORCH_DT,
)
