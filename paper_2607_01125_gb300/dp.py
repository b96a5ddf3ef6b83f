"""Data-parallel exchange of one ZO step: ranks split the tokens, share everything else.

Every rank holds the same W, U, C, m, v and seed, runs the pair forward and the
loss pair on its own token shard, and the ranks then average the loss vector --
[L+, L-, D, a], or [L_0 .. L_q, a_1 .. a_q] for the one-sided q-query estimator
(each entry a mean over the rank's T * n elements, so with equal shards their
average is the global value; every a is linear in the losses).
Each rank then applies the same Adam update with the same regenerated Z, so C
stays identical on every rank without a gradient all-reduce.
"""
import torch.distributed as dist


def allreduce_loss(loss_out, group=None):
    """Average the device (or CPU, for gloo) loss vector over the ranks, in place."""
    world = dist.get_world_size(group)
    if world == 1:
        return loss_out
    dist.all_reduce(loss_out, op=dist.ReduceOp.SUM, group=group)
    loss_out.div_(world)
    return loss_out
