"""Data-parallel exchange of one ZO step: ranks split the tokens, share everything else.

Every rank holds the same W, U, C, m, v and seed, runs the pair forward and the
loss pair on its own token shard, and the ranks then average the loss vector --
[L+, L-, D, a], or [L_0 .. L_q, a_1 .. a_q] for the one-sided q-query estimator
(each entry a mean over the rank's T * n elements, so with equal shards their
average is the global value; every a is linear in the losses).
Each rank then applies the same Adam update with the same regenerated Z, so C
stays identical on every rank without a gradient all-reduce.  check_replicas
compares the ranks' fingerprints of their arenas (zoact_arena_hash) to detect a
replica that diverged anyway (a fault on one rank, a rank fed another seed).

This module only issues collectives and library calls: the division of the
summed loss vector and the fingerprints run in libzoact.  Ranks on the CPU (the
gloo tests) have no device and pass their own `finish` / `fingerprint`.
"""
import torch
import torch.distributed as dist

from . import _lib as Z


def allreduce_loss(loss_out, ctx=None, group=None, finish=None):
    """Average the loss vector over the ranks, in place: one all-reduce (sum), then the division by the
    number of ranks -- zoact_mean_over_ranks on ctx's stream for a device vector, or finish(loss_out, world)
    when given."""
    world = dist.get_world_size(group)
    if world == 1:
        return loss_out
    dist.all_reduce(loss_out, op=dist.ReduceOp.SUM, group=group)
    if finish is not None:
        finish(loss_out, world)
    elif ctx is not None:
        Z.zoact_mean_over_ranks(ctx, loss_out, world)
    else:
        raise ValueError("allreduce_loss: pass the libzoact context (device vector) or a finish function")
    return loss_out


def replica_fingerprints(arenas, ctx=None, group=None, fingerprint=None):
    """Every rank's fingerprints of its arenas: an int64 tensor [world, len(arenas)] (the uint64 bits) on
    every rank.  Device arenas are fingerprinted by zoact_arena_hash on ctx's stream; fingerprint(arena) -> int
    replaces it where given.  One all-gather."""
    if fingerprint is not None:
        vals = [fingerprint(a) for a in arenas]
        local = torch.tensor([v - (1 << 64) if v >= (1 << 63) else v for v in vals], dtype=torch.int64)
    else:
        if ctx is None:
            raise ValueError("replica_fingerprints: pass the libzoact context (device arenas) or a fingerprint")
        local = torch.empty(len(arenas), dtype=torch.int64, device=arenas[0].device)
        for i, a in enumerate(arenas):
            Z.zoact_arena_hash(ctx, a, local[i:i + 1])
    world = dist.get_world_size(group) if dist.is_initialized() else 1
    if world == 1:
        return local.reshape(1, -1).cpu()
    out = [torch.empty_like(local) for _ in range(world)]
    dist.all_gather(out, local, group=group)
    return torch.stack(out).cpu()


def check_replicas(arenas, ctx=None, group=None, fingerprint=None):
    """(status, ranks): ZOACT_OK when every rank's arenas (e.g. [C, m, v]) have the same fingerprints as rank
    0's, else ZOACT_ERR_REPLICA_MISMATCH and the ranks that differ.  The same answer on every rank; syncs."""
    fp = replica_fingerprints(arenas, ctx, group, fingerprint)
    bad = [r for r in range(fp.shape[0]) if not torch.equal(fp[r], fp[0])]
    return (Z.ZOACT_ERR_REPLICA_MISMATCH if bad else Z.ZOACT_OK), bad
