"""Data-parallel ZO step across 2 CPU ranks (gloo): the scalar exchange of dp.allreduce_loss and the
replica check of dp.check_replicas.

Each rank evaluates the oracle's loss pair on its own token shard; after the
all-reduce every rank holds the loss pair of the whole batch, and the Adam
updates the ranks then apply independently are identical to the single-process
update on the concatenated batch.  The ranks have no device, so the division
by the number of ranks (zoact_mean_over_ranks on a GPU) is passed in as
`finish`, and the arena fingerprints (zoact_arena_hash on a GPU) come from the
oracle's definition.  A coefficient perturbed on one rank between steps is
reported by every rank.
"""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import layers, loss as oloss, optim, philox, replica


def _div(v, world):
    v.div_(world)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _problem():
    rng = np.random.default_rng(0)
    d_in, d_out, r, T = 48, 40, 4, 24
    W = rng.standard_normal((d_out, d_in)) / np.sqrt(d_in)
    U = np.linalg.qr(rng.standard_normal((d_in, r)))[0]
    C = 0.1 * rng.standard_normal((d_out, r))
    X = rng.standard_normal((2 * T, d_in))      # the whole batch: two shards of T tokens
    tgt = rng.standard_normal((2 * T, d_out))
    return W, U, C, X, tgt, T


def _rank_step(rank, world, W, U, C, X, tgt, T, eps=1e-3, seed=9, query=1):
    Z = philox.perturbation(seed, 3, query, *C.shape)
    xs, ts = X[rank * T:(rank + 1) * T], tgt[rank * T:(rank + 1) * T]
    Y = layers.pair_forward(W, U, C, Z, xs, eps, T, True)
    out = torch.tensor(oloss.loss_pair(Y, T, ts, eps), dtype=torch.float64)
    return out, Z


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_01125_gb300.dp import allreduce_loss
    W, U, C, X, tgt, T = _problem()
    out, Z = _rank_step(rank, world, W, U, C, X, tgt, T)
    allreduce_loss(out, finish=_div)
    a = float(out[3])
    Cn, _, _ = optim.adam_step(C, 0, 0, optim.zo_gradient(a, Z), 1e-3, 0.9, 0.999, 1e-8, 1)
    gathered = [torch.zeros(Cn.size, dtype=torch.float64) for _ in range(world)]
    dist.all_gather(gathered, torch.from_numpy(Cn.reshape(-1).copy()))
    q.put((rank, out.numpy().tolist(), [g.numpy() for g in gathered]))
    dist.destroy_process_group()


def test_two_rank_scalar_exchange_matches_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    W, U, C, X, tgt, T = _problem()
    Z = philox.perturbation(9, 3, 1, *C.shape)
    # single process on the concatenated batch (both halves see the same x per shard: shared input)
    Yfull = np.concatenate([layers.pair_forward(W, U, C, Z, X[i * T:(i + 1) * T], 1e-3, T, True) for i in range(2)])
    yp = np.concatenate([Yfull[:T], Yfull[2 * T:3 * T]])
    ym = np.concatenate([Yfull[T:2 * T], Yfull[3 * T:]])
    ref = oloss.loss_pair(np.concatenate([yp, ym]), 2 * T, tgt, 1e-3)
    Cref, _, _ = optim.adam_step(C, 0, 0, optim.zo_gradient(ref[3], Z), 1e-3, 0.9, 0.999, 1e-8, 1)
    for rank, out, gathered in results:
        np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-15)
        for g in gathered:                           # every rank holds the same C, equal to the reference
            np.testing.assert_allclose(g, Cref.reshape(-1), rtol=0, atol=1e-15)


def _multi_rank(rank, T, W, U, C, X, tgt, q, mu=1e-3, seed=9):
    Zs = [philox.perturbation(seed, 3, 100 + j, *C.shape) for j in range(q)]
    xs, ts = X[rank * T:(rank + 1) * T], tgt[rank * T:(rank + 1) * T]
    Y = layers.multi_forward(W, U, C, [None] + Zs, [0.0] + [mu] * q, xs, T, True)
    L, a = oloss.loss_queries(Y, T, q + 1, ts, mu)
    return torch.tensor(L + a, dtype=torch.float64), Zs


def _worker_multi(rank, world, port, q, n_queries):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_01125_gb300.dp import allreduce_loss
    W, U, C, X, tgt, T = _problem()
    out, Zs = _multi_rank(rank, T, W, U, C, X, tgt, n_queries)
    allreduce_loss(out, finish=_div)
    a = out.numpy()[n_queries + 1:]
    Cn, _, _ = optim.adam_step(C, 0, 0, optim.zo_gradient_queries(a, Zs), 1e-3, 0.9, 0.999, 1e-8, 1)
    q.put((rank, out.numpy().tolist(), Cn.reshape(-1)))
    dist.destroy_process_group()


def test_two_rank_exchange_of_the_q_query_losses():
    # Algorithm 2's one-sided estimator: the averaged vector [L_0..L_q, a_1..a_q] is that of the whole batch,
    # so both ranks apply the single-process update
    nq = 4
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker_multi, args=(r, 2, port, q, nq)) for r in range(2)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    W, U, C, X, tgt, T = _problem()
    Zs = [philox.perturbation(9, 3, 100 + j, *C.shape) for j in range(nq)]
    blocks = [layers.multi_forward(W, U, C, [None] + Zs, [0.0] + [1e-3] * nq, X[i * T:(i + 1) * T], T, True)
              for i in range(2)]
    # the whole batch: block b holds both shards' rows of evaluation point b
    Yfull = np.concatenate([np.concatenate([blk[b * T:(b + 1) * T] for blk in blocks]) for b in range(nq + 1)])
    L, a = oloss.loss_queries(Yfull, 2 * T, nq + 1, tgt, 1e-3)
    Cref, _, _ = optim.adam_step(C, 0, 0, optim.zo_gradient_queries(a, Zs), 1e-3, 0.9, 0.999, 1e-8, 1)
    for rank, vec, Cn in results:
        np.testing.assert_allclose(vec, L + a, rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(Cn, Cref.reshape(-1), rtol=1e-10, atol=1e-14)


def _worker_replicas(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_01125_gb300.dp import allreduce_loss, check_replicas
    fp = lambda a: replica.arena_hash(a.numpy().astype(np.float32))
    W, U, C, X, tgt, T = _problem()
    C = C.astype(np.float32).astype(np.float64)
    m, v = np.zeros_like(C), np.zeros_like(C)
    statuses = []
    for t in (1, 2, 3):
        out, Z = _rank_step(rank, world, W, U, C, X, tgt, T, query=t)
        allreduce_loss(out, finish=_div)
        C, m, v = optim.adam_step(C, m, v, optim.zo_gradient(float(out[3]), Z), 1e-3, 0.9, 0.999, 1e-8, t)
        C, m, v = (a.astype(np.float32).astype(np.float64) for a in (C, m, v))   # the arenas are fp32
        if t == 2 and rank == 1:
            C[5, 2] = np.nextafter(np.float32(C[5, 2]), np.float32(1.0))         # one rank diverges by 1 ulp
        statuses.append(check_replicas([torch.from_numpy(a.copy()) for a in (C, m, v)], fingerprint=fp))
    q.put((rank, statuses))
    dist.destroy_process_group()


def test_two_rank_replica_check_reports_a_diverged_rank():
    import paper_2607_01125_gb300._lib as Zl
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker_replicas, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank in (0, 1):
        st = results[rank]
        assert st[0] == (Zl.ZOACT_OK, [])                                  # step 1: identical replicas
        assert st[1] == (Zl.ZOACT_ERR_REPLICA_MISMATCH, [1])               # rank 1's C perturbed after step 2
        assert st[2][0] == Zl.ZOACT_ERR_REPLICA_MISMATCH                   # and it stays diverged
