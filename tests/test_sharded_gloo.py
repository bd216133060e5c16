"""The data-parallel step's exchange protocol on CPU ranks (gloo).

A pool is partitioned by prompt group across 2 or 4 gloo processes (one shard
may be empty).  Each rank runs sharded.select_protocol - the same generator the
GPU ranks run, with the same exchanges through torch.distributed - but with the
per-rank kernels replaced by a numpy statement of what they compute (the MSB-first
radix pass over order-preserving 64-bit keys, the tie count at the pivot, the
id lists).  The union of the ranks' lists must equal the oracle's top-k on the
unsharded pool bit for bit, ties across shard boundaries included, and the
loss assembled from the ranks' (numerator, denominator) partials must equal
the oracle's loss on the unsharded batch.  The GPU kernels behind the same
protocol are checked against the oracle in tests/test_gpu_sharded.py."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

SHIFT = (53, 42, 31, 20, 10, 0)
WIDTH = (11, 11, 11, 11, 10, 10)


def order_keys(x):
    b = np.ascontiguousarray(x, np.float64).view(np.uint64).copy()
    b[b == np.uint64(0x8000000000000000)] = np.uint64(0)
    neg = (b >> np.uint64(63)) == 1
    return np.where(neg, ~b, b | np.uint64(0x8000000000000000))


class NumpyShardOps:
    """Per-rank stand-in of pace_select_shard_{pass,ties,write} (CPU tensors)."""

    def __init__(self):
        self.prefix = 0
        self.mask = 0
        self.k_rem = 0

    def _pick(self, hist, p):
        h = hist.numpy().astype(np.int64)
        run = 0
        for d in range((1 << WIDTH[p]) - 1, -1, -1):
            if run < self.k_rem <= run + h[d]:
                self.prefix |= d << SHIFT[p]
                self.mask |= ((1 << WIDTH[p]) - 1) << SHIFT[p]
                self.k_rem -= run
                return
            run += h[d]

    def pass_(self, score, p, k, prev, cur, ws, status, stream):
        if p == 0:
            self.prefix, self.mask, self.k_rem = 0, 0, int(k)
        else:
            self._pick(prev, p - 1)
        keys = order_keys(score.numpy())
        sel = (keys & np.uint64(self.mask)) == np.uint64(self.prefix)
        digit = ((keys[sel] >> np.uint64(SHIFT[p])) & np.uint64((1 << WIDTH[p]) - 1))
        cur.copy_(torch.from_numpy(np.bincount(digit.astype(np.int64),
                                               minlength=2048).astype(np.int32)))

    def ties(self, score, last, tied, ws, status, stream):
        self._pick(last, len(SHIFT) - 1)
        tied.fill_(int((order_keys(score.numpy()) == np.uint64(self.prefix)).sum()))

    def write(self, score, G, k, tied_before, id_base, out, ws, n_rejected, status, stream):
        keys = order_keys(score.numpy())
        U = keys.size
        if k == 0:
            rej = np.zeros(U, bool)
        else:
            pivot = np.uint64(self.prefix)
            eq = keys == pivot
            tie_idx = int(tied_before.item()) + np.cumsum(eq) - 1
            rej = (keys > pivot) | (eq & (tie_idx < self.k_rem))
        traj_rej = np.repeat(rej, G)
        ids = id_base + np.arange(U * G)
        acc_ids, rej_ids = ids[~traj_rej], ids[traj_rej]
        out["accepted"][: acc_ids.size] = torch.from_numpy(acc_ids.astype(np.int32))
        out["rejected"][: rej_ids.size] = torch.from_numpy(rej_ids.astype(np.int32))
        out["flags"][: U * G] = torch.from_numpy((~traj_rej).astype(np.uint8))
        n_rejected.fill_(int(rej.sum()))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _case(seed):
    """A pool of 37 groups of G = 2 with heavy ties, its shard boundaries per world
    size (one empty shard at world 4), and a batch of rows per trajectory."""
    rng = np.random.default_rng(seed)
    U, G = 37, 2
    us = rng.integers(0, 6, size=U).astype(np.float64) / 4.0
    us[5] = -0.0
    us[6] = 0.0
    bounds = {2: [0, 18, 37], 4: [0, 9, 9, 30, 37]}
    lens = rng.integers(3, 9, size=U * G)
    so = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    n_rows = int(so[-1])
    lp = -rng.random(n_rows) * 5
    behav = lp + rng.normal(0, 0.3, n_rows)
    mask = (rng.random(n_rows) < 0.8).astype(np.uint8)
    reward = (rng.random(U * G) < 0.5).astype(np.float32)
    return U, G, us, bounds, so, lp, behav, mask, reward


def _rank_worker(rank, world, port, seed, k, agg, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from paper_2609_36830_gb300 import sharded
    U, G, us, bounds, so, lp, behav, mask, reward = _case(seed)
    u0, u1 = bounds[world][rank], bounds[world][rank + 1]
    buf = sharded.ShardSelectBuffers(u1 - u0, G, "cpu")
    score = torch.from_numpy(us[u0:u1].copy())

    def rank_step():
        yield from sharded.select_protocol(score, G, k, u0 * G, buf, ops=NumpyShardOps())
        # the rank's part of the loss: its groups' rows, advantages over its own
        # accepted members (whole groups are local)
        t0, t1 = u0 * G, u1 * G
        flags = buf.out["flags"][: t1 - t0].numpy().copy()
        r0, r1 = so[t0], so[t1]
        lso = so[t0:t1 + 1] - r0
        part = torch.zeros(2, dtype=torch.float64)
        if t1 > t0:
            _, adv = oracle.group_advantages(reward[t0:t1], G, seq_accepted=flags)
            st, _, _, term = oracle.surrogate(lp[r0:r1], behav[r0:r1], lso, adv,
                                              mask=mask[r0:r1], seq_accepted=flags, agg=agg)
            assert st == 0
            in_loss = np.repeat(flags, np.diff(lso)).astype(bool) & mask[r0:r1].astype(bool)
            if agg == oracle.AGG_TOKEN_MEAN:
                part[0], part[1] = term[in_loss].sum(), in_loss.sum()
            else:
                for i in range(t1 - t0):
                    m = in_loss[lso[i]:lso[i + 1]]
                    if m.any():
                        part[0] += term[lso[i]:lso[i + 1]][m].sum() / m.sum()
                        part[1] += 1
        yield sharded.ALL_REDUCE, part
        buf.partial = part

    sharded.run_process_group(rank_step())
    n = (u1 - u0) * G
    n_rej = int(buf.n_rejected.item())
    q.put((rank, buf.out["accepted"][: n - n_rej * G].numpy().copy(),
           buf.out["rejected"][: n_rej * G].numpy().copy(), buf.out["flags"][:n].numpy().copy(),
           buf.partial.numpy().copy()))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 4])
@pytest.mark.parametrize("k,agg", [(11, 0), (1, 1), (36, 0), (0, 0), (37, 1)])
def test_sharded_selection_and_loss_match_the_unsharded_oracle(world, k, agg):
    import oracle
    oracle.build()  # once, before the ranks load it
    seed = 7 + k
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_worker, args=(r, world, port, seed, k, agg, q))
             for r in range(world)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=180) for _ in range(world)), key=lambda o: o[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    U, G, us, bounds, so, lp, behav, mask, reward = _case(seed)
    st, oacc, orej, oflag = oracle.select(us, G, k)
    assert st == 0
    np.testing.assert_array_equal(np.concatenate([o[1] for o in out]), oacc)
    np.testing.assert_array_equal(np.concatenate([o[2] for o in out]), orej)
    np.testing.assert_array_equal(np.concatenate([o[3] for o in out]), oflag)
    # the loss from the summed partials against the oracle on the whole batch
    part = out[0][4]
    assert all(np.array_equal(o[4], part) for o in out)  # every rank holds the same sums
    _, adv = oracle.group_advantages(reward, G, seq_accepted=oflag)
    st, oloss, _, _ = oracle.surrogate(lp, behav, so, adv, mask=mask, seq_accepted=oflag,
                                       agg=agg)
    loss = part[0] / part[1] if part[1] > 0 else 0.0
    assert abs(loss - oloss) <= 1e-12 * max(abs(oloss), 1e-300) or loss == oloss == 0.0


def test_ties_straddle_the_shard_boundaries():
    """The case above really has tied units at the pivot on both sides of a
    boundary (so the tie scan across ranks is exercised)."""
    import oracle
    U, G, us, bounds, *_ = _case(7 + 11)
    _, _, orej, _ = oracle.select(us, G, 11)
    rej_units = np.unique(orej // G)
    pivot = us[rej_units].min()
    tied = np.nonzero(us == pivot)[0]
    assert (tied < 18).any() and (tied >= 18).any()
    assert len(tied) > len(np.intersect1d(tied, rej_units))  # some ties are accepted
