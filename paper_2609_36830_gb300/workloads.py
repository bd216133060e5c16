"""Seeded synthetic workloads shaped like the paper's experiments.

This module only draws random inputs.  It holds none of the method's
arithmetic (no staleness, percentile, budget, selection, softmax or loss), so
both the CUDA library and the CPU oracle can be fed from it without sharing
any of the computation under test.

Workload recipes (the pool shapes follow the paper's settings: response
budgets of 8,192 and 20,480 tokens, 8-16 responses per prompt, masked tool
output in multi-turn rollouts, version tags bumped at weight-sync
interruptions):

``tiny``       64 trajectories (8 prompts x 8), response lengths U{16..256},
               trainer version j = 20, start version U{j-6 .. j-n_int} with
               n_int ~ U{0..2} interruptions at distinct uniform positions in
               [1, T-1] (each bumps the tag by one), completion version
               c ~ U{start+n_int .. j}, capacity 48, hidden 256, vocab 2048,
               rewards Bernoulli(0.5), clip eps 0.2 / 0.2.
``math7b``     512 trajectories (64 x 8), 256 prompt rows (masked out) plus
               responses lognormal(median 2048, sigma 0.75) clipped to
               [16, 8192], j = 200, start lag Geometric(0.4) on {0,1,..}
               redrawn until n_int <= lag <= 8, n_int ~ U{0..3}, capacity 384,
               hidden 3584, vocab 152064, rewards Bernoulli(0.4).
``multiturn``  256 trajectories (32 x 8), 2-8 turns: model segments
               U{64..1024} interleaved with tool segments U{32..512} (tag -1,
               loss-masked); per-turn tags j - lag_i with lags drawn from
               U{0..10} and sorted non-increasing, capacity 192, hidden 3584,
               vocab 152064, rewards Bernoulli(0.5).
``moe``        1024 trajectories (128 x 8), responses lognormal(median 4096,
               sigma 0.75) clipped to [16, 16384], lag Geometric(0.3) <= 12,
               n_int ~ U{0..4}, capacity 768, hidden 2048, vocab 151936,
               rewards Bernoulli(0.5), clip eps 0.2 / 0.28.
``sweep``      pools of 1k / 16k / 128k / 1M trajectories (groups of 8),
               lognormal(median 2048, sigma 1.0) clipped to [16, 32768],
               j = 1000, n_int ~ U{0..8}, lag ~ U{n_int..32}, capacity N/2.

Prefix scores: a trajectory whose last interruption falls at token m >= 32
carries s_pre ~ |N(0, 0.05 d)| with d its number of interruptions (drift grows
with the number of weight syncs its generation spanned); the others carry NaN
(no prefix rescored).  The window holds 512 draws of the same law with
d ~ U{1..max interruptions}.  Hidden rows are N(0,1), vocabulary rows
N(0, 1/H), targets uniform over the vocabulary, all rounded to bf16 (RNE).
Behaviour log-probs are ``center + N(0, 0.05 (j - v_t))`` per response token,
where the caller passes either the oracle's log-probs (tiny) or the constant
-ln V - 1/2 (the mean log-prob of a uniform target under N(0,1) logits).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import numpy as np

SEED_BASE = 20260000


@dataclass(frozen=True)
class WorkloadSpec:
    name: str
    index: int
    n_traj: int
    group_size: int
    n_target: int
    trainer_version: int
    hidden: int
    vocab: int
    reward_p: float
    eps_low: float
    eps_high: float
    prompt_len: int = 0
    length: tuple = ("uniform", 16, 256)
    lag: tuple = ("start_uniform", 6)
    max_interruptions: int = 2
    multiturn: bool = False


SPECS = {
    "tiny": WorkloadSpec("tiny", 0, 64, 8, 48, 20, 256, 2048, 0.5, 0.2, 0.2,
                         length=("uniform", 16, 256), lag=("start_uniform", 6),
                         max_interruptions=2),
    "math7b": WorkloadSpec("math7b", 1, 512, 8, 384, 200, 3584, 152064, 0.4, 0.2, 0.28,
                           prompt_len=256, length=("lognormal", 2048, 0.75, 8192),
                           lag=("geometric", 0.4, 8), max_interruptions=3),
    "multiturn": WorkloadSpec("multiturn", 2, 256, 8, 192, 200, 3584, 152064, 0.5, 0.2, 0.28,
                              length=("turns", 2, 8), lag=("turns", 10), max_interruptions=7,
                              multiturn=True),
    "moe": WorkloadSpec("moe", 3, 1024, 8, 768, 300, 2048, 151936, 0.5, 0.2, 0.28,
                        length=("lognormal", 4096, 0.75, 16384), lag=("geometric", 0.3, 12),
                        max_interruptions=4),
    "sweep": WorkloadSpec("sweep", 4, 1024, 8, 512, 1000, 0, 0, 0.5, 0.2, 0.28,
                          length=("lognormal", 2048, 1.0, 32768), lag=("uniform", 32),
                          max_interruptions=8),
}

SWEEP_SIZES = (1024, 16384, 131072, 1048576)


@dataclass
class Pool:
    """One pool of completed trajectories plus the rows of its token batch.

    Per-trajectory arrays are numpy.  Per-token arrays (``tags``) and the row
    arrays are numpy unless the pool was expanded on a device, in which case
    they are torch tensors on that device.
    """
    spec: WorkloadSpec
    seed: int
    n_traj: int
    trainer_version: int
    group_size: int
    n_target: int
    offsets: object          # int64 [n_traj+1]  response-token CSR (tags)
    tags: object             # int32 [n_tokens]  v_t, -1 for tool tokens
    c_version: np.ndarray    # int32 [n_traj]    completion (= pool entry) version
    s_pre: np.ndarray        # float32 [n_traj]  prefix forgetting score or NaN
    window: np.ndarray       # float32 [512]     recent prefix scores
    reward: np.ndarray       # float32 [n_traj]
    resp_len: np.ndarray     # int64 [n_traj]
    prompt_len: np.ndarray   # int64 [n_traj]
    n_interruptions: np.ndarray
    meta: dict = field(default_factory=dict)

    @property
    def n_tokens(self) -> int:
        return int(self.resp_len.sum())


def _rng(spec: WorkloadSpec, seed: Optional[int]):
    s = SEED_BASE + spec.index if seed is None else seed
    return s, np.random.SeedSequence(s)


def _lengths(spec, rng, n):
    kind = spec.length[0]
    if kind == "uniform":
        return rng.integers(spec.length[1], spec.length[2] + 1, size=n).astype(np.int64)
    if kind == "lognormal":
        med, sigma, cap = spec.length[1], spec.length[2], spec.length[3]
        x = rng.lognormal(math.log(med), sigma, size=n)
        return np.clip(np.rint(x), 16, cap).astype(np.int64)
    raise ValueError(kind)


def _geometric_lags(rng, p, lo, hi):
    """Geometric(p) lags on {0, 1, ...}, each redrawn until lo[i] <= lag <= hi."""
    lag = rng.geometric(p, size=lo.size) - 1
    bad = (lag < lo) | (lag > hi)
    while bad.any():
        lag[bad] = rng.geometric(p, size=int(bad.sum())) - 1
        bad = (lag < lo) | (lag > hi)
    return lag


def _interruption_positions(rng, lens, n_int, max_k):
    """Per trajectory, n_int distinct positions uniform in [1, T-1], ascending; -1 pads."""
    n = lens.size
    col = np.arange(max_k)[None, :]
    used = col < n_int[:, None]
    pos = rng.integers(1, np.maximum(lens, 2)[:, None], size=(n, max_k))
    big = np.iinfo(np.int64).max
    while True:
        srt = np.sort(np.where(used, pos, big), axis=1)
        dup = ((srt[:, 1:] == srt[:, :-1]) & (srt[:, 1:] != big)).any(axis=1)
        if not dup.any():
            break
        rows = np.nonzero(dup)[0]
        pos[rows] = rng.integers(1, np.maximum(lens[rows], 2)[:, None], size=(rows.size, max_k))
    return np.where(used, srt, -1)


def make_pool(name: str, seed: Optional[int] = None, n_traj: Optional[int] = None,
              device=None) -> Pool:
    """Draw a pool.  ``n_traj`` overrides the occupancy (whole groups only).

    With ``device`` set (a torch device string), the per-token tag array is
    expanded on that device with torch; otherwise with numpy on the host.  The
    per-trajectory draws are identical either way.
    """
    spec = SPECS[name]
    seed, ss = _rng(spec, seed)
    n = spec.n_traj if n_traj is None else int(n_traj)
    G = spec.group_size
    assert n % G == 0, "pools hold whole prompt groups"
    s_len, s_ver, s_int, s_pre, s_win, s_rew = ss.spawn(6)
    r_len, r_ver, r_int = (np.random.default_rng(s) for s in (s_len, s_ver, s_int))
    r_pre, r_win, r_rew = (np.random.default_rng(s) for s in (s_pre, s_win, s_rew))
    j = spec.trainer_version

    if spec.multiturn:
        return _make_multiturn(spec, seed, n, r_len, r_ver, r_int, r_pre, r_win, r_rew, device)

    lens = _lengths(spec, r_len, n)
    n_int = r_int.integers(0, spec.max_interruptions + 1, size=n)
    n_int = np.minimum(n_int, lens - 1)
    kind = spec.lag[0]
    if kind == "start_uniform":
        start = r_ver.integers(j - spec.lag[1], j - n_int + 1)
    elif kind == "geometric":
        start = j - _geometric_lags(r_ver, spec.lag[1], n_int, spec.lag[2])
    elif kind == "uniform":
        start = j - r_ver.integers(n_int, spec.lag[1] + 1)
    else:
        raise ValueError(kind)
    start = start.astype(np.int64)
    end = start + n_int
    c = r_ver.integers(end, j + 1).astype(np.int64)
    pos = _interruption_positions(r_int, lens, n_int, max(spec.max_interruptions, 1))
    last = np.where(n_int > 0, pos[np.arange(n), np.maximum(n_int - 1, 0)], -1)
    s_pre_v = np.full(n, np.nan, np.float32)
    has = (n_int > 0) & (last >= 32)
    s_pre_v[has] = np.abs(r_pre.normal(0.0, 0.05 * n_int[has])).astype(np.float32)
    d = r_win.integers(1, max(spec.max_interruptions, 1) + 1, size=512)
    window = np.abs(r_win.normal(0.0, 0.05 * d)).astype(np.float32)
    reward = (r_rew.random(n) < spec.reward_p).astype(np.float32)
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tags = _expand_tags(offsets, start, pos, n_int, device)
    return Pool(spec, seed, n, j, G, _target_for(spec, n), offsets if device is None else
                _to_device(offsets, device), tags, c.astype(np.int32), s_pre_v, window, reward,
                lens, np.full(n, spec.prompt_len, np.int64), n_int,
                meta={"offsets_host": offsets, "last_interrupt": last.astype(np.int64)})


def _target_for(spec, n):
    if spec.name == "sweep":
        return n // 2
    return spec.n_target


def _to_device(a, device):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def _expand_tags(offsets, start, pos, n_int, device):
    """tag_t = start + #(interruption positions <= t) within each trajectory."""
    n = start.size
    total = int(offsets[-1])
    lens = np.diff(offsets)
    valid = pos >= 0
    traj_idx = np.nonzero(valid)[0]
    gpos = offsets[traj_idx] + pos[valid]
    if device is None:
        # positions are distinct, so a plain store marks them
        delta = np.zeros(total, np.int32)
        delta[gpos] = 1
        cum = np.cumsum(delta, dtype=np.int32)
        del delta
        before = np.concatenate([[0], cum])[offsets[:-1]].astype(np.int64)
        cum += np.repeat((start - before).astype(np.int32), lens)
        return cum
    import torch
    dev = torch.device(device)
    lens_t = torch.from_numpy(lens).to(dev)
    delta = torch.zeros(total, dtype=torch.int32, device=dev)
    if gpos.size:
        delta.index_put_((torch.from_numpy(gpos).to(dev),),
                         torch.ones(gpos.size, dtype=torch.int32, device=dev), accumulate=True)
    cum = torch.cumsum(delta, 0, dtype=torch.int32)
    del delta
    zero = torch.zeros(1, dtype=torch.int32, device=dev)
    before = torch.cat([zero, cum])[torch.from_numpy(offsets[:-1]).to(dev)]
    tags = cum
    tags -= torch.repeat_interleave(before, lens_t, output_size=total)
    tags += torch.repeat_interleave(torch.from_numpy(start.astype(np.int32)).to(dev), lens_t,
                                    output_size=total)
    return tags


def _make_multiturn(spec, seed, n, r_len, r_ver, r_int, r_pre, r_win, r_rew, device):
    j = spec.trainer_version
    max_lag = spec.lag[1]
    seg_tags, lens, c, n_int, last_pos = [], [], [], [], []
    for i in range(n):
        turns = int(r_len.integers(spec.length[1], spec.length[2] + 1))
        lags = np.sort(r_ver.integers(0, max_lag + 1, size=turns))[::-1]
        parts = []
        p = 0
        last = -1
        k = 0
        for t in range(turns):
            if t > 0:
                tl = int(r_len.integers(32, 513))
                parts.append(np.full(tl, -1, np.int32))
                p += tl
            ml = int(r_len.integers(64, 1025))
            if t > 0 and lags[t] != lags[t - 1]:
                last, k = p, k + 1
            parts.append(np.full(ml, j - lags[t], np.int32))
            p += ml
        seg = np.concatenate(parts)
        seg_tags.append(seg)
        lens.append(seg.size)
        c.append(int(r_ver.integers(j - lags[-1], j + 1)))
        n_int.append(k)
        last_pos.append(last)
    lens = np.array(lens, np.int64)
    n_int = np.array(n_int, np.int64)
    last = np.array(last_pos, np.int64)
    s_pre_v = np.full(n, np.nan, np.float32)
    has = (n_int > 0) & (last >= 32)
    s_pre_v[has] = np.abs(r_pre.normal(0.0, 0.05 * n_int[has])).astype(np.float32)
    d = r_win.integers(1, spec.max_interruptions + 1, size=512)
    window = np.abs(r_win.normal(0.0, 0.05 * d)).astype(np.float32)
    reward = (r_rew.random(n) < spec.reward_p).astype(np.float32)
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tags = np.concatenate(seg_tags)
    if device is not None:
        tags = _to_device(tags, device)
    return Pool(spec, seed, n, j, spec.group_size, spec.n_target,
                offsets if device is None else _to_device(offsets, device), tags,
                np.array(c, np.int32), s_pre_v, window, reward, lens,
                np.zeros(n, np.int64), n_int,
                meta={"offsets_host": offsets, "last_interrupt": last})


# ---------------------------------------------------------------------------
# Rows of the token batch (the LM-head / surrogate half of the step)
# ---------------------------------------------------------------------------

@dataclass
class Rows:
    """Row arrays of a pool's token batch: one row per prompt or response token.

    ``row_offsets`` is the per-trajectory CSR over rows; ``mask`` is 1 for a
    response token generated by the policy, 0 for prompt and tool rows;
    ``row_version`` is the tag of the row's token (-1 for prompt / tool rows).
    """
    row_offsets: np.ndarray   # int64 [n_traj+1]
    mask: np.ndarray          # uint8 [n_rows]
    targets: np.ndarray       # int32 [n_rows]
    row_version: np.ndarray   # int32 [n_rows]
    n_rows: int


def make_rows(pool: Pool, seed_offset: int = 0) -> Rows:
    """Row layout, loss mask and targets for every trajectory of ``pool`` (host)."""
    n = pool.n_traj
    per = pool.prompt_len + pool.resp_len
    row_offsets = np.concatenate([[0], np.cumsum(per)]).astype(np.int64)
    n_rows = int(row_offsets[-1])
    tags = pool.tags
    if not isinstance(tags, np.ndarray):
        tags = tags.cpu().numpy()
    row_version = np.full(n_rows, -1, np.int32)
    resp_rows = np.ones(n_rows, bool)
    if pool.prompt_len.any():
        starts = row_offsets[:-1]
        prompt_idx = np.repeat(starts, pool.prompt_len) + _ramp(pool.prompt_len)
        resp_rows[prompt_idx] = False
    row_version[resp_rows] = tags
    mask = (row_version != -1).astype(np.uint8)
    rng = np.random.default_rng(np.random.SeedSequence(pool.seed + 7919 + seed_offset))
    V = pool.spec.vocab if pool.spec.vocab else 2
    targets = rng.integers(0, V, size=n_rows).astype(np.int32)
    return Rows(row_offsets, mask, targets, row_version, n_rows)


def _ramp(lens):
    """0..len-1 for each entry of ``lens``, concatenated."""
    total = int(lens.sum())
    starts = np.repeat(np.cumsum(lens) - lens, lens)
    return np.arange(total) - starts


def behaviour_logprob(rows: Rows, trainer_version: int, center, seed: int) -> np.ndarray:
    """ell^mu_t = center_t + N(0, 0.05 (j - v_t)) on policy rows; center on others.

    ``center`` is a scalar or an array of per-row log-probs (float64).
    """
    rng = np.random.default_rng(np.random.SeedSequence(seed + 104729))
    lag = np.where(rows.row_version >= 0, trainer_version - rows.row_version, 0)
    noise = rng.standard_normal(rows.n_rows) * (0.05 * lag)
    return (np.asarray(center, np.float64) + noise).astype(np.float32)


def uniform_center(vocab: int) -> float:
    """Mean log-prob of a uniform target under N(0,1) logits: about -ln V - 1/2."""
    return -math.log(vocab) - 0.5


def bf16_normal_host(shape, std: float, seed: int) -> np.ndarray:
    """N(0, std^2) rounded to bf16 (RNE); returned as uint16 bit patterns."""
    import torch
    rng = np.random.default_rng(np.random.SeedSequence(seed))
    x = torch.from_numpy(rng.standard_normal(shape).astype(np.float32) * np.float32(std))
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


def bf16_normal_device(shape, std: float, seed: int, device="cuda", chunk_rows: int = 65536):
    """N(0, std^2) in bf16 on ``device`` from a seeded torch generator, drawn in row chunks."""
    import torch
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    rows = shape[0]
    for r0 in range(0, rows, chunk_rows):
        r1 = min(rows, r0 + chunk_rows)
        x = torch.randn((r1 - r0,) + tuple(shape[1:]), generator=gen, device=device,
                        dtype=torch.float32)
        if std != 1.0:
            x.mul_(std)
        out[r0:r1].copy_(x)
    return out


@dataclass
class PrefixBatch:
    """Prefixes of the pool's interrupted rollouts, for re-scoring (Eq. 6).

    Prefix i is trajectory ``traj[i]``'s prompt plus the response tokens generated
    before its last weight-sync interruption; ``rows`` are its row indices in the
    pool's row layout and ``mask`` marks the eligible (policy-generated) rows.
    """
    traj: np.ndarray         # int64 [n_prefix]
    seq_offsets: np.ndarray  # int64 [n_prefix+1]
    rows: np.ndarray         # int64 [n_rows] pool row of each prefix row
    mask: np.ndarray         # uint8 [n_rows]
    n_rows: int


def make_prefixes(pool: Pool, rows: Rows) -> PrefixBatch:
    last = pool.meta["last_interrupt"]
    traj = np.nonzero(last >= 1)[0].astype(np.int64)
    plen = pool.prompt_len[traj] + last[traj]
    seq_offsets = np.concatenate([[0], np.cumsum(plen)]).astype(np.int64)
    starts = rows.row_offsets[traj]
    idx = np.repeat(starts, plen) + _ramp(plen)
    return PrefixBatch(traj, seq_offsets, idx.astype(np.int64), rows.mask[idx].copy(),
                       int(seq_offsets[-1]))
