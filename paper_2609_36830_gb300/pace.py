"""Python binding of libpace (include/pace.h): argument marshalling only.

Every step of the path runs in the library's CUDA kernels; torch provides the
device memory (outputs and workspace are allocated here, never by the library)
and the current stream.  Loading fails loudly if the library was not built:
there is no fallback of any kind.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpace.so")
_lock = threading.Lock()
_lib = None

# status codes (include/pace.h)
OK = 0
ERR_INVALID_ARG = 1
ERR_VERSION_ORDER = 2
ERR_NAN_INPUT = 3
ERR_UNSUPPORTED_SHAPE = 4
ERR_WORKSPACE = 5
ERR_TIMEOUT = 6
ERR_CUDA = 7

SCORE_EFF, SCORE_RAW, SCORE_GEN = 0, 1, 2
PROFILE_LMHEAD, PROFILE_TAG_REDUCE = 0, 1
AGG_TOKEN_MEAN, AGG_SEQ_MEAN_TOKEN_MEAN = 0, 1

_P = ctypes.c_void_p
_I32, _I64, _F32, _F64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_double
_SZ = ctypes.c_size_t


class PaceScoreParams(ctypes.Structure):
    _fields_ = [("mode", _I32), ("gamma", _I32), ("min_obs", _I32), ("group_size", _I32),
                ("f_missing", _F64)]


class PaceBudgetParams(ctypes.Structure):
    _fields_ = [("n_target", _I64), ("beta", _F64), ("r_max", _F64), ("r_hat_prev", _F64)]


class PaceLossParams(ctypes.Structure):
    _fields_ = [("eps_low", _F32), ("eps_high", _F32), ("dual_clip", _F32), ("adv_eps", _F32),
                ("agg", _I32), ("std_unbiased", _I32)]


class PaceBatch(ctypes.Structure):
    _fields_ = [("seq_offsets", _P), ("seq_accepted", _P), ("mask", _P), ("n_seq", _I64),
                ("n_rows", _I64)]


class PaceLossArgs(ctypes.Structure):
    _fields_ = [("behav_lp", _P), ("reward", _P), ("group_size", _I32),
                ("params", PaceLossParams), ("loss", _P), ("adv", _P), ("ratio", _P),
                ("partial", _P)]


# every symbol include/pace.h declares, with its C signature
SIGNATURES = {
    "pace_status_string": ([_I32], ctypes.c_char_p),
    "pace_version": ([], _I32),
    "pace_score_params_default": ([_P], None),
    "pace_score_pool": ([_P, _P, _P, _P, _I64, _I64, _I32, _P, _I64, _P, _P, _P, _P, _P, _P, _P,
                         _SZ, _P, _P], _I32),
    "pace_score_pool_workspace_size": ([_I64, _I64], _SZ),
    "pace_budget_params_default": ([_P], None),
    "pace_budget": ([_I64, _I64, _P, _P, _P, _P], _I32),
    "pace_select": ([_P, _I64, _I32, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_select_k": ([_P, _I64, _I32, _I64, _P, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_select_workspace_size": ([_I64], _SZ),
    "pace_select_k_noalloc": ([_P, _I64, _I32, _I64, _P, _P, _P, _P, _P], _I32),
    "pace_select_shard_workspace_size": ([_I64], _SZ),
    "pace_select_shard_pass": ([_P, _I64, _I32, _I64, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_select_shard_ties": ([_P, _I64, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_select_shard_write": ([_P, _I64, _I32, _I64, _P, _I64, _P, _P, _P, _P, _P, _SZ, _P,
                                 _P], _I32),
    "pace_loss_params_default": ([_P], None),
    "pace_group_advantages": ([_P, _P, _I64, _I32, _F32, _I32, _P, _P], _I32),
    "pace_token_logprob": ([_P, _P, _P, _P, _I32, _I32, _F32, _P, _P, _P, _P, _SZ, _P, _P],
                           _I32),
    "pace_token_logprob_workspace_size": ([_I64, _I64, _I32, _I32], _SZ),
    "pace_surrogate_loss": ([_P, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_surrogate_loss_workspace_size": ([_I64, _I64], _SZ),
    "pace_loss_from_partial": ([_P, _P, _P], _I32),
    "pace_prefix_score": ([_P, _P, _P, _P, _P, _I32, _I32, _F32, _I32, _I32, _P, _P, _P, _SZ,
                           _P, _P], _I32),
    "pace_prefix_score_workspace_size": ([_I64, _I64, _I32, _I32], _SZ),
    "pace_stale_k": ([_P, _P, _I64, _I64, _I32, _F64, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_stale_k_workspace_size": ([_I64], _SZ),
    "pace_staleness_histogram": ([_P, _P, _I64, _F64, _F64, _I32, _P, _P, _P], _I32),
    "pace_quantile_admit": ([_P, _I64, _F64, _I64, _I32, _P, _I64, _P, _P, _P, _P, _P], _I32),
    "pace_surrogate_backward": ([_P, _P, _P, _P, _P, _SZ, _P, _P], _I32),
    "pace_surrogate_backward_workspace_size": ([_I64, _I64], _SZ),
    "pace_token_logprob_backward": ([_P, _P, _P, _P, _I32, _I32, _F32, _P, _P, _P, _P, _P, _SZ,
                                     _P, _P], _I32),
    "pace_token_logprob_backward_workspace_size": ([_I64, _I64, _I32, _I32], _SZ),
    "pace_set_profile_events": ([_I32, _P, _P], _I32),
    "pace_set_lmhead_splits": ([_I32], _I32),
    "pace_set_score_fused_min_traj": ([_I64], _I32),
    "pace_score_fused_min_traj_default": ([], _I64),
    "pace_kernel_launches": ([], ctypes.c_uint64),
    "pace_wait_timeout_selftest": ([ctypes.c_uint64, _P, _P], _I32),
    "pace_div_selftest": ([_P, _P, _I64, _P, _P, _P, _P, _P], _I32),
}


class PaceError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


def lib():
    """The loaded libpace.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"{LIB_PATH} is missing: build it with "
                    "`python -c 'import __graft_entry__ as g; g.build()'` "
                    "(there is no fallback implementation)")
            L = ctypes.CDLL(LIB_PATH)
            for name, (args, res) in SIGNATURES.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = res
            _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().pace_status_string(int(status)).decode()


def _check(st: int, where: str):
    if st != OK:
        raise PaceError(st, where)


def _arg(t: Optional[torch.Tensor], dtype, n: Optional[int] = None, name: str = "tensor"):
    """Device pointer of a contiguous tensor of `dtype` with at least `n` elements on
    the current CUDA device; None passes as NULL.  Anything else raises here, before
    the library sees a pointer its kernels could not use."""
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor, got {type(t).__name__}")
    if not t.is_cuda:
        raise ValueError(f"{name}: expected a CUDA tensor")
    if t.get_device() != torch.cuda.current_device():
        raise ValueError(f"{name}: on cuda:{t.get_device()}, the current device is "
                         f"cuda:{torch.cuda.current_device()}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name}: expected {dtype}, got {t.dtype}")
    if n is not None and t.numel() < n:
        raise ValueError(f"{name}: needs at least {n} elements, has {t.numel()}")
    return ctypes.c_void_p(t.data_ptr())


_U8, _I32T, _I64T = torch.uint8, torch.int32, torch.int64
_F32T, _F64T, _BF16 = torch.float32, torch.float64, torch.bfloat16


# The current stream's handle without building a torch.cuda.Stream object (0.08 us
# against ~3 us per call, a tenth of a small pool's scoring call); the public
# call is the fallback where torch does not provide it.
_raw_current_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream=None):
    if stream is not None:
        return ctypes.c_void_p(stream.cuda_stream)
    if _raw_current_stream is not None:
        return ctypes.c_void_p(_raw_current_stream(torch.cuda.current_device()))
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def workspace(nbytes: int, device) -> torch.Tensor:
    """A caller-owned workspace buffer (torch's allocator aligns to >= 256 bytes)."""
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def new_status(device) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device)


def check_status(status: torch.Tensor, where: str = "device"):
    """Synchronises and raises if a device-side error was recorded."""
    v = int(status.item())
    _check(v, where)


# ---------------------------------------------------------------- (a) pool

def score_params(mode=SCORE_EFF, gamma=4, min_obs=32, group_size=8, f_missing=1.0):
    return PaceScoreParams(int(mode), int(gamma), int(min_obs), int(group_size),
                           float(f_missing))


def score_pool(tags, offsets, c_version, s_pre, trainer_version, window, params=None,
               out=None, ws=None, status=None, stream=None):
    """pace_score_pool.  Returns dict kgen, kwait, weight, score, unit_score (float64)."""
    p = params or score_params()
    dev = offsets.device
    n = offsets.numel() - 1
    if out is None:
        out = {k: torch.empty(n, dtype=torch.float64, device=dev)
               for k in ("kgen", "kwait", "weight", "score")}
        out["unit_score"] = torch.empty(n // max(p.group_size, 1), dtype=torch.float64,
                                        device=dev)
    wl = 0 if window is None else window.numel()
    if ws is None:
        ws = workspace(lib().pace_score_pool_workspace_size(n, wl), dev)
    units = n // max(p.group_size, 1)
    st = lib().pace_score_pool(
        _arg(tags, _I32T, None, "tags"), _arg(offsets, _I64T, n + 1, "offsets"),
        _arg(c_version, _I32T, n, "c_version"), _arg(s_pre, _F32T, n, "s_pre"), n,
        tags.numel(), int(trainer_version), _arg(window, _F32T, wl, "window"), wl,
        ctypes.byref(p), _arg(out.get("kgen"), _F64T, n, "kgen"),
        _arg(out.get("kwait"), _F64T, n, "kwait"), _arg(out.get("weight"), _F64T, n, "weight"),
        _arg(out["score"], _F64T, n, "score"),
        _arg(out.get("unit_score"), _F64T, units, "unit_score"), _arg(ws, _U8, None, "ws"),
        ws.numel(), _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_score_pool")
    return out


def budget_params(n_target, beta=0.0, r_max=0.9, r_hat_prev=0.0):
    return PaceBudgetParams(int(n_target), float(beta), float(r_max), float(r_hat_prev))


def budget(n_traj, n_units, params):
    """pace_budget (host only): (r, r_hat, k_units)."""
    r, rh, k = _F64(), _F64(), _I64()
    st = lib().pace_budget(int(n_traj), int(n_units), ctypes.byref(params), ctypes.byref(r),
                           ctypes.byref(rh), ctypes.byref(k))
    _check(st, "pace_budget")
    return r.value, rh.value, k.value


def select(unit_score, group_size, params, out=None, ws=None, status=None, stream=None):
    """pace_select: budget on the host, rejection on the device.

    Returns (r_hat, k_units, accepted_ids, rejected_ids, traj_accepted) where the id
    tensors are views of the first (U-k)*G / k*G entries of full-size buffers.
    """
    dev = unit_score.device
    u = unit_score.numel()
    n = u * group_size
    if out is None:
        out = {"accepted": torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               "rejected": torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               "flags": torch.empty(max(n, 1), dtype=torch.uint8, device=dev)}
    if ws is None:
        ws = workspace(lib().pace_select_workspace_size(u), dev)
    rh, k = _F64(), _I64()
    st = lib().pace_select(_arg(unit_score, _F64T, u, "unit_score"), u, int(group_size),
                           ctypes.byref(params), ctypes.byref(rh), ctypes.byref(k),
                           _arg(out["accepted"], _I32T, n, "accepted"),
                           _arg(out["rejected"], _I32T, n, "rejected"),
                           _arg(out["flags"], _U8, n, "flags"), _arg(ws, _U8, None, "ws"),
                           ws.numel(), _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_select")
    kk = k.value
    return (rh.value, kk, out["accepted"][:(u - kk) * group_size],
            out["rejected"][:kk * group_size], out["flags"][:n])


def select_k(unit_score, group_size, k, out=None, ws=None, status=None, stream=None):
    dev = unit_score.device
    u = unit_score.numel()
    n = u * group_size
    if out is None:
        out = {"accepted": torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               "rejected": torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               "flags": torch.empty(max(n, 1), dtype=torch.uint8, device=dev)}
    if ws is None:
        ws = workspace(lib().pace_select_workspace_size(u), dev)
    st = lib().pace_select_k(_arg(unit_score, _F64T, u, "unit_score"), u, int(group_size),
                             int(k), _arg(out["accepted"], _I32T, n, "accepted"),
                             _arg(out["rejected"], _I32T, n, "rejected"),
                             _arg(out["flags"], _U8, n, "flags"), _arg(ws, _U8, None, "ws"),
                             ws.numel(), _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_select_k")
    return (out["accepted"][:(u - k) * group_size], out["rejected"][:k * group_size],
            out["flags"][:n])


# Sharded rejection (pool partitioned by unit across ranks); histograms are
# int32 tensors of SHARD_HIST_BINS (the library's uint32 bins; counts < 2^31).
SHARD_PASSES = 6
SHARD_HIST_BINS = 2048


def select_shard_workspace(n_units, device):
    return workspace(lib().pace_select_shard_workspace_size(int(n_units)), device)


def select_shard_pass(unit_score, pass_, k, hist_prev, hist_out, ws, status=None, stream=None):
    u = unit_score.numel()
    st = lib().pace_select_shard_pass(_arg(unit_score, _F64T, u, "unit_score"), u, int(pass_),
                                      int(k), _arg(hist_prev, _I32T, SHARD_HIST_BINS, "hist_prev"),
                                      _arg(hist_out, _I32T, SHARD_HIST_BINS, "hist_out"),
                                      _arg(ws, _U8, None, "ws"), ws.numel(),
                                      _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_select_shard_pass")


def select_shard_ties(unit_score, hist_last, n_tied_out, ws, status=None, stream=None):
    u = unit_score.numel()
    st = lib().pace_select_shard_ties(_arg(unit_score, _F64T, u, "unit_score"), u,
                                      _arg(hist_last, _I32T, SHARD_HIST_BINS, "hist_last"),
                                      _arg(n_tied_out, _I64T, 1, "n_tied"),
                                      _arg(ws, _U8, None, "ws"), ws.numel(),
                                      _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_select_shard_ties")


def select_shard_write(unit_score, group_size, k, tied_before, id_base, out, ws,
                       n_rejected_out=None, status=None, stream=None):
    """out: {"accepted", "rejected", "flags"} of n_units * group_size entries."""
    u = unit_score.numel()
    n = u * group_size
    st = lib().pace_select_shard_write(_arg(unit_score, _F64T, u, "unit_score"), u,
                                       int(group_size), int(k),
                                       _arg(tied_before, _I64T, 1, "tied_before"), int(id_base),
                                       _arg(out["accepted"], _I32T, n, "accepted"),
                                       _arg(out["rejected"], _I32T, n, "rejected"),
                                       _arg(out["flags"], _U8, n, "flags"),
                                       _arg(n_rejected_out, _I64T, 1, "n_rejected"),
                                       _arg(ws, _U8, None, "ws"), ws.numel(),
                                       _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_select_shard_write")


# ---------------------------------------------------------------- (b) batch

def loss_params(eps_low=0.2, eps_high=0.28, dual_clip=10.0, adv_eps=1e-6,
                agg=AGG_TOKEN_MEAN, std_unbiased=True):
    return PaceLossParams(float(eps_low), float(eps_high), float(dual_clip), float(adv_eps),
                          int(agg), int(bool(std_unbiased)))


def make_batch(seq_offsets, n_rows, seq_accepted=None, mask=None):
    n_seq = seq_offsets.numel() - 1
    b = PaceBatch(_arg(seq_offsets, _I64T, None, "seq_offsets"),
                  _arg(seq_accepted, _U8, n_seq, "seq_accepted"),
                  _arg(mask, _U8, int(n_rows), "mask"), n_seq, int(n_rows))
    b._keep = (seq_offsets, seq_accepted, mask)  # keep the tensors alive with the struct
    return b


def make_loss_args(behav_lp, reward, group_size, params, loss_out, adv_out=None,
                   ratio_out=None, partial_out=None):
    """partial_out (float64 [2], optional) receives the aggregate's numerator and
    denominator, which ranks holding parts of one batch add before dividing."""
    a = PaceLossArgs(_arg(behav_lp, _F32T, None, "behav_lp"), _arg(reward, _F32T, None, "reward"),
                     int(group_size), params, _arg(loss_out, _F64T, 1, "loss"),
                     _arg(adv_out, _F32T, reward.numel(), "adv"),
                     _arg(ratio_out, _F32T, behav_lp.numel(), "ratio"),
                     _arg(partial_out, _F64T, 2, "partial"))
    a._keep = (behav_lp, reward, loss_out, adv_out, ratio_out, partial_out)
    return a


def loss_from_partial(partial, loss_out, stream=None):
    """loss = partial[0] / partial[1] (0 if the denominator is 0), on the device."""
    st = lib().pace_loss_from_partial(_arg(partial, _F64T, 2, "partial"),
                                      _arg(loss_out, _F64T, 1, "loss"), _stream(stream))
    _check(st, "pace_loss_from_partial")


def group_advantages(reward, group_size, seq_accepted=None, adv_eps=1e-6, std_unbiased=True,
                     out=None, stream=None):
    n = reward.numel()
    if out is None:
        out = torch.empty(n, dtype=torch.float32, device=reward.device)
    st = lib().pace_group_advantages(_arg(reward, _F32T, n, "reward"),
                                     _arg(seq_accepted, _U8, n, "seq_accepted"), n,
                                     int(group_size), float(adv_eps), int(bool(std_unbiased)),
                                     _arg(out, _F32T, n, "out"), _stream(stream))
    _check(st, "pace_group_advantages")
    return out


def token_logprob_workspace_size(n_rows, n_seq, hidden, vocab):
    return lib().pace_token_logprob_workspace_size(int(n_rows), int(n_seq), int(hidden),
                                                   int(vocab))


def _head_shapes(batch: PaceBatch, hidden, w_vocab):
    """(H, V) of a bf16 hidden [>= n_rows, H] / w_vocab [V, H] pair, checked."""
    if hidden.dim() != 2 or w_vocab.dim() != 2 or hidden.shape[1] != w_vocab.shape[1]:
        raise ValueError("hidden must be [n_rows, H] and w_vocab [V, H]")
    if hidden.shape[0] < batch.n_rows:
        raise ValueError(f"hidden has {hidden.shape[0]} rows, the batch {batch.n_rows}")
    return int(hidden.shape[1]), int(w_vocab.shape[0])


def token_logprob(batch: PaceBatch, hidden, w_vocab, targets, temperature=1.0, loss=None,
                  logprob=None, lse=None, ws=None, status=None, stream=None):
    """pace_token_logprob.  hidden [n_rows, H] and w_vocab [V, H] are bf16 tensors."""
    H, V = _head_shapes(batch, hidden, w_vocab)
    n_rows = batch.n_rows
    dev = hidden.device
    if logprob is None:
        logprob = torch.empty(n_rows, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(token_logprob_workspace_size(n_rows, batch.n_seq, H, V), dev)
    st = lib().pace_token_logprob(ctypes.byref(batch), _arg(hidden, _BF16, None, "hidden"),
                                  _arg(w_vocab, _BF16, None, "w_vocab"),
                                  _arg(targets, _I32T, n_rows, "targets"), H, V,
                                  float(temperature), _arg(logprob, _F32T, n_rows, "logprob"),
                                  _arg(lse, _F32T, n_rows, "lse"),
                                  ctypes.byref(loss) if loss is not None else None,
                                  _arg(ws, _U8, None, "ws"), ws.numel(),
                                  _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_token_logprob")
    return logprob


def surrogate_loss(batch: PaceBatch, logprob, loss: PaceLossArgs, ws=None, status=None,
                   stream=None):
    dev = logprob.device
    if ws is None:
        ws = workspace(lib().pace_surrogate_loss_workspace_size(batch.n_rows, batch.n_seq), dev)
    st = lib().pace_surrogate_loss(ctypes.byref(batch),
                                   _arg(logprob, _F32T, batch.n_rows, "logprob"),
                                   ctypes.byref(loss), _arg(ws, _U8, None, "ws"), ws.numel(),
                                   _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_surrogate_loss")


def set_profile_events(kernel: int, begin=None, end=None):
    """Record torch.cuda.Event ``begin`` / ``end`` around every launch of ``kernel``
    (PROFILE_LMHEAD or PROFILE_TAG_REDUCE) on this thread; None turns it off."""
    def handle(ev):
        if ev is None:
            return None
        if not ev.cuda_event:  # torch creates the CUDA event on its first record
            ev.record()
        return ctypes.c_void_p(ev.cuda_event)
    b, e = handle(begin), handle(end)
    _check(lib().pace_set_profile_events(int(kernel), b, e), "pace_set_profile_events")


def set_score_fused_min_traj(min_traj: Optional[int] = None):
    """pace_set_score_fused_min_traj: pools of at least min_traj trajectories finalise
    their scores inside the tag reduction's launch (None: the library's default)."""
    if min_traj is None:
        min_traj = lib().pace_score_fused_min_traj_default()
    _check(lib().pace_set_score_fused_min_traj(int(min_traj)), "pace_set_score_fused_min_traj")


def set_lmhead_splits(splits: int):
    """pace_set_lmhead_splits: vocabulary splits of the LM head on large batches
    (0 = automatic), for the whole process."""
    _check(lib().pace_set_lmhead_splits(int(splits)), "pace_set_lmhead_splits")


def kernel_launches() -> int:
    """Kernels the library has launched from this thread so far."""
    return int(lib().pace_kernel_launches())


def prefix_score(batch: PaceBatch, hidden, w_vocab, targets, behav_lp, temperature=1.0,
                 min_tokens=32, cap_tokens=1024, s_pre=None, logprob=None, ws=None, status=None,
                 stream=None):
    """pace_prefix_score (Eq. 6): float32 s_pre per prefix (NaN = not scored)."""
    H, V = _head_shapes(batch, hidden, w_vocab)
    n_rows = batch.n_rows
    dev = hidden.device
    if s_pre is None:
        s_pre = torch.empty(batch.n_seq, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib().pace_prefix_score_workspace_size(n_rows, batch.n_seq, H, V), dev)
    st = lib().pace_prefix_score(ctypes.byref(batch), _arg(hidden, _BF16, None, "hidden"),
                                 _arg(w_vocab, _BF16, None, "w_vocab"),
                                 _arg(targets, _I32T, n_rows, "targets"),
                                 _arg(behav_lp, _F32T, n_rows, "behav_lp"), H, V,
                                 float(temperature), int(min_tokens), int(cap_tokens),
                                 _arg(s_pre, _F32T, batch.n_seq, "s_pre"),
                                 _arg(logprob, _F32T, n_rows, "logprob"),
                                 _arg(ws, _U8, None, "ws"), ws.numel(),
                                 _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_prefix_score")
    return s_pre


def stale_k(tags, offsets, trainer_version, k_max, kbar=None, admitted=None, ws=None,
            status=None, stream=None):
    """pace_stale_k: (kbar float64, admitted uint8) per trajectory."""
    dev = offsets.device
    n = offsets.numel() - 1
    if kbar is None:
        kbar = torch.empty(n, dtype=torch.float64, device=dev)
    if admitted is None:
        admitted = torch.empty(n, dtype=torch.uint8, device=dev)
    if ws is None:
        ws = workspace(lib().pace_stale_k_workspace_size(n), dev)
    st = lib().pace_stale_k(_arg(tags, _I32T, None, "tags"),
                            _arg(offsets, _I64T, n + 1, "offsets"), n, tags.numel(),
                            int(trainer_version), float(k_max), _arg(kbar, _F64T, n, "kbar"),
                            _arg(admitted, _U8, n, "admitted"), _arg(ws, _U8, None, "ws"),
                            ws.numel(), _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_stale_k")
    return kbar, admitted


def staleness_histogram(values, flags, lo, hi, n_bins, hist=None, status=None, stream=None):
    """pace_staleness_histogram: int32-viewable uint32 counts [2, n_bins] (rejected, accepted)."""
    if hist is None:
        hist = torch.empty(2 * n_bins, dtype=torch.int32, device=values.device)
    n = values.numel()
    st = lib().pace_staleness_histogram(_arg(values, _F64T, n, "values"),
                                        _arg(flags, _U8, n, "flags"), n, float(lo), float(hi),
                                        int(n_bins), _arg(hist, _I32T, 2 * int(n_bins), "hist"),
                                        _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_staleness_histogram")
    return hist.view(2, n_bins)


class ScoreWindow:
    """Device ring window of recent unit scores for quantile_admit (state kept across steps)."""

    def __init__(self, capacity=512, device="cuda"):
        self.values = torch.zeros(capacity, dtype=torch.float64, device=device)
        self.state = torch.zeros(2, dtype=torch.int64, device=device)  # count, next slot


def quantile_admit(unit_score, r_hat, batch_units, window: ScoreWindow, min_obs=32,
                   decision=None, kappa=None, status=None, stream=None):
    """pace_quantile_admit: (decision uint8 [n], kappa float64 [1]); updates ``window``."""
    n = unit_score.numel()
    dev = unit_score.device
    if decision is None:
        decision = torch.empty(max(n, 1), dtype=torch.uint8, device=dev)
    if kappa is None:
        kappa = torch.empty(1, dtype=torch.float64, device=dev)
    st = lib().pace_quantile_admit(_arg(unit_score, _F64T, n, "unit_score"), n, float(r_hat),
                                   int(batch_units), int(min_obs),
                                   _arg(window.values, _F64T, None, "window.values"),
                                   window.values.numel(),
                                   _arg(window.state, _I64T, 2, "window.state"),
                                   _arg(decision, _U8, n, "decision"),
                                   _arg(kappa, _F64T, 1, "kappa"),
                                   _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_quantile_admit")
    return decision[:n], kappa


def surrogate_backward(batch: PaceBatch, logprob, loss: PaceLossArgs, dlp=None, ws=None,
                       status=None, stream=None):
    """pace_surrogate_backward: float32 dLoss/dlp per row."""
    dev = logprob.device
    if dlp is None:
        dlp = torch.empty(batch.n_rows, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib().pace_surrogate_backward_workspace_size(batch.n_rows, batch.n_seq),
                       dev)
    st = lib().pace_surrogate_backward(ctypes.byref(batch),
                                       _arg(logprob, _F32T, batch.n_rows, "logprob"),
                                       ctypes.byref(loss), _arg(dlp, _F32T, batch.n_rows, "dlp"),
                                       _arg(ws, _U8, None, "ws"), ws.numel(),
                                       _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_surrogate_backward")
    return dlp


def token_logprob_backward(batch: PaceBatch, hidden, w_vocab, targets, lse, dlp,
                           temperature=1.0, grad_hidden=None, grad_w=None, ws=None, status=None,
                           stream=None):
    """pace_token_logprob_backward: (grad_hidden fp32 [n_rows, H], grad_w fp32 [V, H])."""
    H, V = _head_shapes(batch, hidden, w_vocab)
    n_rows = batch.n_rows
    dev = hidden.device
    if grad_hidden is None:
        grad_hidden = torch.empty(n_rows, H, dtype=torch.float32, device=dev)
    if grad_w is None:
        grad_w = torch.empty(V, H, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib().pace_token_logprob_backward_workspace_size(n_rows, batch.n_seq, H,
                                                                        V), dev)
    st = lib().pace_token_logprob_backward(ctypes.byref(batch),
                                           _arg(hidden, _BF16, None, "hidden"),
                                           _arg(w_vocab, _BF16, None, "w_vocab"),
                                           _arg(targets, _I32T, n_rows, "targets"), H, V,
                                           float(temperature), _arg(lse, _F32T, n_rows, "lse"),
                                           _arg(dlp, _F32T, n_rows, "dlp"),
                                           _arg(grad_hidden, _F32T, n_rows * H, "grad_hidden"),
                                           _arg(grad_w, _F32T, V * H, "grad_w"),
                                           _arg(ws, _U8, None, "ws"), ws.numel(),
                                           _arg(status, _I32T, 1, "status"), _stream(stream))
    _check(st, "pace_token_logprob_backward")
    return grad_hidden, grad_w
