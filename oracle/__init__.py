"""PACE oracle: plain fp64 CPU implementation of the hot path, for testing only.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package.  The
CUDA library never calls it, and it shares no code with the CUDA library; the
two meet only in the seeded input generators of
``paper_2609_36830_gb300.workloads``.

The arithmetic lives in ``pace_oracle.c`` (plain C, fp64, FP contraction off);
this module compiles it with gcc on first use and wraps each function with
numpy marshalling.  Every wrapper returns ``(status, outputs...)``; status 0
is success and the other codes read the same as the library's.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pace_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libpace_oracle.so")
_lock = threading.Lock()
_lib = None

OK, ERR_INVALID_ARG, ERR_VERSION_ORDER, ERR_NAN_INPUT = 0, 1, 2, 3
MODE_EFF, MODE_RAW, MODE_GEN = 0, 1, 2
AGG_TOKEN_MEAN, AGG_SEQ_MEAN_TOKEN_MEAN = 0, 1

_P = ctypes.c_void_p
_I32, _I64, _F64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double


def build(force: bool = False) -> str:
    """Compile ``pace_oracle.c`` into ``oracle/_build/libpace_oracle.so``."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-pthread", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            sig = {
                "oracle_policy_lag": [_P, _P, _I64, _I32, _P, _P, _P],
                "oracle_staleness": [_P, _P, _P, _I64, _I64, _I32, _P, _P, _P, _P],
                "oracle_score_pool": [_P, _P, _P, _P, _I64, _I64, _I32, _P, _I64, _I32, _I32,
                                      _I32, _F64, _I32, _P, _P, _P, _P, _P],
                "oracle_budget": [_I64, _I64, _F64, _F64, _F64, _I64, _P, _P, _P],
                "oracle_select": [_P, _I64, _I32, _I64, _P, _P, _P],
                "oracle_token_logprob": [_P, _P, _P, _P, _I64, _I32, _I32, _F64, _P, _P, _I32],
                "oracle_group_advantages": [_P, _P, _I64, _I32, _F64, _I32, _P],
                "oracle_surrogate": [_P, _P, _P, _P, _P, _I64, _P, _F64, _F64, _F64, _I32, _P,
                                     _P, _P],
                "oracle_prefix_score": [_P, _P, _P, _P, _I64, _I32, _I32, _P],
                "oracle_stale_k": [_P, _P, _I64, _I32, _F64, _P, _P],
                "oracle_histogram": [_P, _P, _I64, _F64, _F64, _I32, _P],
                "oracle_quantile_admit": [_P, _I64, _F64, _I64, _I32, _P, _I64, _P, _P, _P, _P],
                "oracle_surrogate_grad": [_P, _P, _P, _P, _P, _I64, _P, _F64, _F64, _F64, _I32,
                                          _P],
                "oracle_lmhead_backward": [_P, _P, _P, _P, _I64, _I32, _I32, _F64, _P, _P, _I32],
                "oracle_lmhead_backward_magnitude": [_P, _P, _P, _P, _I64, _I32, _I32, _F64, _P,
                                                     _P, _I32],
            }
            for name, args in sig.items():
                fn = getattr(lib, name)
                fn.argtypes = args
                fn.restype = ctypes.c_int
            lib.oracle_ecdf.argtypes = [_P, _I64, ctypes.c_float]
            lib.oracle_ecdf.restype = ctypes.c_double
            lib.oracle_sharpen.argtypes = [ctypes.c_double, _I32]
            lib.oracle_sharpen.restype = ctypes.c_double
            _lib = lib
    return _lib


def _c(a, dtype):
    """Contiguous numpy copy of ``a`` in ``dtype`` (None stays None)."""
    if a is None:
        return None
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def _ptr(a):
    return None if a is None else a.ctypes.data


def policy_lag(tags, offsets, j):
    """Eq. 1: token-weighted policy lag per trajectory."""
    tags, offsets = _c(tags, np.int32), _c(offsets, np.int64)
    n = offsets.size - 1
    s, t, k = np.zeros(n, np.int64), np.zeros(n, np.int64), np.zeros(n, np.float64)
    st = _load().oracle_policy_lag(_ptr(tags), _ptr(offsets), n, int(j), _ptr(s), _ptr(t), _ptr(k))
    return st, s, t, k


def staleness(tags, offsets, c_version, j):
    """Lemma 1 / Eq. 2: (status, gen_sum, n_policy_tokens, K_gen, K_wait)."""
    tags, offsets, c = _c(tags, np.int32), _c(offsets, np.int64), _c(c_version, np.int32)
    n = offsets.size - 1
    s, t = np.zeros(n, np.int64), np.zeros(n, np.int64)
    kg, kw = np.zeros(n, np.float64), np.zeros(n, np.float64)
    st = _load().oracle_staleness(_ptr(tags), _ptr(offsets), _ptr(c), n, tags.size, int(j),
                                  _ptr(s), _ptr(t), _ptr(kg), _ptr(kw))
    return st, s, t, kg, kw


def ecdf(window, s):
    """Eq. 9: right-continuous empirical CDF of the float32 window at s."""
    w = _c(window, np.float32)
    return _load().oracle_ecdf(_ptr(w), w.size, float(np.float32(s)))


def sharpen(q, gamma):
    """Eq. 10: phi_gamma(q) for integer gamma."""
    return _load().oracle_sharpen(float(q), int(gamma))


def score_pool(tags, offsets, c_version, s_pre, j, window, mode=MODE_EFF, gamma=4, min_obs=32,
               f_missing=1.0, group_size=8):
    """Eqs. 2, 7-10 and group means: (status, kgen, kwait, weight, score, unit_score)."""
    tags, offsets = _c(tags, np.int32), _c(offsets, np.int64)
    c, sp, w = _c(c_version, np.int32), _c(s_pre, np.float32), _c(window, np.float32)
    n = offsets.size - 1
    out = [np.zeros(n, np.float64) for _ in range(4)]
    us = np.zeros(max(n // max(group_size, 1), 0), np.float64)
    st = _load().oracle_score_pool(_ptr(tags), _ptr(offsets), _ptr(c), _ptr(sp), n, tags.size,
                                   int(j), _ptr(w), w.size, int(mode), int(gamma), int(min_obs),
                                   float(f_missing), int(group_size), *[_ptr(o) for o in out],
                                   _ptr(us))
    return (st, *out, us)


def budget(n_traj, n_target, beta, r_max, r_hat_prev, n_units):
    """Eqs. 3-4 with the cap: (status, r, r_hat, k_units)."""
    r, rh, k = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    st = _load().oracle_budget(int(n_traj), int(n_target), float(beta), float(r_max),
                               float(r_hat_prev), int(n_units), ctypes.byref(r),
                               ctypes.byref(rh), ctypes.byref(k))
    return st, r.value, rh.value, k.value


def select(unit_score, group_size, k):
    """Top-k rejection: (status, accepted_ids, rejected_ids, traj_accepted)."""
    us = _c(unit_score, np.float64)
    u = us.size
    acc = np.zeros((u - k) * group_size, np.int32)
    rej = np.zeros(k * group_size, np.int32)
    flag = np.zeros(u * group_size, np.uint8)
    st = _load().oracle_select(_ptr(us), u, int(group_size), int(k), _ptr(acc), _ptr(rej),
                               _ptr(flag))
    return st, acc, rej, flag


def token_logprob(hidden_bits, w_bits, targets, rows=None, temperature=1.0, n_threads=None):
    """Per-row log-probabilities in fp64 from bf16 bit patterns (uint16 arrays).

    ``hidden_bits`` is [n_rows_total, H], ``w_bits`` is [V, H]; ``rows`` picks the
    rows to compute (default: all).  Returns (status, logprob, lse) for those rows.
    """
    hb = _c(hidden_bits, np.uint16)
    wb = _c(w_bits, np.uint16)
    tg = _c(targets, np.int32)
    H = hb.shape[1]
    V = wb.shape[0]
    assert wb.shape[1] == H
    rid = _c(rows, np.int64) if rows is not None else None
    n = rid.size if rid is not None else hb.shape[0]
    lp, lse = np.zeros(n, np.float64), np.zeros(n, np.float64)
    if n_threads is None:
        n_threads = os.cpu_count() or 1
    st = _load().oracle_token_logprob(_ptr(hb), _ptr(wb), _ptr(tg), _ptr(rid), n, H, V,
                                      float(temperature), _ptr(lp), _ptr(lse), int(n_threads))
    return st, lp, lse


def group_advantages(reward, group_size, seq_accepted=None, eps=1e-6, unbiased=True):
    """GRPO within-group standardisation: (status, adv fp64)."""
    r = _c(reward, np.float32)
    acc = _c(seq_accepted, np.uint8)
    adv = np.zeros(r.size, np.float64)
    st = _load().oracle_group_advantages(_ptr(r), _ptr(acc), r.size, int(group_size), float(eps),
                                         int(bool(unbiased)), _ptr(adv))
    return st, adv


def surrogate(logprob, behav_lp, seq_offsets, adv, mask=None, seq_accepted=None, eps_low=0.2,
              eps_high=0.28, dual_clip=10.0, agg=AGG_TOKEN_MEAN):
    """Clipped surrogate: (status, loss, ratio per row, loss term per row)."""
    lp, bl = _c(logprob, np.float64), _c(behav_lp, np.float64)
    so, a = _c(seq_offsets, np.int64), _c(adv, np.float64)
    m, sa = _c(mask, np.uint8), _c(seq_accepted, np.uint8)
    n_rows = lp.size
    loss = ctypes.c_double()
    ratio, term = np.zeros(n_rows, np.float64), np.zeros(n_rows, np.float64)
    st = _load().oracle_surrogate(_ptr(lp), _ptr(bl), _ptr(m), _ptr(so), _ptr(sa), so.size - 1,
                                  _ptr(a), float(eps_low), float(eps_high), float(dual_clip),
                                  int(agg), ctypes.byref(loss), _ptr(ratio), _ptr(term))
    return st, loss.value, ratio, term


def prefix_score(logprob, behav_lp, seq_offsets, mask=None, min_tokens=32, cap_tokens=1024):
    """Eq. 6 Prefix Forgetting Score per prefix: (status, s_pre fp64, NaN = not scored)."""
    lp, bl = _c(logprob, np.float64), _c(behav_lp, np.float64)
    so, m = _c(seq_offsets, np.int64), _c(mask, np.uint8)
    out = np.zeros(so.size - 1, np.float64)
    st = _load().oracle_prefix_score(_ptr(lp), _ptr(bl), _ptr(m), _ptr(so), so.size - 1,
                                     int(min_tokens), int(cap_tokens), _ptr(out))
    return st, out


def stale_k(tags, offsets, j, k_max):
    """Stale-k admission: (status, kbar fp64, admitted uint8)."""
    tags, offsets = _c(tags, np.int32), _c(offsets, np.int64)
    n = offsets.size - 1
    kbar, adm = np.zeros(n, np.float64), np.zeros(n, np.uint8)
    st = _load().oracle_stale_k(_ptr(tags), _ptr(offsets), n, int(j), float(k_max), _ptr(kbar),
                                _ptr(adm))
    return st, kbar, adm


def histogram(values, flags, lo, hi, n_bins):
    """(status, hist uint32 [2, n_bins]): row 0 rejected (flag 0), row 1 accepted."""
    v = _c(values, np.float64)
    f = _c(flags, np.uint8)
    h = np.zeros(2 * n_bins, np.uint32)
    st = _load().oracle_histogram(_ptr(v), _ptr(f), v.size, float(lo), float(hi), int(n_bins),
                                  _ptr(h))
    return st, h.reshape(2, n_bins)


class Window:
    """Ring window of recently observed scores (state of oracle_quantile_admit)."""

    def __init__(self, capacity):
        self.values = np.zeros(capacity, np.float64)
        self.count = 0
        self.head = 0


def quantile_admit(scores, r, batch_units, window: Window, min_obs=32):
    """Sec. 3.1 / Algorithm 1 rule; updates ``window``: (status, decision uint8, kappa)."""
    sc = _c(scores, np.float64)
    dec = np.zeros(sc.size, np.uint8)
    cnt, hd, kap = ctypes.c_int64(window.count), ctypes.c_int64(window.head), ctypes.c_double()
    st = _load().oracle_quantile_admit(_ptr(sc), sc.size, float(r), int(batch_units),
                                       int(min_obs), _ptr(window.values), window.values.size,
                                       ctypes.byref(cnt), ctypes.byref(hd), _ptr(dec),
                                       ctypes.byref(kap))
    window.count, window.head = cnt.value, hd.value
    return st, dec, kap.value


def surrogate_grad(logprob, behav_lp, seq_offsets, adv, mask=None, seq_accepted=None,
                   eps_low=0.2, eps_high=0.28, dual_clip=10.0, agg=AGG_TOKEN_MEAN):
    """dLoss/dlp per row of the clipped surrogate: (status, dlp fp64)."""
    lp, bl = _c(logprob, np.float64), _c(behav_lp, np.float64)
    so, a = _c(seq_offsets, np.int64), _c(adv, np.float64)
    m, sa = _c(mask, np.uint8), _c(seq_accepted, np.uint8)
    out = np.zeros(lp.size, np.float64)
    st = _load().oracle_surrogate_grad(_ptr(lp), _ptr(bl), _ptr(m), _ptr(so), _ptr(sa),
                                       so.size - 1, _ptr(a), float(eps_low), float(eps_high),
                                       float(dual_clip), int(agg), _ptr(out))
    return st, out


def lmhead_backward(hidden_bits, w_bits, targets, g, temperature=1.0, with_dw=True,
                    n_threads=None, magnitude=False):
    """(status, dH fp64 [n_rows, H], dW fp64 [V, H] or None) for dLoss/dlp = g.

    magnitude=True returns instead the error scales sum_v |G_rv| |W_vk| and
    sum_r |G_rv| |h_rk| (a relative error e in each G_rv moves dH and dW by at
    most e times these, element by element)."""
    hb, wb = _c(hidden_bits, np.uint16), _c(w_bits, np.uint16)
    tg, gg = _c(targets, np.int32), _c(g, np.float64)
    n, H = hb.shape
    V = wb.shape[0]
    dh = np.zeros((n, H), np.float64)
    dw = np.zeros((V, H), np.float64) if with_dw else None
    if n_threads is None:
        n_threads = min(os.cpu_count() or 1, 64)
    fn = (_load().oracle_lmhead_backward_magnitude if magnitude
          else _load().oracle_lmhead_backward)
    st = fn(_ptr(hb), _ptr(wb), _ptr(tg), _ptr(gg), n, H, V,
                                        float(temperature), _ptr(dh), _ptr(dw), int(n_threads))
    return st, dh, dw
