"""The C ABI from plain C programs, with no Python or torch in their process.

- tests/c/pace_host_c.c (strict C99, -pedantic -Werror) includes include/pace.h,
  links libpace.so and runs the host-only entry points on a machine without a
  GPU: version, status strings, defaults and the rejection budget (Eqs. 3-4),
  compared bit for bit with the oracle.
- tests/c/pace_gpu_c.c (C11) allocates with cudaMalloc and runs scoring,
  selection, the fused log-probs and the fused loss (PaceLossArgs filled in C)
  on the tiny 64-trajectory pool; its outputs are compared with the oracle
  (scores bit for bit, ids exactly, log-probs within 5e-3, loss within 1e-3
  relative)."""
import math
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from paper_2609_36830_gb300 import build as pace_build
from paper_2609_36830_gb300 import workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CDIR = os.path.join(ROOT, "tests", "c")
LIBDIR = os.path.join(ROOT, "paper_2609_36830_gb300")
CUDA_HOME = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _compile(src, out, flags, extra_libs=()):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    pace_build.build()
    cmd = [gcc] + flags + ["-I" + os.path.join(ROOT, "include"), os.path.join(CDIR, src),
                           "-L" + LIBDIR, "-lpace"] + list(extra_libs) + \
          ["-Wl,-rpath," + LIBDIR, "-o", out]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out


def test_host_entry_points_from_c99(tmp_path):
    exe = _compile("pace_host_c.c", str(tmp_path / "pace_host_c"),
                   ["-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror"])
    rng = np.random.default_rng(5)
    cases = [(47, 35, 0.0, 0.9, 0.0, 47), (64, 48, 0.0, 0.9, 0.0, 8), (10, 20, 0.3, 0.9, 0.5, 10)]
    for _ in range(300):
        n = int(rng.integers(0, 2_000_000))
        cases.append((n, int(rng.integers(0, n + 2)), float(rng.choice([0.0, 0.25, 0.9])),
                      float(rng.choice([0.9, 1.0])), float(rng.random()),
                      n // int(rng.choice([1, 8]))))
    stdin = "".join(f"{n} {nt} {b!r} {m!r} {p!r} {u}\n" for n, nt, b, m, p, u in cases)
    r = subprocess.run([exe], input=stdin, capture_output=True, text=True, check=True)
    lines = r.stdout.strip().splitlines()
    assert lines[0] == "version 300"
    assert lines[1] == "status PACE_OK PACE_ERR_TIMEOUT PACE_ERR_UNKNOWN"
    assert lines[2].split()[1:5] == ["0", "4", "32", "8"]
    assert float.fromhex(lines[3].split()[3]) == 0.9
    body = lines[5:]
    assert len(body) == len(cases)
    for (n, nt, b, m, p, u), line in zip(cases, body):
        st, r_, rh, k = line.split()
        ost, orr, orh, ok = oracle.budget(n, nt, b, m, p, u)
        assert int(st) == ost == 0
        assert (float.fromhex(r_), float.fromhex(rh), int(k)) == (orr, orh, ok), (n, nt, b, m, p)


@pytest.mark.gpu
def test_score_select_logprob_from_c(tmp_path):
    if not os.path.exists(os.path.join(CUDA_HOME, "include", "cuda_runtime.h")):
        pytest.skip("no CUDA toolkit headers")
    exe = _compile("pace_gpu_c.c", str(tmp_path / "pace_gpu_c"),
                   ["-std=c11", "-Wall", "-Wextra", "-Werror",
                    "-I" + os.path.join(CUDA_HOME, "include")],
                   ["-L" + os.path.join(CUDA_HOME, "lib64"), "-lcudart",
                    "-Wl,-rpath," + os.path.join(CUDA_HOME, "lib64")])
    pool = workloads.make_pool("tiny")
    rows = workloads.make_rows(pool)
    H, V, G = pool.spec.hidden, pool.spec.vocab, pool.group_size
    hb = workloads.bf16_normal_host((rows.n_rows, H), 1.0, pool.seed + 1)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H), pool.seed + 2)
    offsets = pool.meta["offsets_host"].astype(np.int64)
    tags = np.ascontiguousarray(pool.tags, np.int32)
    n = pool.n_traj
    st_o, olp, _ = oracle.token_logprob(hb, wb, rows.targets)
    assert st_o == 0
    behav = workloads.behaviour_logprob(rows, pool.trainer_version, olp, pool.seed)
    inp = tmp_path / "in.bin"
    with open(inp, "wb") as f:
        np.array([n, tags.size, rows.n_rows, H, V, pool.window.size, G, pool.n_target,
                  pool.trainer_version], np.int64).tofile(f)
        for a, dt in ((tags, np.int32), (offsets, np.int64), (pool.c_version, np.int32),
                      (pool.s_pre, np.float32), (pool.window, np.float32),
                      (rows.row_offsets, np.int64), (rows.mask, np.uint8),
                      (rows.targets, np.int32), (hb, np.uint16), (wb, np.uint16),
                      (behav, np.float32), (pool.reward, np.float32)):
            np.ascontiguousarray(a, dt).tofile(f)
    out = tmp_path / "out.bin"
    eps_l, eps_h = pool.spec.eps_low, pool.spec.eps_high
    r = subprocess.run([exe, str(inp), str(out), repr(eps_l), repr(eps_h)], capture_output=True,
                       text=True)
    assert r.returncode == 0, r.stderr
    raw = out.read_bytes()
    U = n // G
    st = np.frombuffer(raw, np.int32, 5, 0)
    k = int(np.frombuffer(raw, np.int64, 1, 20)[0])
    r_hat = float(np.frombuffer(raw, np.float64, 1, 28)[0])
    o = 36
    unit = np.frombuffer(raw, np.float64, U, o)
    flags = np.frombuffer(raw, np.uint8, n, o + 8 * U)
    lp = np.frombuffer(raw, np.float32, rows.n_rows, o + 8 * U + n)
    o2 = o + 8 * U + n + 4 * rows.n_rows
    loss = float(np.frombuffer(raw, np.float64, 1, o2)[0])
    adv = np.frombuffer(raw, np.float32, n, o2 + 8)
    assert (st == 0).all(), st

    _, *_, ous = oracle.score_pool(tags, offsets, pool.c_version, pool.s_pre,
                                   pool.trainer_version, pool.window, group_size=G)
    assert (unit.view(np.uint64) == ous.view(np.uint64)).all()
    _, _, orh, ok = oracle.budget(n, pool.n_target, 0.0, 0.9, 0.0, U)
    assert (k, r_hat) == (ok, orh)
    _, _, _, oflag = oracle.select(ous, G, ok)
    np.testing.assert_array_equal(flags, oflag)
    in_loss = np.repeat(oflag, np.diff(rows.row_offsets)).astype(bool) & rows.mask.astype(bool)
    assert in_loss.any() and (~in_loss).any()
    assert float(np.abs(lp[in_loss] - olp[in_loss]).max()) <= 5e-3
    assert (lp[~in_loss] == 0).all()
    _, oadv = oracle.group_advantages(pool.reward, G, seq_accepted=oflag,
                                      eps=float(np.float32(1e-6)))
    np.testing.assert_allclose(adv, oadv, rtol=1e-5, atol=1e-6)
    _, oloss, _, _ = oracle.surrogate(olp, behav, rows.row_offsets, oadv, mask=rows.mask,
                                      seq_accepted=oflag, eps_low=float(np.float32(eps_l)),
                                      eps_high=float(np.float32(eps_h)))
    assert abs(loss - oloss) <= 1e-3 * abs(oloss), (loss, oloss)
