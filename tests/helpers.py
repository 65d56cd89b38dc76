"""Shared test helpers: tolerances, oracle fan-out over a spawn pool, device transfer."""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np
import torch

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import synth

RTOL = 2e-3          # scores: relative error bound for bf16 inputs with fp32 accumulation


def assert_scores_close(got, ref, rtol=RTOL, atol_frac=1e-6, atol=0.0, what=""):
    """|got - ref| <= rtol |ref| + atol_frac max|ref| + atol, element by element."""
    got = np.asarray(got, dtype=np.float64).reshape(-1)
    ref = np.asarray(ref, dtype=np.float64).reshape(-1)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    if ref.size == 0:
        return
    scale = float(np.abs(ref).max())
    tol = rtol * np.abs(ref) + atol_frac * scale + atol
    err = np.abs(got - ref)
    bad = np.nonzero(~(err <= tol))[0]
    assert bad.size == 0, (f"{what}: {bad.size}/{ref.size} out of tolerance; worst idx {bad[np.argmax(err[bad])]} "
                           f"got {got[bad[np.argmax(err[bad])]]} ref {ref[bad[np.argmax(err[bad])]]}; "
                           f"max rel err {np.max(err / np.maximum(np.abs(ref), 1e-300)):.3e}")


def assert_distances_close(got, ref, what=""):
    """APC distances d_i (Eq. 4): |got - ref| <= 2e-3 |ref| + 1e-5 element by element.

    The 1e-5 absolute term is there for distances whose exact value is 0 (identical tokens);
    every other d_i is held to the relative bound alone."""
    assert_scores_close(got, ref, rtol=RTOL, atol_frac=0.0, atol=1e-5, what=what)


def assert_kept_matches(kept_gpu, s_final_ref, K, offset=0, rtol=RTOL):
    """Kept set equals the oracle's except for tokens within rtol of the K-th score."""
    kept = np.asarray(kept_gpu, dtype=np.int64) - offset
    assert kept.size == K, (kept.size, K)
    if K == 0:
        return
    assert np.all(np.diff(kept) > 0), "kept indices must be strictly ascending"
    n = len(s_final_ref)
    assert kept.min() >= 0 and kept.max() < n
    ref = O.top_k_ascending(s_final_ref, K)
    thr = np.sort(s_final_ref)[::-1][K - 1]
    ambiguous = np.abs(s_final_ref - thr) <= rtol * abs(thr) + 1e-12
    a, b = set(kept.tolist()), set(ref.tolist())
    diff = (a ^ b)
    assert all(ambiguous[i] for i in diff), f"{len(diff)} kept tokens differ away from the threshold"


def oracle_vit(Q64, K64, cu, scale, merge=4, pool=None):
    """Oracle S_vis; with a pool, each (image, head) goes to one worker."""
    if pool is None:
        return O.vit_attn_importance(Q64, K64, cu, scale, merge)
    jobs, keys = [], []
    for b in range(len(cu) - 1):
        s0, s1 = int(cu[b]), int(cu[b + 1])
        for h in range(Q64.shape[1]):
            jobs.append((np.ascontiguousarray(Q64[s0:s1, h]), np.ascontiguousarray(K64[s0:s1, h]), scale))
            keys.append(b)
    res = pool.starmap(O.received_attention, jobs, chunksize=1)
    out = []
    for b in range(len(cu) - 1):
        a = sum(r for r, kb in zip(res, keys) if kb == b)
        out.append(a.reshape(-1, merge).sum(axis=1))
    return np.concatenate(out)


def spawn_pool(n=None):
    """Process pool for the oracle, started with 'spawn' (never forked from a CUDA process)."""
    n = n or os.cpu_count() or 4
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"
    try:
        return mp.get_context("spawn").Pool(n)
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def bf16_tensor(bits: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 bf16 bit patterns -> torch.bfloat16 tensor on the device (bit-exact)."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device)


def f64(bits: np.ndarray) -> np.ndarray:
    return synth.bf16_bits_to_f64(bits)
