"""Host check of the FMA-pipe exp2 used by the attention epilogue (`exp2_fma2`).

The device function splits x = j + f (j = floor(x), f in [0, 1)) and evaluates 2^f with a
cubic; this test re-evaluates the same float32 steps in numpy from the coefficients written
in pace_ptx.cuh and checks them against exp2 in double precision, so that a change of the
coefficients or of the range reduction that loses accuracy fails on the CPU.
"""
import re
from pathlib import Path

import numpy as np

PTX = Path(__file__).resolve().parents[1] / "paper_2608_27206_gb300" / "csrc" / "pace_ptx.cuh"


def _coefficients():
    src = PTX.read_text()
    body = src[src.index("float2 exp2_fma2(float2 x)"):]
    body = body[:body.index("\n}\n")]
    vals = [float(v) for v in re.findall(r"make_float2\(([0-9.e+-]+)f,", body)]
    # Horner order in the source: c3, c2, then c1, then c0
    c3, c2, c1, c0 = vals[1], vals[2], vals[3], vals[4]
    return np.float32(c0), np.float32(c1), np.float32(c2), np.float32(c3)


def _emulate(x):
    c0, c1, c2, c3 = _coefficients()
    x = np.maximum(x.astype(np.float32), np.float32(-126.0))
    j = np.floor(x).astype(np.float32)                 # what x + 1.5 * 2^23 rounded down encodes
    f = (x - j).astype(np.float32)
    q = (f * c3 + c2).astype(np.float32)
    q = (q * f + c1).astype(np.float32)
    q = (q * f + c0).astype(np.float32)
    bits = q.view(np.uint32).astype(np.int64) + (j.astype(np.int64) << 23)
    return (bits & 0xFFFFFFFF).astype(np.uint32).view(np.float32)


def test_relative_error_over_range():
    x = np.linspace(-125.0, 0.0, 2_000_001, dtype=np.float32)
    got = _emulate(x).astype(np.float64)
    ref = np.exp2(x.astype(np.float64))
    rel = np.abs(got - ref) / ref
    assert rel.max() < 1e-4, rel.max()
    assert abs(np.mean((got - ref) / ref)) < 2e-5      # no bias that sums would accumulate


def test_lower_clamp_is_tiny_and_non_negative():
    x = np.array([-np.inf, -1e30, -300.0, -127.0, -126.5, -126.0], np.float32)
    y = _emulate(x)
    assert np.all(y >= 0) and np.all(y <= np.float32(2.0 ** -125))
    assert np.all(np.isfinite(y))
