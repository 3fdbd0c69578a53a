"""The polynomial 2^x of the scoring epilogues (ex2_poly in csrc/ptx.cuh): its constants are
read from the source and its fp32 arithmetic replayed step by step, then compared with 2^x in
fp64.  The bound 3e-7 relative is that of the hardware ex2.approx it stands in for."""
import os
import re

import numpy as np

SRC = os.path.join(os.path.dirname(__file__), "..", "paper_2607_16213_gb300", "csrc", "ptx.cuh")


def _poly_constants():
    body = open(SRC).read()
    body = body[body.index("float ex2_poly(float x)"):]
    body = body[:body.index("\n}\n")]
    c5 = float(re.search(r"float p = ([0-9.eE+-]+)f;", body).group(1))
    rest = [float(v) for v in re.findall(r"p = fmaf\(p, f, ([0-9.eE+-]+)f\);", body)]
    return np.float32(c5), [np.float32(v) for v in rest]


def ex2_poly_replay(x):
    """The kernel's steps in fp32: clamp, round by 1.5 * 2^23, Horner, exponent add."""
    f32 = np.float32
    c5, rest = _poly_constants()
    x = np.maximum(x.astype(f32), f32(-127.0))
    magic = f32(12582912.0)
    t = (x + magic).astype(f32)
    f = (x - (t - magic).astype(f32)).astype(f32)
    p = np.full_like(f, c5)
    for c in rest:
        p = (p.astype(np.float64) * f + c).astype(f32)  # fmaf: one rounding
    n = t.view(np.int32) - np.array([magic], dtype=f32).view(np.int32)[0]
    return (p.view(np.int32) + (n << 23)).view(f32)


def test_constants_are_five_fmas():
    c5, rest = _poly_constants()
    assert len(rest) == 5 and abs(float(rest[-1]) - 1.0) < 1e-6 and abs(float(rest[-2]) - np.log(2)) < 1e-4


def test_relative_error_bound():
    x = np.concatenate([np.linspace(-126.0, 0.0, 2_000_001), -np.geomspace(1e-8, 126.0, 200_001), [0.0, -0.5, -1.0]])
    x = x.astype(np.float32)
    got = ex2_poly_replay(x).astype(np.float64)
    want = np.exp2(x.astype(np.float64))
    rel = np.abs(got / want - 1.0)
    assert rel.max() < 3e-7, rel.max()


def test_integers_and_halves_exact_enough():
    x = np.arange(-126, 1, dtype=np.float32)
    got = ex2_poly_replay(x).astype(np.float64)
    assert np.all(np.abs(got / np.exp2(x.astype(np.float64)) - 1.0) < 2e-7)
