"""The error bound behind the keys-only re-encode's fast rotation (host arithmetic, no GPU).

The kernel rotates a key pair (x, y) by cos/sin held as float pairs (hi, lo) split from
fp64.  Its fast form drops the low parts and rounds one product:
    r = RN32(x ch - RN32(y sh)),   t = RN32(y ch + RN32(x sh)),
and it falls back to the compensated products wherever |r| or |t| < 2^-13 max(|x|, |y|) (or
max(|x|, |y|) < 2^-100).  The bound in kvlink_rope.cuh says every result kept from the fast
form rounds to bf16 within one ulp of the correctly rounded fp64 rotation (Sec. 2.2: the key
rotated by its position delta).  This test draws bf16 keys at random angles up to the
workloads' positions, half of them chosen to cancel, emulates the fast form in float32
(numpy: the product inside the FMA is exact in float64, then one rounding to float32), and
checks (a) the kept results are within one bf16 ulp, (b) without the fallback they would not
be (so the threshold is doing work), (c) random keys rarely need the fallback.
"""
import numpy as np


def _bf16(x64):
    """Round to nearest even bf16, returned as float32 values."""
    u = np.asarray(x64, np.float64).astype(np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def _ordinal(b):
    u = (b.view(np.uint32) >> 16).astype(np.int64)
    return np.where(u & 0x8000, -(u & 0x7FFF), u)


def _f32(x):
    return np.asarray(x, np.float64).astype(np.float32).astype(np.float64)


def test_fast_rotation_within_one_ulp_where_kept():
    rng = np.random.default_rng(20250222)
    n = 1_000_000
    x = _bf16(rng.standard_normal(n)).astype(np.float64)
    ang = rng.uniform(0.0, 2 * np.pi, n) * rng.uniform(0.0, 52000.0, n)
    c64, s64 = np.cos(ang), np.sin(ang)
    adv = rng.random(n) < 0.5
    near = x * c64 / np.where(np.abs(s64) > 1e-3, s64, 1.0)
    y = np.where(adv, near * (1 + rng.standard_normal(n) * 2.0 ** -rng.integers(6, 30, n)), rng.standard_normal(n))
    y = _bf16(y).astype(np.float64)
    ch, sh = _f32(c64), _f32(s64)
    r = _f32(x * ch - _f32(y * sh))
    t = _f32(y * ch + _f32(x * sh))
    m = np.maximum(np.abs(x), np.abs(y))
    lim = _f32(2.0 ** -13 * m)
    hard = (np.abs(r) < lim) | (np.abs(t) < lim) | (m < 2.0 ** -100)
    dr = np.abs(_ordinal(_bf16(r)) - _ordinal(_bf16(x * c64 - y * s64)))
    dt = np.abs(_ordinal(_bf16(t)) - _ordinal(_bf16(y * c64 + x * s64)))
    kept = ~hard
    assert dr[kept].max() <= 1 and dt[kept].max() <= 1
    assert max(dr.max(), dt.max()) > 100          # cancellation: the fallback is needed
    assert hard[~adv].mean() < 1e-3               # random keys rarely take it
