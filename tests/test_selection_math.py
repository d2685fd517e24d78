"""Host checks of the arithmetic the coverage vote (csrc/select.cu) rests on.

1. Fixed-point weights. The kernel weighs a key of non-negative float value x
   as x * 2^shift rounded to the nearest integer (ties to even), saturated at
   2^64 - 1, in integer arithmetic: x = mant * 2^(e - 150) with the 24-bit
   significand mant, shifted left by s = e - 150 + shift, or right by r = -s
   as (mant + 2^(r-1) - 1 + bit r of mant) >> r with r clamped to [1, 31].
   The same steps are restated here with numpy integers and compared with
   float64 rounding of the exact product (x has 24 significant bits, so
   x * 2^shift is exact in float64 and numpy's rint rounds half to even).

2. The bound on the cover set's last key. With weights w (key desc, index
   asc order), target = min(total, ceil(tau * total)) and the cover set the
   shortest prefix whose weight reaches the target, its last key weighs at
   least (total - target + 1) // n when target >= 1: the keys before it
   weigh at most target - 1 and the at most n - 1 after it at most as much as
   it does. The kernel decides the cover among the keys above that bound
   alone (with total 0 no key reaches the bound and it takes its first-digit
   path).
"""
import math

import numpy as np
import pytest


def weight_steps(bits: np.ndarray, shift: int) -> np.ndarray:
    """The kernel's integer weight of float32 bit patterns (non-negative)."""
    u = bits.astype(np.int64) & 0x7FFFFFFF
    e = u >> 23
    mant = (u & 0x7FFFFF) | 0x800000
    s = e - 150 + shift
    r = np.clip(-s, 1, 31)
    small = (mant + ((np.int64(1) << (r - 1)) - 1) + ((mant >> r) & 1)) >> r
    big = mant.astype(np.uint64) << np.clip(s, 0, 40).astype(np.uint64)
    w = np.where(s >= 0, big, small.astype(np.uint64))
    return np.where((e == 255) | (s > 40), np.uint64(2**64 - 1), w)


def weight_reference(bits: np.ndarray, shift: int) -> np.ndarray:
    with np.errstate(invalid="ignore"):   # NaN patterns (saturated below, as in the kernel)
        x = bits.astype(np.uint32).view(np.float32).astype(np.float64)
    v = x * 2.0 ** shift
    out = np.empty(bits.shape, dtype=np.uint64)
    sat = ~np.isfinite(v) | (v >= 2.0 ** 64)
    out[sat] = np.uint64(2**64 - 1)
    ok = ~sat
    out[ok] = np.rint(v[ok]).astype(np.uint64)
    return out


def _patterns(rng):
    # every exponent with edge significands, halfway cases at each right shift,
    # and random patterns
    exps = np.arange(0, 256, dtype=np.int64)
    sig = np.array([0, 1, 2, 0x3FFFFF, 0x400000, 0x400001, 0x7FFFFE, 0x7FFFFF], dtype=np.int64)
    edge = (exps[:, None] << 23) | sig[None, :]
    half = []
    for r in range(1, 26):   # significands with exactly the half bit below the cut
        for low in (1 << (r - 1), (1 << (r - 1)) | 1, (1 << r) - 1):
            m = ((0x2A5A5A5 >> 0) & ~((1 << r) - 1) & 0x7FFFFF) | (low & 0x7FFFFF)
            for e in range(100, 140):
                half.append((e << 23) | m)
                half.append((e << 23) | (m ^ (1 << r)))
    rnd = rng.integers(0, 0x7F800001, size=400_000, dtype=np.int64)
    return np.concatenate([edge.ravel(), np.array(half, dtype=np.int64), rnd])


@pytest.mark.parametrize("shift", [40, 39, 24, 17, 1, 0])
def test_fixed_point_weight_is_round_half_even(shift):
    bits = _patterns(np.random.default_rng(shift))
    got = weight_steps(bits, shift)
    want = weight_reference(bits, shift)
    bad = np.nonzero(got != want)[0]
    assert bad.size == 0, [(hex(int(bits[i])), int(got[i]), int(want[i])) for i in bad[:5]]


def _cover_last(w: np.ndarray, target: int) -> int:
    """Position (in key desc, index asc order) of the cover set's last key."""
    order = np.lexsort((np.arange(w.size), -w.astype(np.float64)))
    # the weights fit in 2^53 here, so float64 keys order them exactly
    cum = np.cumsum(w[order].astype(object))
    for pos, c in enumerate(cum):
        if c >= target:
            return int(order[pos])
    return int(order[-1])


@pytest.mark.parametrize("tau", [0.5, 0.95, float(np.float32(0.95)), 0.999])
@pytest.mark.parametrize("kind", ["lognormal", "flat", "ties", "zeros"])
def test_last_cover_key_weighs_at_least_the_bound(tau, kind):
    rng = np.random.default_rng([int(tau * 1e6), ["lognormal", "flat", "ties", "zeros"].index(kind)])
    # (seeded per case, independent of the interpreter's hash seed)
    for n in (1, 2, 7, 300, 4000):
        if kind == "lognormal":
            x = np.exp(rng.normal(0.0, 3.0, n))
        elif kind == "flat":
            x = rng.uniform(0.5, 1.0, n)
        elif kind == "ties":
            x = rng.integers(1, 4, n) * 0.25
        else:
            x = np.where(rng.random(n) < 0.7, 0.0, rng.uniform(0.0, 1.0, n))
        x = (x / max(x.sum(), 1e-30) * 112.0).astype(np.float32)
        w = weight_steps(x.view(np.uint32).astype(np.int64), 40).astype(object)
        total = int(sum(w))
        target = min(total, math.ceil(tau * total))
        lb = (total - target + 1) // n
        if target == 0:
            # all weights 0: no key reaches a positive bound, the kernel
            # collects no candidate and takes its first-digit path instead
            assert max(w) == 0 and (lb == 0 or lb > max(w))
            continue
        last = _cover_last(np.array(w, dtype=np.float64), target)
        assert int(w[last]) >= lb, (kind, tau, n, int(w[last]), lb)
