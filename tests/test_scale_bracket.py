"""The division-free scale decision of the tensor-core row encoder (CPU, float32 arithmetic).

The encoder decides the fp16 scale s = fp16(fl((max - min) / qmax)) of a block from the two ends
d of its range interval without dividing: it forms fl(fl(d * fl(1/qmax)) * (1 -+ 2^-21)) and
takes the scale as decided when both ends round to the same fp16 value. That is exact only if
the two products bracket the IEEE quotients fl(d / qmax) (fp16 rounding is monotone). numpy's
float32 operations are the same IEEE round-to-nearest operations, so this checks the bracket for
every code width, on random ranges and on ranges whose quotient sits on an fp16 rounding
midpoint or next to it.
"""
import numpy as np
import pytest

F = np.float32
BELOW = F(1.0 - 2.0 ** -21)
ABOVE = F(1.0 + 2.0 ** -21)


def _bracket(d, qmax):
    rq = F(1.0) / F(qmax)
    p = (d * rq).astype(np.float32)
    return (p * BELOW).astype(np.float32), (p * ABOVE).astype(np.float32)


def _fp16_midpoints():
    """Every rounding midpoint between consecutive positive finite fp16 values, as float32."""
    h = np.arange(0, 0x7BFF, dtype=np.uint16)  # finite positive patterns but the largest
    lo = h.view(np.float16).astype(np.float64)
    hi = (h + 1).view(np.float16).astype(np.float64)
    return ((lo + hi) / 2).astype(np.float32)


@pytest.mark.parametrize("bits", [2, 3, 4, 6, 8])
def test_products_bracket_the_quotient(bits):
    qmax = F((1 << bits) - 1)
    rng = np.random.default_rng(bits)
    # ranges over the whole useful fp32 span (log-uniform), with random mantissas
    d = np.exp2(rng.uniform(-40.0, 40.0, 2_000_000)).astype(np.float32)
    n_random = d.size
    # and ranges whose quotient is an fp16 rounding midpoint, or one or two fp32 ulps off it
    mid = _fp16_midpoints()
    for k in (-2, -1, 0, 1, 2):
        t = (mid * qmax).astype(np.float32)
        t = np.nextafter(t, np.float32(np.inf if k > 0 else 0.0)) if k else t
        if abs(k) == 2:
            t = np.nextafter(t, np.float32(np.inf if k > 0 else 0.0))
        d = np.concatenate([d, t[np.isfinite(t) & (t > 0)]])
    q = (d / qmax).astype(np.float32)  # IEEE division, round to nearest even
    lo, hi = _bracket(d, qmax)
    assert np.all(lo <= q) and np.all(q <= hi)
    # hence equal fp16 roundings of the bracket give the quotient's fp16 value (inf above the
    # fp16 range on both sides); the midpoint cases are meant to stay undecided
    with np.errstate(over="ignore"):
        l16, h16, q16 = lo.astype(np.float16), hi.astype(np.float16), q.astype(np.float16)
    same = l16 == h16
    assert same[:n_random].mean() > 0.99
    assert np.array_equal(q16[same], l16[same])


def test_bracket_is_tight_enough_to_decide():
    """The widening is far below the fp16 spacing: away from a midpoint by more than 2^-20
    relative, the bracket always decides."""
    qmax = F(15)
    rng = np.random.default_rng(7)
    d = np.exp2(rng.uniform(-10.0, 10.0, 500_000)).astype(np.float32)
    q = (d / qmax).astype(np.float64)
    h = q.astype(np.float16).astype(np.float64)
    nxt = np.nextafter(q.astype(np.float16), np.float16(np.inf)).astype(np.float64)
    prv = np.nextafter(q.astype(np.float16), np.float16(0)).astype(np.float64)
    dist = np.minimum(np.abs(q - (h + nxt) / 2), np.abs(q - (h + prv) / 2)) / q
    lo, hi = _bracket(d, qmax)
    far = dist > 2.0 ** -20
    assert np.all(lo.astype(np.float16)[far] == hi.astype(np.float16)[far])
