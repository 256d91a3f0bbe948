"""The decode comparison itself (CPU): what the tight check accepts and what it rejects.

The GPU parity tests compare decoded bf16 values with the fp64 oracle decode through
cgcheck.compare_decode. Here the oracle's own decode, rounded to bf16, stands in for a perfect
decoder: it must pass with no value outside bf16(ref), while a value moved by two ulps, or by
one ulp where ref is far from a rounding midpoint, must be rejected.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import bf16_rne, compare_decode, decode_eval_bound


def _case(backend):
    if backend == 0:
        w = synth.Workload(name="c", L=1, B=1, H=1, T=200, d=128, group=128, backend=0, bits=4, block=64, residual=0)
    else:
        w = synth.Workload(name="k", L=1, B=1, H=1, T=300, d=128, group=64, backend=1, bits=3, block=128,
                           residual=128)
    x = synth.kv_cache(w, threads=2)
    G = synth.gauges(w)
    ref = oracle.encode(w.shape, w.params, x, G)
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    return w, G, ref, xr


def _bits(v):
    return (v.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def test_bf16_rne_ties_to_even():
    v = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 1.0 + 2.0 ** -8 + 2.0 ** -30])
    np.testing.assert_array_equal(bf16_rne(v), [1.0, 1.0 + 2 * 2.0 ** -7, -1.0, 1.0 + 2.0 ** -7])


@pytest.mark.parametrize("backend", [0, 1])
def test_tight_check_accepts_rounded_reference_and_rejects_slips(backend):
    w, G, ref, xr = _case(backend)
    r = bf16_rne(xr.reshape(-1))
    st = compare_decode(w, _bits(r), xr, G, None, codes=ref["codes"], scales_u16=ref["scales"])
    assert st["tight"] == xr.size and st["tight_not_rne"] == 0
    eb = decode_eval_bound(w, G, ref["codes"], ref["scales"])
    ulp = np.ldexp(1.0, np.frexp(np.abs(r))[1] - 8)
    # the bound is a small fraction of an ulp for typical values
    big = np.abs(r) > 0.5 * np.sqrt(np.mean(r ** 2))
    assert np.median(eb[big] / ulp[big]) < 0.2
    # two ulps off: rejected anywhere
    b2 = _bits(r)
    k = int(np.flatnonzero(big)[7])
    b2[k] += 2
    with pytest.raises(AssertionError):
        compare_decode(w, b2, xr, G, None, codes=ref["codes"], scales_u16=ref["scales"])
    # one ulp off where ref is far (in units of eb) from the rounding midpoint: rejected
    mid_dist = np.abs(np.abs(xr.reshape(-1)) - (np.abs(r) + 0.5 * ulp))
    far = big & (mid_dist > 4 * eb)
    k = int(np.flatnonzero(far)[3])
    b1 = _bits(r)
    b1[k] += 1
    with pytest.raises(AssertionError):
        compare_decode(w, b1, xr, G, None, codes=ref["codes"], scales_u16=ref["scales"])
