"""Pins of the oracle's KIVI streaming append (CPU only).

A KIVI cache that grows token by token (Sec. 4.3 KIVI-style path with a full-precision
window; the rolling cache of Sec. 4.4) must hold, after every append, exactly what the batch
KIVI encode of all tokens so far holds: the same quantized key groups and value tokens, and
the newest tokens raw. The batch encode is pinned in test_oracle_pins.py; here the stream
state is checked against it through the flush boundaries T = R + Gt - 1, R + Gt, R + Gt + 1,
for one-token appends, ragged chunks and a bulk prefill, and the stream decode against the
batch decode.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import stream_to_batch


def _wl(**kw):
    base = dict(name="k", L=2, B=2, H=2, T=0, d=64, group=16, backend=1, bits=3, block=16, residual=20)
    base.update(kw)
    return synth.Workload(**base)


def _check_state(w, x, G, T, T_cap, st):
    codes, scales, ring = st
    wt = w.replace(T=T)
    ref = oracle.encode(wt.shape, wt.params, np.ascontiguousarray(x[..., :T, :]), G)
    c, s, r = stream_to_batch(w, T, T_cap, codes, scales, ring)
    np.testing.assert_array_equal(c, ref["codes"])
    np.testing.assert_array_equal(s, ref["scales"])
    np.testing.assert_array_equal(r, ref["residual"])
    xs = oracle.kivi_stream_decode(dict(wt.shape, T_cap=T_cap), wt.params, codes, scales, ring, G)
    xb = oracle.decode(wt.shape, wt.params, ref["codes"], ref["scales"], ref["residual"], G)
    np.testing.assert_array_equal(xs, xb)


@pytest.mark.parametrize("bits,Gt,R,g", [(3, 16, 20, 16), (4, 32, 0, 32), (2, 8, 8, 8), (8, 16, 40, 64)])
def test_one_token_appends_equal_batch_encode(bits, Gt, R, g):
    T_cap = R + 3 * Gt + 5
    w = _wl(bits=bits, block=Gt, residual=R, group=g, T=T_cap)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    st = oracle.kivi_stream_alloc(dict(w.shape, T=0, T_cap=T_cap), w.params)
    check_at = {1, R, R + Gt - 1, R + Gt, R + Gt + 1, R + 2 * Gt, T_cap}
    for t in range(T_cap):
        sh = dict(w.shape, T=1, t0=t, T_cap=T_cap)
        oracle.kivi_append(sh, w.params, np.ascontiguousarray(x[..., t:t + 1, :]), G, *st)
        if t + 1 in check_at:
            _check_state(w, x, G, t + 1, T_cap, st)


def test_chunked_appends_and_prefill():
    """A prefill of 45 tokens, then ragged chunks (1, 7, 16, 3, 40, 1): the chunks cross flush
    boundaries and one is longer than a key group."""
    w = _wl(T=120)
    T_cap = 130
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    st = oracle.kivi_stream_alloc(dict(w.shape, T=0, T_cap=T_cap), w.params)
    t = 0
    for n in (45, 1, 7, 16, 3, 40, 1):
        sh = dict(w.shape, T=n, t0=t, T_cap=T_cap)
        oracle.kivi_append(sh, w.params, np.ascontiguousarray(x[..., t:t + n, :]), G, *st)
        t += n
        _check_state(w, x, G, t, T_cap, st)


def test_stream_bytes_closed_form():
    """Codes and scales as the batch layout at T_cap tokens; the ring holds R + Gt tokens."""
    w = _wl()
    for T_cap in (1, 20, 36, 37, 100):
        cap = dict(w.shape, T=0, T_cap=T_cap)
        c, s, r = oracle.kivi_stream_bytes(cap, w.params)
        bc, bs, _ = oracle.packed_bytes(dict(w.shape, T=T_cap), w.params)
        assert (c, s) == (bc, bs)
        assert r == w.L * 2 * w.B * w.H * (w.residual + w.block) * w.d * 2


def test_stream_rejects_bad_shapes():
    w = _wl()
    with pytest.raises(ValueError):
        oracle.kivi_stream_bytes(dict(w.shape, T=5, t0=10, T_cap=12), w.params)   # t0 + T > T_cap
    with pytest.raises(ValueError):
        oracle.kivi_stream_bytes(dict(w.shape, T=0, T_cap=0), w.params)           # no capacity
    with pytest.raises(ValueError):
        oracle.kivi_stream_bytes(dict(w.shape, T=1, T_cap=8), dict(w.params, backend=0))
