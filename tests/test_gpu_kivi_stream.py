"""GPU parity of the KIVI streaming append and stream decode against the CPU oracle.

A KIVI cache that grows by appends (Sec. 4.3 KIVI-style path with a full-precision window)
must hold after every append what the batch KIVI encode of all tokens so far holds (the
oracle's stream functions are pinned to that in test_oracle_stream_pins.py). The GPU stream
state, read back in the batch layout, is compared with the batch oracle element by element
(codes bit-exact except oracle-flagged near-boundary values, scales exact, the raw window
bit-exact) at the flush boundaries T = R + k Gt - 1, R + k Gt, R + k Gt + 1, after a prefill,
one-token appends and ragged chunks; the stream decode is checked against the oracle decode,
also on the oracle's own stream bytes (identical packed input, tight check).
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_codes, compare_decode, compare_scales, scales_as_elements, stream_to_batch

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _wl(**kw):
    base = dict(name="kstream", L=2, B=2, H=2, T=0, d=128, group=64, backend=1, bits=3, block=128, residual=128)
    base.update(kw)
    return synth.Workload(**base)


# (workload, capacity, prefill, append chunk sizes after the prefill)
CASES = {
    # tensor-core keys and values (d = 128, 128-token groups)
    "kivi3_g64_Gt128_R128": (_wl(), 560, 300, [1] * 86 + [128, 3, 40]),
    # CUDA-core keys (16-token groups), small head dim
    "kivi4_g16_Gt16_d64_R8": (_wl(d=64, group=16, bits=4, block=16, residual=8), 120, 5, [1] * 30 + [16, 7, 16, 1, 9]),
    # no window (R = 0): a group flushes as soon as it is complete
    "kivi2_g128_Gt32_R0": (_wl(group=128, bits=2, block=32, residual=0), 200, 31, [1, 1, 30, 32, 2, 31, 1]),
}


def _dev(a, dtype=np.int16):
    return torch.from_numpy(np.ascontiguousarray(a).reshape(-1).view(dtype)).cuda()


def _check(w, x, G, dG, T, T_cap, bufs):
    codes, scales, ring, _ = bufs
    wt = w.replace(T=T)
    ref = oracle.encode(wt.shape, wt.params, np.ascontiguousarray(x[..., :T, :]), G, want_flags=True)
    c, s, r = stream_to_batch(w, T, T_cap, codes.cpu().numpy().view(np.uint8),
                              scales.cpu().numpy().view(np.uint16), ring.cpu().numpy().view(np.uint16))
    mism = compare_codes(wt, c, ref["codes"], ref["flags"])
    compare_scales(s, ref["scales"])
    np.testing.assert_array_equal(r, ref["residual"])
    xr = oracle.decode(wt.shape, wt.params, ref["codes"], ref["scales"], ref["residual"], G)
    out = torch.full((max(xr.size, 8),), -1, dtype=torch.int16, device="cuda")
    sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=T, d=w.d, t0=0, T_cap=T_cap)
    cg.kivi_stream_decode(sh, cg.Params(**w.params), codes, scales, ring, dG, out)
    assert cg.get_status() == 0
    step = scales_as_elements(wt, ref["scales"]) * mism if mism.any() else None
    compare_decode(wt, out.cpu().numpy().view(np.uint16)[: xr.size], xr, G, step, codes=ref["codes"],
                   scales_u16=ref["scales"])
    return int(mism.sum())


@pytest.mark.parametrize("name", list(CASES))
def test_stream_appends_match_batch_encode(name):
    w, T_cap, prefill, chunks = CASES[name]
    T_end = prefill + sum(chunks)
    assert T_end <= T_cap
    x = synth.kv_cache(w.replace(T=T_end), threads=4)
    G = synth.gauges(w)
    dG = _dev(G, np.float32)
    params = cg.Params(**w.params)
    cap = cg.Shape(L=w.L, B=w.B, H=w.H, T=0, d=w.d, t0=0, T_cap=T_cap)
    bufs = cg.kivi_stream_alloc(cap, params)
    R, Gt = w.residual, w.block
    boundaries = {R + k * Gt + o for k in range(1, T_cap // Gt + 1) for o in (-1, 0, 1)}
    t = 0
    for n in [prefill] + chunks:
        sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=n, d=w.d, t0=t, T_cap=T_cap)
        cg.kivi_append(sh, params, _dev(x[..., t:t + n, :]), dG, *bufs)
        t += n
        if t in boundaries or n > 1 or t == T_end:
            _check(w, x, G, dG, t, T_cap, bufs)
    assert cg.get_status() == 0


@pytest.mark.parametrize("name", list(CASES))
def test_stream_decode_of_oracle_bytes(name):
    """The GPU stream decode of the oracle's own stream state: identical packed input, so every
    value gets the tight check."""
    w, T_cap, prefill, chunks = CASES[name]
    T = prefill + sum(chunks[:len(chunks) // 2])
    x = synth.kv_cache(w.replace(T=T), threads=4)
    G = synth.gauges(w)
    shp = dict(L=w.L, B=w.B, H=w.H, d=w.d)
    st = oracle.kivi_stream_alloc(dict(shp, T=0, t0=0, T_cap=T_cap), w.params)
    oracle.kivi_append(dict(shp, T=T, t0=0, T_cap=T_cap), w.params, x, G, *st)
    codes, scales, ring = st
    xr = oracle.kivi_stream_decode(dict(shp, T=T, t0=0, T_cap=T_cap), w.params, codes, scales, ring, G)
    dc = torch.from_numpy(np.concatenate([codes, np.zeros(16, np.uint8)])).cuda()
    ds = _dev(np.concatenate([scales, np.zeros(8, np.uint16)]))
    dr = _dev(ring)
    out = torch.full((xr.size,), -1, dtype=torch.int16, device="cuda")
    cg.kivi_stream_decode(cg.Shape(T=T, t0=0, T_cap=T_cap, **shp), cg.Params(**w.params), dc, ds, dr,
                          _dev(G, np.float32), out)
    assert cg.get_status() == 0
    wt = w.replace(T=T)
    cb, sb, _ = stream_to_batch(w, T, T_cap, codes, scales, ring)
    stt = compare_decode(wt, out.cpu().numpy().view(np.uint16), xr, G, None, codes=cb, scales_u16=sb)
    assert stt["tight"] == xr.size


def test_stream_rejects_long_appends_and_small_workspace():
    w = _wl(L=1, B=1, H=1)
    params = cg.Params(**w.params)
    T_cap = 600
    bufs = cg.kivi_stream_alloc(cg.Shape(L=1, B=1, H=1, T=0, d=w.d, T_cap=T_cap), params)
    x = synth.kv_cache(w.replace(T=400), threads=1)
    dG = _dev(synth.gauges(w), np.float32)
    cg.kivi_append(cg.Shape(L=1, B=1, H=1, T=200, d=w.d, t0=0, T_cap=T_cap), params, _dev(x[..., :200, :]), dG, *bufs)
    with pytest.raises(cg.CodecGaugeError) as e:
        cg.kivi_append(cg.Shape(L=1, B=1, H=1, T=129, d=w.d, t0=200, T_cap=T_cap), params,
                       _dev(x[..., 200:329, :]), dG, *bufs)
    assert e.value.code == -2
    # the append that completes the group at 256 tokens needs the workspace
    with pytest.raises(cg.CodecGaugeError) as e:
        cg.kivi_append(cg.Shape(L=1, B=1, H=1, T=56, d=w.d, t0=200, T_cap=T_cap), params,
                       _dev(x[..., 200:256, :]), dG, *bufs[:3], None)
    assert e.value.code == -1
    assert cg.get_status() == 0
