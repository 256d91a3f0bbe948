"""GPU parity: the CUDA path through the C ABI against the CPU oracle, element by element.

Sizes span several 128-token tiles and a ragged tail, every bit width, group size and
block shape the library accepts, KIVI splits with and without a residual window, the
no-compression sanity rows (Sec. 4.4), a rolling append into a history (Sec. 4.4 rolling
compressed-history scoring), empty inputs and the device status bits.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_codes, compare_decode, compare_scales, scales_as_elements

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _wl(**kw):
    base = dict(name="case", L=2, B=1, H=2, T=300, d=128, group=128, backend=0, bits=4, block=64, residual=0)
    base.update(kw)
    return synth.Workload(**base)


CASES = {
    "tiny": synth.WORKLOADS["tiny"],
    "bu4_g128_blk64": _wl(),
    "bu6_g32_blk32": _wl(B=2, T=257, group=32, bits=6, block=32),
    "bu3_g8_blk8_d64": _wl(d=64, group=8, bits=3, block=8, T=130),
    "bu2_g16_blk16_d32": _wl(d=32, group=16, bits=2, block=16, T=129),
    "bu8_g64_blk128_d256": _wl(d=256, group=64, bits=8, block=128, T=140, H=1),
    "bu3_g128_blk128_T1": _wl(group=128, bits=3, block=128, T=1, B=3),
    "bu4_g64_blk16": _wl(group=64, bits=4, block=16, T=384),
    "bu4_g16_blk64_B3": _wl(group=16, bits=4, block=64, T=77, B=3, L=1),
    "kivi3_g64": _wl(backend=1, group=64, bits=3, block=128, residual=128, T=700, B=2),
    "kivi3_T_lt_R": _wl(backend=1, group=64, bits=3, block=128, residual=128, T=100),
    "kivi3_T_eq_R_plus_Gt": _wl(backend=1, group=64, bits=3, block=128, residual=128, T=256),
    "kivi4_g16_blk16_d64": _wl(backend=1, d=64, group=16, bits=4, block=16, residual=8, T=90),
    "kivi2_g32_blk32_R0": _wl(backend=1, group=32, bits=2, block=32, residual=0, T=96),
    "kivi6_g128_blk32": _wl(backend=1, group=128, bits=6, block=32, residual=20, T=150),
    "kivi4_g128_blk128": _wl(backend=1, group=128, bits=4, block=128, residual=16, T=400),
    "kivi3_g32_blk128_B3_R0": _wl(backend=1, group=32, bits=3, block=128, residual=0, T=300, B=3),
    "kivi8_g64_blk128": _wl(backend=1, group=64, bits=8, block=128, residual=128, T=520, L=1, H=3),
    "kivi3_g8_blk128_R0": _wl(backend=1, group=8, bits=3, block=128, residual=0, T=256),
    "kivi4_g16_blk128": _wl(backend=1, group=16, bits=4, block=128, residual=32, T=300),
    "none_g128": _wl(backend=2, group=128, T=260),
    "none_g8_d64": _wl(backend=2, d=64, group=8, T=33),
}


def _dev(x, G):
    return (torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda(),
            torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda())


def _host_u8(t, n):
    return t.cpu().numpy().view(np.uint8)[:n]


def _host_u16(t, nbytes):
    return t.cpu().numpy().view(np.uint16)[: nbytes // 2]


def gpu_encode(w, dx, dG):
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    return codes, scales, resid


def gpu_decode(w, codes, scales, resid, dG, T=None):
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    n = w.L * 2 * w.B * w.H * (T or w.T) * w.d
    out = torch.full((max(n, 8),), -1, dtype=torch.int16, device="cuda")
    cg.decode(shape, params, codes, scales, resid, dG, out)
    return out.cpu().numpy().view(np.uint16)[:n]


@pytest.mark.parametrize("name", list(CASES))
def test_encode_decode_parity(name):
    w = CASES[name]
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx, dG = _dev(x, G)
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, nr = cg.packed_bytes(shape, params)
    assert (nc, ns, nr) == oracle.packed_bytes(w.shape, w.params)
    codes, scales, resid = gpu_encode(w, dx, dG)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G, want_z=True, want_flags=True)
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    if w.backend == 2:
        zg = codes.cpu().numpy().view(np.float32)[: nc // 4]
        np.testing.assert_array_equal(zg, ref["z"])
        step_mism = None
    else:
        mism = compare_codes(w, _host_u8(codes, nc), ref["codes"], ref["flags"])
        compare_scales(_host_u16(scales, ns), ref["scales"])
        step_mism = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    if nr:
        np.testing.assert_array_equal(_host_u16(resid, nr), ref["residual"])
    # end to end: GPU decode of the GPU's own buffers
    got = gpu_decode(w, codes, scales, resid, dG)
    packed = {} if w.backend == 2 else dict(codes=ref["codes"], scales_u16=ref["scales"])
    compare_decode(w, got, xr, G, step_mism, **packed)
    # identical packed input: GPU decode of the oracle's bytes, no flag allowance
    oc = torch.from_numpy(np.concatenate([ref["codes"], np.zeros(16, np.uint8)])).cuda()
    os_ = torch.from_numpy(np.concatenate([ref["scales"], np.zeros(8, np.uint16)]).view(np.int16)).cuda()
    orr = torch.from_numpy(np.concatenate([ref["residual"], np.zeros(8, np.uint16)]).view(np.int16)).cuda()
    got2 = gpu_decode(w, oc, os_, orr, dG)
    st = compare_decode(w, got2, xr, G, None, **packed)
    assert st["tight"] == (xr.size if packed else 0)
    assert cg.get_status() == 0


@pytest.mark.parametrize("kind", ["identity", "hadamard", "dct"])
def test_structured_gauges(kind):
    w = _wl(group=32, bits=4, block=32, T=200)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w, kind)
    dx, dG = _dev(x, G)
    codes, scales, _ = gpu_encode(w, dx, dG)
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    nc, ns, _ = oracle.packed_bytes(w.shape, w.params)
    compare_codes(w, _host_u8(codes, nc), ref["codes"], ref["flags"])
    compare_scales(_host_u16(scales, ns), ref["scales"])


def test_no_compression_round_trip():
    """Sec. 4.4 sanity rows: gauge then inverse with no quantization restores X (1e-5)."""
    w = _wl(backend=2, group=128, T=256, L=2, B=2)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx, dG = _dev(x, G)
    codes, _, _ = gpu_encode(w, dx, dG)
    got = synth.bf16_bits_to_f32(gpu_decode(w, codes, None, None, dG)).astype(np.float64)
    xf = synth.bf16_bits_to_f32(x).astype(np.float64).ravel()
    # bf16 output: the round trip is exact up to the final bf16 rounding
    rel = np.linalg.norm(got - xf) / np.linalg.norm(xf)
    assert rel <= 1e-5, rel
    Gi = synth.gauges(w, "identity")
    codes, _, _ = gpu_encode(w, dx, torch.from_numpy(Gi.reshape(-1)).cuda())
    got = gpu_decode(w, codes, None, None, torch.from_numpy(Gi.reshape(-1)).cuda())
    np.testing.assert_array_equal(got, x.ravel())  # identity clone: zero error


def test_rolling_append_and_window_decode():
    """Rolling history (Sec. 4.4): append one token per sequence at t0 into a T_cap history,
    then decode the whole window; equals the oracle's full encode + decode."""
    w = _wl(L=2, B=3, H=2, T=21, group=128, bits=4, block=64)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dG = torch.from_numpy(G.reshape(-1)).cuda()
    Tc = 24
    hist = cg.Shape(L=w.L, B=w.B, H=w.H, T=20, d=w.d, t0=0, T_cap=Tc)
    app = cg.Shape(L=w.L, B=w.B, H=w.H, T=1, d=w.d, t0=20, T_cap=Tc)
    params = cg.Params(**w.params)
    codes, scales, _ = cg.alloc_outputs(cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d), params)
    cg.encode(hist, params, torch.from_numpy(np.ascontiguousarray(x[..., :20, :]).reshape(-1).view(np.int16)).cuda(), dG, codes, scales)
    snap = codes.clone()
    cg.encode(app, params, torch.from_numpy(np.ascontiguousarray(x[..., 20:21, :]).reshape(-1).view(np.int16)).cuda(), dG, codes, scales)
    rowb = w.d * w.bits // 8
    c_before = snap.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)
    c_after = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)
    np.testing.assert_array_equal(c_before[..., :20, :], c_after[..., :20, :])
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    got_codes = np.ascontiguousarray(c_after[..., :21, :]).ravel()
    mism = compare_codes(w, got_codes, ref["codes"], ref["flags"])
    got_sc = scales.cpu().numpy().view(np.uint16).reshape(w.L, 2, w.B, w.H, Tc, -1)[..., :21, :]
    compare_scales(np.ascontiguousarray(got_sc).ravel(), ref["scales"])
    win = cg.Shape(L=w.L, B=w.B, H=w.H, T=21, d=w.d, t0=0, T_cap=Tc)
    out = torch.empty(w.L * 2 * w.B * w.H * 21 * w.d, dtype=torch.int16, device="cuda")
    cg.decode(win, params, codes, scales, None, dG, out)
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    step = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    compare_decode(w, out.cpu().numpy().view(np.uint16), xr, G, step, codes=ref["codes"], scales_u16=ref["scales"])
    # a window in the middle of the history: tokens [5, 17)
    mid = cg.Shape(L=w.L, B=w.B, H=w.H, T=12, d=w.d, t0=5, T_cap=Tc)
    out2 = torch.empty(w.L * 2 * w.B * w.H * 12 * w.d, dtype=torch.int16, device="cuda")
    cg.decode(mid, params, codes, scales, None, dG, out2)
    o_full = out.cpu().numpy().view(np.uint16).reshape(w.L, 2, w.B, w.H, 21, w.d)
    np.testing.assert_array_equal(out2.cpu().numpy().view(np.uint16).reshape(w.L, 2, w.B, w.H, 12, w.d),
                                  o_full[..., 5:17, :])


def test_empty_and_status():
    w = _wl(T=0)
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    assert cg.packed_bytes(shape, params) == (0, 0, 0)
    z = torch.zeros(16, dtype=torch.int16, device="cuda")
    cg.encode(shape, params, z, z.float(), z, z, None)
    cg.decode(shape, params, z, z, None, z.float(), z)
    assert cg.get_status() == 0
    # non-finite input raises the status bit, which then clears
    w = _wl(T=3, L=1, H=1)
    x = synth.kv_cache(w, threads=1)
    x[0, 1, 0, 0, 2, 7] = 0x7FC0  # NaN
    G = synth.gauges(w)
    dx, dG = _dev(x, G)
    gpu_encode(w, dx, dG)
    assert cg.get_status() & 1
    assert cg.get_status() == 0
    # fp16 overflow of a block zero
    x = synth.kv_cache(w, threads=1)
    x[0, 0, 0, 0, 1, :] = synth.f32_to_bf16_bits(np.full(w.d, -1.0e6, np.float32))
    dx, dG = _dev(x, synth.gauges(w, "identity"))
    gpu_encode(w, dx, dG)
    assert cg.get_status() & 2


def test_per_layer_calls_match_whole_call():
    """Layer-major layout: L=1 calls with offset pointers reproduce the L=2 call."""
    w = _wl(L=2, T=130)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx, dG = _dev(x, G)
    codes, scales, _ = gpu_encode(w, dx, dG)
    shape1 = cg.Shape(L=1, B=w.B, H=w.H, T=w.T, d=w.d)
    params = cg.Params(**w.params)
    nc1, ns1, _ = cg.packed_bytes(shape1, params)
    c2 = torch.zeros_like(codes)
    s2 = torch.zeros_like(scales)
    per_x = dx.numel() // 2
    per_g = dG.numel() // 2
    for l in range(2):
        cg.encode(shape1, params, dx[l * per_x:(l + 1) * per_x], dG[l * per_g:(l + 1) * per_g],
                  c2[l * nc1:(l + 1) * nc1], s2[l * ns1 // 4:(l + 1) * ns1 // 4], None)
    assert torch.equal(codes, c2) and torch.equal(scales, s2)


@pytest.mark.parametrize("name,kw", [
    ("bu4_g128_blk64", dict(group=128, bits=4, block=64)),
    ("bu6_g32_blk32", dict(group=32, bits=6, block=32)),
    ("kivi3_g64", dict(backend=1, group=64, bits=3, block=128, residual=128)),
])
def test_many_tiles_per_cta(name, kw):
    """Every CTA of the persistent tensor-core kernels walks tens of 128-token tiles and
    several gauge changes (8 tiles per (layer, cache, head) set): the warpgroup rotation,
    the accumulator and stage rings and the gauge conversion at each change, element by
    element against the oracle."""
    w = _wl(L=4, B=1, H=8, T=1024 + (128 if kw.get("backend") == 1 else 0), **kw)
    x = synth.kv_cache(w, threads=8)
    G = synth.gauges(w)
    dx, dG = _dev(x, G)
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, nr = cg.packed_bytes(shape, params)
    codes, scales, resid = gpu_encode(w, dx, dG)
    got = gpu_decode(w, codes, scales, resid, dG)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    mism = compare_codes(w, _host_u8(codes, nc), ref["codes"], ref["flags"])
    compare_scales(_host_u16(scales, ns), ref["scales"])
    if nr:
        np.testing.assert_array_equal(_host_u16(resid, nr), ref["residual"])
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    step = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    compare_decode(w, got, xr, G, step)
