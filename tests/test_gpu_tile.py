"""GPU parity of the block-uniform tile backend (CG_BLOCK_TILE) against the CPU oracle.

One range per 16-token x block tile (Sec. 4.3, T_b = 16 from Sec. 4.2; block = d is the
paper's T_b x d_l tile). The tile encode computes every gauge-space value in the library's
fixed fp32 order, so codes, scales and zeros must equal the oracle's bit for bit, with no
near-boundary allowance. Decode runs the block-uniform decode kernels with the tile's
scale map. Cases span ragged last tiles, every bit width, the head dims 32..256 and appends
at tile boundaries, including the re-encode of an open tile in a rolling history.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_decode

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu

TILE = 3


def _wl(**kw):
    base = dict(name="tile", L=2, B=1, H=2, T=300, d=128, group=128, backend=TILE, bits=4, block=128, residual=0)
    base.update(kw)
    return synth.Workload(**base)


CASES = {
    "tile4_g128_blk128": _wl(),
    "tile6_g32_blk32_B2": _wl(B=2, T=257, group=32, bits=6, block=32),
    "tile3_g16_blk16_d64": _wl(d=64, group=16, bits=3, block=16, T=37),
    "tile2_g8_blk8_d32": _wl(d=32, group=8, bits=2, block=8, T=129),
    "tile8_g64_blk128_d256": _wl(d=256, group=64, bits=8, block=128, T=140, H=1),
    "tile4_g128_blk256_d256": _wl(d=256, group=128, bits=4, block=256, T=50, H=1),
    "tile3_g128_blk64_T1": _wl(bits=3, block=64, T=1, B=3),
    "tile4_g64_blk16_T384": _wl(group=64, bits=4, block=16, T=384),
}


def _dev_bf16(x):
    return torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda()


def _dev_f32(G):
    return torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()


def _decode(w, shape, params, codes, scales, dG, T):
    out = torch.full((w.L * 2 * w.B * w.H * T * w.d,), -1, dtype=torch.int16, device="cuda")
    cg.decode(shape, params, codes, scales, None, dG, out)
    return out.cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("name", list(CASES))
def test_tile_encode_decode_parity(name):
    w = CASES[name]
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx, dG = _dev_bf16(x), _dev_f32(G)
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, nr = cg.packed_bytes(shape, params)
    assert (nc, ns, nr) == oracle.packed_bytes(w.shape, w.params)
    codes, scales, _ = cg.alloc_outputs(shape, params)
    cg.encode(shape, params, dx, dG, codes, scales)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G)
    np.testing.assert_array_equal(codes.cpu().numpy().view(np.uint8)[:nc], ref["codes"])
    got_s = scales.cpu().numpy().view(np.uint16)[: ns // 2]
    np.testing.assert_array_equal(got_s.view(np.float16).astype(np.float32),
                                  ref["scales"].view(np.float16).astype(np.float32))
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], None, G)
    got = _decode(w, shape, params, codes, scales, dG, w.T)
    st = compare_decode(w, got, xr, G, None, codes=ref["codes"], scales_u16=ref["scales"])
    assert st["tight"] == xr.size
    assert cg.get_status() == 0


def test_tile_appends_at_tile_boundaries():
    """Calls of 16, 16 and a ragged 9 tokens into a 48-token history equal one call over the
    41 tokens; bytes of earlier tiles stay unchanged by later calls."""
    w = _wl(L=1, B=2, H=2, T=41, group=32, bits=3, block=64)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dG = _dev_f32(G)
    params = cg.Params(**w.params)
    Tc = 48
    hist = cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d)
    codes, scales, _ = cg.alloc_outputs(hist, params)
    rowb = w.d * w.bits // 8
    for t0, n in ((0, 16), (16, 16), (32, 9)):
        before = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)[..., :t0, :].copy()
        sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=n, d=w.d, t0=t0, T_cap=Tc)
        cg.encode(sh, params, _dev_bf16(x[..., t0:t0 + n, :]), dG, codes, scales)
        after = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)[..., :t0, :]
        np.testing.assert_array_equal(before, after)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G)
    got_c = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)[..., :w.T, :]
    np.testing.assert_array_equal(np.ascontiguousarray(got_c).ravel(), ref["codes"])
    nt = -(-w.T // 16)
    got_s = scales.cpu().numpy().view(np.uint16).reshape(w.L, 2, w.B, w.H, Tc // 16, -1)[..., :nt, :]
    np.testing.assert_array_equal(np.ascontiguousarray(got_s).ravel().view(np.float16).astype(np.float32),
                                  ref["scales"].view(np.float16).astype(np.float32))
    # decode a window that starts at a tile boundary
    win = cg.Shape(L=w.L, B=w.B, H=w.H, T=25, d=w.d, t0=16, T_cap=Tc)
    out = _decode(w, win, params, codes, scales, dG, 25)
    full = _decode(w, cg.Shape(L=w.L, B=w.B, H=w.H, T=w.T, d=w.d, t0=0, T_cap=Tc), params, codes, scales, dG, w.T)
    np.testing.assert_array_equal(out.reshape(w.L, 2, w.B, w.H, 25, w.d),
                                  full.reshape(w.L, 2, w.B, w.H, w.T, w.d)[..., 16:41, :])


def test_tile_rolling_reencode_of_open_tile():
    """A rolling step appends one token to an open tile by re-encoding the tile from its first
    token: after tokens 0..19 (one full tile, one open tile of 4), the call for token 20
    re-encodes tokens 16..20 at t0 = 16; the history equals one call over 21 tokens."""
    w = _wl(L=2, B=3, H=2, T=21, group=128, bits=4, block=128)
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dG = _dev_f32(G)
    params = cg.Params(**w.params)
    Tc = 32
    codes, scales, _ = cg.alloc_outputs(cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d), params)
    cg.encode(cg.Shape(L=w.L, B=w.B, H=w.H, T=20, d=w.d, t0=0, T_cap=Tc), params, _dev_bf16(x[..., :20, :]), dG,
              codes, scales)
    cg.encode(cg.Shape(L=w.L, B=w.B, H=w.H, T=5, d=w.d, t0=16, T_cap=Tc), params, _dev_bf16(x[..., 16:21, :]), dG,
              codes, scales)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G)
    rowb = w.d * w.bits // 8
    got_c = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)[..., :21, :]
    np.testing.assert_array_equal(np.ascontiguousarray(got_c).ravel(), ref["codes"])
    got_s = scales.cpu().numpy().view(np.uint16).reshape(w.L, 2, w.B, w.H, 2, -1)
    np.testing.assert_array_equal(np.ascontiguousarray(got_s).ravel().view(np.float16).astype(np.float32),
                                  ref["scales"].view(np.float16).astype(np.float32))


def test_tile_append_inside_a_tile_is_rejected():
    w = _wl(T=4)
    params = cg.Params(**w.params)
    sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=4, d=w.d, t0=8, T_cap=32)
    with pytest.raises(cg.CodecGaugeError) as e:
        cg.packed_bytes(sh, params)
    assert e.value.code == -2
