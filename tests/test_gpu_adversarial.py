"""GPU parity on inputs aimed at the tensor-core encode's error bound.

The tensor-core encode computes z~ = G x with the exact three-term bf16 split of G and fp32
accumulation, bounds |z~ - z| per block, and recomputes exactly (in the library's fixed fp32
order) every extreme or code that this bound leaves undecided (Sec. 3, Z = G X; Sec. 4.3
block-uniform and KIVI quantizers). The bound is largest, relative to the values, where
|z_i| is far below ||G_i|| ||x||. These inputs go there, with dense gauges:

  - rows whose entries mix magnitudes from 2^-20 to 2^11 (random signs): most products are
    negligible next to a few large ones, and small z values carry large absolute errors;
  - cancelling rows: x = bf16(c G^T e_k) per gauge group, so z = G x is one large value and
    g - 1 values that are rounding residue, |z_i| ~ 2^-9 ||G_i|| ||x||;
  - near-identity gauges (I plus off-diagonal entries of 1e-6): z_i = x_i + tiny terms, so
    block extremes and zeros sit next to fp16-representable values.

Codes must match the oracle except flagged elements, scales and zeros bit for bit, for
block-uniform rows (one, two and four blocks per row) and KIVI keys and values.
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
    base = dict(name="adv", L=1, B=2, H=2, T=384, d=128, group=128, backend=0, bits=4, block=64, residual=0)
    base.update(kw)
    return synth.Workload(**base)


def mixed_magnitudes(w, rng):
    shp = (w.L, 2, w.B, w.H, w.T, w.d)
    e = rng.integers(-20, 12, size=shp)
    mant = 1.0 + rng.integers(0, 128, size=shp) / 128.0
    v = np.ldexp(mant, e) * rng.choice([-1.0, 1.0], size=shp)
    return synth.f32_to_bf16_bits(v.astype(np.float32)).reshape(shp)


def cancelling(w, G, rng):
    """x = bf16(c G^T e_k) per gauge group, k and c random per (token, group)."""
    g = w.group
    x = np.empty((w.L, 2, w.B, w.H, w.T, w.d), np.float32)
    for l, s, b, h in np.ndindex(w.L, 2, w.B, w.H):
        Gs = G[l, s, h].astype(np.float64)  # [d/g][g][g]
        k = rng.integers(0, g, size=(w.T, w.d // g))
        c = np.exp(rng.normal(0.0, 1.0, size=(w.T, w.d // g))) * rng.choice([-1.0, 1.0], size=(w.T, w.d // g))
        for r in range(w.d // g):
            x[l, s, b, h, :, r * g:(r + 1) * g] = c[:, r:r + 1] * Gs[r][k[:, r], :]  # row k of G = (G^T e_k)^T
    return synth.f32_to_bf16_bits(x).reshape(x.shape)


def near_identity(w, rng, eps=1e-6):
    g = w.group
    G = np.empty((w.L, 2, w.H, w.d // g, g, g), np.float32)
    for idx in np.ndindex(w.L, 2, w.H, w.d // g):
        S = rng.normal(0.0, 1.0, size=(g, g))
        G[idx] = (np.eye(g) + eps * (S - S.T)).astype(np.float32)
    return G


def _run(w, x, G):
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    dx = torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    out = torch.empty_like(dx)
    cg.decode(shape, params, codes, scales, resid, dG, out)
    assert cg.get_status() == 0
    nc, ns, nr = cg.packed_bytes(shape, params)
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    mism = compare_codes(w, codes.cpu().numpy().view(np.uint8)[:nc], ref["codes"], ref["flags"])
    compare_scales(scales.cpu().numpy().view(np.uint16)[: ns // 2], ref["scales"])
    if nr:
        np.testing.assert_array_equal(resid.cpu().numpy().view(np.uint16)[: nr // 2], ref["residual"])
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    step = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    compare_decode(w, out.cpu().numpy().view(np.uint16)[: xr.size], xr, G, step, codes=ref["codes"],
                   scales_u16=ref["scales"])


SHAPES = {
    "bu4_g128_blk64": _wl(),
    "bu6_g32_blk32": _wl(group=32, bits=6, block=32),
    "bu3_g64_blk128": _wl(group=64, bits=3, block=128),
    "kivi3_g64": _wl(backend=1, group=64, bits=3, block=128, residual=128, T=512),
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_mixed_magnitudes(name):
    w = SHAPES[name]
    rng = np.random.default_rng(11)
    _run(w, mixed_magnitudes(w, rng), synth.gauges(w))


@pytest.mark.parametrize("name", list(SHAPES))
def test_cancelling_rows(name):
    w = SHAPES[name]
    rng = np.random.default_rng(12)
    G = synth.gauges(w)
    _run(w, cancelling(w, G, rng), G)


@pytest.mark.parametrize("name", list(SHAPES))
def test_near_identity_gauges(name):
    w = SHAPES[name]
    rng = np.random.default_rng(13)
    _run(w, synth.kv_cache(w, threads=4), near_identity(w, rng))
