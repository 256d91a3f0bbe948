"""GPU parity of the Hadamard gauge by fast Walsh-Hadamard transform (cg_encode_hadamard,
cg_decode_hadamard; the structured Hadamard control of Sec. 4.3).

The transform path applies G = H_g / sqrt(g) without a gauge tensor. Every product of the
quantization rule is +-fl(c x_j) with c = fp32(1/sqrt(g)), and the rule's pairwise order is the
butterfly order, so its codes, scales and zeros must equal the oracle's (given the fp32 Hadamard
gauge tensor) bit for bit, with no near-boundary allowance, for every group size, including
inputs whose magnitudes span 2^-20 .. 2^11. Decode of the oracle's bytes gets the tight check.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_decode

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _wl(**kw):
    base = dict(name="had", L=2, B=2, H=2, T=130, d=128, group=128, backend=0, bits=4, block=64, residual=0)
    base.update(kw)
    return synth.Workload(**base)


CASES = {
    "g128_b4_blk64": _wl(),
    "g64_b3_blk32": _wl(group=64, bits=3, block=32),
    "g32_b6_blk32": _wl(group=32, bits=6, block=32, T=77),
    "g16_b2_blk16": _wl(group=16, bits=2, block=16),
    "g8_b8_blk8": _wl(group=8, bits=8, block=8, T=33),
    "d64_g64_b4_blk64": _wl(d=64, group=64, T=300),
    "d32_g16_b3_blk32": _wl(d=32, group=16, bits=3, block=32),
    "d256_g128_b4_blk128": _wl(d=256, group=128, block=128, H=1),
}


def _mixed(w, rng):
    shp = (w.L, 2, w.B, w.H, w.T, w.d)
    v = np.ldexp(1.0 + rng.integers(0, 128, size=shp) / 128.0, rng.integers(-20, 12, size=shp))
    return synth.f32_to_bf16_bits((v * rng.choice([-1.0, 1.0], size=shp)).astype(np.float32)).reshape(shp)


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("inputs", ["cache", "mixed"])
def test_hadamard_transform_matches_oracle(name, inputs):
    w = CASES[name]
    x = synth.kv_cache(w, threads=4) if inputs == "cache" else _mixed(w, np.random.default_rng(21))
    G = synth.gauges(w, "hadamard")
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, _ = cg.packed_bytes(shape, params)
    codes, scales, _ = cg.alloc_outputs(shape, params)
    cg.encode_hadamard(shape, params, torch.from_numpy(x.reshape(-1).view(np.int16)).cuda(), codes, scales)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G)
    np.testing.assert_array_equal(codes.cpu().numpy().view(np.uint8)[:nc], ref["codes"])
    np.testing.assert_array_equal(scales.cpu().numpy().view(np.uint16)[: ns // 2].view(np.float16).astype(np.float32),
                                  ref["scales"].view(np.float16).astype(np.float32))
    # decode of the oracle's bytes: tight check against the fp64 decode
    oc = torch.from_numpy(np.concatenate([ref["codes"], np.zeros(16, np.uint8)])).cuda()
    os_ = torch.from_numpy(np.concatenate([ref["scales"], np.zeros(8, np.uint16)]).view(np.int16)).cuda()
    out = torch.empty(x.size, dtype=torch.int16, device="cuda")
    cg.decode_hadamard(shape, params, oc, os_, out)
    assert cg.get_status() == 0
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], None, G)
    st = compare_decode(w, out.cpu().numpy().view(np.uint16), xr, G, None, codes=ref["codes"],
                        scales_u16=ref["scales"])
    assert st["tight"] == xr.size


def test_hadamard_rolling_append():
    """Appending at t0 into a T_cap history through the transform path equals one call."""
    w = _wl(T=20, group=64, bits=4, block=64)
    x = synth.kv_cache(w, threads=4)
    params = cg.Params(**w.params)
    Tc = 24
    codes, scales, _ = cg.alloc_outputs(cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d), params)
    for t0, n in ((0, 19), (19, 1)):
        sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=n, d=w.d, t0=t0, T_cap=Tc)
        cg.encode_hadamard(sh, params, torch.from_numpy(np.ascontiguousarray(x[..., t0:t0 + n, :]).reshape(-1)
                                                        .view(np.int16)).cuda(), codes, scales)
    ref = oracle.encode(w.shape, w.params, x, synth.gauges(w, "hadamard"))
    rowb = w.d * w.bits // 8
    got = codes.cpu().numpy().reshape(w.L, 2, w.B, w.H, Tc, rowb)[..., :w.T, :]
    np.testing.assert_array_equal(np.ascontiguousarray(got).ravel(), ref["codes"])
