"""GPU parity on planted inputs that drive the tensor-core encode through its repair paths.

With identity gauges the gauge-space values are the bf16 inputs themselves, so blocks can be
built whose fp16 scale or zero sits exactly on a rounding midpoint (Sec. 4.3 quantizer: the
scale is the fp16 rounding of (max - min) / (2^b - 1), the zero the fp16 rounding of min),
whose pre-rounding code values are exact half-integers, or whose extremes repeat across the
block. The tensor-core kernel cannot decide such blocks from its approximate values: it must
recompute the candidates exactly, often more of them than one repair round holds. The
expected scales, zeros and codes are worked out by hand in planted.py (fp16 round-half-even), so
the test pins the oracle and the kernel alike, and the oracle comparison covers the rest.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import codes_as_elements, compare_codes, compare_decode, compare_scales, scales_as_elements
from planted import N_KINDS, block_values, expected_scale_zero, planted_rows

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _gpu_encode(w, x, G):
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    dx = torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    nc, ns, _ = cg.packed_bytes(shape, params)
    return codes.cpu().numpy().view(np.uint8)[:nc], scales.cpu().numpy().view(np.uint16)[: ns // 2]


@pytest.mark.parametrize("bits,block", [(4, 64), (3, 32), (6, 128), (2, 64)])
def test_planted_block_uniform(bits, block):
    w = synth.Workload(name="planted", L=1, B=2, H=2, T=300, d=128, group=128, backend=0, bits=bits,
                       block=block, residual=0)
    qmax = (1 << bits) - 1
    x, kind = planted_rows(w, np.random.default_rng(100 + bits))
    G = synth.gauges(w, "identity")
    gc, gs = _gpu_encode(w, x, G)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    compare_scales(gs, ref["scales"])
    compare_codes(w, gc, ref["codes"], ref["flags"])
    # the hand-worked values
    sm = gs.reshape(kind.shape + (2,))
    for k in range(N_KINDS):
        es, em = expected_scale_zero(k, qmax)
        sel = kind == k
        if es is not None:
            assert (sm[..., 0][sel] == es).all(), (k, np.unique(sm[..., 0][sel]))
        if em is not None:
            assert (sm[..., 1][sel] == em).all(), (k, np.unique(sm[..., 1][sel]))
    q = codes_as_elements(w, gc)
    xv = synth.bf16_bits_to_f32(x)
    per_elem = np.repeat(kind, w.block, axis=-1)
    # kind 0: t = z exactly; half-integers round to the even neighbour
    tie = per_elem == 0
    np.testing.assert_array_equal(q[tie], np.rint(xv[tie]).astype(q.dtype))
    # constant and zero blocks: all codes 0
    assert (q[(per_elem == 2) | (per_elem == 3)] == 0).all()


def test_planted_kivi_keys_and_values():
    """KIVI (Sec. 4.3): key blocks are channels over a 128-token group, value blocks token rows;
    the planted kinds run along the tokens for keys and along the channels for values."""
    w = synth.Workload(name="planted_kivi", L=1, B=2, H=2, T=256 + 40, d=128, group=64, backend=1, bits=3,
                       block=128, residual=40)
    qmax = (1 << w.bits) - 1
    rng = np.random.default_rng(7)
    x = np.empty((w.L, 2, w.B, w.H, w.T, w.d), np.float32)
    for idx in np.ndindex(w.L, w.B, w.H):
        l, b, h = idx
        for c in range(w.d):  # keys: one block per channel and 128-token group
            for t0 in range(0, w.T, 128):
                n = min(128, w.T - t0)
                x[l, 0, b, h, t0:t0 + n, c] = block_values((c + t0 // 128) % N_KINDS, 128, qmax, rng)[:n]
        for t in range(w.T):  # values: one block per token row
            x[l, 1, b, h, t, :] = block_values(t % N_KINDS, w.d, qmax, rng)
    xb = synth.f32_to_bf16_bits(x).reshape(x.shape)
    G = synth.gauges(w, "identity")
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    dx = torch.from_numpy(np.ascontiguousarray(xb).reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    assert cg.get_status() == 0
    nc, ns, nr = cg.packed_bytes(shape, params)
    ref = oracle.encode(w.shape, w.params, xb, G, want_flags=True)
    compare_scales(scales.cpu().numpy().view(np.uint16)[: ns // 2], ref["scales"])
    mism = compare_codes(w, codes.cpu().numpy().view(np.uint8)[:nc], ref["codes"], ref["flags"])
    np.testing.assert_array_equal(resid.cpu().numpy().view(np.uint16)[: nr // 2], ref["residual"])
    # decode of the planted cache stays within the decode tolerance
    out = torch.empty(xb.size, dtype=torch.int16, device="cuda")
    cg.decode(shape, params, codes, scales, resid, dG, out)
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    step = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    compare_decode(w, out.cpu().numpy().view(np.uint16), xr, G, step, codes=ref["codes"], scales_u16=ref["scales"])
