"""Pins of the oracle's block-uniform tile backend (CPU only).

Sec. 4.3 gives block-uniform one range per T_b x d_l block, with T_b = 16 tokens (Sec. 4.2).
The library reads a tile as T_b consecutive tokens of one (l, s, b, h) by `block` channels
(block = d_l is the paper's tile); codes keep the per-token layout of the block-uniform rows
and the {scale, zero} pairs are per tile. The checks below pin that reading against
brute-force numpy (identity gauge: the tile quantizer applied to X itself), against the
oracle's own pinned gauge-space values, against the per-token backend it reduces to, and
against invariants (monotone fp16 rounding of the tile minimum, append at tile
boundaries, closed-form byte counts).
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

TB = oracle.TILE_TOKENS


def _wl(**kw):
    base = dict(name="t", L=1, B=2, H=2, T=37, d=64, group=16, backend=oracle.TILE, bits=4, block=32)
    base.update(kw)
    return synth.Workload(**base)


def _np_quantize(v, bits):
    """Block quantizer in numpy fp32 / float16 over the flattened values of one range."""
    v = v.astype(np.float32).ravel()
    qmax = np.float32(2 ** bits - 1)
    mn, mx = v.min(), v.max()
    s16 = np.float16(np.float32(mx - mn) / qmax)
    m16 = np.float16(mn)
    s, m = np.float32(s16), np.float32(m16)
    if s == 0:
        return s16, m16, np.zeros(v.size, np.uint8)
    q = np.clip(np.rint((v - m) / s), 0, qmax).astype(np.uint8)
    return s16, m16, q


def _np_pack(q, bits):
    bits_arr = ((np.asarray(q, np.uint32)[:, None] >> np.arange(bits, dtype=np.uint32)) & 1).astype(np.uint8)
    return np.packbits(bits_arr.reshape(-1), bitorder="little")


def _h(v):
    return int(np.array(v, np.float16).view(np.uint16))


def _brute_force(w, vals):
    """Codes and scales of the tile backend rebuilt from the values vals [L][2][B][H][T][d]."""
    nb, blk, bits = w.d // w.block, w.block, w.bits
    ntiles = -(-w.T // TB)
    codes = np.zeros((w.L, 2, w.B, w.H, w.T, nb, blk * bits // 8), np.uint8)
    scales = np.zeros((w.L, 2, w.B, w.H, ntiles, nb, 2), np.uint16)
    for idx in np.ndindex(w.L, 2, w.B, w.H):
        for k in range(ntiles):
            t_lo, t_hi = k * TB, min(w.T, (k + 1) * TB)
            for b in range(nb):
                tile = vals[idx][t_lo:t_hi, b * blk:(b + 1) * blk]   # [tokens][channels]
                s16, m16, q = _np_quantize(tile, bits)
                scales[idx][k, b] = (_h(s16), _h(m16))
                q = q.reshape(t_hi - t_lo, blk)
                for tt in range(t_hi - t_lo):
                    codes[idx][t_lo + tt, b] = _np_pack(q[tt], bits)
    return codes.ravel(), scales.ravel()


@pytest.mark.parametrize("bits,blk,T", [(4, 32, 37), (3, 64, 16), (6, 16, 5), (2, 64, 48), (8, 32, 33)])
def test_tile_identity_gauge_is_bare_tile_quantizer(bits, blk, T):
    """Identity gauge: Z = X, so each tile's range, codes and packing follow from X alone."""
    w = _wl(T=T, bits=bits, block=blk)
    x = synth.kv_cache(w, threads=1)
    r = oracle.encode(w.shape, w.params, x, synth.gauges(w, "identity"))
    want_c, want_s = _brute_force(w, synth.bf16_bits_to_f32(x).reshape(w.L, 2, w.B, w.H, w.T, w.d))
    np.testing.assert_array_equal(r["codes"], want_c)
    np.testing.assert_array_equal(r["scales"].view(np.float16).astype(np.float32),
                                  want_s.view(np.float16).astype(np.float32))


@pytest.mark.parametrize("bits,blk,g", [(4, 128, 128), (3, 64, 32), (6, 32, 64)])
def test_tile_ranges_brute_force_on_z(bits, blk, g):
    """Dense gauges: ranges, scales, zeros and codes from the oracle's own gauge-space values."""
    w = _wl(T=40, d=128, group=g, bits=bits, block=blk, B=1)
    x = synth.kv_cache(w, threads=1)
    r = oracle.encode(w.shape, w.params, x, synth.gauges(w), want_z=True)
    want_c, want_s = _brute_force(w, r["z"].reshape(w.L, 2, w.B, w.H, w.T, w.d))
    np.testing.assert_array_equal(r["codes"], want_c)
    np.testing.assert_array_equal(r["scales"], want_s)


def test_one_token_tile_is_the_per_token_backend():
    """A call of one token fills one tile with one token: its range is that token's block range."""
    w = _wl(T=1, d=128, group=32, block=64, bits=4)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    a = oracle.encode(w.shape, w.params, x, G)
    b = oracle.encode(w.shape, dict(w.params, backend=oracle.BU), x, G)
    np.testing.assert_array_equal(a["codes"], b["codes"])
    np.testing.assert_array_equal(a["scales"], b["scales"])


def test_tile_zero_is_min_of_token_zeros():
    """fp16 rounding is monotone, so the tile's zero fp16(min) is the least per-token zero of
    the per-token backend over the tile's tokens, and the tile's scale is at least each
    token's scale (the tile range contains every token range)."""
    w = _wl(T=64, d=128, group=128, block=64, bits=4)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    t = oracle.encode(w.shape, w.params, x, G)
    p = oracle.encode(w.shape, dict(w.params, backend=oracle.BU), x, G)
    nb = w.d // w.block
    ts = t["scales"].view(np.float16).astype(np.float32).reshape(w.L, 2, w.B, w.H, w.T // TB, nb, 2)
    ps = p["scales"].view(np.float16).astype(np.float32).reshape(w.L, 2, w.B, w.H, w.T // TB, TB, nb, 2)
    np.testing.assert_array_equal(ts[..., 1], ps[..., 1].min(axis=-2))
    assert (ts[..., 0] >= ps[..., 0].max(axis=-2)).all()
    assert (ts[..., 0] > ps[..., 0].max(axis=-2)).mean() > 0.5  # the tile range is genuinely wider


def test_tile_append_at_tile_boundaries_matches_one_call():
    """Calls that start at tile boundaries fill disjoint tiles: three appends (16, 16 and a
    ragged 7 tokens) into a 39-token history equal one call over all 39 tokens."""
    w = _wl(T=39, d=64, group=32, block=32, bits=3)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    full = oracle.encode(w.shape, w.params, x, G)
    codes = np.zeros_like(full["codes"])
    scales = np.zeros_like(full["scales"])
    for t0, n in ((0, 16), (16, 16), (32, 7)):
        sh = dict(w.shape, T=n, t0=t0, T_cap=39)
        r = oracle.encode(sh, w.params, np.ascontiguousarray(x[..., t0:t0 + n, :]), G)
        codes |= r["codes"]
        scales |= r["scales"]
        # bytes of earlier tiles stay untouched
        assert not r["codes"].reshape(w.L, 2, w.B, w.H, 39, -1)[..., :t0, :].any()
    np.testing.assert_array_equal(codes, full["codes"])
    np.testing.assert_array_equal(scales, full["scales"])


def test_tile_append_inside_a_tile_is_unsupported():
    w = _wl()
    with pytest.raises(ValueError, match="rc=-2"):
        oracle.packed_bytes(dict(w.shape, T=4, t0=17, T_cap=64), w.params)
    assert oracle.packed_bytes(dict(w.shape, T=4, t0=32, T_cap=64), w.params)


def test_tile_packed_bytes_closed_form():
    """Codes as for the per-token backend; one fp16 pair per tile block: bits + 32/(T_b block)
    bits per value (4.0156 at the 8B shape with block = d = 128)."""
    w = synth.WORKLOADS["llama3_8b"].replace(backend=oracle.TILE, block=128)
    c, s, r = oracle.packed_bytes(w.shape, w.params)
    n = w.n_elems
    assert (c, s, r) == (n * 4 // 8, n // (16 * 128) * 4, 0)
    assert (c + s) * 8 / n == 4 + 32 / (16 * 128)
    w = _wl(T=37, d=64, block=16, bits=6)
    units = w.L * 2 * w.B * w.H
    assert oracle.packed_bytes(w.shape, w.params) == (units * 37 * 64 * 6 // 8, units * 3 * 4 * 4, 0)


@pytest.mark.parametrize("bits,blk,g", [(4, 128, 128), (3, 32, 16)])
def test_tile_decode_error_within_quantization_bound(bits, blk, g):
    """Decode with tile ranges (Sec. 3: Xhat = G^T Zhat): per gauge group ||Xhat - X||_2 is at
    most sqrt(sum_j e_j^2), e_j = s/2 + qmax |s32 - s| + |min - m| of element j's tile, since G
    is orthogonal; and the decode of the identity gauge is q s + m exactly."""
    w = _wl(T=45, d=128, group=g, bits=bits, block=blk, B=1)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True)
    xh = oracle.decode(w.shape, w.params, r["codes"], r["scales"], None, G)
    z = r["z"].reshape(w.L, 2, w.B, w.H, w.T, w.d).astype(np.float64)
    qmax = 2 ** bits - 1
    nb = w.d // blk
    sc = r["scales"].view(np.float16).astype(np.float64).reshape(w.L, 2, w.B, w.H, -1, nb, 2)
    e = np.zeros_like(z)
    for idx in np.ndindex(w.L, 2, w.B, w.H):
        for t in range(w.T):
            for b in range(nb):
                k = t // TB
                v = z[idx][k * TB:min(w.T, (k + 1) * TB), b * blk:(b + 1) * blk]
                s, m = sc[idx][k, b]
                s32 = float(np.float32(np.float32(v.max()) - np.float32(v.min())) / np.float32(qmax))
                e[idx][t, b * blk:(b + 1) * blk] = s / 2 * (1 + 1e-6) + qmax * abs(s32 - s) + abs(v.min() - m) + 1e-7
    xf = synth.bf16_bits_to_f32(x).astype(np.float64).reshape(z.shape)
    err = np.linalg.norm((xh.reshape(z.shape) - xf).reshape(-1, g), axis=-1)
    bound = np.linalg.norm(e.reshape(-1, g), axis=-1) + 1e-5 * (1 + np.linalg.norm(xf.reshape(-1, g), axis=-1))
    assert np.all(err <= bound)
    assert np.median(err / bound) > 0.05
    Gi = synth.gauges(w, "identity")
    ri = oracle.encode(w.shape, w.params, x, Gi)
    xi = oracle.decode(w.shape, w.params, ri["codes"], ri["scales"], None, Gi).reshape(z.shape)
    qs = oracle.unpack(ri["codes"], w.n_elems, bits).reshape(z.shape).astype(np.float64)
    si = ri["scales"].view(np.float16).astype(np.float64).reshape(w.L, 2, w.B, w.H, -1, nb, 2)
    tok_tile = np.arange(w.T) // TB
    s_el = np.repeat(si[..., 0][:, :, :, :, tok_tile, :], blk, axis=-1)
    m_el = np.repeat(si[..., 1][:, :, :, :, tok_tile, :], blk, axis=-1)
    np.testing.assert_array_equal(xi, qs * s_el + m_el)
