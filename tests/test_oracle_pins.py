"""Pins of the CPU oracle against what the paper and the mathematics fix (CPU only).

Each test checks the oracle against something other than itself: IEEE conversions of
numpy/torch, fp64 matrix products within the fp32 chain's rounding-error bound,
hand-worked examples (tests/golden), brute-force numpy recomputation, invariants of
the method (Sec. 3: G^{-1} G X = X; gauge locality; identity gauge = bare backend), and
closed-form byte counts (Appendix metric table: actual bits/value from measured bytes).
"""
import os

import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
U = 2.0 ** -24


def _golden(name):
    recs, cur = [], {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        k, *v = line.split()
        if k in cur:
            recs.append(cur)
            cur = {}
        cur[k] = v
    recs.append(cur)
    return recs


def _bf16(a):
    return synth.f32_to_bf16_bits(np.asarray(a, np.float32))


def _f32(b):
    return synth.bf16_bits_to_f32(b)


def _wl(**kw):
    base = dict(name="t", L=1, B=1, H=1, T=4, d=32, group=8, backend=0, bits=4, block=16)
    base.update(kw)
    return synth.Workload(**base)


# ---------------------------------------------------------------- IEEE conversions
def test_f16_to_f32_all_patterns():
    for h in range(0, 65536, 1):
        e = (h >> 10) & 31
        ref = np.array([h], np.uint16).view(np.float16).astype(np.float32)[0]
        got = oracle.f16_bits_to_f32(h)
        if e == 31 and h & 0x3FF:
            assert np.isnan(got)
        else:
            assert got == ref or (got == 0 and ref == 0), h


def test_f32_to_f16_round_to_nearest_even_vs_numpy():
    rng = np.random.default_rng(0)
    # every half value, the midpoints between neighbours (ties), and points just off them
    hv = np.arange(0, 0x7C00, dtype=np.uint16).view(np.float16).astype(np.float64)
    mids = (hv[:-1] + hv[1:]) / 2
    cand = np.concatenate([hv, mids, np.nextafter(mids.astype(np.float32), np.float32(np.inf)).astype(np.float64),
                           np.nextafter(mids.astype(np.float32), np.float32(0)).astype(np.float64),
                           [65504.0, 65519.0, 65520.0, 65536.0, 1e6, 2.0 ** -25, 2.0 ** -26, 3 * 2.0 ** -26]])
    cand = np.concatenate([cand, -cand, rng.standard_normal(20000) * 10.0 ** rng.uniform(-9, 5, 20000)])
    f = cand.astype(np.float32)
    with np.errstate(over="ignore"):
        ref = f.astype(np.float16).view(np.uint16)
    got = np.array([oracle.f32_to_f16_bits(float(v)) for v in f], np.uint16)
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, [(float(f[i]), hex(got[i]), hex(ref[i])) for i in bad[:5]]


# ---------------------------------------------------------------- gauge application
def _order_terms(g):
    """Rounding steps on the longest path of the fixed summation order: the product, then
    log2(g) levels of pairwise sums."""
    return 1 + int(np.log2(g))


@pytest.mark.parametrize("g", [8, 16, 32, 64, 128])
def test_gauge_coord_within_fp32_dot_product_bound(g):
    """Z = G X (Sec. 3): the fp32 evaluation lies within gamma_n * sum|G_ij x_j| of the exact
    product, n the rounding steps on the longest path of its summation tree (Higham's
    bound for a recursively summed dot product with fma)."""
    rng = np.random.default_rng(g)
    n = _order_terms(g)
    for _ in range(50):
        G = synth.random_orthogonal(g, rng).astype(np.float32)
        x = _f32(_bf16(rng.standard_normal(g) * 3))
        for i in range(g):
            z = float(oracle.gauge_coord(G[i], x))
            exact = float(np.dot(G[i].astype(np.float64), x.astype(np.float64)))
            bound = (n * U / (1 - n * U)) * float(np.abs(G[i].astype(np.float64)) @ np.abs(x.astype(np.float64)))
            assert abs(z - exact) <= bound + 1e-45


def test_summation_order_hand_worked():
    rec = _golden("order_pairwise.txt")[0]
    g = int(rec["g"][0])
    row = np.array([float(v) for v in rec["row"]], np.float32)
    x = np.ones(g, np.float32)
    assert float(oracle.gauge_coord(row, x)) == float(rec["z0"][0])
    # the same value through the encoder's no-compression path (z stored as fp32)
    w = _wl(T=1, d=g, group=g, backend=2)
    G = np.zeros((1, 2, 1, 1, g, g), np.float32)
    G[...] = np.eye(g, dtype=np.float32)
    G[0, :, 0, 0, 0] = row
    xb = np.zeros((1, 2, 1, 1, 1, g), np.uint16)
    xb[...] = _bf16(x)
    r = oracle.encode(w.shape, w.params, xb, G, want_z=True)
    assert r["z"][0] == float(rec["z0"][0]) and r["z"][g] == float(rec["z0"][0])
    np.testing.assert_array_equal(r["z"].reshape(2, g)[:, 1:], 1.0)


def test_chain_identity_rows_exact():
    rng = np.random.default_rng(1)
    x = _f32(_bf16(rng.standard_normal(16)))
    I = np.eye(16, dtype=np.float32)
    for i in range(16):
        assert oracle.gauge_coord(I[i], x) == x[i]


@pytest.mark.parametrize("kind", ["random", "hadamard", "dct"])
def test_encode_z_matches_fp64_matvec(kind):
    """The oracle's z is G X, not G^T X or another index order: compare with numpy fp64
    using non-symmetric random gauges (and the structured Hadamard/DCT controls)."""
    w = _wl(L=1, B=2, H=2, T=5, d=64, group=32)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w, kind)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True)
    z = r["z"].reshape(w.L, 2, w.B, w.H, w.T, w.d)
    xf = _f32(x).astype(np.float64).reshape(w.L, 2, w.B, w.H, w.T, w.d // 32, 32)
    Gd = G.astype(np.float64)  # [L][2][H][R][g][g]
    ref = np.einsum("lshrij,lsbhtrj->lsbhtri", Gd, xf).reshape(z.shape)
    absdot = np.einsum("lshrij,lsbhtrj->lsbhtri", np.abs(Gd), np.abs(xf)).reshape(z.shape)
    n = _order_terms(32)
    assert np.all(np.abs(z - ref) <= n * U * 1.01 * absdot + 1e-45)


def test_generated_gauges_orthogonal():
    """Generated gauges are orthogonal to 1e-6 (evaluated in fp64)."""
    for name in ("tiny", "kivi3_qwen"):
        w = synth.WORKLOADS[name].replace(L=2)
        G = synth.gauges(w).astype(np.float64)
        eye = np.eye(w.group)
        err = np.abs(np.einsum("...ij,...kj->...ik", G, G) - eye).max()
        assert err <= 1e-6, err
    for kind in ("hadamard", "dct"):
        G = synth.gauges(_wl(group=32, d=64), kind).astype(np.float64)
        assert np.abs(np.einsum("...ij,...kj->...ik", G, G) - np.eye(32)).max() <= 1e-6


# ---------------------------------------------------------------- packing
@pytest.mark.parametrize("name", ["pack_3bit.txt", "pack_4bit_6bit.txt"])
def test_pack_hand_worked(name):
    for rec in _golden(name):
        bits = int(rec["bits"][0])
        q = np.array([int(v) for v in rec["codes"]], np.uint8)
        want = np.array([int(v, 16) for v in rec["bytes"]], np.uint8)
        # pad to a whole number of bytes for the packer's n*bits/8 size
        assert (q.size * bits) % 8 == 0
        np.testing.assert_array_equal(oracle.pack(q, bits), want)
        np.testing.assert_array_equal(oracle.unpack(want, q.size, bits), q)


@pytest.mark.parametrize("bits", [2, 3, 4, 6, 8])
def test_pack_unpack_identity(bits):
    rng = np.random.default_rng(bits)
    q = rng.integers(0, 2 ** bits, size=128).astype(np.uint8)
    np.testing.assert_array_equal(oracle.unpack(oracle.pack(q, bits), 128, bits), q)


@pytest.mark.parametrize("name", ["block_4bit_identity.txt", "block_4bit_offset.txt"])
def test_block_hand_worked_identity(name):
    rec = _golden(name)[0]
    d, g, blk, bits = (int(rec[k][0]) for k in ("d", "group", "block", "bits"))
    w = _wl(T=1, d=d, group=g, block=blk, bits=bits)
    xv = np.array([float(v) for v in rec["x"]], np.float32)
    x = np.zeros((1, 2, 1, 1, 1, d), np.uint16)
    x[...] = _bf16(xv)
    G = synth.gauges(w, "identity")
    r = oracle.encode(w.shape, w.params, x, G)
    want_codes = np.array([int(v, 16) for v in rec["codes"]], np.uint8)
    want_scales = np.array([int(v, 16) for v in rec["scales"]], np.uint16)
    np.testing.assert_array_equal(r["codes"][:d * bits // 8], want_codes)
    np.testing.assert_array_equal(r["scales"][:2 * d // blk], want_scales)
    xh = oracle.decode(w.shape, w.params, r["codes"], r["scales"], r["residual"], G)
    np.testing.assert_array_equal(xh[:d], xv.astype(np.float64))


# ---------------------------------------------------------------- quantizer
def _np_quantize(v, bits):
    """Block quantizer recomputed with numpy fp32 / float16 (independent of the oracle's C)."""
    v = v.astype(np.float32)
    qmax = np.float32(2 ** bits - 1)
    mn, mx = v.min(), v.max()
    s16 = np.float16(np.float32(mx - mn) / qmax)
    m16 = np.float16(mn)
    s, m = np.float32(s16), np.float32(m16)
    if s == 0:
        return s16, m16, np.zeros(v.size, np.uint8)
    t = (v - m) / s
    q = np.clip(np.rint(t), 0, qmax).astype(np.uint8)
    return s16, m16, q


@pytest.mark.parametrize("bits,blk", [(4, 64), (3, 32), (6, 128), (2, 64)])
def test_planted_midpoints_hand_worked(bits, blk):
    """fp16 round-half-even on exact midpoints of the scale (max - min) / qmax and of the
    zero (an fp16 subnormal midpoint), exact half-integer codes, constant and zero blocks
    (Sec. 4.3 quantizer): the values worked out by hand in planted.py."""
    from planted import N_KINDS, expected_scale_zero, planted_rows
    w = _wl(T=12, d=128, group=128, block=blk, bits=bits)
    qmax = 2 ** bits - 1
    x, kind = planted_rows(w, np.random.default_rng(bits))
    r = oracle.encode(w.shape, w.params, x, synth.gauges(w, "identity"))
    sm = r["scales"].reshape(kind.shape + (2,))
    for k in range(N_KINDS):
        es, em = expected_scale_zero(k, qmax)
        if es is not None:
            assert (sm[..., 0][kind == k] == es).all(), k
        if em is not None:
            assert (sm[..., 1][kind == k] == em).all(), k
    q = oracle.unpack(r["codes"], x.size, bits).reshape(x.shape)
    per_elem = np.repeat(kind, blk, axis=-1)
    xv = _f32(x)
    np.testing.assert_array_equal(q[per_elem == 0], np.rint(xv[per_elem == 0]))
    assert (q[(per_elem == 2) | (per_elem == 3)] == 0).all()


@pytest.mark.parametrize("bits,blk,g", [(4, 16, 8), (3, 32, 32), (6, 32, 16), (2, 8, 8), (8, 64, 64)])
def test_identity_gauge_is_bare_backend(bits, blk, g):
    """Sec. 4.3: the identity gauge compresses the raw cache, so encode must equal the
    backend applied to X directly (brute-force numpy min/max per block)."""
    w = _wl(L=1, B=2, H=2, T=7, d=64, group=g, block=blk, bits=bits)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w, "identity")
    r = oracle.encode(w.shape, w.params, x, G)
    xf = _f32(x).reshape(-1, w.d)
    nb, pay = w.d // blk, blk * bits // 8
    codes = r["codes"].reshape(-1, nb, pay)
    sc = r["scales"].reshape(-1, nb, 2)
    for row in range(xf.shape[0]):
        for b in range(nb):
            s16, m16, q = _np_quantize(xf[row, b * blk:(b + 1) * blk], bits)
            assert sc[row, b, 0] == np.array(s16).view(np.uint16)
            assert sc[row, b, 1] == np.array(m16).view(np.uint16)
            np.testing.assert_array_equal(oracle.unpack(codes[row, b], blk, bits), q)


def _np_pack(q, bits):
    """Little-endian bit stream of b-bit codes (bit 0 = LSB of byte 0), numpy only."""
    bits_arr = ((np.asarray(q, np.uint32)[:, None] >> np.arange(bits, dtype=np.uint32)) & 1).astype(np.uint8)
    return np.packbits(bits_arr.reshape(-1), bitorder="little")


@pytest.mark.parametrize("bits,Gt,R", [(3, 32, 20), (4, 16, 0), (2, 32, 40)])
def test_kivi_identity_gauge_is_bare_kivi(bits, Gt, R):
    """Sec. 4.3 KIVI with the identity gauge: keys quantized per channel over groups of Gt
    tokens, values per token over blocks of Gt channels, the newest T - n_q tokens kept raw.
    The codes, scales and residual are rebuilt with numpy from the layouts alone (per-channel
    key streams, then per-token value blocks) and the numpy block quantizer."""
    w = _wl(L=1, B=2, H=2, T=150, d=32, group=8, backend=1, bits=bits, block=Gt, residual=R)
    x = synth.kv_cache(w, threads=1)
    r = oracle.encode(w.shape, w.params, x, synth.gauges(w, "identity"))
    xf = _f32(x)
    nq = max(0, (w.T - R) // Gt) * Gt
    codes, scales = [], []
    for b in range(w.B):          # keys [B][H][n_q/Gt][d]: one channel's Gt-token stream each
        for h in range(w.H):
            for grp in range(nq // Gt):
                for c in range(w.d):
                    s16, m16, q = _np_quantize(xf[0, 0, b, h, grp * Gt:(grp + 1) * Gt, c], bits)
                    codes.append(_np_pack(q, bits))
                    scales += [np.array(s16).view(np.uint16), np.array(m16).view(np.uint16)]
    for b in range(w.B):          # values [B][H][n_q][d/Gt]: one token's Gt-channel block each
        for h in range(w.H):
            for t in range(nq):
                for k in range(w.d // Gt):
                    s16, m16, q = _np_quantize(xf[0, 1, b, h, t, k * Gt:(k + 1) * Gt], bits)
                    codes.append(_np_pack(q, bits))
                    scales += [np.array(s16).view(np.uint16), np.array(m16).view(np.uint16)]
    want_codes = np.concatenate(codes) if codes else np.zeros(0, np.uint8)
    np.testing.assert_array_equal(r["codes"][:want_codes.size], want_codes)
    got_s = r["scales"][:len(scales)].view(np.float16).astype(np.float32)
    want_s = np.array(scales, np.uint16).view(np.float16).astype(np.float32)
    np.testing.assert_array_equal(got_s, want_s)
    np.testing.assert_array_equal(r["residual"].reshape(w.L, 2, w.B, w.H, w.T - nq, w.d), x[..., nq:, :])
    assert oracle.packed_bytes(w.shape, w.params) == (want_codes.size, 2 * len(scales), 2 * x[..., nq:, :].size)


@pytest.mark.parametrize("bits,blk,g", [(4, 64, 128), (6, 32, 32), (3, 128, 64)])
def test_block_ranges_brute_force_on_z(bits, blk, g):
    """Per-block min/max, scale, zero and codes recomputed by brute force from the
    oracle's own gauge-space values (numpy fp32/float16)."""
    w = _wl(L=1, B=1, H=2, T=9, d=128, group=g, block=blk, bits=bits)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True, want_flags=True)
    z = r["z"].reshape(-1, w.d)
    nb, pay = w.d // blk, blk * bits // 8
    codes = r["codes"].reshape(-1, nb, pay)
    sc = r["scales"].reshape(-1, nb, 2)
    for row in range(z.shape[0]):
        for b in range(nb):
            v = z[row, b * blk:(b + 1) * blk]
            s16, m16, q = _np_quantize(v, bits)
            assert sc[row, b, 0] == np.array(s16).view(np.uint16)
            assert sc[row, b, 1] == np.array(m16).view(np.uint16)
            np.testing.assert_array_equal(oracle.unpack(codes[row, b], blk, bits), q)
            # the extremes map to the ends of the code range
            assert q[np.argmax(v)] == 2 ** bits - 1
            assert q[np.argmin(v)] == 0
            # reconstruction error of each value is at most half a step (plus fp16 slack)
            s, m = np.float32(s16), np.float32(m16)
            zh = q.astype(np.float64) * s + m
            assert np.all(np.abs(zh - v) <= s / 2 * (1 + 1e-6) + abs(float(m) - float(v.min())) + 1e-7)


def test_clamp_when_fp16_zero_rounds():
    """fp16 rounding of the block zero can push values outside the code range; the rule
    clamps them to [0, 2^bits - 1]. A non-orthogonal diagonal gauge makes z = RN(G_ii x_i)
    (exact in numpy) a narrow cluster far from 0, where fp16(min) is coarse."""
    w = _wl(T=1, d=32, group=32, block=32, bits=4)
    G = np.zeros((1, 2, 1, 1, 32, 32), np.float32)
    eps = np.linspace(1e-4, 2.1e-3, 32).astype(np.float32)  # min 10.001: fp16 zero 10.0
    for s in range(2):
        G[0, s, 0, 0] = np.diag(np.float32(1.0) + eps * (1 + s))
    x = np.zeros((1, 2, 1, 1, 1, 32), np.uint16)
    x[...] = _bf16(np.full(32, 10.0))
    r = oracle.encode(w.shape, w.params, x, G, want_z=True)
    z_ref = (np.float64(10.0) * G[0, :, 0, 0].diagonal(axis1=-2, axis2=-1).astype(np.float64)).astype(np.float32)
    z = r["z"].reshape(2, 32)
    np.testing.assert_array_equal(z, z_ref)
    for s in range(2):
        s16, m16, q = _np_quantize(z[s], 4)
        assert q.max() == 15 and np.any(((z[s] - np.float32(m16)) / np.float32(s16)) > 15.5)
        np.testing.assert_array_equal(oracle.unpack(r["codes"][s * 16:(s + 1) * 16], 32, 4), q)


@pytest.mark.parametrize("backend,bits,blk,g", [(0, 4, 64, 128), (0, 3, 16, 16), (0, 6, 32, 32), (1, 3, 16, 64)])
def test_decode_error_within_quantization_bound(backend, bits, blk, g):
    """Decode (Sec. 3: Xhat = G^T Zhat): per gauge group, ||Xhat - X||_2 is at most the
    gauge-space bound sqrt(sum_j e_j^2) with e_j = s/2 + qmax*|s32 - s| + |min - m| (half a
    step, plus the fp16 rounding of scale and zero), since G is orthogonal."""
    w = _wl(L=1, B=2, H=2, T=48, d=128, group=g, backend=backend, bits=bits, block=blk, residual=8)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True)
    xh = oracle.decode(w.shape, w.params, r["codes"], r["scales"], r["residual"], G)
    z = r["z"].reshape(w.L, 2, w.B, w.H, w.T, w.d).astype(np.float64)
    qmax = 2 ** bits - 1
    e = np.zeros_like(z)
    nq = oracle.kivi_nq(w.T, w.residual, blk) if backend == 1 else w.T

    def ebound(v, s16, m16):
        s, m = float(np.float16(s16)), float(np.float16(m16))
        s32 = float(np.float32(np.float32(v.max()) - np.float32(v.min())) / np.float32(qmax))
        return s / 2 * (1 + 1e-6) + qmax * abs(s32 - s) + abs(float(v.min()) - m) + 1e-7

    sc = r["scales"].view(np.float16).reshape(-1, 2)
    if backend == 0:
        sc = sc.reshape(w.L, 2, w.B, w.H, w.T, w.d // blk, 2)
        for idx in np.ndindex(w.L, 2, w.B, w.H, w.T):
            for b in range(w.d // blk):
                v = z[idx][b * blk:(b + 1) * blk]
                e[idx][b * blk:(b + 1) * blk] = ebound(v, *sc[idx][b])
    else:
        kpb, vpb = (nq // blk) * w.d, nq * (w.d // blk)
        ks = sc[:w.B * w.H * kpb].reshape(w.B, w.H, nq // blk, w.d, 2)
        vs = sc[w.B * w.H * kpb:].reshape(w.B, w.H, nq, w.d // blk, 2)
        for b, h in np.ndindex(w.B, w.H):
            for tg in range(nq // blk):
                for c in range(w.d):
                    v = z[0, 0, b, h, tg * blk:(tg + 1) * blk, c]
                    e[0, 0, b, h, tg * blk:(tg + 1) * blk, c] = ebound(v, *ks[b, h, tg, c])
            for t in range(nq):
                for k in range(w.d // blk):
                    v = z[0, 1, b, h, t, k * blk:(k + 1) * blk]
                    e[0, 1, b, h, t, k * blk:(k + 1) * blk] = ebound(v, *vs[b, h, t, k])
    xf = _f32(x).astype(np.float64).reshape(z.shape)
    err = np.linalg.norm((xh.reshape(z.shape) - xf)[..., :nq, :].reshape(-1, g), axis=-1)
    bound = np.linalg.norm(e[..., :nq, :].reshape(-1, g), axis=-1) + 1e-5 * (1 + np.linalg.norm(xf[..., :nq, :].reshape(-1, g), axis=-1))
    assert np.all(err <= bound)
    # and the bound is not vacuous: the typical error is within a few times smaller
    assert np.median(err / bound) > 0.05


def test_flags_mark_near_boundary_values():
    w = _wl(L=1, B=1, H=1, T=64, d=64, group=16, block=32, bits=4)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True, want_flags=True)
    z = r["z"].reshape(-1, w.d)
    sc = r["scales"].reshape(-1, 2, 2)
    fl = r["flags"].reshape(-1, w.d)
    for row in range(z.shape[0]):
        for b in range(2):
            s = np.float32(sc[row, b, 0:1].view(np.float16)[0])
            m = np.float32(sc[row, b, 1:2].view(np.float16)[0])
            t = ((z[row, b * 32:(b + 1) * 32] - m) / s).astype(np.float64)
            near = np.abs(t - np.floor(t) - 0.5) < 1e-4
            np.testing.assert_array_equal(fl[row, b * 32:(b + 1) * 32].astype(bool), near)


# ---------------------------------------------------------------- invariants
@pytest.mark.parametrize("g", [8, 16, 32, 64, 128])
def test_no_compression_round_trip(g):
    """Sec. 3: without backend error G^{-1} G X = X up to numerical precision; the accepted
    bound is 1e-5 relative (the sanity rows of Sec. 4.4 report < 5.1e-8 NRMSE)."""
    w = _wl(L=2, B=1, H=2, T=6, d=128, group=g, backend=2)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G)
    xh = oracle.decode(w.shape, w.params, r["codes"], None, None, G)
    xf = _f32(x).astype(np.float64).ravel()
    rel = np.linalg.norm(xh - xf) / np.linalg.norm(xf)
    assert rel <= 1e-5, rel
    assert np.abs(xh - xf).max() <= 1e-5 * np.abs(xf).max()


def test_identity_clone_zero_error():
    """Sec. 4.4 sanity rows: the identity clone has zero cache error."""
    w = _wl(L=1, B=1, H=2, T=8, d=64, group=16, backend=2)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w, "identity")
    r = oracle.encode(w.shape, w.params, x, G)
    xh = oracle.decode(w.shape, w.params, r["codes"], None, None, G)
    np.testing.assert_array_equal(xh, _f32(x).astype(np.float64).ravel())


@pytest.mark.parametrize("backend,bits,blk,g", [(0, 4, 64, 128), (0, 6, 32, 32), (1, 3, 16, 64)])
def test_decode_error_equals_gauge_space_error(backend, bits, blk, g):
    """Orthogonality: within each group ||Xhat - X||_2 = ||Zhat - Z||_2 (Sec. 4.1), up to the
    fp32 chain's rounding of Z."""
    w = _wl(L=1, B=1, H=2, T=40, d=128, group=g, backend=backend, bits=bits, block=blk, residual=8)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    r = oracle.encode(w.shape, w.params, x, G, want_z=True)
    xh = oracle.decode(w.shape, w.params, r["codes"], r["scales"], r["residual"], G).reshape(-1, w.d // g, g)
    xf = _f32(x).astype(np.float64).reshape(-1, w.d // g, g)
    z = r["z"].astype(np.float64).reshape(-1, w.d // g, g)
    Gd = G.astype(np.float64)
    nq = oracle.kivi_nq(w.T, w.residual, blk) if backend == 1 else w.T
    rows = np.arange(xf.shape[0]).reshape(w.L, 2, w.B, w.H, w.T)[..., :nq].ravel()
    err_x = np.linalg.norm(xh[rows] - xf[rows], axis=-1)
    # ||Xhat - X|| = ||G^T Zhat - X|| = ||Zhat - G X|| and G X = z up to the chain error
    gz = np.einsum("lshrij,lsbhtrj->lsbhtri", Gd, xf.reshape(w.L, 2, w.B, w.H, w.T, w.d // g, g))
    assert np.abs(gz.reshape(z.shape)[rows] - z[rows]).max() <= 1e-5 * np.abs(xf).max()
    zhat = np.einsum("lshrij,lsbhtrj->lsbhtri", Gd, xh.reshape(w.L, 2, w.B, w.H, w.T, w.d // g, g)).reshape(z.shape)
    err_z = np.linalg.norm(zhat[rows] - z[rows], axis=-1)
    assert np.all(np.abs(err_x - err_z) <= 1e-5 * (1 + np.linalg.norm(xf[rows], axis=-1)))
    if backend == 1:  # residual window round-trips bit-exactly
        rr = np.setdiff1d(np.arange(xf.shape[0]), rows)
        np.testing.assert_array_equal(xh[rr], xf[rr])


def test_gauge_locality():
    """Sec. 3: the gauge mixes channels only inside a group and never mixes tokens, heads
    or layers: perturbing one group of one token changes only the blocks it overlaps."""
    w = _wl(L=2, B=2, H=2, T=5, d=64, group=16, block=32, bits=4)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    base = oracle.encode(w.shape, w.params, x, G)
    x2 = x.copy()
    l, s, b, h, t, grp = 1, 0, 1, 0, 3, 2
    x2[l, s, b, h, t, grp * 16:(grp + 1) * 16] = _bf16(np.full(16, 7.5))
    pert = oracle.encode(w.shape, w.params, x2, G)
    nb, pay = 2, 16
    c0 = base["codes"].reshape(w.L, 2, w.B, w.H, w.T, nb, pay)
    c1 = pert["codes"].reshape(w.L, 2, w.B, w.H, w.T, nb, pay)
    s0 = base["scales"].reshape(w.L, 2, w.B, w.H, w.T, nb, 2)
    s1 = pert["scales"].reshape(w.L, 2, w.B, w.H, w.T, nb, 2)
    changed = np.any(c0 != c1, axis=-1) | np.any(s0 != s1, axis=-1)
    expect = np.zeros_like(changed)
    expect[l, s, b, h, t, (grp * 16) // 32] = True
    assert changed[l, s, b, h, t, (grp * 16) // 32]
    np.testing.assert_array_equal(changed, expect)


def test_gauge_locality_kivi_keys():
    """KIVI keys: one token's perturbation changes only its own token group's key ranges of
    the channels in the perturbed gauge group (and nothing in other heads/layers)."""
    w = _wl(L=1, B=1, H=2, T=40, d=64, group=16, backend=1, bits=3, block=8, residual=8)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    base = oracle.encode(w.shape, w.params, x, G)
    x2 = x.copy()
    x2[0, 0, 0, 1, 10, 16:32] = _bf16(np.full(16, -6.0))
    pert = oracle.encode(w.shape, w.params, x2, G)
    nq = oracle.kivi_nq(40, 8, 8)
    key_bytes_per_bh = (nq // 8) * 64 * 3
    k0 = base["codes"][:2 * key_bytes_per_bh].reshape(2, nq // 8, 64, 3)
    k1 = pert["codes"][:2 * key_bytes_per_bh].reshape(2, nq // 8, 64, 3)
    changed = np.any(k0 != k1, axis=-1)
    assert changed[1, 1, 16:32].any()
    changed[1, 1, 16:32] = False
    assert not changed.any()
    np.testing.assert_array_equal(base["codes"][2 * key_bytes_per_bh:], pert["codes"][2 * key_bytes_per_bh:])


# ---------------------------------------------------------------- sizes and splits
def test_kivi_split():
    R = Gt = 128
    want = {1: 0, R - 1: 0, R: 0, R + Gt - 1: 0, R + Gt: 128, 32768: 32640}
    for T, nq in want.items():
        assert oracle.kivi_nq(T, R, Gt) == nq
        assert R <= T - nq < R + Gt or T < R


def test_packed_bytes_closed_form():
    """Measured bytes (Appendix metric table). Block-uniform with fp16 scale+zero stores
    bits + 32/block bits per value; KIVI adds a bf16 residual window."""
    for name, bpv in (("tiny", 5.0), ("llama3_8b", 4.5), ("gemma27b", 7.0), ("rolling", 4.5)):
        w = synth.WORKLOADS[name]
        c, s, r = oracle.packed_bytes(w.shape, w.params)
        n = w.L * 2 * w.B * w.H * (w.T_cap or w.T) * w.d
        assert r == 0
        assert (c + s) * 8 == bpv * n
        assert c * 8 == w.bits * n
    w = synth.WORKLOADS["llama3_8b"]
    assert oracle.packed_bytes(w.shape, w.params) == (268_435_456, 33_554_432, 0)
    w = synth.WORKLOADS["gemma27b"]
    assert oracle.packed_bytes(w.shape, w.params) == (2_315_255_808, 385_875_968, 0)
    w = synth.WORKLOADS["kivi3_qwen"]
    c, s, r = oracle.packed_bytes(w.shape, w.params)
    nq = 32640
    lbh = w.L * w.B * w.H
    assert c == 2 * lbh * nq * w.d * 3 // 8 == 1_403_781_120
    assert s == lbh * (nq // 128 * w.d + nq) * 4 == 116_981_760
    assert r == 2 * lbh * (w.T - nq) * w.d * 2 == 29_360_128
    w = w.replace(backend=2)
    assert oracle.packed_bytes(w.shape, w.params)[0] == w.n_elems * 4


# ---------------------------------------------------------------- rolling history
def test_rolling_append_matches_full_encode():
    """Sec. 4.4 rolling history: each new token passes through gauge and backend; earlier
    tokens' bytes never change and the history equals a full re-encode."""
    w = _wl(L=2, B=3, H=2, T=9, d=64, group=32, block=32, bits=4)
    x = synth.kv_cache(w, threads=1)
    G = synth.gauges(w)
    full = oracle.encode(w.shape, w.params, x, G)
    hist_shape = dict(w.shape, T=8, T_cap=9)
    h1 = oracle.encode(hist_shape, w.params, np.ascontiguousarray(x[..., :8, :]), G)
    app_shape = dict(w.shape, T=1, t0=8, T_cap=9)
    # the oracle writes only the appended rows; merge into the history buffers
    h2 = oracle.encode(app_shape, w.params, np.ascontiguousarray(x[..., 8:9, :]), G)
    c = h1["codes"].reshape(w.L, 2, w.B, w.H, 9, -1).copy()
    c[..., 8, :] = h2["codes"].reshape(w.L, 2, w.B, w.H, 9, -1)[..., 8, :]
    np.testing.assert_array_equal(c.ravel(), full["codes"])
    sc = h1["scales"].reshape(w.L, 2, w.B, w.H, 9, -1).copy()
    sc[..., 8, :] = h2["scales"].reshape(w.L, 2, w.B, w.H, 9, -1)[..., 8, :]
    np.testing.assert_array_equal(sc.ravel(), full["scales"])
    # rows before t0 are untouched by the append call
    assert not h2["codes"].reshape(w.L, 2, w.B, w.H, 9, -1)[..., :8, :].any()


# ---------------------------------------------------------------- status
def test_status_flags():
    w = _wl(T=2, d=32, group=8, block=16)
    G = synth.gauges(w, "identity")
    x = np.zeros((1, 2, 1, 1, 2, 32), np.uint16)
    x[0, 0, 0, 0, 1, 5] = 0x7F80  # +inf
    assert oracle.encode(w.shape, w.params, x, G)["status"] & 1
    x = np.zeros((1, 2, 1, 1, 2, 32), np.uint16)
    x[0, 1, 0, 0, 0, :16] = _bf16(np.linspace(-1e5, 1e5, 16))
    assert oracle.encode(w.shape, w.params, x, G)["status"] & 2
