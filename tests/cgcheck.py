"""Parity helpers: run the CUDA path through the C ABI and compare with the CPU oracle.

Tolerances (the accepted error of the method's outputs, with the library's readings):
  - packed byte counts and layout: exact;
  - codes: bit-exact, except elements the oracle flags (pre-rounding value within 1e-4
    steps of a rounding boundary), which may differ by +-1; at most 1e-4 of all elements;
  - scales and zeros: equal as fp16 values (1e-6 relative on an fp16 value is equality);
  - recovered cache, gauge groups whose packed input equals the oracle's (all of them for
    the oracle's own bytes; end to end, every group without a differing code): the bf16
    value must be a bf16 rounding of a value within the GPU's fp32 evaluation bound of the
    fp64 reference (decode_eval_bound), so it equals bf16(ref) unless ref lies that close
    to a rounding midpoint;
  - recovered cache, groups with a differing code: |xhat - ref| <= a + half a bf16 ulp at
    magnitude |ref| + a (the bf16 store), a = 1e-3 * max(|ref|, rms of ref over the gauge
    group) plus one quantization step times |G[j][i]| for every code j of the group that
    differs (the benchmark spec: 1e-3 relative plus one step on flagged elements). The values that
    pass only through the rms floor are counted.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2607_20538_gb300 import synth


def unpack_stream(buf: np.ndarray, n_codes: int, bits: int) -> np.ndarray:
    """Little-endian bit stream of `bits`-bit codes -> uint8 codes (numpy bit ops)."""
    b = np.unpackbits(np.ascontiguousarray(buf, np.uint8), bitorder="little")[: n_codes * bits]
    b = b.reshape(n_codes, bits).astype(np.uint16)
    return (b << np.arange(bits, dtype=np.uint16)).sum(axis=1).astype(np.uint8)


def codes_as_elements(w, codes: np.ndarray, T: int | None = None) -> np.ndarray:
    """Codes laid out like the cache, [L][2][B][H][T][d] (KIVI residual tokens = 0)."""
    T = w.T if T is None else T
    L, B, H, d, bits = w.L, w.B, w.H, w.d, w.bits
    if w.backend in (0, 3):  # block-uniform rows and tiles share the per-token code layout
        q = unpack_stream(codes, L * 2 * B * H * T * d, bits)
        return q.reshape(L, 2, B, H, T, d)
    Gt = w.block
    nq = oracle.kivi_nq(T, w.residual, Gt)
    out = np.zeros((L, 2, B, H, T, d), np.uint8)
    pay = Gt * bits // 8
    kpb, vpb = (nq // Gt) * d * pay, nq * d * bits // 8
    per_layer = B * H * (kpb + vpb)
    for l in range(L):
        lay = codes[l * per_layer:(l + 1) * per_layer]
        kq = unpack_stream(lay[:B * H * kpb], B * H * (nq // Gt) * d * Gt, bits).reshape(B, H, nq // Gt, d, Gt)
        out[l, 0, :, :, :nq, :] = kq.transpose(0, 1, 2, 4, 3).reshape(B, H, nq, d)
        vq = unpack_stream(lay[B * H * kpb:], B * H * nq * d, bits).reshape(B, H, nq, d)
        out[l, 1, :, :, :nq, :] = vq
    return out


def scales_as_elements(w, scales_u16: np.ndarray, T: int | None = None, which: int = 0) -> np.ndarray:
    """Per-element fp32 step size s (which = 0) or zero-point m (which = 1) of the element's block."""
    T = w.T if T is None else T
    L, B, H, d = w.L, w.B, w.H, w.d
    s = scales_u16.view(np.float16).reshape(-1, 2)[:, which].astype(np.float32)
    if w.backend == 0:
        nb = d // w.block
        return np.repeat(s.reshape(L, 2, B, H, T, nb), w.block, axis=-1)
    if w.backend == 3:  # one pair per 16-token tile block
        nb, TB = d // w.block, oracle.TILE_TOKENS
        st = s.reshape(L, 2, B, H, -1, nb)[:, :, :, :, np.arange(T) // TB, :]
        return np.repeat(st, w.block, axis=-1)
    Gt = w.block
    nq = oracle.kivi_nq(T, w.residual, Gt)
    out = np.zeros((L, 2, B, H, T, d), np.float32)
    kps, vps = (nq // Gt) * d, nq * (d // Gt)
    per_layer = B * H * (kps + vps)
    for l in range(L):
        lay = s[l * per_layer:(l + 1) * per_layer]
        ks = lay[:B * H * kps].reshape(B, H, nq // Gt, 1, d)
        out[l, 0, :, :, :nq, :] = np.broadcast_to(ks, (B, H, nq // Gt, Gt, d)).reshape(B, H, nq, d)
        vs = lay[B * H * kps:].reshape(B, H, nq, d // Gt)
        out[l, 1, :, :, :nq, :] = np.repeat(vs, Gt, axis=-1)
    return out


def compare_codes(w, gpu_codes, ref_codes, flags, T=None, max_frac=1e-4):
    """Element-wise code check; returns the boolean mismatch mask [L][2][B][H][T][d]."""
    qg = codes_as_elements(w, gpu_codes, T)
    qr = codes_as_elements(w, ref_codes, T)
    mism = qg != qr
    n = int(mism.sum())
    if n:
        fl = flags.reshape(qr.shape).astype(bool)
        assert fl[mism].all(), f"{int((~fl[mism]).sum())} unflagged code mismatches"
        diff = np.abs(qg[mism].astype(np.int32) - qr[mism].astype(np.int32))
        assert (diff == 1).all(), "flagged codes differ by more than one"
        assert n <= max_frac * qr.size, f"{n} flagged mismatches > {max_frac} of {qr.size}"
    else:
        assert np.array_equal(gpu_codes, ref_codes), "codes equal element-wise but bytes differ"
    return mism


def compare_scales(gpu_u16, ref_u16):
    a = gpu_u16.view(np.float16).astype(np.float32)
    b = ref_u16.view(np.float16).astype(np.float32)
    both_nan = np.isnan(a) & np.isnan(b)
    bad = ~((a == b) | both_nan)
    assert not bad.any(), f"{int(bad.sum())} scale/zero values differ, first at {np.argmax(bad)}"


def decode_tolerance(w, ref: np.ndarray, G: np.ndarray, step_mism: np.ndarray | None = None,
                     rms_floor: bool = True) -> np.ndarray:
    """Per-element bound for |xhat_gpu - ref| (ref: fp64 oracle decode, cache layout)."""
    g = w.group
    shp = (w.L, 2, w.B, w.H, -1, w.d // g, g)
    r = ref.reshape(shp)
    rms = np.sqrt(np.mean(r ** 2, axis=-1, keepdims=True))
    tol = 1e-3 * (np.maximum(np.abs(r), rms) if rms_floor else np.abs(r))
    if step_mism is not None and step_mism.any():
        # one quantization step through |G^T|: sum_j s_j |G[j][i]| over differing codes j
        sm = step_mism.reshape(shp).astype(np.float64)
        tol = tol + np.einsum("lshrji,lsbhtrj->lsbhtri", np.abs(G.astype(np.float64)), sm)
    # the bf16 store rounds the GPU's value, which lies within `tol` of ref: half an ulp at
    # that value's magnitude, bounded by the ulp at |ref| + tol (it may cross a power of two)
    half_ulp = np.ldexp(1.0, np.frexp(np.abs(r) + tol)[1] - 9)
    return (tol + half_ulp + 1e-30).reshape(ref.shape)


def bf16_rne(v: np.ndarray) -> np.ndarray:
    """Round fp64 values to bf16 (nearest, ties to even), returned as fp64 (normal range)."""
    m, e = np.frexp(v)  # v = m 2^e, 0.5 <= |m| < 1: keep 8 significant bits
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def decode_eval_bound(w, G: np.ndarray, codes: np.ndarray, scales_u16: np.ndarray, T: int | None = None):
    """Bound on |v - xhat| for the GPU's fp32 value v of xhat_i = sum_j G[j][i] zhat_j before its
    bf16 store, given the exact packed input (cache layout, fp64).

    M1 = sum_j |G[j][i]| |zhat_j| bounds what the bf16 splits leave out: G^T as hi + lo
    (residual <= 2^-16 |G|) and, for KIVI keys, zhat as hi + lo with the lo x lo product
    dropped (3 x 2^-16 in all); the CUDA-core kernels' fp32 sums stay below 2^-17 M1.
    M2 = sum_j |G[j][i]| (s_j (o + q_j) + |m_j - o s_j|), o = 2^b (0 for 8-bit codes), bounds
    the magnitudes of the fp32 terms of the row kernels, which multiply the integer codes
    offset by o (exact in bf16) and add the zero-point term (m - o s) c_k: their tensor-core
    accumulation and epilogue roundings stay below 12 u M2 (u = 2^-24; K / 16 + 4 steps, K <= 64
    per sub-block, or <= 128 with one sub-block and g = 128). The bound takes 2^-15 M1 (rows) or
    2^-14 M1 (KIVI, keys) plus 2^-20 M2 (16 u).
    """
    g = w.group
    q = codes_as_elements(w, codes, T).astype(np.float64)
    s = scales_as_elements(w, scales_u16, T).astype(np.float64)
    m = scales_as_elements(w, scales_u16, T, which=1).astype(np.float64)
    o = float(1 << w.bits) if w.bits < 8 else 0.0
    zhat = q * s + m
    shp = (w.L, 2, w.B, w.H, -1, w.d // g, g)
    aG = np.abs(G.astype(np.float64))
    M1 = np.einsum("lshrji,lsbhtrj->lsbhtri", aG, np.abs(zhat).reshape(shp))
    M2 = np.einsum("lshrji,lsbhtrj->lsbhtri", aG, (s * (o + q) + np.abs(m - o * s)).reshape(shp))
    c1 = 2.0 ** -14 if w.backend == 1 else 2.0 ** -15
    return (c1 * M1 + 2.0 ** -20 * M2).reshape(-1)


def compare_decode(w, got_bf16: np.ndarray, ref: np.ndarray, G: np.ndarray, step_mism=None,
                   codes=None, scales_u16=None, T=None) -> dict:
    """Decoded bf16 values against the fp64 oracle decode `ref`.

    Given the oracle's packed input (`codes`, `scales_u16`), every gauge group whose codes
    equal the oracle's gets the tight check: the GPU value must be a bf16 rounding of some
    value within decode_eval_bound of ref, bf16(ref - eb) <= got <= bf16(ref + eb); so it
    equals bf16(ref) except where ref lies within eb of a rounding midpoint. Groups with a
    differing code (end to end), and calls without the packed input, get decode_tolerance.
    Returns counts: values checked tightly, those of them that differ from bf16(ref), and
    (loose groups) those that pass only through the rms floor of the tolerance.
    """
    got = synth.bf16_bits_to_f32(got_bf16).astype(np.float64).reshape(-1)
    r = ref.reshape(-1)
    g = w.group
    ngrp = r.size // g
    loose_grp = np.zeros(ngrp, bool) if codes is not None else np.ones(ngrp, bool)
    if step_mism is not None and step_mism.any():
        loose_grp |= step_mism.reshape(ngrp, g).any(axis=1)
    loose = np.repeat(loose_grp, g)
    stats = {"tight": int((~loose).sum()), "tight_not_rne": 0, "rms_floor_only": 0}
    if stats["tight"]:
        eb = decode_eval_bound(w, G, codes, scales_u16, T)[~loose]
        rt, gt = r[~loose], got[~loose]
        lo, hi = bf16_rne(rt - eb), bf16_rne(rt + eb)
        bad = (gt < lo) | (gt > hi)
        assert not bad.any(), (f"{int(bad.sum())} decoded values are not a bf16 rounding of a value within the "
                               f"evaluation bound of the reference; first at element "
                               f"{np.flatnonzero(~loose)[np.argmax(bad)]}")
        stats["tight_not_rne"] = int((gt != bf16_rne(rt)).sum())
    if loose.any():
        tol = decode_tolerance(w, ref, G, step_mism).reshape(-1)
        err = np.abs(got - r)
        bad = loose & (err > tol)
        assert not bad.any(), (f"{int(bad.sum())} decoded values outside tolerance; worst err {err[bad].max():.3g} "
                               f"at element {np.argmax(np.where(loose, err - tol, -np.inf))}")
        tol_rel = decode_tolerance(w, ref, G, step_mism, rms_floor=False).reshape(-1)
        stats["rms_floor_only"] = int((loose & (err > tol_rel)).sum())
    return stats


def stream_to_batch(w, T: int, T_cap: int, codes: np.ndarray, scales_u16: np.ndarray, ring_u16: np.ndarray):
    """The state of a KIVI stream of capacity T_cap holding T tokens, in the batch layout of a
    T-token KIVI encode: (codes, scales, residual). Keys [B][H][n_q/Gt][d][pay] and values
    [B][H][n_q][d/Gt][pay] per layer are cut from the capacity layout; the residual tokens
    [n_q, T) come from ring slot t mod (R + Gt)."""
    L, B, H, d, Gt, bits, R = w.L, w.B, w.H, w.d, w.block, w.bits, w.residual
    pay, nb, W = Gt * bits // 8, d // Gt, R + Gt
    nq, ncap = oracle.kivi_nq(T, R, Gt), oracle.kivi_nq(T_cap, R, Gt)
    kc_cap, vc_cap = (ncap // Gt) * d * pay, ncap * nb * pay
    ks_cap, vs_cap = (ncap // Gt) * d, ncap * nb
    c = codes.reshape(L, -1)
    s = scales_u16.reshape(-1, 2).reshape(L, -1, 2)
    out_c, out_s = [], []
    for l in range(L):
        kc = c[l, :B * H * kc_cap].reshape(B, H, kc_cap)[:, :, :(nq // Gt) * d * pay]
        vc = c[l, B * H * kc_cap:].reshape(B, H, vc_cap)[:, :, :nq * nb * pay]
        ks = s[l, :B * H * ks_cap].reshape(B, H, ks_cap, 2)[:, :, :(nq // Gt) * d]
        vs = s[l, B * H * ks_cap:].reshape(B, H, vs_cap, 2)[:, :, :nq * nb]
        out_c += [kc.ravel(), vc.ravel()]
        out_s += [ks.ravel(), vs.ravel()]
    ring = ring_u16.reshape(L, 2, B, H, W, d)
    resid = ring[:, :, :, :, np.arange(nq, T) % W, :]
    return np.concatenate(out_c), np.concatenate(out_s), np.ascontiguousarray(resid).ravel()
