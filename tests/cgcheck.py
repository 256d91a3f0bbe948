"""Parity helpers: run the CUDA path through the C ABI and compare with the CPU oracle.

Tolerances (the accepted error of the method's outputs, with the library's readings):
  - packed byte counts and layout: exact;
  - codes: bit-exact, except elements the oracle flags (pre-rounding value within 1e-4
    steps of a rounding boundary), which may differ by +-1; at most 1e-4 of all elements;
  - scales and zeros: equal as fp16 values (1e-6 relative on an fp16 value is equality);
  - recovered cache: |xhat - ref| <= a + half a bf16 ulp at magnitude |ref| + a (the bf16
    store), a = 1e-3 * max(|ref|, rms of ref over the gauge group) plus, end to end, one
    quantization step times |G[j][i]| for every code j of the group that differs.
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
    if w.backend == 0:
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


def scales_as_elements(w, scales_u16: np.ndarray, T: int | None = None) -> np.ndarray:
    """Per-element fp32 step size s (the fp16 scale of the element's block)."""
    T = w.T if T is None else T
    L, B, H, d = w.L, w.B, w.H, w.d
    s = scales_u16.view(np.float16).reshape(-1, 2)[:, 0].astype(np.float32)
    if w.backend == 0:
        nb = d // w.block
        return np.repeat(s.reshape(L, 2, B, H, T, nb), w.block, axis=-1)
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


def decode_tolerance(w, ref: np.ndarray, G: np.ndarray, step_mism: np.ndarray | None = None) -> np.ndarray:
    """Per-element bound for |xhat_gpu - ref| (ref: fp64 oracle decode, cache layout)."""
    g = w.group
    shp = (w.L, 2, w.B, w.H, -1, w.d // g, g)
    r = ref.reshape(shp)
    rms = np.sqrt(np.mean(r ** 2, axis=-1, keepdims=True))
    tol = 1e-3 * np.maximum(np.abs(r), rms)
    if step_mism is not None and step_mism.any():
        # one quantization step through |G^T|: sum_j s_j |G[j][i]| over differing codes j
        sm = step_mism.reshape(shp).astype(np.float64)
        tol = tol + np.einsum("lshrji,lsbhtrj->lsbhtri", np.abs(G.astype(np.float64)), sm)
    # the bf16 store rounds the GPU's value, which lies within `tol` of ref: half an ulp at
    # that value's magnitude, bounded by the ulp at |ref| + tol (it may cross a power of two)
    half_ulp = np.ldexp(1.0, np.frexp(np.abs(r) + tol)[1] - 9)
    return (tol + half_ulp + 1e-30).reshape(ref.shape)


def compare_decode(w, got_bf16: np.ndarray, ref: np.ndarray, G: np.ndarray, step_mism=None):
    got = synth.bf16_bits_to_f32(got_bf16).astype(np.float64).reshape(ref.shape)
    tol = decode_tolerance(w, ref, G, step_mism)
    err = np.abs(got - ref)
    bad = err > tol
    assert not bad.any(), (f"{int(bad.sum())} decoded values outside tolerance; worst err {err.max():.3g} "
                           f"at {np.unravel_index(np.argmax(err - tol), err.shape)}")
