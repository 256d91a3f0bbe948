"""Planted quantization blocks with hand-worked fp16 scales, zeros and codes (Sec. 4.3).

Every value is bf16-exact. With identity gauges the gauge-space values equal the inputs, so
each block kind fixes its fp16 scale (max - min) / (2^b - 1) and zero (min) by hand:

  0  half-integer codes: min 0, max 2^b - 1, so scale 1.0, zero 0 and t = z exactly;
  1  scale on an fp16 midpoint, (max - min) / qmax = 1 + 2^-11, rounds to 1.0 (even);
     the max repeats across the block;
  2  constant block 2.5: scale 0, zero 2.5, all codes 0;
  3  zeros: scale 0, zero 0;
  4  zero on an fp16 subnormal midpoint, 1.5 * 2^-24, rounds to 2^-23 (even);
  5  scale on the other midpoint, 1 + 3 * 2^-11, rounds to 1 + 2^-9 (even).
"""
import numpy as np

from paper_2607_20538_gb300 import synth

H16_ONE = 0x3C00        # 1.0
H16_ONE_2M9 = 0x3C02    # 1 + 2^-9
H16_2P5 = 0x4100        # 2.5
H16_2M23 = 0x0002       # 2^-23 (subnormal, mantissa 2)
N_KINDS = 6


def block_values(kind: int, n: int, qmax: int, rng) -> np.ndarray:
    """fp32 values (all bf16-exact) of one quantization block of n values."""
    if kind == 0:
        # code ties: min 0, max qmax, so s = 1, m = 0 and t = z exactly
        v = rng.integers(0, qmax, n).astype(np.float32) + 0.5
        i = rng.choice(n, 2, replace=False)
        v[i[0]], v[i[1]] = 0.0, float(qmax)
        return v
    if kind == 1:
        # scale on an fp16 midpoint: (max - min) / qmax = 1 + 2^-11 (rounds to 1.0, even),
        # max repeated all over the block (many exact candidates)
        v = np.full(n, float(qmax), np.float32)
        i = rng.choice(n, 4, replace=False)
        v[i[0]] = -qmax * 2.0 ** -11
        v[i[1:]] = 1.25
        return v
    if kind == 2:
        # constant block: scale 0, every code 0; every value is a candidate extreme
        return np.full(n, 2.5, np.float32)
    if kind == 3:
        return np.zeros(n, np.float32)
    if kind == 4:
        # zero on an fp16 subnormal midpoint: min = 1.5 * 2^-24 rounds to 2^-23 (even)
        v = rng.uniform(0.125, 1.0, n).astype(np.float32)
        v = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(v))
        v[rng.integers(0, n, 4)] = 1.5 * 2.0 ** -24
        return v
    # the other midpoint direction: (max - min) / qmax = 1 + 3 * 2^-11 rounds to 1 + 2^-9
    v = np.full(n, float(qmax), np.float32)
    i = rng.choice(n, 7, replace=False)
    v[i[:2]] = -3 * qmax * 2.0 ** -11
    v[i[2:]] = 0.75
    return v


def planted_rows(w, rng) -> tuple[np.ndarray, np.ndarray]:
    """bf16 cache whose token rows cycle through the block kinds, and the kind per row."""
    qmax = (1 << w.bits) - 1
    nbk = w.d // w.block
    x = np.empty((w.L, 2, w.B, w.H, w.T, w.d), np.float32)
    kind = np.empty((w.L, 2, w.B, w.H, w.T, nbk), np.int64)
    for idx in np.ndindex(w.L, 2, w.B, w.H, w.T):
        for b in range(nbk):
            k = (idx[-1] + b) % N_KINDS
            kind[idx + (b,)] = k
            x[idx + (slice(b * w.block, (b + 1) * w.block),)] = block_values(k, w.block, qmax, rng)
    return synth.f32_to_bf16_bits(x).reshape(x.shape), kind


def expected_scale_zero(kind: int, qmax: int):
    """(scale bits, zero bits) fixed by hand for each block kind."""
    return {0: (H16_ONE, 0), 1: (H16_ONE, None), 2: (0, H16_2P5), 3: (0, 0), 4: (None, H16_2M23),
            5: (H16_ONE_2M9, None)}[kind]
