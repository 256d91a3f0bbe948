"""Seeded synthetic inputs: KV caches shaped like the paper's models, and gauges.

This module draws random numbers and rounds them to bf16; it holds none of the codec's
arithmetic, and both the CUDA path and the CPU oracle take their inputs from it.

KV recipe (stands in for the frozen-model caches of the paper's six-model matrix and its
27B check, Sec. 4.4, which are not available here):
  keys   K[l,b,h,t,c] = N(0,1) * sk[l,h,c],  sk ~ lognormal(0, 0.5), and n_outlier seeded
         distinct channels per (l,h) multiplied by outlier_mult; sk is shared over b and t;
  values V[l,b,h,t,c] = N(0,1) * sv[l,b,h,t], sv ~ lognormal(0, sigma_v);
  both rounded to bf16 (round to nearest even).
Every (l, s, b, h) unit is drawn from its own counter-derived seed, so any unit can be
regenerated alone (the oracle checks sampled units of the full-size workloads).

Gauges: random orthogonal g x g matrices, Q of the QR factorisation of a seeded Gaussian
with the sign fix Q * diag(sign(diag R)) (the random-orthogonal control of Sec. 4.3),
computed in fp64 and stored fp32 as [L][2][H][d/g][g][g]. Identity, Hadamard and DCT-II
gauges (the fixed controls of Sec. 4.3) are provided as well.
"""
from __future__ import annotations

import math
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

_TAG_KEY_SCALE, _TAG_UNIT, _TAG_GAUGE, _TAG_OUTLIER = 11, 12, 13, 14


@dataclass(frozen=True)
class Workload:
    """A named cache workload: shape, KV distribution and codec parameters."""
    name: str
    L: int
    B: int
    H: int
    T: int
    d: int
    group: int
    backend: int          # 0 block-uniform, 1 KIVI, 2 none, 3 block-uniform tiles
    bits: int
    block: int
    residual: int = 0
    n_outlier: int = 4
    outlier_mult: float = 10.0
    sigma_v: float = 0.3
    kv_seed: int = 1000
    gauge_seed: int = 2000
    T_cap: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def shape(self) -> dict:
        return dict(L=self.L, B=self.B, H=self.H, T=self.T, d=self.d, t0=0, T_cap=self.T_cap)

    @property
    def params(self) -> dict:
        return dict(backend=self.backend, group=self.group, bits=self.bits, block=self.block,
                    residual=self.residual)

    @property
    def n_elems(self) -> int:
        return self.L * 2 * self.B * self.H * self.T * self.d

    def replace(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# The cache workloads: a tiny case, a Llama-3-8B-shaped cache (per-token blocks, and the
# paper's 16-token tiles), a Qwen/Mistral-shaped KIVI case (whole cache, and a KIVI decode loop
# over a 32k history), a Gemma-2-27B-shaped 6-bit case and a rolling decode step over a 16k
# history.
WORKLOADS = {
    "tiny": Workload("tiny", L=1, B=1, H=2, T=256, d=64, group=16, backend=0, bits=4, block=32,
                     n_outlier=2, outlier_mult=10.0, sigma_v=0.3, kv_seed=1000, gauge_seed=2000),
    "llama3_8b": Workload("llama3_8b", L=32, B=1, H=8, T=8192, d=128, group=128, backend=0, bits=4,
                          block=64, n_outlier=4, outlier_mult=10.0, sigma_v=0.3, kv_seed=1001,
                          gauge_seed=2001),
    "kivi3_qwen": Workload("kivi3_qwen", L=28, B=4, H=4, T=32768, d=128, group=64, backend=1, bits=3,
                           block=128, residual=128, n_outlier=4, outlier_mult=10.0, sigma_v=0.3,
                           kv_seed=1002, gauge_seed=2002),
    "gemma27b": Workload("gemma27b", L=46, B=2, H=16, T=8192, d=128, group=32, backend=0, bits=6,
                         block=32, n_outlier=8, outlier_mult=20.0, sigma_v=0.5, kv_seed=1003,
                         gauge_seed=2003),
    # the rolling step with attention read straight from the codes (4 query heads per KV head)
    "rolling_attn": Workload("rolling_attn", L=32, B=64, H=8, T=16384, d=128, group=128, backend=0, bits=4,
                             block=64, n_outlier=4, outlier_mult=10.0, sigma_v=0.3, kv_seed=1004,
                             gauge_seed=2004, T_cap=16384, extra={"n_rep": 4}),
    # a KIVI decode loop over the Qwen-shaped cache: a 32k history, one token appended per step
    "kivi3_stream": Workload("kivi3_stream", L=28, B=4, H=4, T=32768, d=128, group=64, backend=1, bits=3,
                             block=128, residual=128, n_outlier=4, outlier_mult=10.0, sigma_v=0.3,
                             kv_seed=1002, gauge_seed=2002, T_cap=32768),
    # the 8B cache under the Hadamard gauge, applied by fast Walsh-Hadamard transform
    "llama3_8b_hadamard": Workload("llama3_8b_hadamard", L=32, B=1, H=8, T=8192, d=128, group=128, backend=0,
                                   bits=4, block=64, n_outlier=4, outlier_mult=10.0, sigma_v=0.3, kv_seed=1001,
                                   gauge_seed=2001, extra={"gauge": "hadamard"}),
    # the paper's block-uniform block shape on the 8B cache: one range per 16-token x d tile
    "llama3_8b_tile": Workload("llama3_8b_tile", L=32, B=1, H=8, T=8192, d=128, group=128, backend=3,
                               bits=4, block=128, n_outlier=4, outlier_mult=10.0, sigma_v=0.3,
                               kv_seed=1001, gauge_seed=2001),
    # rolling: history of T_cap=16384 tokens; T is the decode length of one step
    "rolling": Workload("rolling", L=32, B=64, H=8, T=16384, d=128, group=128, backend=0, bits=4,
                        block=64, n_outlier=4, outlier_mult=10.0, sigma_v=0.3, kv_seed=1004,
                        gauge_seed=2004, T_cap=16384),
}


def _rng(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(entropy=seed, spawn_key=tuple(key))))


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(a, np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def key_scales(w: Workload, l: int, h: int) -> np.ndarray:
    """Per-channel key scale of layer l, head h (shared over batch and tokens)."""
    sk = _rng(w.kv_seed, _TAG_KEY_SCALE, l, h).lognormal(0.0, 0.5, size=w.d)
    if w.n_outlier:
        ch = _rng(w.kv_seed, _TAG_OUTLIER, l, h).choice(w.d, size=min(w.n_outlier, w.d), replace=False)
        sk[ch] *= w.outlier_mult
    return sk


def kv_unit(w: Workload, l: int, s: int, b: int, h: int, T: int | None = None, t_start: int = 0) -> np.ndarray:
    """bf16 bit patterns [T][d] of unit (l, s, b, h), tokens [t_start, t_start + T)."""
    T = w.T if T is None else T
    r = _rng(w.kv_seed, _TAG_UNIT, l, s, b, h)
    n_before = t_start * w.d
    if n_before:
        r.standard_normal(size=n_before, dtype=np.float32)  # advance past tokens before t_start
    x = r.standard_normal(size=(T, w.d), dtype=np.float32)
    if s == 0:
        x *= key_scales(w, l, h)[None, :].astype(np.float32)
    else:
        rv = _rng(w.kv_seed, _TAG_UNIT + 100, l, b, h)
        sv = rv.lognormal(0.0, w.sigma_v, size=t_start + T)[t_start:]
        x *= sv[:, None].astype(np.float32)
    return f32_to_bf16_bits(x)


def kv_cache(w: Workload, T: int | None = None, threads: int = 8) -> np.ndarray:
    """Full cache as bf16 bit patterns [L][2][B][H][T][d] (uint16)."""
    T = w.T if T is None else T
    out = np.empty((w.L, 2, w.B, w.H, T, w.d), np.uint16)

    def fill(idx):
        l, s, b, h = idx
        out[l, s, b, h] = kv_unit(w, l, s, b, h, T)

    units = [(l, s, b, h) for l in range(w.L) for s in range(2) for b in range(w.B) for h in range(w.H)]
    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        list(ex.map(fill, units))
    return out


def rolling_history_layer(w: Workload, threads: int = 8) -> np.ndarray:
    """History tokens [0, T_cap - 1) of the rolling workload for ONE layer, [1][2][B][H][T_cap-1][d].

    Every layer's history is this one draw (layer 0's units); the per-layer gauges still
    differ. A full independent draw of the 32-layer, batch-64, 16k-token history is 137 GB
    of bf16, too much to generate on the host for a test or a benchmark."""
    return kv_cache(w.replace(L=1, T=w.T_cap - 1), threads=threads)


def rolling_new_token(w: Workload, threads: int = 8) -> np.ndarray:
    """The token appended at position T_cap - 1 of every sequence, [L][2][B][H][1][d] (its own seed)."""
    return kv_cache(w.replace(T=1, kv_seed=w.kv_seed + 500), threads=threads)


def random_orthogonal(g: int, rng: np.random.Generator) -> np.ndarray:
    a = rng.standard_normal((g, g))
    q, r = np.linalg.qr(a)
    q = q * np.sign(np.diag(r))[None, :]
    return q


def gauges(w: Workload, kind: str = "random") -> np.ndarray:
    """fp32 [L][2][H][d/g][g][g] gauges of the given kind: random, identity, hadamard, dct."""
    g, R = w.group, w.d // w.group
    out = np.empty((w.L, 2, w.H, R, g, g), np.float32)
    if kind == "identity":
        out[...] = np.eye(g, dtype=np.float32)
        return out
    if kind == "hadamard":
        out[...] = hadamard(g).astype(np.float32)
        return out
    if kind == "dct":
        out[...] = dct2_matrix(g).astype(np.float32)
        return out
    assert kind == "random", kind
    for l in range(w.L):
        for s in range(2):
            for h in range(w.H):
                for r in range(R):
                    out[l, s, h, r] = random_orthogonal(g, _rng(w.gauge_seed, _TAG_GAUGE, l, s, h, r))
    return out


def hadamard(g: int) -> np.ndarray:
    """Sylvester Hadamard matrix scaled to be orthonormal (g a power of two)."""
    H = np.ones((1, 1))
    while H.shape[0] < g:
        H = np.block([[H, H], [H, -H]])
    return H / math.sqrt(g)


def dct2_matrix(g: int) -> np.ndarray:
    """Orthonormal DCT-II matrix C[k][n] = a_k cos(pi (2n+1) k / (2g))."""
    k = np.arange(g)[:, None]
    n = np.arange(g)[None, :]
    C = np.sqrt(2.0 / g) * np.cos(np.pi * (2 * n + 1) * k / (2 * g))
    C[0] /= math.sqrt(2.0)
    return C


def gauge_for(w: Workload, G: np.ndarray, l: int, s: int, h: int) -> np.ndarray:
    return G[l, s, h]
