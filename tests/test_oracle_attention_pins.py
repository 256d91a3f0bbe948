"""Pins of the oracle's attention over the recovered cache (CPU only).

The decoded cache is consumed by standard softmax attention (Fig. 1: the inverse gauge restores
the cache before attention; Sec. 3 leaves attention semantics unchanged), with grouped query
heads. The oracle's fp64 attention is pinned against torch's scaled_dot_product_attention in
float64 (a library routine), and against special cases: one token gives its value row, equal
keys give the mean of the values, permuting tokens changes nothing, and scores far above the
exp range still give the dominant value.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

torch = pytest.importorskip("torch")


def _rand(shape, rng, s=1.0):
    return rng.normal(0.0, s, size=shape)


def _qbf16(q):
    return synth.f32_to_bf16_bits(np.asarray(q, np.float32))


@pytest.mark.parametrize("n_rep,T,d", [(4, 37, 64), (1, 16, 32), (2, 130, 128)])
def test_attention_matches_torch_sdpa(n_rep, T, d):
    rng = np.random.default_rng(5)
    L, B, H = 2, 2, 3
    xh = _rand((L, 2, B, H, T, d), rng)
    qb = _qbf16(_rand((L, B, H, n_rep, d), rng, 0.5))
    scale = 1.0 / np.sqrt(d)
    got = oracle.attention(dict(L=L, B=B, H=H, T=T, d=d), n_rep, qb, xh, scale)
    q = torch.from_numpy(synth.bf16_bits_to_f32(qb).astype(np.float64))         # [L][B][H][n_rep][d]
    K = torch.from_numpy(xh[:, 0]).unsqueeze(3).expand(L, B, H, n_rep, T, d)     # KV head shared by n_rep
    V = torch.from_numpy(xh[:, 1]).unsqueeze(3).expand(L, B, H, n_rep, T, d)
    ref = torch.nn.functional.scaled_dot_product_attention(q.unsqueeze(-2), K, V, scale=scale).squeeze(-2)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(6)
    L, B, H, d, n_rep = 1, 1, 2, 32, 2
    sh = lambda T: dict(L=L, B=B, H=H, T=T, d=d)
    qb = _qbf16(_rand((L, B, H, n_rep, d), rng))
    # one token: the output is its value row
    xh = _rand((L, 2, B, H, 1, d), rng)
    o = oracle.attention(sh(1), n_rep, qb, xh, 0.125)
    np.testing.assert_array_equal(o, np.broadcast_to(xh[:, 1][:, :, :, None, 0, :], o.shape))
    # equal keys: the mean of the values
    T = 9
    xh = _rand((L, 2, B, H, T, d), rng)
    xh[:, 0] = xh[:, 0, :, :, :1, :]
    o = oracle.attention(sh(T), n_rep, qb, xh, 0.125)
    np.testing.assert_allclose(o, np.broadcast_to(xh[:, 1].mean(axis=-2)[:, :, :, None, :], o.shape), rtol=1e-13,
                               atol=1e-15)
    # token permutation (keys and values together)
    xh = _rand((L, 2, B, H, T, d), rng)
    perm = rng.permutation(T)
    o1 = oracle.attention(sh(T), n_rep, qb, xh, 0.125)
    o2 = oracle.attention(sh(T), n_rep, qb, np.ascontiguousarray(xh[:, :, :, :, perm, :]), 0.125)
    np.testing.assert_allclose(o1, o2, rtol=1e-12, atol=1e-14)
    # scores of order 1e4: the largest dominates, nothing overflows
    xh = _rand((L, 2, B, H, T, d), rng)
    q = synth.bf16_bits_to_f32(qb).astype(np.float64)
    xh[0, 0, 0, :, 4, :] = 1e4 * np.sign(q[0, 0, :, 0, :])     # token 4 aligned with query 0 of every head
    o = oracle.attention(sh(T), n_rep, qb, xh, 1.0)
    assert np.isfinite(o).all()
    np.testing.assert_allclose(o[0, 0, :, 0, :], xh[0, 1, 0, :, 4, :], rtol=1e-12, atol=1e-12)
