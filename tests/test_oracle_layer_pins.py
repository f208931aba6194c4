"""Pins of the fp64 reader-layer oracle (CPU).

* block-skip exactness at layer level (arXiv 2609.32395, Sec. 3.1 and App.
  "Serving measurements": the final block computed alone equals the full
  reader pass): a masked full pass of the whole layer over B blocks (torch
  SDPA, block-diagonal causal self-attention, block-causal cross-attention
  with the null column) equals the one-block pass of every block;
* a decode step equals the one-block pass at its token;
* closed forms: GELU at textbook values of the normal CDF, LayerNorm moments,
  zero residual branches.
"""
import math

import numpy as np
import pytest
import torch

from oracle.reader_layer import LayerWeights, gelu, layer_norm, reader_layer_decode, reader_layer_prefill


def rand_weights(rng, d, scale=None):
    s = 1.0 / math.sqrt(d) if scale is None else scale
    r = lambda *shape: rng.standard_normal(shape) * s  # noqa: E731
    g = lambda: 1.0 + 0.1 * rng.standard_normal(d)  # noqa: E731
    bb = lambda: 0.1 * rng.standard_normal(d)  # noqa: E731
    return LayerWeights(ln1_g=g(), ln1_b=bb(), w_qkv=r(d, 3 * d), w_os=r(d, d), ln2_g=g(), ln2_b=bb(),
                        w_qc=r(d, d), w_oc=r(d, d), w_kc=r(d, d), w_vc=r(d, d), ln3_g=g(), ln3_b=bb(),
                        w_1=r(d, 4 * d), w_2=rng.standard_normal((4 * d, d)) / math.sqrt(4 * d))


def _sdpa(q, k, v, mask):
    """q [H][n][D], k/v [H][m][D], boolean mask [n][m]; rows without keys -> 0."""
    o = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q), torch.from_numpy(k),
                                                         torch.from_numpy(v), attn_mask=torch.from_numpy(mask))
    o = o.numpy().copy()
    o[:, ~mask.any(axis=1), :] = 0.0
    return o


def full_layer_pass(X, mu, w, H, D, b, nu=None):
    """The reader layer over all B*b tokens at once with explicit masks.
    X: [B*b][d]; mu: [B][R][d] memory rows of every block."""
    n, d = X.shape
    B, R, _ = mu.shape
    pos = np.arange(n)
    blk = pos // b
    h1 = layer_norm(X, w.ln1_g, w.ln1_b)
    qkv = h1 @ w.w_qkv
    q, k, v = (qkv[:, i * d:(i + 1) * d].reshape(n, H, D).transpose(1, 0, 2) for i in range(3))
    sa_mask = (blk[:, None] == blk[None, :]) & (pos[None, :] <= pos[:, None])
    sa = _sdpa(q, k, v, sa_mask).transpose(1, 0, 2).reshape(n, d)
    X1 = X + sa @ w.w_os
    h2 = layer_norm(X1, w.ln2_g, w.ln2_b)
    qc = (h2 @ w.w_qc).reshape(n, H, D).transpose(1, 0, 2)
    rows = mu.reshape(B * R, d)                          # memory rows in block order
    mk = (rows @ w.w_kc).reshape(B * R, H, D).transpose(1, 0, 2)
    mv = (rows @ w.w_vc).reshape(B * R, H, D).transpose(1, 0, 2)
    ca_mask = np.repeat(np.arange(B), R)[None, :] < blk[:, None]
    if nu is not None:
        kn = (nu @ w.w_kc).reshape(H, D)
        vn = (nu @ w.w_vc).reshape(H, D)
        mk = np.concatenate([kn[:, None], mk], axis=1)
        mv = np.concatenate([vn[:, None], mv], axis=1)
        ca_mask = np.concatenate([np.ones((n, 1), bool), ca_mask], axis=1)
    ca = _sdpa(qc, mk, mv, ca_mask).transpose(1, 0, 2).reshape(n, d)
    X2 = X1 + ca @ w.w_oc
    h3 = layer_norm(X2, w.ln3_g, w.ln3_b)
    return X2 + gelu(h3 @ w.w_1) @ w.w_2


@pytest.mark.parametrize("with_null", [False, True])
def test_one_block_layer_equals_full_pass(with_null):
    rng = np.random.default_rng(31 + with_null)
    B, b, H, D = 4, 8, 2, 8
    d = H * D
    w = rand_weights(rng, d)
    X = rng.standard_normal((B * b, d))
    mu = rng.standard_normal((B, b, d))
    nu = rng.standard_normal(d) if with_null else None
    full = full_layer_pass(X, mu, w, H, D, b, nu)
    perm = rng.permutation(B)
    for i in range(B):
        sl = slice(i * b, (i + 1) * b)
        out, _, _ = reader_layer_prefill(X[sl], perm, mu[perm], i, w, H, D, nu)
        np.testing.assert_allclose(out, full[sl], rtol=0, atol=1e-11)


@pytest.mark.parametrize("rope_window", [0, 2])
def test_decode_step_equals_one_block_row(rope_window):
    rng = np.random.default_rng(37)
    b, H, D, nblk = 8, 2, 8, 3
    d = H * D
    w = rand_weights(rng, d)
    X = rng.standard_normal((b, d))
    mu = rng.standard_normal((nblk, b, d))
    nu = rng.standard_normal(d)
    out, ks, vs = reader_layer_prefill(X, np.arange(nblk), mu, nblk, w, H, D, nu, rope_window=rope_window)
    for p in (0, 3, b - 1):
        xo, kn, vn = reader_layer_decode(X[p], np.arange(nblk), mu, nblk, p, ks[:p], vs[:p], w, H, D, nu,
                                         rope_window=rope_window)
        np.testing.assert_allclose(xo, out[p], rtol=0, atol=1e-12)
        np.testing.assert_allclose(kn, ks[p], rtol=0, atol=1e-12)


def test_gelu_textbook_values():
    # GELU(x) = x Phi(x); Phi(1), Phi(2) from normal-distribution tables
    np.testing.assert_allclose(gelu(np.array([1.0, -1.0, 2.0, 0.0])),
                               [0.8413447460685429, -0.15865525393145707, 2 * 0.9772498680518208, 0.0],
                               rtol=0, atol=1e-15)
    assert abs(gelu(np.array([8.0]))[0] - 8.0) < 1e-12      # identity for large x
    assert abs(gelu(np.array([-8.0]))[0]) < 1e-12           # zero for very negative x


def test_layer_norm_moments_and_constant_row():
    rng = np.random.default_rng(41)
    x = 3.0 + 2.0 * rng.standard_normal((5, 64))
    y = layer_norm(x, np.ones(64), np.zeros(64))
    np.testing.assert_allclose(y.mean(axis=1), 0.0, atol=1e-12)
    var = x.var(axis=1)
    np.testing.assert_allclose((y ** 2).mean(axis=1), var / (var + 1e-5), rtol=1e-12)
    c = np.full((1, 64), 7.0)
    bias = rng.standard_normal(64)
    np.testing.assert_array_equal(layer_norm(c, rng.standard_normal(64), bias)[0], bias)


def test_zero_branches_leave_the_stream_unchanged():
    rng = np.random.default_rng(43)
    b, H, D, nblk = 8, 2, 8, 2
    d = H * D
    w = rand_weights(rng, d)
    w.w_os[:] = 0.0
    w.w_oc[:] = 0.0
    w.w_2[:] = 0.0
    X = rng.standard_normal((b, d))
    out, _, _ = reader_layer_prefill(X, np.arange(nblk), rng.standard_normal((nblk, b, d)), nblk, w, H, D)
    np.testing.assert_array_equal(out, X)


def test_grouped_kv_heads_equal_repeated_full_heads():
    """Grouped-query attention (H_kv key/value heads, query head h reading
    head h // G) equals ordinary multi-head attention whose key/value maps
    repeat each grouped head's columns G times."""
    rng = np.random.default_rng(47)
    b, H, D, nblk, G = 8, 4, 8, 3, 2
    d, kvd = H * D, H * D // G
    w = rand_weights(rng, d)
    w.w_qkv = rng.standard_normal((d, d + 2 * kvd)) / np.sqrt(d)
    w.w_kc = rng.standard_normal((d, kvd)) / np.sqrt(d)
    w.w_vc = rng.standard_normal((d, kvd)) / np.sqrt(d)

    def expand(m):  # [d][H_kv*D] -> [d][H*D], head h = grouped head h // G
        return np.repeat(m.reshape(m.shape[0], H // G, D), G, axis=1).reshape(m.shape[0], d)

    full = LayerWeights(**{**w.__dict__})
    full.w_qkv = np.concatenate([w.w_qkv[:, :d], expand(w.w_qkv[:, d:d + kvd]), expand(w.w_qkv[:, d + kvd:])], axis=1)
    full.w_kc, full.w_vc = expand(w.w_kc), expand(w.w_vc)
    X = rng.standard_normal((b, d))
    mu = rng.standard_normal((nblk, b, d))
    nu = rng.standard_normal(d)
    a, ks, vs = reader_layer_prefill(X, np.arange(nblk), mu, nblk, w, H, D, nu)
    c, ks_full, _ = reader_layer_prefill(X, np.arange(nblk), mu, nblk, full, H, D, nu)
    np.testing.assert_allclose(a, c, rtol=0, atol=1e-12)
    assert ks.shape == (b, H // G, D)
    np.testing.assert_allclose(np.repeat(ks, G, axis=1), ks_full, rtol=0, atol=1e-12)
    xo, _, _ = reader_layer_decode(X[3], np.arange(nblk), mu, nblk, 3, ks[:3], vs[:3], w, H, D, nu)
    np.testing.assert_allclose(xo, a[3], rtol=0, atol=1e-12)
