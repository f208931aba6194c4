"""Pins of the fp64 SMem+RoPE composite oracle (CPU).

* the rotation equals the matrix exponential of the rotary generator
  (scipy), composes additively and preserves norms;
* closed forms of a one-row cross-attention with the null row, with and
  without the saturating window (arXiv 2609.32395, App. "Needle": key phase
  max(j, i - W), query phase i);
* saturation is the identity inside the trained range (i <= W); without the
  null row the cross-attention depends only on block offsets (shift
  invariance); far blocks share one phase; values are never rotated;
* the one-block pass equals the masked full pass with per-token phases, and
  a decode step equals the one-block row at its token.
"""
import numpy as np
import pytest
import torch
from scipy.linalg import expm

from oracle.rope import key_phase, reader_decode_rope, reader_prefill_rope, rope


def generator(D, base=1e4):
    G = np.zeros((D, D))
    for m in range(D // 2):
        th = base ** (-2.0 * m / D)
        G[2 * m + 1, 2 * m] = th
        G[2 * m, 2 * m + 1] = -th
    return G


@pytest.mark.parametrize("D", [2, 8, 64])
def test_rotation_is_the_exponential_of_the_generator(D):
    rng = np.random.default_rng(D)
    x = rng.standard_normal(D)
    for phi in (0.0, 1.0, 7.0, 15.0, 63.0):
        # expm of a 63-radian rotation carries ~1e-12 of its own error
        np.testing.assert_allclose(rope(x, phi), expm(phi * generator(D)) @ x, rtol=0, atol=1e-9)


def test_rotation_group_and_norm():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((5, 4, 32))
    np.testing.assert_allclose(rope(rope(x, 3.0), 9.0), rope(x, 12.0), atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(rope(x, 11.0), axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(rope(rope(x, 4.0), -4.0), x, atol=1e-13)


def _one_row(i, j, window):
    """H = 1, D = 2, b = 1, one memory row (1, 0) with value (1, 0), the
    null row (1, 0) with value (0, 0); query (sqrt 2, 0)."""
    qc = np.array([[[np.sqrt(2.0), 0.0]]])
    z = np.zeros((1, 1, 2))
    bk = np.array([[[[1.0, 0.0]]]])
    bv = np.array([[[[1.0, 0.0]]]])
    kn = np.array([[1.0, 0.0]])
    vn = np.array([[0.0, 0.0]])
    _, oca = reader_prefill_rope([j], bk, bv, i, z, z, z, qc, kn, vn, window=window)
    return oca[0, 0, 0]


def test_cross_attention_closed_forms():
    # theta_0 = 1: score = cos(i - phase) (scale 1/sqrt(2) cancels |q| = sqrt 2)
    s_mem, s_null = np.cos(5 - 2), np.cos(5 - 0)
    want = np.exp(s_mem) / (np.exp(s_mem) + np.exp(s_null))
    assert abs(_one_row(5, 2, None) - want) < 1e-14
    assert abs(_one_row(5, 2, 15) - want) < 1e-14          # i <= W: saturation is the identity
    # W = 2: the row's phase max(2, 3) = 3 and the null row's max(0, 3) = 3 -> equal scores
    assert abs(_one_row(5, 2, 2) - 0.5) < 1e-14
    assert key_phase(2, 5, 2) == 3 and key_phase(0, 5, 2) == 3 and key_phase(4, 5, 2) == 4


def _random_case(rng, n, H=2, D=8, R=4, b=4):
    blocks = rng.standard_normal((n, H, R, D))
    vals = rng.standard_normal((n, H, R, D))
    q = [rng.standard_normal((b, H, D)) for _ in range(4)]
    kn, vn = rng.standard_normal((H, D)), rng.standard_normal((H, D))
    return blocks, vals, q, kn, vn


def test_shift_invariance_without_null_row():
    rng = np.random.default_rng(11)
    blocks, vals, (qs, ks, vs, qc), _, _ = _random_case(rng, 5)
    idx = np.array([0, 2, 3, 6, 7])
    a = reader_prefill_rope(idx, blocks, vals, 9, qs, ks, vs, qc, window=None)
    b = reader_prefill_rope(idx + 13, blocks, vals, 9 + 13, qs, ks, vs, qc, window=None)
    np.testing.assert_allclose(a[1], b[1], atol=1e-12)
    np.testing.assert_array_equal(a[0], b[0])


def test_far_blocks_share_one_phase_and_values_are_not_rotated():
    rng = np.random.default_rng(12)
    blocks, vals, (qs, ks, vs, qc), kn, vn = _random_case(rng, 6)
    idx = np.arange(6)
    # W = 2 at i = 8: blocks 0..5 all read at phase 6; swapping two blocks' contents
    # swaps nothing in the result
    a = reader_prefill_rope(idx, blocks, vals, 8, qs, ks, vs, qc, kn, vn, window=2)
    perm = np.array([3, 1, 2, 0, 4, 5])
    b = reader_prefill_rope(idx, blocks[perm], vals[perm], 8, qs, ks, vs, qc, kn, vn, window=2)
    np.testing.assert_allclose(a[1], b[1], atol=1e-12)
    # a zero query weighs every row (and the null row) equally, whatever the phases
    z = np.zeros_like(qc)
    _, oca = reader_prefill_rope(idx, blocks, vals, 8, qs, ks, vs, z, kn, vn, window=2)
    want = (vals.sum(axis=(0, 2)) + vn) / (6 * 4 + 1)
    np.testing.assert_allclose(oca, np.broadcast_to(want, oca.shape), atol=1e-12)


def test_one_block_pass_equals_full_pass_with_token_phases():
    """Unsaturated (each key has one phase for every reader): the full pass over
    B blocks with per-token rotated queries/keys and explicit masks equals the
    one-block pass of every block."""
    rng = np.random.default_rng(21)
    B, b, H, D = 4, 4, 2, 8
    n = B * b
    qs, ks, vs, qc = (rng.standard_normal((n, H, D)) for _ in range(4))
    mk, mv = rng.standard_normal((B, H, b, D)), rng.standard_normal((B, H, b, D))
    pos = np.arange(n)
    blk = pos // b
    t = pos % b
    qs_r, ks_r = rope(qs, t[:, None].astype(float)), rope(ks, t[:, None].astype(float))
    qc_r = rope(qc, blk[:, None].astype(float))
    mk_r = rope(mk, np.arange(B, dtype=float)[:, None, None])
    sdpa = torch.nn.functional.scaled_dot_product_attention
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a))  # noqa: E731
    sa_mask = (blk[:, None] == blk[None, :]) & (pos[None, :] <= pos[:, None])
    osa = sdpa(T(qs_r.transpose(1, 0, 2)), T(ks_r.transpose(1, 0, 2)), T(vs.transpose(1, 0, 2)),
               attn_mask=T(sa_mask)).numpy().transpose(1, 0, 2)
    keys = mk_r.transpose(1, 0, 2, 3).reshape(H, B * b, D)
    values = mv.transpose(1, 0, 2, 3).reshape(H, B * b, D)
    ca_mask = np.repeat(np.arange(B), b)[None, :] < blk[:, None]
    oca = np.zeros((n, H, D))
    rows = ca_mask.any(axis=1)
    oca[rows] = sdpa(T(qc_r[rows].transpose(1, 0, 2)), T(keys), T(values),
                     attn_mask=T(ca_mask[rows])).numpy().transpose(1, 0, 2)
    for i in range(B):
        sl = slice(i * b, (i + 1) * b)
        a_sa, a_ca = reader_prefill_rope(np.arange(i), mk[:i], mv[:i], i, qs[sl], ks[sl], vs[sl], qc[sl],
                                         window=None)
        np.testing.assert_allclose(a_sa, osa[sl], atol=1e-12)
        np.testing.assert_allclose(a_ca, oca[sl], atol=1e-12)


def test_decode_step_equals_one_block_row():
    rng = np.random.default_rng(31)
    blocks, vals, (qs, ks, vs, qc), kn, vn = _random_case(rng, 5, b=8)
    idx = np.array([1, 2, 4, 7, 9])
    for window in (15, 3):
        osa, oca = reader_prefill_rope(idx, blocks, vals, 12, qs, ks, vs, qc, kn, vn, window=window)
        for p in (0, 3, 7):
            a, c = reader_decode_rope(idx, blocks, vals, 12, p, ks[:p], vs[:p], qs[p], ks[p], vs[p], qc[p], kn, vn,
                                      window=window)
            np.testing.assert_allclose(a, osa[p], atol=1e-12)
            np.testing.assert_allclose(c, oca[p], atol=1e-12)
