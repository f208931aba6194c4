"""Pins of the fp64 oracle to facts outside itself (CPU only).

Each test ties the oracle to something the paper or the mathematics fixes:
a library routine on a brute-force masked "full pass" (block-skip exactness,
arXiv 2609.32395 Sec. 3.1, App. "Serving measurements"), closed forms, the
leak test (App. "Leak tests"), exact composition / deletion / path
independence (Proposition 1, Theorem 1, gates G5-G8), and Lemma 1's
Jacobian and bound (gates G1, G2, G4).
"""
import numpy as np
import pytest
import torch

import oracle
from oracle.bookkeeping import CacheMirror

RNG = np.random.default_rng(1234)


def _rand(*shape, rng=RNG):
    return rng.standard_normal(shape)


# ---------------------------------------------------------------------------
# brute-force full pass with torch's SDPA (library routine) and explicit masks
# ---------------------------------------------------------------------------
def full_pass(qs, ks, vs, qc, mem_k, mem_v, b, k_null=None, v_null=None):
    """Reader attention for every position of a B-block context at once.

    qs/ks/vs/qc: [B*b][H][D]; mem_k/v: [B][H][R][D] (block j = index j).
    Self-attention mask: same block and key position <= query position.
    Cross-attention mask: memory block index < the query's block index;
    the null row (if any) is visible to every query.
    Returns (osa, oca) [B*b][H][D]; rows with no visible key give 0.
    """
    n, H, D = qs.shape
    B, _, R, _ = mem_k.shape
    pos = np.arange(n)
    blk = pos // b
    sa_mask = (blk[:, None] == blk[None, :]) & (pos[None, :] <= pos[:, None])
    row_blk = np.repeat(np.arange(B), R)
    ca_mask = row_blk[None, :] < blk[:, None]
    mk = mem_k.transpose(1, 0, 2, 3).reshape(H, B * R, D)
    mv = mem_v.transpose(1, 0, 2, 3).reshape(H, B * R, D)
    if k_null is not None:
        mk = np.concatenate([k_null[:, None, :], mk], axis=1)
        mv = np.concatenate([v_null[:, None, :], mv], axis=1)
        ca_mask = np.concatenate([np.ones((n, 1), bool), ca_mask], axis=1)

    def sdpa(q, k, v, mask):
        q = torch.from_numpy(np.ascontiguousarray(q))
        k = torch.from_numpy(np.ascontiguousarray(k))
        v = torch.from_numpy(np.ascontiguousarray(v))
        m = torch.from_numpy(mask)
        o = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=m)
        o = o.numpy().copy()
        o[:, ~mask.any(axis=1), :] = 0.0
        return o

    osa = sdpa(qs.transpose(1, 0, 2), ks.transpose(1, 0, 2), vs.transpose(1, 0, 2), sa_mask)
    oca = sdpa(qc.transpose(1, 0, 2), mk, mv, ca_mask)
    return osa.transpose(1, 0, 2), oca.transpose(1, 0, 2)


@pytest.mark.parametrize("with_null", [False, True])
@pytest.mark.parametrize("B,b,H,D", [(4, 8, 2, 8), (3, 16, 3, 16)])
def test_prefill_equals_full_pass(B, b, H, D, with_null):
    """Block-skip exactness: the one-block pass over cached memory equals the
    final (and every) block of a full masked pass."""
    rng = np.random.default_rng(B * 100 + b + with_null)
    n = B * b
    qs, ks, vs, qc = (_rand(n, H, D, rng=rng) for _ in range(4))
    mem_k, mem_v = _rand(B, H, b, D, rng=rng), _rand(B, H, b, D, rng=rng)
    kn = _rand(H, D, rng=rng) if with_null else None
    vn = _rand(H, D, rng=rng) if with_null else None
    fsa, fca = full_pass(qs, ks, vs, qc, mem_k, mem_v, b, kn, vn)
    perm = rng.permutation(B)  # memory handed over in a scrambled order
    for i in range(B):
        sl = slice(i * b, (i + 1) * b)
        osa, oca = oracle.reader_prefill(perm, mem_k[perm], mem_v[perm], i, qs[sl], ks[sl], vs[sl], qc[sl], kn, vn)
        np.testing.assert_allclose(osa, fsa[sl], rtol=0, atol=1e-12)
        np.testing.assert_allclose(oca, fca[sl], rtol=0, atol=1e-12)


@pytest.mark.parametrize("with_null", [False, True])
def test_decode_equals_full_pass(with_null):
    """A decode step at in-block offset p equals the full pass at that token."""
    rng = np.random.default_rng(7 + with_null)
    B, b, H, D = 4, 8, 2, 16
    n = B * b
    qs, ks, vs, qc = (_rand(n, H, D, rng=rng) for _ in range(4))
    mem_k, mem_v = _rand(B, H, b, D, rng=rng), _rand(B, H, b, D, rng=rng)
    kn = _rand(H, D, rng=rng) if with_null else None
    vn = _rand(H, D, rng=rng) if with_null else None
    fsa, fca = full_pass(qs, ks, vs, qc, mem_k, mem_v, b, kn, vn)
    for i in range(B):
        for p in (0, 1, b // 2, b - 1):
            t = i * b + p
            osa, oca = oracle.reader_decode(np.arange(B), mem_k, mem_v, i, p, ks[i * b:t], vs[i * b:t],
                                            qs[t], ks[t], vs[t], qc[t], kn, vn)
            np.testing.assert_allclose(osa, fsa[t], rtol=0, atol=1e-12)
            np.testing.assert_allclose(oca, fca[t], rtol=0, atol=1e-12)


def test_paper_shape_full_pass():
    """b = R = 64, d_h = 64 (the configured reader block): last block only."""
    rng = np.random.default_rng(99)
    B, b, H, D = 3, 64, 2, 64
    n = B * b
    qs, ks, vs, qc = (_rand(n, H, D, rng=rng) for _ in range(4))
    mem_k, mem_v = _rand(B, H, b, D, rng=rng), _rand(B, H, b, D, rng=rng)
    fsa, fca = full_pass(qs, ks, vs, qc, mem_k, mem_v, b)
    sl = slice((B - 1) * b, B * b)
    osa, oca = oracle.reader_prefill(np.arange(B), mem_k, mem_v, B - 1, qs[sl], ks[sl], vs[sl], qc[sl])
    np.testing.assert_allclose(osa, fsa[sl], rtol=0, atol=1e-12)
    np.testing.assert_allclose(oca, fca[sl], rtol=0, atol=1e-12)


# ---------------------------------------------------------------------------
# closed forms and special cases
# ---------------------------------------------------------------------------
def _one_layer(rng, nblk=3, b=8, H=2, D=8, R=None):
    R = b if R is None else R
    return (_rand(nblk, H, R, D, rng=rng), _rand(nblk, H, R, D, rng=rng),
            *(_rand(b, H, D, rng=rng) for _ in range(4)))


def test_first_position_returns_its_value_exactly():
    rng = np.random.default_rng(3)
    mk, mv, qs, ks, vs, qc = _one_layer(rng)
    osa, _ = oracle.reader_prefill(np.arange(3), mk, mv, 3, qs, ks, vs, qc)
    assert np.array_equal(osa[0], vs[0])


def test_single_memory_row_returns_its_value_exactly():
    rng = np.random.default_rng(4)
    b, H, D = 8, 2, 8
    mk, mv = _rand(1, H, 1, D, rng=rng), _rand(1, H, 1, D, rng=rng)
    qs, ks, vs, qc = (_rand(b, H, D, rng=rng) for _ in range(4))
    _, oca = oracle.reader_prefill([0], mk, mv, 1, qs, ks, vs, qc)
    for t in range(b):
        assert np.array_equal(oca[t], mv[0, :, 0, :])


def test_zero_query_gives_row_mean():
    rng = np.random.default_rng(5)
    mk, mv, qs, ks, vs, qc = _one_layer(rng)
    qc[:] = 0.0
    _, oca = oracle.reader_prefill(np.arange(3), mk, mv, 3, qs, ks, vs, qc)
    mean = mv.transpose(1, 0, 2, 3).reshape(2, -1, 8).mean(axis=1)
    for t in range(qc.shape[0]):
        np.testing.assert_allclose(oca[t], mean, rtol=0, atol=1e-14)


def test_equal_keys_give_row_mean():
    rng = np.random.default_rng(6)
    mk, mv, qs, ks, vs, qc = _one_layer(rng)
    mk[:] = mk[0, :, 0:1, :][None]  # every row of every block: same key per head
    _, oca = oracle.reader_prefill(np.arange(3), mk, mv, 3, qs, ks, vs, qc)
    mean = mv.transpose(1, 0, 2, 3).reshape(2, -1, 8).mean(axis=1)
    for t in range(qc.shape[0]):
        np.testing.assert_allclose(oca[t], mean, rtol=0, atol=1e-14)


def test_dominant_row_gives_one_hot():
    rng = np.random.default_rng(8)
    mk, mv, qs, ks, vs, qc = _one_layer(rng)
    D = 8
    for h in range(2):
        mk[1, h, 5, :] = qc[0, h, :] * 1e4  # score gap far beyond exp underflow
    _, oca = oracle.reader_prefill(np.arange(3), mk, mv, 3, qs, ks, vs, qc)
    assert np.array_equal(oca[0], mv[1, :, 5, :])
    assert D == mk.shape[-1]


def test_null_row_only_and_empty_memory():
    rng = np.random.default_rng(9)
    b, H, D = 8, 2, 8
    qs, ks, vs, qc = (_rand(b, H, D, rng=rng) for _ in range(4))
    kn, vn = _rand(H, D, rng=rng), _rand(H, D, rng=rng)
    _, oca = oracle.reader_prefill([], None, None, 0, qs, ks, vs, qc, kn, vn)
    for t in range(b):
        assert np.array_equal(oca[t], vn)  # block 1 reads the null row only
    _, oca0 = oracle.reader_prefill([], None, None, 0, qs, ks, vs, qc)
    assert np.array_equal(oca0, np.zeros_like(oca0))


def test_null_row_with_equal_scores_halves():
    """One memory row and the null row with equal scores: the average."""
    rng = np.random.default_rng(10)
    b, H, D = 4, 1, 8
    qs, ks, vs, qc = (_rand(b, H, D, rng=rng) for _ in range(4))
    k = _rand(H, D, rng=rng)
    mk = k[None, :, None, :].copy()
    mv = _rand(1, H, 1, D, rng=rng)
    vn = _rand(H, D, rng=rng)
    _, oca = oracle.reader_prefill([0], mk, mv, 1, qs, ks, vs, qc, k_null=k.copy(), v_null=vn)
    for t in range(b):
        np.testing.assert_allclose(oca[t], 0.5 * (vn + mv[0, :, 0, :]), rtol=0, atol=1e-15)


# ---------------------------------------------------------------------------
# leak test: structural masks, exact-zero change
# ---------------------------------------------------------------------------
def test_leak_future_positions_and_blocks():
    rng = np.random.default_rng(11)
    nblk, b, H, D = 5, 8, 2, 8
    mk, mv, qs, ks, vs, qc = _one_layer(rng, nblk=nblk, b=b, H=H, D=D)
    q_idx = 3
    osa, oca = oracle.reader_prefill(np.arange(nblk), mk, mv, q_idx, qs, ks, vs, qc)
    for t in range(b):
        ks2, vs2 = ks.copy(), vs.copy()
        ks2[t + 1:] = _rand(b - t - 1, H, D, rng=rng)
        vs2[t + 1:] = _rand(b - t - 1, H, D, rng=rng)
        osa2, _ = oracle.reader_prefill(np.arange(nblk), mk, mv, q_idx, qs, ks2, vs2, qc)
        assert np.array_equal(osa2[: t + 1], osa[: t + 1])
    mk2, mv2 = mk.copy(), mv.copy()
    mk2[q_idx:] = _rand(nblk - q_idx, H, b, D, rng=rng)
    mv2[q_idx:] = _rand(nblk - q_idx, H, b, D, rng=rng)
    _, oca2 = oracle.reader_prefill(np.arange(nblk), mk2, mv2, q_idx, qs, ks, vs, qc)
    assert np.array_equal(oca2, oca)


def test_rowset_is_block_causal_and_canonical():
    idx = np.array([7, 2, 9, 0, 5])
    assert list(oracle.rowset(idx, 6)) == [3, 1, 4]       # blocks 0, 2, 5
    assert list(oracle.rowset(idx, 0)) == []
    assert list(oracle.rowset(idx, 100)) == [3, 1, 4, 0, 2]
    with pytest.raises(oracle.OracleError):
        oracle.rowset([1, 1], 5)


# ---------------------------------------------------------------------------
# composition, deletion, path independence (Prop. 1, Thm. 1, gates G5-G8)
# ---------------------------------------------------------------------------
def _read_via_mirror(mirror, store, seq, q_idx, qs, ks, vs, qc):
    """Reader pass over a sequence's memory as held in slots of a store."""
    idx, slots = mirror.table(seq)
    mk = np.stack([store[s][0] for s in slots]) if slots else None
    mv = np.stack([store[s][1] for s in slots]) if slots else None
    return oracle.reader_prefill(idx, mk, mv, q_idx, qs, ks, vs, qc)


def test_composition_is_exact():
    """Per-block appends in any order equal one bulk memory (bitwise)."""
    rng = np.random.default_rng(12)
    nblk, b, H, D = 6, 8, 2, 8
    mk, mv, qs, ks, vs, qc = _one_layer(rng, nblk=nblk, b=b, H=H, D=D)
    ref = oracle.reader_prefill(np.arange(nblk), mk, mv, nblk, qs, ks, vs, qc)
    for trial in range(5):
        order = rng.permutation(nblk)
        m = CacheMirror(16, 1, 16, free_order=rng.permutation(16))
        store = {}
        for j in order:
            rc, s = m.append(0, int(j))
            assert rc == 0
            store[s] = (mk[j], mv[j])
        out = _read_via_mirror(m, store, 0, nblk, qs, ks, vs, qc)
        assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


def test_deletion_equals_never_inserted():
    rng = np.random.default_rng(13)
    nblk, b, H, D = 6, 8, 2, 8
    mk, mv, qs, ks, vs, qc = _one_layer(rng, nblk=nblk, b=b, H=H, D=D)
    keep = [0, 1, 2, 4, 5]
    ref = oracle.reader_prefill(np.array(keep), mk[keep], mv[keep], nblk, qs, ks, vs, qc)
    m = CacheMirror(8, 1, 8)
    store = {}
    for j in range(nblk):
        rc, s = m.append(0, j)
        store[s] = (mk[j], mv[j])
    assert m.delete(0, 3) == 0
    out = _read_via_mirror(m, store, 0, nblk, qs, ks, vs, qc)
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])
    # re-append block 3: it lands in a different slot, reads return to the full set
    rc, s = m.append(0, 3)
    assert rc == 0 and s == 6
    store[s] = (mk[3], mv[3])
    full = oracle.reader_prefill(np.arange(nblk), mk, mv, nblk, qs, ks, vs, qc)
    out = _read_via_mirror(m, store, 0, nblk, qs, ks, vs, qc)
    assert np.array_equal(out[1], full[1])


def test_path_independence_100_orders():
    """100 random edit sequences ending at the same block set: identical."""
    rng = np.random.default_rng(14)
    nblk, b, H, D = 8, 8, 2, 8
    universe_k, universe_v = _rand(12, H, b, D, rng=rng), _rand(12, H, b, D, rng=rng)
    qs, ks, vs, qc = (_rand(b, H, D, rng=rng) for _ in range(4))
    target = sorted(rng.choice(12, size=nblk, replace=False).tolist())
    ref = None
    for trial in range(100):
        m = CacheMirror(32, 1, 16, free_order=rng.permutation(32))
        store = {}
        live = set()
        # random churn, then converge on the target set
        for _ in range(20):
            j = int(rng.integers(0, 12))
            if j in live and rng.random() < 0.5:
                assert m.delete(0, j) == 0
                live.discard(j)
            elif j not in live:
                rc, s = m.append(0, j)
                assert rc == 0
                store[s] = (universe_k[j], universe_v[j])
                live.add(j)
        for j in sorted(live - set(target), key=lambda _: rng.random()):
            assert m.delete(0, j) == 0
        for j in sorted(set(target) - live, key=lambda _: rng.random()):
            rc, s = m.append(0, j)
            store[s] = (universe_k[j], universe_v[j])
        out = _read_via_mirror(m, store, 0, 12, qs, ks, vs, qc)
        if ref is None:
            ref = out
        assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


# ---------------------------------------------------------------------------
# Lemma 1: Jacobian closed form and the size-free bound (gates G1, G2, G4)
# ---------------------------------------------------------------------------
def _ca_single(q, K, V):
    """Cross-attention output of the oracle for one query and one head."""
    N, D = K.shape
    mk = K.reshape(N, 1, 1, D)
    mv = V.reshape(N, 1, 1, D)
    z = np.zeros((1, 1, D))
    _, oca = oracle.reader_prefill(np.arange(N), mk, mv, N, z, z, z, q.reshape(1, 1, D))
    return oca[0, 0]


def _fd_jacobian(q, K, V, h=1e-6):
    D = q.shape[0]
    J = np.zeros((V.shape[1], D))
    for j in range(D):
        e = np.zeros(D)
        e[j] = h
        J[:, j] = (_ca_single(q + e, K, V) - _ca_single(q - e, K, V)) / (2 * h)
    return J


def test_lemma1_jacobian_closed_form():
    """G1: d c / d q = (1/sqrt(d)) Cov_a(v, k) with W_Q = I."""
    rng = np.random.default_rng(15)
    N, D = 24, 8
    K, V, q = _rand(N, D, rng=rng), _rand(N, D, rng=rng), _rand(D, rng=rng)
    s = q @ K.T / np.sqrt(D)
    a = np.exp(s - s.max())
    a /= a.sum()
    vbar, kbar = a @ V, a @ K
    cov = ((V - vbar).T * a) @ (K - kbar)
    J = _fd_jacobian(q, K, V)
    np.testing.assert_allclose(J, cov / np.sqrt(D), rtol=0, atol=1e-8)


def test_lemma1_two_item_worst_case_attains_bound():
    """G4: with two rows the bound is met at a_1 = 1/2 and not elsewhere."""
    rng = np.random.default_rng(16)
    D = 8
    k1, k2, v1, v2 = (_rand(D, rng=rng) for _ in range(4))
    K, V = np.stack([k1, k2]), np.stack([v1, v2])
    bound = np.linalg.norm(k1 - k2) * np.linalg.norm(v1 - v2) / (4 * np.sqrt(D))
    dk = k1 - k2
    q0 = _rand(D, rng=rng)
    q_half = q0 - (q0 @ dk) / (dk @ dk) * dk  # equal scores: a_1 = 1/2
    n_half = np.linalg.norm(_fd_jacobian(q_half, K, V), 2)
    np.testing.assert_allclose(n_half, bound, rtol=1e-7)
    q_off = q_half + 0.7 * dk / np.linalg.norm(dk)
    assert np.linalg.norm(_fd_jacobian(q_off, K, V), 2) < bound * (1 - 1e-3)


def test_lemma1_bound_is_size_free():
    """G2: at fixed key/value diameters the bound holds from 16 to 4096 rows."""
    rng = np.random.default_rng(17)
    D = 8
    for N in (16, 64, 256, 1024, 4096):
        K = _rand(N, D, rng=rng)
        K /= np.linalg.norm(K, axis=1, keepdims=True)  # rows on the unit sphere
        V = _rand(N, D, rng=rng)
        V /= np.linalg.norm(V, axis=1, keepdims=True)
        q = 3.0 * _rand(D, rng=rng)
        nrm = np.linalg.norm(_fd_jacobian(q, K, V, h=1e-5), 2)
        assert nrm <= 2.0 * 2.0 / (4 * np.sqrt(D)) + 1e-7  # diam <= 2 on the sphere
