"""GPU parity of the recompute-K/V regime (the pool holds only the memory rows
mu; every reader-layer call re-derives the layer's cross-attention from them,
arXiv 2609.32395, Sec. 3.1 and App. "Serving") against the same fp64 layer
oracle as the materialized path -- keys mu W_kc and values mu W_vc are the
oracle's definition; the kernel's re-association is checked against it:

* one-block prefill and batched decode per layer, with and without the null
  row, d_h 64/128, at test shapes and at the 160M / 410M / 1.5B widths;
* bitwise edit-path independence (Theorem 1) of prefill and decode outputs;
* agreement with the materialized cache on the same inputs;
* entry points that take projected K/V refuse a recompute cache.
"""
import numpy as np
import pytest
import torch

import synth
from oracle.reader_layer import reader_layer_decode, reader_layer_prefill
from paper_2609_32395_gb300 import smem
from tests.layer_helpers import B_TOK, LayerModel, assert_layer_close, bits_dev, mu_bits
from tests.test_gpu_layer import LayerCache, _decode_setup, _np, x_rows

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("D,H,has_null", [(64, 4, True), (64, 4, False), (128, 2, True), (32, 8, True)])
def test_recompute_layer_prefill_matches_oracle(D, H, has_null):
    model = LayerModel(2, H * D, seed=601 + D)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=16, capacity=24, has_null=has_null,
                    free_order=synth.slot_permutation(3, 24), recompute=True)
    for j in (5, 0, 7, 2, 6, 1, 4, 3):
        lc.append(0, j)
    for q_idx in (8, 3, 0):
        x = torch.from_numpy(x_rows(model.seed, 0, q_idx, lc.d)).cuda()
        for layer in range(model.L):
            x_in = _np(x)
            lc.prefill(0, layer, q_idx, x)
            ref, _, _ = lc.oracle_prefill(0, layer, q_idx, x_in)
            assert_layer_close(_np(x), ref, x_in, f"layer {layer} q_idx {q_idx}")
    assert smem.smem_check_device_error(lc.h) == smem.OK


@pytest.mark.parametrize("H,D,nblk", [(12, 64, 256), (12, 64, 64), (16, 64, 40), (16, 128, 24), (16, 32, 64)])
def test_recompute_prefill_at_model_widths(H, D, nblk):
    """d = 768 / 1024 / 2048 (the 160M / 410M / 1.5B reader widths) and 512:
    every query-tile width of the kernel (32 queries per CTA at d = 768 and
    1024, 16 at d = 2048, 64 at d = 512, where two score buffers of 64
    queries fit tensor memory)."""
    d = H * D
    model = LayerModel(1, d, seed=701 + d)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=nblk + 4, capacity=nblk + 4, recompute=True)
    for j in range(nblk):
        lc.append(0, j)
    x = torch.from_numpy(x_rows(model.seed, 0, nblk, d)).cuda()
    x_in = _np(x)
    lc.prefill(0, 0, nblk, x)
    ref, _, _ = lc.oracle_prefill(0, 0, nblk, x_in)
    assert_layer_close(_np(x), ref, x_in, f"d {d}")


def _decode_check(model, lc, xs, ctx, pos, H, D):
    x = torch.from_numpy(np.stack([xs[s][0][0][pos[s]] for s in range(len(ctx))]).astype(np.float32)).cuda()
    for layer in range(model.L):
        x_in = _np(x)
        lc.decode(layer, list(range(len(ctx))), pos, ctx, x)
        got = _np(x)
        for s in range(len(ctx)):
            ids, mu = lc.memory(s, ctx[s])
            _, ks, vs = reader_layer_prefill(xs[s][0][layer], ids, mu, ctx[s], model.oracle[layer], H, D, lc.nu)
            ref, _, _ = reader_layer_decode(x_in[s], ids, mu, ctx[s], pos[s], ks[:pos[s]], vs[:pos[s]],
                                            model.oracle[layer], H, D, lc.nu)
            assert_layer_close(got[s], ref, x_in[s], f"decode layer {layer} seq {s}")
    return _np(x)


@pytest.mark.parametrize("H,D", [(4, 64), (16, 64), (12, 128)])
def test_recompute_decode_after_prefill_matches_oracle(H, D):
    """Batched decode (contexts 5, 0, 9, 30 blocks; offsets 17, 0, 63, 5)
    after each sequence's layer prefill."""
    model = LayerModel(2, H * D, seed=809 + H)
    ctx, pos = [5, 0, 9, 30], [17, 0, 63, 5]
    lc, xs = _decode_setup(model, H, D, ctx, recompute=True)
    _decode_check(model, lc, xs, ctx, pos, H, D)
    assert smem.smem_check_device_error(lc.h) == smem.OK


def test_recompute_outputs_are_edit_path_independent():
    H, D, L = 4, 64, 2
    model = LayerModel(L, H * D, seed=907)
    ctx = [20, 3]
    a, xa = _decode_setup(model, H, D, ctx, recompute=True)
    b, xb = _decode_setup(model, H, D, ctx, free_order=synth.slot_permutation(5, sum(ctx) + 16), history=True,
                          recompute=True)
    assert a.mirror.table(0)[1] != b.mirror.table(0)[1]
    for s in range(2):
        np.testing.assert_array_equal(xa[s][1], xb[s][1])
    pos = [11, 40]
    x0 = np.stack([xa[s][0][0][pos[s]] for s in range(2)]).astype(np.float32)
    outs = []
    for lc in (a, b):
        x = torch.from_numpy(x0).cuda()
        for layer in range(L):
            lc.decode(layer, [0, 1], pos, ctx, x)
        outs.append(_np(x))
    np.testing.assert_array_equal(outs[0], outs[1])


def test_recompute_agrees_with_materialized_cache():
    """The same blocks, weights and inputs through both regimes: the outputs
    agree within the layer tolerance (they round at different places)."""
    H, D = 4, 64
    model = LayerModel(1, H * D, seed=1009)
    ctx = [12]
    m, xm = _decode_setup(model, H, D, ctx)
    r, xr = _decode_setup(model, H, D, ctx, recompute=True)
    assert_layer_close(xr[0][1], xm[0][1].astype(np.float64), xm[0][0][0], "prefill: recompute vs materialized")


def test_recompute_cache_refuses_projected_kv_entries():
    H, D = 4, 64
    d = H * D
    model = LayerModel(2, d, seed=1103)
    mat = smem.make_config(2, H, D, 2, 8, 8, has_null_row=True)
    rec = smem.make_config(2, H, D, 2, 8, 8, has_null_row=True, recompute_kv=True)
    # the pool shrinks from L*H*2*R*d_h to R*d elements per slot (2L = 4 times)
    pool_m = 8 * 2 * H * 2 * 64 * D * 2
    pool_r = 8 * 64 * d * 2
    assert smem.smem_cache_required_bytes(mat) - smem.smem_cache_required_bytes(rec) >= pool_m - pool_r - (1 << 20)
    lc = LayerCache(model, H, D, max_seqs=2, max_blocks=8, capacity=8, recompute=True)
    t = torch.zeros(B_TOK, H, D, dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros(2, H, 64, D, dtype=torch.bfloat16, device="cuda")
    for call in (lambda: smem.smem_append_block(lc.h, 0, 0, kv, kv),
                 lambda: smem.smem_set_null_row(lc.h, t[0], t[0]),
                 lambda: smem.smem_prefill_block(lc.h, 0, 0, 0, t, t, t, t, t, t),
                 lambda: smem.smem_decode(lc.h, 0, [0], [0], [0], t[:1], t[:1], t[:1], t[:1], t[:1], t[:1])):
        with pytest.raises(smem.SmemError) as e:
            call()
        assert e.value.code == smem.ERR_UNSUPPORTED
    # memory rows need no weights on a recompute cache
    slot = smem.smem_append_block_rows(lc.h, 1, 0, bits_dev(mu_bits(1, 1, 0, d)), [], lc.ws)
    assert slot == lc.mirror.append(1, 0)[1]


def _qprime(seed, shape, d, fields):
    """Folded queries q' (bf16): N(0, 1/d), so that base-2 scores q'.mu have
    unit spread over N(0,1) memory rows."""
    z = torch.from_numpy(bits_f64_arr(synth.tensor_np(seed, synth.KIND_QDEC_C, shape, *fields)))
    return (z.float() * float(np.float32(1.0 / np.sqrt(d)))).to(torch.bfloat16)


def bits_f64_arr(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _oracle_mu(q, mus, nu):
    """The oracle's attention with every query reading the same rows: keys =
    values = the memory rows (broadcast over the queries), scale chosen so
    that the oracle's exp(q.k / sqrt(d)) equals the kernel's 2^(q'.mu)."""
    import oracle
    nq, d = q.shape
    qo = q * (np.log(2.0) * np.sqrt(d))
    n = len(mus)
    bk = np.broadcast_to(np.asarray(mus)[:, None], (n, nq, 64, d)) if n else None
    kn = np.broadcast_to(nu, (nq, d)) if nu is not None else None
    zero = np.zeros((nq, d))
    _, oca = oracle.reader_decode(np.arange(n), bk, bk, n, 0, None, None, zero, zero, zero, qo, kn, kn)
    return oca


@pytest.mark.parametrize("has_null", [True, False])
def test_mu_decode_kernel_matches_oracle(has_null):
    """The memory-row attention primitive alone: items with 0, 3, 9 and 300
    blocks (one to sixteen splits), H = 4 queries of width d = 256 each."""
    from tests.gpu_helpers import MAX_ABS, MEAN_ABS
    H, D = 4, 64
    d = H * D
    model = LayerModel(1, d, seed=1201)
    ctx = [0, 3, 9, 300]
    lc = LayerCache(model, H, D, max_seqs=4, max_blocks=310, capacity=320, has_null=has_null, recompute=True)
    for s, n in enumerate(ctx):
        for j in range(n):
            lc.append(s, j)
    qp = _qprime(1201, (4, H, d), d, (0,))
    op = torch.empty(4, H, d, dtype=torch.bfloat16, device="cuda")
    smem.smem_mu_decode(lc.h, [0, 1, 2, 3], ctx, qp.cuda(), op, lc.ws)
    got = op.float().cpu().numpy().astype(np.float64)
    for s, n in enumerate(ctx):
        _, mus = lc.memory(s, n)
        ref = _oracle_mu(qp[s].double().numpy(), list(mus), lc.nu)
        err = np.abs(got[s] - ref)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (s, err.max(), err.mean())
    assert smem.smem_check_device_error(lc.h) == smem.OK


@pytest.mark.parametrize("H,D,nblk", [(4, 64, 7), (12, 64, 40), (16, 64, 20), (16, 128, 12), (16, 32, 64)])
def test_mu_prefill_kernel_matches_oracle(H, D, nblk):
    """The block form: H x 64 queries over one row set, every query-tile
    width (16 at 7 blocks or d = 2048, 32 at d = 768 / 1024, 64 at d = 512)."""
    from tests.gpu_helpers import MAX_ABS, MEAN_ABS
    d = H * D
    model = LayerModel(1, d, seed=1301 + d)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=nblk + 2, capacity=nblk + 2, recompute=True)
    for j in range(nblk):
        lc.append(0, j)
    qp = _qprime(1301, (H, B_TOK, d), d, (1,))
    op = torch.empty(H, B_TOK, d, dtype=torch.bfloat16, device="cuda")
    smem.smem_mu_prefill(lc.h, 0, nblk, qp.cuda(), op, lc.ws)
    got = op.float().cpu().numpy().astype(np.float64)
    _, mus = lc.memory(0, nblk)
    for h in range(H):
        q = qp[h].double().numpy()
        # a few queries at a time keeps the oracle's broadcast rows small
        ref = np.concatenate([_oracle_mu(q[i:i + 8], list(mus), lc.nu) for i in range(0, B_TOK, 8)])
        err = np.abs(got[h] - ref)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (h, err.max(), err.mean())


def _mu_cache(H, D, ctx, has_null=True, free_order=None, history=False, seed=1401):
    d = H * D
    model = LayerModel(1, d, seed=seed)
    cap = sum(ctx) + 4 * len(ctx) + 8
    lc = LayerCache(model, H, D, max_seqs=len(ctx), max_blocks=max(ctx) + 8, capacity=cap, has_null=has_null,
                    free_order=free_order, recompute=True)
    for s, n in enumerate(ctx):
        order = list(range(n))[::-1] if history else list(range(n))
        if history:
            lc.append(s, n + 2, content_seq=77)   # appended and deleted again
        for j in order:
            lc.append(s, j)
        if history:
            lc.delete(s, n + 2)
            if n > 3:
                lc.delete(s, 2)
                lc.append(s, 2)
    return lc


def _mu_run(lc, H, d, ctx, seed):
    qp = _qprime(seed, (len(ctx), H, d), d, (2,))
    op = torch.empty(len(ctx), H, d, dtype=torch.bfloat16, device="cuda")
    smem.smem_mu_decode(lc.h, list(range(len(ctx))), ctx, qp.cuda(), op, lc.ws)
    assert smem.smem_check_device_error(lc.h) == smem.OK
    return qp, op


def _check_mu_decode(lc, H, d, ctx, qp, op):
    from tests.gpu_helpers import MAX_ABS, MEAN_ABS
    got = op.float().cpu().numpy().astype(np.float64)
    for s, n in enumerate(ctx):
        _, mus = lc.memory(s, n)
        q = qp[s].double().numpy()
        # one query at a time keeps the oracle's broadcast rows small
        ref = np.stack([_oracle_mu(q[i:i + 1], list(mus), lc.nu)[0] for i in range(H)])
        err = np.abs(got[s] - ref)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (s, n, err.max(), err.mean())


@pytest.mark.parametrize("H,D,cluster", [(4, 64, 1), (12, 64, 3), (16, 64, 4), (16, 128, 8), (32, 64, 0),
                                         (20, 64, 0)])
@pytest.mark.parametrize("has_null", [True, False])
@pytest.mark.parametrize("slices", [False, True])
def test_mu_decode_at_model_widths(H, D, cluster, has_null, slices, monkeypatch):
    """The decode form at d = 256 .. 2048, with the two-pass kernel and with
    the column-slice kernel switched on (clusters of 1, 3, 4 and 8 CTAs at
    d = 256, 768 = 160M, 1024 = 410M, 2048 = 1.5B; the two-pass kernel
    stays where the exchange would not fit). H = 32 at d = 2048 takes two
    16-query tiles per item, H = 20 one 32-query tile. Contexts of 0, 1,
    31, 33 and 70 blocks: no readable block, one short split, and one to
    three splits with a ragged last (splits of at least 24 blocks, 32 with
    column slices)."""
    d = H * D
    ctx = [0, 1, 31, 33, 70]
    monkeypatch.setenv("SMEM_MU_CLUSTERS", "1" if slices else "0")
    lc = _mu_cache(H, D, ctx, has_null=has_null)
    nq, cl, wsl = smem.smem_mu_decode_plan(lc.h)
    assert cl == (cluster if slices else 0)
    if cl:
        assert wsl * cl == d and nq == (H + 15) // 16 * 16
    else:
        assert nq in (16, 32) and nq * ((H + nq - 1) // nq) >= H
    qp, op = _mu_run(lc, H, d, ctx, 1401 + d)
    _check_mu_decode(lc, H, d, ctx, qp, op)


@pytest.mark.parametrize("slices", [False, True])
def test_mu_decode_sixteen_splits(slices, monkeypatch):
    """600 blocks at d = 256: 16 splits of 38 blocks, the last ragged; 300
    blocks: 13 splits of 24 (two-pass) or 10 of 32 (column slices, clusters
    of one CTA)."""
    H, D = 4, 64
    ctx = [600, 300, 5]
    monkeypatch.setenv("SMEM_MU_CLUSTERS", "1" if slices else "0")
    lc = _mu_cache(H, D, ctx)
    assert smem.smem_mu_decode_plan(lc.h)[1] == (1 if slices else 0)
    qp, op = _mu_run(lc, H, H * D, ctx, 1501)
    _check_mu_decode(lc, H, H * D, ctx, qp, op)


def test_mu_decode_slice_kernel_is_edit_path_independent(monkeypatch):
    """Theorem 1 through the column-slice kernel (d = 1024, clusters of 4):
    the same block sets reached by different edit paths and slot orders
    give bitwise-equal outputs."""
    H, D = 16, 64
    ctx = [70, 40, 9]
    monkeypatch.setenv("SMEM_MU_CLUSTERS", "1")
    a = _mu_cache(H, D, ctx)
    b = _mu_cache(H, D, ctx, free_order=synth.slot_permutation(11, sum(ctx) + 4 * len(ctx) + 8), history=True)
    assert smem.smem_mu_decode_plan(a.h)[1] == 4
    assert a.mirror.table(0)[1] != b.mirror.table(0)[1]
    _, oa = _mu_run(a, H, H * D, ctx, 1601)
    _, ob = _mu_run(b, H, H * D, ctx, 1601)
    assert torch.equal(oa.view(torch.int16), ob.view(torch.int16))


def test_mu_decode_two_kernels_agree(monkeypatch):
    """The two-pass kernel (clusters switched off for the cache) and the
    column-slice kernel on the same rows and queries: both within the
    tolerance of the oracle, and of each other."""
    from tests.gpu_helpers import MAX_ABS
    H, D = 16, 64
    ctx = [45, 12]
    monkeypatch.setenv("SMEM_MU_CLUSTERS", "1")
    s = _mu_cache(H, D, ctx)
    monkeypatch.setenv("SMEM_MU_CLUSTERS", "0")
    t = _mu_cache(H, D, ctx)
    assert smem.smem_mu_decode_plan(s.h)[1] == 4 and smem.smem_mu_decode_plan(t.h)[1] == 0
    qs, os_ = _mu_run(s, H, H * D, ctx, 1701)
    _, ot = _mu_run(t, H, H * D, ctx, 1701)
    _check_mu_decode(t, H, H * D, ctx, qs, ot)
    assert float((os_.float() - ot.float()).abs().max()) <= MAX_ABS
