"""GPU parity of the full reader layer (LayerNorm, projections and the GELU
FFN around the attention kernels, through the C ABI) against the fp64 layer
oracle on the same seeded bf16 weights and inputs:

* one-block prefill per layer, with and without the null row, d_h 64/128,
  every / some / no memory block readable;
* the layer-level block-skip gate: the one-block pass of every block equals
  the masked full pass over all blocks (arXiv 2609.32395, Sec. 3.1);
* decode steps after a layer prefill (in-block rows handed over), batched
  over sequences with different contexts, including an empty one;
* bitwise edit-path independence (Theorem 1) of prefill and decode outputs;
* argument errors of the layer entry points.
"""
import numpy as np
import pytest
import torch

import synth
from oracle.bookkeeping import CacheMirror
from oracle.reader_layer import reader_layer_decode, reader_layer_prefill
from paper_2609_32395_gb300 import smem
from tests.layer_helpers import (B_TOK, LayerModel, assert_layer_close, bits_dev, bits_f64, mu_bits, nu_bits,
                                 x_rows)
from tests.test_oracle_layer_pins import full_layer_pass

pytestmark = pytest.mark.gpu


class LayerCache:
    """A device cache filled through the reader-layer entry points."""

    def __init__(self, model: LayerModel, H, D, max_seqs, max_blocks, capacity, has_null=True, free_order=None,
                 max_batch=None, recompute=False, rope_window=0, n_kv_heads=0):
        self.m, self.H, self.D, self.d = model, H, D, H * D
        self.cfg = smem.make_config(model.L, H, D, max_seqs, max_blocks, capacity, has_null_row=has_null,
                                    max_decode_batch=max_batch, free_order=free_order, recompute_kv=recompute,
                                    rope_window=rope_window, n_kv_heads=n_kv_heads)
        self.cache = smem.SmemCache(self.cfg, device="cuda")
        self.h = self.cache.h
        self.mirror = CacheMirror(capacity, max_seqs, max_blocks, free_order=free_order)
        nmax = max(B_TOK, max_seqs if max_batch is None else max_batch)
        self.ws = torch.empty(smem.smem_layer_workspace_bytes(self.h, nmax), dtype=torch.uint8, device="cuda")
        self.mu = {}  # (seq, idx) -> bf16 bits [R][d]
        self.nu = None
        if has_null:
            nb = nu_bits(model.seed, self.d)
            smem.smem_set_null_vector(self.h, bits_dev(nb), model.sw, self.ws)
            self.nu = bits_f64(nb)

    def append(self, seq, idx, content_seq=None):
        mb = mu_bits(self.m.seed, seq if content_seq is None else content_seq, idx, self.d)
        slot = smem.smem_append_block_rows(self.h, seq, idx, bits_dev(mb), self.m.sw, self.ws)
        rc, s_m = self.mirror.append(seq, idx)
        assert rc == 0 and s_m == slot
        self.mu[(seq, idx)] = mb
        return slot

    def delete(self, seq, idx):
        smem.smem_delete_block(self.h, seq, idx)
        assert self.mirror.delete(seq, idx) == 0
        del self.mu[(seq, idx)]

    def memory(self, seq, q_idx):
        ids = sorted(i for (s, i) in self.mu if s == seq and i < q_idx)
        mu = np.stack([bits_f64(self.mu[(seq, i)]) for i in ids]) if ids else np.zeros((0, 64, self.d))
        return np.array(ids, dtype=np.int64), mu

    def prefill(self, seq, layer, q_idx, x):
        smem.smem_reader_layer_prefill(self.h, seq, layer, q_idx, self.m.sw[layer], x, self.ws)

    def oracle_prefill(self, seq, layer, q_idx, x_in):
        ids, mu = self.memory(seq, q_idx)
        return reader_layer_prefill(x_in, ids, mu, q_idx, self.m.oracle[layer], self.H, self.D, self.nu)

    def decode(self, layer, seqs, pos, qidx, x):
        smem.smem_reader_layer_decode(self.h, layer, seqs, pos, qidx, self.m.sw[layer], x, self.ws)


def _np(t):
    return t.detach().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("D,H,has_null", [(64, 4, True), (64, 4, False), (128, 2, True), (32, 8, True)])
def test_layer_prefill_matches_oracle(D, H, has_null):
    """Two chained layers, 8 memory blocks appended out of order into a
    shuffled pool; blocks 8 (all readable), 3 and 0 (null row only)."""
    model = LayerModel(2, H * D, seed=101 + D)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=16, capacity=24, has_null=has_null,
                    free_order=synth.slot_permutation(7, 24))
    for j in (5, 0, 7, 2, 6, 1, 4, 3):
        lc.append(0, j)
    assert list(smem.smem_get_table(lc.h, 0)[1]) == lc.mirror.table(0)[1]
    for q_idx in (8, 3, 0):
        x = torch.from_numpy(x_rows(model.seed, 0, q_idx, lc.d)).cuda()
        for layer in range(model.L):
            x_in = _np(x)
            lc.prefill(0, layer, q_idx, x)
            ref, _, _ = lc.oracle_prefill(0, layer, q_idx, x_in)
            assert_layer_close(_np(x), ref, x_in, f"layer {layer} q_idx {q_idx}")
    assert smem.smem_check_device_error(lc.h) == smem.OK


def test_layer_block_skip_equals_full_pass():
    """Sec. 3.1 at layer level: the one-block pass of block i over the cache
    equals rows i*b .. i*b+b-1 of the masked full pass over all blocks."""
    H, D, B = 4, 64, 4
    d = H * D
    model = LayerModel(1, d, seed=211)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=8, capacity=8)
    for j in range(B):
        lc.append(0, j)
    X = np.concatenate([x_rows(model.seed, 0, i, d) for i in range(B)]).astype(np.float64)
    mu = np.stack([bits_f64(lc.mu[(0, j)]) for j in range(B)])
    full = full_layer_pass(X, mu, model.oracle[0], H, D, B_TOK, lc.nu)
    for i in range(B):
        sl = slice(i * B_TOK, (i + 1) * B_TOK)
        x = torch.from_numpy(X[sl].astype(np.float32)).cuda()
        lc.prefill(0, 0, i, x)
        assert_layer_close(_np(x), full[sl], X[sl], f"block {i}")


def _decode_setup(model, H, D, ctx, free_order=None, history=False, recompute=False):
    """Sequences with the given contexts; each sequence's current block
    (index ctx[s]) runs the layer prefill on all layers first, leaving its
    in-block rows. history=True reaches the same block set by another edit
    path (extra blocks appended and deleted, a delete/re-append)."""
    S = len(ctx)
    cap = sum(ctx) + 4 * S + 8
    lc = LayerCache(model, H, D, max_seqs=S, max_blocks=max(ctx) + 8, capacity=cap, free_order=free_order,
                    recompute=recompute)
    for s, n in enumerate(ctx):
        order = list(range(n))
        if history:
            order = order[::-1]
            lc.append(s, n + 3, content_seq=99)  # a block that is deleted again
        for j in order:
            lc.append(s, j)
        if history:
            lc.delete(s, n + 3)
            if n > 2:
                lc.delete(s, 1)
                lc.append(s, 1)
    xs = []
    for s, n in enumerate(ctx):
        x = torch.from_numpy(x_rows(model.seed, s, n, lc.d)).cuda()
        layer_in = []
        for layer in range(model.L):
            layer_in.append(_np(x))
            lc.prefill(s, layer, n, x)
        xs.append((layer_in, _np(x)))
    return lc, xs


def test_layer_decode_after_prefill_matches_oracle():
    """A batched decode step over sequences with 5, 0 and 9 memory blocks at
    in-block positions 17, 0 and 63: each token's layer input is its row of
    the block's prefill input, the earlier tokens' k/v are the rows the layer
    prefill stored."""
    H, D, L = 4, 64, 2
    d = H * D
    model = LayerModel(L, d, seed=307)
    ctx = [5, 0, 9]
    pos = [17, 0, 63]
    lc, xs = _decode_setup(model, H, D, ctx)
    x = torch.from_numpy(np.stack([xs[s][0][0][pos[s]] for s in range(3)]).astype(np.float32)).cuda()
    for layer in range(L):
        x_in = _np(x)
        lc.decode(layer, [0, 1, 2], pos, ctx, x)
        got = _np(x)
        for s in range(3):
            ids, mu = lc.memory(s, ctx[s])
            # the oracle's in-block rows: its own prefill of the same layer input
            _, ks, vs = reader_layer_prefill(xs[s][0][layer], ids, mu, ctx[s], model.oracle[layer], H, D, lc.nu)
            ref, _, _ = reader_layer_decode(x_in[s], ids, mu, ctx[s], pos[s], ks[:pos[s]], vs[:pos[s]],
                                            model.oracle[layer], H, D, lc.nu)
            assert_layer_close(got[s], ref, x_in[s], f"decode layer {layer} seq {s}")
    assert smem.smem_check_device_error(lc.h) == smem.OK


def test_layer_outputs_are_edit_path_independent():
    """Theorem 1 through the whole layer: two caches reaching the same block
    sets by different edit paths and slot orders give bitwise-equal prefill
    and decode outputs."""
    H, D, L = 4, 64, 2
    d = H * D
    model = LayerModel(L, d, seed=401)
    ctx = [6, 3]
    a, xa = _decode_setup(model, H, D, ctx)
    b, xb = _decode_setup(model, H, D, ctx, free_order=synth.slot_permutation(9, sum(ctx) + 16), history=True)
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


def test_layer_argument_errors():
    H, D = 2, 64
    d = H * D
    model = LayerModel(1, d, seed=503)
    lc = LayerCache(model, H, D, max_seqs=2, max_blocks=4, capacity=4, has_null=False)
    x = torch.zeros(B_TOK, d, device="cuda")
    need = smem.smem_layer_workspace_bytes(lc.h, B_TOK)
    assert need > 0 and smem.smem_layer_workspace_bytes(lc.h, 10 ** 6) == 0
    with pytest.raises(smem.SmemError) as e:
        smem.smem_reader_layer_prefill(lc.h, 0, 0, 0, model.sw[0], x, lc.ws[: need - 256])
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:
        smem.smem_reader_layer_prefill(lc.h, 0, 0, 0, model.sw[0], x, lc.ws[16:])
    assert e.value.code == smem.ERR_ALIGN
    partial = dict(model.dev[0])
    partial["w_1"] = None
    with pytest.raises(smem.SmemError) as e:
        smem.smem_reader_layer_prefill(lc.h, 0, 0, 0, smem.layer_weights(partial), x, lc.ws)
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:  # no null row in this cache
        smem.smem_set_null_vector(lc.h, bits_dev(nu_bits(1, d)), model.sw, lc.ws)
    assert e.value.code == smem.ERR_INVALID_ARG
    # a failing append changes nothing
    fifo = smem.smem_get_free_fifo(lc.h)
    smem.smem_debug_fail_after(lc.h, 1)
    with pytest.raises(smem.SmemError) as e:
        smem.smem_append_block_rows(lc.h, 0, 0, bits_dev(mu_bits(1, 0, 0, d)), model.sw, lc.ws)
    assert e.value.code == smem.ERR_CUDA
    assert smem.smem_get_free_fifo(lc.h) == fifo and smem.smem_get_table(lc.h, 0) == ([], [])
