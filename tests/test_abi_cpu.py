"""C ABI checks that need no GPU: the library loads, exports every symbol the
header declares, validates geometry, and its host bookkeeping matches the
independent mirror bit for bit (bookkeeping-only caches make no CUDA call)."""
import os
import re

import numpy as np
import pytest

from oracle import bookkeeping as bk
from oracle.bookkeeping import CacheMirror
from paper_2609_32395_gb300 import smem
from tests.test_bookkeeping_mirror import parse_golden

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "smem.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(smem_\w+)\s*\(", text)))


def test_exports_every_declared_symbol():
    names = declared_functions()
    assert len(names) >= 15
    L = smem.lib()
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(smem.EXPORTED)
    assert smem.smem_abi_version() == 8


def test_required_bytes_validation():
    ok = smem.make_config(2, 4, 64, 3, 16, 32)
    assert smem.smem_cache_required_bytes(ok) > 32 * 2 * 4 * 2 * 64 * 64 * 2
    for bad in (smem.make_config(2, 4, 96, 3, 16, 32),           # d_h unsupported
                smem.make_config(2, 4, 64, 3, 16, 32, block_tokens=32),
                smem.make_config(0, 4, 64, 3, 16, 32),
                smem.make_config(2, 4, 64, 3, 16, 32, max_decode_batch=4)):
        assert smem.smem_cache_required_bytes(bad) == 0


def test_bad_free_order_rejected():
    with pytest.raises(smem.SmemError) as e:
        smem.smem_cache_create(smem.make_config(1, 1, 64, 1, 4, 4, free_order=[0, 1, 1, 2]))
    assert e.value.code == smem.ERR_INVALID_ARG


def test_device_ops_refused_without_device():
    h = smem.smem_cache_create(smem.make_config(1, 2, 64, 2, 8, 8))
    try:
        L = smem.lib()
        assert L.smem_decode(h, 0, 1, None, None, None, None, None, None, None, None, None, None) != 0
        assert L.smem_prefill_block(h, 0, 0, 1, None, None, None, None, None, None, None) == smem.ERR_NO_DEVICE
        assert L.smem_check_device_error(h, None) == smem.ERR_NO_DEVICE
        assert L.smem_write_inblock(h, 0, 0, 1, None, None, None) == smem.ERR_NO_DEVICE
    finally:
        smem.smem_cache_destroy(h)


def _tables(h, n_seqs):
    return [list(zip(*smem.smem_get_table(h, s))) for s in range(n_seqs)]


def test_golden_example_matches_library():
    h = smem.smem_cache_create(smem.make_config(1, 1, 64, 2, 3, 4))
    try:
        for st in parse_golden():
            if st["op"] == "append":
                rc = smem.lib().smem_append_block(h, st["seq"], st["blk"], None, None, None, None)
            elif st["op"] == "delete":
                rc = smem.lib().smem_delete_block(h, st["seq"], st["blk"], None)
            else:
                rc = smem.lib().smem_release_seq(h, st["seq"], None)
            assert rc == st["rc"], st
            for seq in range(2):
                idx, slots = smem.smem_get_table(h, seq)
                assert list(zip(idx, slots)) == st["tables"][seq], st
            assert smem.smem_get_free_fifo(h) == st["fifo"], st
    finally:
        smem.smem_cache_destroy(h)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_random_ops_match_mirror(seed):
    rng = np.random.default_rng(seed)
    C, S, MB = 48, 5, 12
    order = rng.permutation(C)
    m = CacheMirror(C, S, MB, free_order=order)
    h = smem.smem_cache_create(smem.make_config(2, 2, 64, S, MB, C, free_order=order))
    L = smem.lib()
    slot = smem.ctypes.c_int32(-1)
    try:
        for step in range(4000):
            seq = int(rng.integers(-1, S + 1))
            blk = int(rng.integers(-2, 30))
            u = rng.random()
            if u < 0.55:
                rc_m, s_m = m.append(seq, blk)
                rc = L.smem_append_block(h, seq, blk, None, None, None, smem.ctypes.byref(slot))
                assert rc == rc_m
                if rc == 0:
                    assert slot.value == s_m
            elif u < 0.97:
                assert L.smem_delete_block(h, seq, blk, None) == m.delete(seq, blk)
            else:
                assert L.smem_release_seq(h, seq, None) == m.release(seq)
            if step % 25 == 0 or step > 3900:
                for s in range(S):
                    assert smem.smem_get_table(h, s) == m.table(s)
                assert smem.smem_get_free_fifo(h) == m.free_list()
        assert smem.smem_free_slots(h) == len(m.free_list())
    finally:
        smem.smem_cache_destroy(h)


def test_error_codes_agree_with_mirror_constants():
    assert (smem.ERR_INVALID_ARG, smem.ERR_NO_SUCH_SEQ, smem.ERR_DUPLICATE_BLOCK, smem.ERR_NO_SUCH_BLOCK,
            smem.ERR_POOL_FULL, smem.ERR_TABLE_FULL) == (bk.ERR_INVALID_ARG, bk.ERR_NO_SUCH_SEQ,
                                                         bk.ERR_DUPLICATE_BLOCK, bk.ERR_NO_SUCH_BLOCK,
                                                         bk.ERR_POOL_FULL, bk.ERR_TABLE_FULL)


def test_layer_entry_points_on_a_bookkeeping_cache():
    """Workspace sizing is host arithmetic; the layer calls need a device."""
    cfg = smem.make_config(2, 4, 64, 3, 16, 32, has_null_row=True)
    h = smem.smem_cache_create(cfg, None)
    try:
        d = 4 * 64
        w0 = smem.smem_layer_workspace_bytes(h, 0)
        w64 = smem.smem_layer_workspace_bytes(h, 64)
        assert w0 == 256  # the memory-row projections need no scratch (a nominal minimum)
        # h (LayerNorm output, bf16 d), qkv (bf16 3d), att and qc (bf16 d each), g (bf16 4d) per row
        assert w64 == 64 * (d * 2 + 3 * d * 2 + 2 * d * 2 + 4 * d * 2)
        assert smem.smem_layer_workspace_bytes(h, 65) == 0      # above max(b, max_decode_batch)
        assert smem.smem_layer_workspace_bytes(h, -1) == 0
        w = [smem.SmemLayerWeights()] * 2
        L = smem.lib()
        import ctypes
        arr = (smem.SmemLayerWeights * 2)(*w)
        assert L.smem_reader_layer_prefill(h, 0, 0, 0, arr, None, None, 0, None) == smem.ERR_NO_DEVICE
        assert L.smem_append_block_rows(h, 0, 0, None, arr, None, 0, None, None) == smem.ERR_NO_DEVICE
        assert L.smem_set_null_vector(h, None, arr, None, 0, None) == smem.ERR_NO_DEVICE
        seq = (ctypes.c_int32 * 1)(0)
        assert L.smem_reader_layer_decode(h, 0, 1, seq, seq, seq, arr, None, None, 0, None) == smem.ERR_NO_DEVICE
        assert smem.smem_get_table(h, 0) == ([], [])
    finally:
        smem.smem_cache_destroy(h)


def test_recompute_geometry():
    """A recompute cache's slot holds R*d bf16 memory rows instead of the
    L*H*2*R*d_h of the materialized K/V; unsupported widths are refused."""
    mat = smem.make_config(4, 4, 64, 2, 8, 64)
    rec = smem.make_config(4, 4, 64, 2, 8, 64, recompute_kv=True)
    diff = smem.smem_cache_required_bytes(mat) - smem.smem_cache_required_bytes(rec)
    assert abs(diff - 64 * (4 * 4 * 2 * 64 * 64 * 2 - 64 * 256 * 2)) < 8192
    assert smem.smem_cache_required_bytes(smem.make_config(1, 1, 64, 1, 4, 4, recompute_kv=True)) == 0  # d = 64
    h = smem.smem_cache_create(rec, None)
    try:
        d = 4 * 64
        w0 = smem.smem_layer_workspace_bytes(h, 0)
        w2 = smem.smem_layer_workspace_bytes(h, 2)
        # per row: the dense buffers, q' and O' [H][d] bf16, split partials
        dense = 6 * d * 2 + 4 * d * 4 + 4 * d * 2
        assert w2 - w0 >= 2 * (dense + 2 * 4 * d * 2)
        # the decode kernel is chosen on a device only
        with pytest.raises(smem.SmemError) as e:
            smem.smem_mu_decode_plan(h)
        assert e.value.code == smem.ERR_NO_DEVICE
    finally:
        smem.smem_cache_destroy(h)
    h = smem.smem_cache_create(mat, None)
    try:
        with pytest.raises(smem.SmemError) as e:
            smem.smem_mu_decode_plan(h)
        assert e.value.code == smem.ERR_UNSUPPORTED
    finally:
        smem.smem_cache_destroy(h)


def test_recompute_workspace_covers_every_query_tile():
    """H = 32 heads at d = 2048 need two 16-query tiles per decode item (the
    two-pass kernel's accumulators fit 16 queries at that width); the
    workspace holds the split partials of both tiles."""
    cfg = smem.make_config(1, 32, 64, 4, 8, 16, recompute_kv=True)
    h = smem.smem_cache_create(cfg, None)
    try:
        d = 32 * 64
        w0 = smem.smem_layer_workspace_bytes(h, 0)
        w4 = smem.smem_layer_workspace_bytes(h, 4)
        assert w4 - w0 >= 4 * 32 * 16 * (d + 4) * 4  # 4 items x 32 query rows x 16 splits
    finally:
        smem.smem_cache_destroy(h)


def test_memory_row_and_static_scratch_entry_points_need_a_device():
    """Without a device the memory-row attention entry points and the
    static-scratch decode refuse with SMEM_ERR_NO_DEVICE before touching any
    argument; a NULL cache is SMEM_ERR_INVALID_ARG."""
    import ctypes
    L = smem.lib()
    seq = (ctypes.c_int32 * 1)(0)
    for recompute in (False, True):
        h = smem.smem_cache_create(smem.make_config(1, 4, 64, 2, 8, 8, recompute_kv=recompute), None)
        try:
            assert L.smem_mu_decode(h, 1, seq, seq, None, None, None, 0, None) == smem.ERR_NO_DEVICE
            assert L.smem_mu_prefill(h, 0, 1, None, None, None, 0, None) == smem.ERR_NO_DEVICE
            assert L.smem_decode_static_scratch(h, 0, 1, seq, seq, seq, None, None, None, None, None, None,
                                                None) == smem.ERR_NO_DEVICE
        finally:
            smem.smem_cache_destroy(h)
    assert L.smem_mu_decode(None, 1, seq, seq, None, None, None, 0, None) == smem.ERR_INVALID_ARG
    assert L.smem_mu_prefill(None, 0, 1, None, None, None, 0, None) == smem.ERR_INVALID_ARG
    assert L.smem_mu_decode_plan(None, None, None, None) == smem.ERR_INVALID_ARG
