"""GPU parity of the batched decode step (C ABI -> CUDA kernels) against the
fp64 oracle on identical seeded inputs, plus bitwise edit-path independence
and bit-exact bookkeeping on the device."""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, assert_close, out_f64

pytestmark = pytest.mark.gpu


def _check_decode(dc, layer, seqs, pos, qidx, step=0):
    ins, osa, oca = dc.decode(layer, seqs, pos, qidx, step)
    qs, kn, vn, qc = ins
    got_sa, got_ca = out_f64(osa), out_f64(oca)
    for i, s in enumerate(seqs):
        ref_sa, ref_ca = dc.oracle_decode(layer, s, pos[i], qidx[i], qs[i], kn[i], vn[i], qc[i])
        assert_close(got_sa[i], ref_sa, f"osa seq {s} p {pos[i]}")
        assert_close(got_ca[i], ref_ca, f"oca seq {s} nblk<{qidx[i]}")
    return osa, oca


def test_tiny_config_decode_and_delete_reappend():
    """Tiny reader (H=4, d_h=64, 8 blocks of 64 rows): decode, then delete
    block 3 and re-append it; it lands in another slot and the outputs are
    bitwise unchanged."""
    dc = DeviceCache(L=1, H=4, D=64, max_seqs=1, max_blocks=16, capacity=16)
    for j in range(8):
        dc.append(0, j)
    dc.write_inblock(0, 0, 63)
    dc.check_tables([0])
    osa0, oca0 = _check_decode(dc, 0, [0], [63], [8])
    dc.delete(0, 3)
    dc.check_tables([0])
    slot = dc.append(0, 3)
    assert slot == 8
    dc.check_tables([0])
    dc.write_inblock(0, 0, 63)
    _, osa1, oca1 = dc.decode(0, [0], [63], [8])
    assert torch.equal(oca0.view(torch.int16), oca1.view(torch.int16))
    assert torch.equal(osa0.view(torch.int16), osa1.view(torch.int16))
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("D", [32, 64, 128])
@pytest.mark.parametrize("has_null", [False, True])
def test_ragged_batch(D, has_null):
    """Ragged contexts spanning one to many splits with a ragged last split,
    an empty context, mid-table query blocks, and in-block offsets 0..63."""
    nblks = [0, 1, 4, 5, 33, 70, 130]
    S = len(nblks)
    perm = synth.slot_permutation(3, 400)
    dc = DeviceCache(L=2, H=3, D=D, max_seqs=S, max_blocks=160, capacity=400, seed=1, free_order=perm,
                     has_null=has_null)
    rng = np.random.default_rng(5)
    for s, n in enumerate(nblks):
        for j in rng.permutation(n):  # append out of order: the table sorts
            dc.append(s, int(j))
    dc.check_tables(range(S))
    pos = [0, 63, 17, 1, 40, 5, 62]
    for layer in range(2):
        for s, p in enumerate(pos):
            dc.write_inblock(s, layer, p, tag=layer)
    qidx = [n for n in nblks]
    qidx[4] = 20   # mid-table: blocks 0..19 only
    qidx[6] = 129  # all but the last block
    for layer in range(2):
        _check_decode(dc, layer, list(range(S)), pos, qidx, step=layer)
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_consecutive_steps_grow_inblock_rows():
    """Steps p = 0, 1, 2, ... write the new token's k, v and attend to all
    earlier in-block rows of the block."""
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=2, max_blocks=32, capacity=64, seed=2)
    for s in range(2):
        for j in range(10 + s):
            dc.append(s, j)
    for p in range(5):
        _check_decode(dc, 0, [1, 0], [p, p], [11, 10], step=p)


def test_path_independence_bitwise():
    """Two caches reaching the same block set through different edit paths
    and different slot orders give bitwise-identical decode outputs."""
    H, D, L = 4, 64, 1
    target = [0, 1, 2, 5, 6, 9, 11, 12, 13, 20, 21, 22, 23, 30]
    outs = []
    for trial in range(3):
        perm = synth.slot_permutation(100 + trial, 96)
        dc = DeviceCache(L=L, H=H, D=D, max_seqs=1, max_blocks=64, capacity=96, seed=7, free_order=perm)
        rng = np.random.default_rng(trial)
        live = set()
        for _ in range(40):
            j = int(rng.integers(0, 32))
            if j in live and rng.random() < 0.5:
                dc.delete(0, j)
                live.discard(j)
            elif j not in live:
                dc.append(0, j)
                live.add(j)
        for j in sorted(live - set(target)):
            dc.delete(0, j)
        for j in rng.permutation(sorted(set(target) - live)):
            dc.append(0, int(j))
        dc.check_tables([0])
        dc.write_inblock(0, 0, 10)
        _, osa, oca = dc.decode(0, [0], [10], [40])
        outs.append((osa.view(torch.int16).clone(), oca.view(torch.int16).clone()))
    for o in outs[1:]:
        assert torch.equal(o[0], outs[0][0]) and torch.equal(o[1], outs[0][1])


def test_injected_failure_leaves_state_unchanged():
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=1, max_blocks=8, capacity=8)
    for j in range(3):
        dc.append(0, j)
    before = (smem.smem_get_table(dc.h, 0), smem.smem_get_free_fifo(dc.h))
    K, V = dc.block_bits(0, 5)
    smem.smem_debug_fail_after(dc.h, 1)
    with pytest.raises(smem.SmemError) as e:
        smem.smem_append_block(dc.h, 0, 5, synth.bits_to_torch_bf16(K).cuda(), synth.bits_to_torch_bf16(V).cuda())
    assert e.value.code == smem.ERR_CUDA
    smem.smem_debug_fail_after(dc.h, 1)
    with pytest.raises(smem.SmemError):
        smem.smem_delete_block(dc.h, 0, 1)
    assert (smem.smem_get_table(dc.h, 0), smem.smem_get_free_fifo(dc.h)) == before
    dc.check_tables([0])


def test_decode_rejects_bad_arguments():
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=2, max_blocks=8, capacity=8)
    x = torch.zeros((2, 2, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode(dc.h, 0, [0, 0], [0, 0], [1, 1], x, x, x, x, x, x)  # duplicate sequence
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode(dc.h, 0, [0], [64], [1], x, x, x, x, x, x)  # offset beyond the block
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode(dc.h, 1, [0], [0], [1], x, x, x, x, x, x)  # no such layer
    assert e.value.code == smem.ERR_INVALID_ARG


@pytest.mark.gpu
def test_shared_blocks_read_like_private_copies():
    """Exact reuse (Sec. 2): sequence 1 shares sequence 0's cached blocks by
    reference, sequence 2 holds private copies of the same rows; prefill and
    decode outputs of 1 and 2 are bitwise equal. Deleting 0's references
    keeps 1 unchanged and frees no shared slot; releasing 1 frees them."""
    import torch

    import synth
    from paper_2609_32395_gb300 import smem
    from tests.gpu_helpers import DeviceCache, to_dev

    dc = DeviceCache(L=2, H=4, D=64, max_seqs=3, max_blocks=16, capacity=40)
    for j in range(10):
        dc.append(0, j)
        dc.append(2, j, content_seq=0)            # private copy of the same rows
    for j in range(10):
        smem.smem_share_block(dc.h, 0, j, 1, j)
        assert dc.mirror.share(0, j, 1, j)[0] == 0
    fifo0 = smem.smem_get_free_fifo(dc.h)
    assert fifo0 == dc.mirror.free_list()

    def outputs():
        res = []
        for s in (1, 2):
            _, sa, ca = dc.prefill(s, 1, 10, tag=3)
            res.append((sa, ca))
        return res

    (sa1, ca1), (sa2, ca2) = outputs()
    assert torch.equal(sa1, sa2) and torch.equal(ca1, ca2)
    for j in range(10):
        smem.smem_delete_block(dc.h, 0, j)
        assert dc.mirror.delete(0, j) == 0
    assert smem.smem_get_free_fifo(dc.h) == fifo0   # no shared slot came free
    (_, ca1b), (_, ca2b) = outputs()
    assert torch.equal(ca1b, ca1) and torch.equal(ca2b, ca2)
    # a decode step of each with identical inputs and identical in-block rows
    Kb = to_dev(synth.tensor_np(7, synth.KIND_KIN, (5, 4, 64), 0))
    Vb = to_dev(synth.tensor_np(7, synth.KIND_VIN, (5, 4, 64), 0))
    q = [to_dev(synth.tensor_np(7, k, (1, 4, 64), 1)) for k in (synth.KIND_QDEC_S, synth.KIND_KNEW,
                                                               synth.KIND_VNEW, synth.KIND_QDEC_C)]
    outs = []
    for s in (1, 2):
        smem.smem_write_inblock(dc.h, s, 0, 5, Kb, Vb)
        osa = torch.empty(1, 4, 64, dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_decode(dc.h, 0, [s], [5], [10], *q, osa, oca)
        outs.append((osa, oca))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    smem.smem_release_seq(dc.h, 1)
    assert dc.mirror.release(1) == 0
    assert smem.smem_get_free_fifo(dc.h) == dc.mirror.free_list()
    assert len(dc.mirror.free_list()) == len(fifo0) + 10
