"""GPU parity of the one-block prefill (tcgen05 tensor-core kernel, through
the C ABI) against the fp64 oracle on identical seeded inputs, plus bitwise
edit-path independence."""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, assert_close, out_f64, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(params=["clusters", "no_clusters"])
def cluster_mode(request, monkeypatch):
    """d_h = 64 prefill with one cluster per head, or the cluster-free kernel."""
    if request.param == "no_clusters":
        monkeypatch.setenv("SMEM_PREFILL_CLUSTERS", "0")
    else:
        monkeypatch.delenv("SMEM_PREFILL_CLUSTERS", raising=False)
    return request.param


def _check_prefill(dc, seq, layer, q_idx, tag=0):
    ins, osa, oca = dc.prefill(seq, layer, q_idx, tag)
    ref_sa, ref_ca = dc.oracle_prefill(seq, layer, q_idx, *ins)
    assert_close(out_f64(osa), ref_sa, f"osa seq {seq} layer {layer}")
    assert_close(out_f64(oca), ref_ca, f"oca seq {seq} layer {layer} q_idx {q_idx}")
    return osa, oca


def test_tiny_config_prefill_and_delete_reappend(cluster_mode):
    """Tiny reader: H=4, d_h=64, 8 memory blocks (512 rows), one 64-token
    query block; delete block 3, re-append it to another slot: bitwise equal."""
    dc = DeviceCache(L=1, H=4, D=64, max_seqs=1, max_blocks=16, capacity=16)
    for j in range(8):
        dc.append(0, j)
    osa0, oca0 = _check_prefill(dc, 0, 0, 8)
    dc.delete(0, 3)
    _check_prefill(dc, 0, 0, 8)  # 7 blocks: parity with block 3 absent
    assert dc.append(0, 3) == 8
    dc.check_tables([0])
    _, osa1, oca1 = dc.prefill(0, 0, 8)
    assert torch.equal(oca0.view(torch.int16), oca1.view(torch.int16))
    assert torch.equal(osa0.view(torch.int16), osa1.view(torch.int16))
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("D", [32, 64, 128])
@pytest.mark.parametrize("has_null", [False, True])
def test_ragged_contexts(D, has_null, cluster_mode):
    """Contexts from empty to many splits with a ragged last split, and a
    query block in the middle of the table."""
    nblks = [0, 1, 2, 5, 33, 64, 130]
    S = len(nblks)
    perm = synth.slot_permutation(4, 300)
    dc = DeviceCache(L=2, H=3, D=D, max_seqs=S, max_blocks=160, capacity=300, seed=3, free_order=perm,
                     has_null=has_null)
    rng = np.random.default_rng(8)
    for s, n in enumerate(nblks):
        for j in rng.permutation(n):
            dc.append(s, int(j))
    for s, n in enumerate(nblks):
        _check_prefill(dc, s, s % 2, n, tag=s)
    _check_prefill(dc, 6, 1, 77, tag=9)  # blocks 0..76 of 130
    _check_prefill(dc, 4, 0, 0, tag=10)  # query block 0: no memory at all
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("nblk", [16, 64, 256])
def test_160m_shape_one_layer(nblk, cluster_mode):
    """160M reader shape (H=12, d_h=64) at 16 / 64 / 256 cached blocks."""
    dc = DeviceCache(L=1, H=12, D=64, max_seqs=1, max_blocks=nblk + 1, capacity=nblk + 8, seed=5,
                     free_order=synth.slot_permutation(5, nblk + 8))
    for j in range(nblk):
        dc.append(0, j)
    _check_prefill(dc, 0, 0, nblk)
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("nblk,has_null,rope", [(1, False, 0), (7, True, 0), (64, True, 0), (256, False, 0),
                                                (40, True, 15)])
def test_cluster_and_cluster_free_bitwise_equal(nblk, has_null, rope, monkeypatch):
    """At d_h = 64 the split plan depends on the block and head counts alone;
    the cluster kernel and the cluster-free one (a device that cannot hold
    the clusters) merge the same partials in the same order, null row
    first, so the same block set gives the same bits in either mode."""
    outs = []
    for clusters in (True, False):
        if clusters:
            monkeypatch.delenv("SMEM_PREFILL_CLUSTERS", raising=False)
        else:
            monkeypatch.setenv("SMEM_PREFILL_CLUSTERS", "0")
        dc = DeviceCache(L=1, H=12, D=64, max_seqs=1, max_blocks=nblk + 2, capacity=nblk + 2, seed=71,
                         has_null=has_null, rope_window=rope)
        for j in range(nblk):
            dc.append(0, j)
        ins, osa, oca = dc.prefill(0, 0, nblk + 1)
        if clusters and nblk <= 64 and not rope:
            ref_sa, ref_ca = dc.oracle_prefill(0, 0, nblk + 1, *ins)
            assert_close(out_f64(osa), ref_sa, "osa")
            assert_close(out_f64(oca), ref_ca, "oca")
        outs.append((osa.view(torch.int16).clone(), oca.view(torch.int16).clone()))
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])


@pytest.mark.parametrize("D", [32, 64, 128])
def test_path_independence_bitwise(D):
    outs = []
    target = list(range(0, 40, 2)) + [41, 45]
    for trial in range(3):
        dc = DeviceCache(L=1, H=2, D=D, max_seqs=1, max_blocks=64, capacity=100, seed=13,
                         free_order=synth.slot_permutation(50 + trial, 100))
        rng = np.random.default_rng(100 + trial)
        live = set()
        for _ in range(50):
            j = int(rng.integers(0, 48))
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
        _, osa, oca = dc.prefill(0, 0, 50)
        outs.append((osa.view(torch.int16).clone(), oca.view(torch.int16).clone()))
    for o in outs[1:]:
        assert torch.equal(o[0], outs[0][0]) and torch.equal(o[1], outs[0][1])


def test_prefills_interleaved_with_edits_without_host_sync():
    """Prefills are launched with programmatic dependent launch, so a launch
    may begin while the previous kernel still runs. Appends, deletes and
    prefills enqueued back to back with no host synchronisation must give,
    output for output, the bits of the same calls each followed by a full
    synchronisation (every read of the pool and the block table sees every
    edit enqueued before it)."""
    def run(sync):
        dc = DeviceCache(L=2, H=12, D=64, max_seqs=1, max_blocks=64, capacity=80, seed=91, has_null=True,
                         free_order=synth.slot_permutation(17, 80))
        outs = []

        def pf(layer, q_idx, tag):
            qs, ks, vs, qc = [to_dev(x) for x in dc.prefill_inputs(layer, tag)]
            osa = torch.empty((64, 12, 64), dtype=torch.bfloat16, device="cuda")
            oca = torch.empty_like(osa)
            smem.smem_prefill_block(dc.h, 0, layer, q_idx, qs, ks, vs, qc, osa, oca)
            outs.append((osa, oca))
            if sync:
                torch.cuda.synchronize()

        def edit(fn, *a):
            fn(*a)
            if sync:
                torch.cuda.synchronize()

        for j in range(40):
            edit(dc.append, 0, j)
        pf(0, 40, 0)
        pf(1, 40, 1)
        pf(0, 40, 2)
        edit(dc.delete, 0, 7)
        pf(0, 40, 3)
        pf(1, 40, 4)
        edit(dc.append, 0, 7)
        edit(dc.append, 0, 45)
        pf(0, 50, 5)
        pf(1, 50, 6)
        pf(0, 50, 7)
        torch.cuda.synchronize()
        assert smem.smem_check_device_error(dc.h) == smem.OK
        return dc, [(a.view(torch.int16).clone(), b.view(torch.int16).clone()) for a, b in outs]

    dc, fast = run(False)
    _, slow = run(True)
    assert len(fast) == len(slow)
    for i, (f, s2) in enumerate(zip(fast, slow)):
        assert torch.equal(f[0], s2[0]) and torch.equal(f[1], s2[1]), f"prefill {i}"
    # the last prefill against the oracle (the final block set: 0..39 and 45)
    ins = dc.prefill_inputs(0, 7)
    ref_sa, ref_ca = dc.oracle_prefill(0, 0, 50, *ins)
    got_sa = out_f64(fast[-1][0].view(torch.bfloat16))
    got_ca = out_f64(fast[-1][1].view(torch.bfloat16))
    assert_close(got_sa, ref_sa, "osa")
    assert_close(got_ca, ref_ca, "oca")


def test_prefill_ks_feed_decode():
    """The prefill's in-block K/V written as in-block rows give a decode step
    that agrees with the oracle (prefill -> decode hand-off)."""
    dc = DeviceCache(L=1, H=4, D=64, max_seqs=1, max_blocks=16, capacity=16, seed=21)
    for j in range(6):
        dc.append(0, j)
    (qs, ks, vs, qc), _, _ = dc.prefill(0, 0, 6)
    p = 40
    from tests.gpu_helpers import to_dev
    smem.smem_write_inblock(dc.h, 0, 0, p, to_dev(ks[:p]), to_dev(vs[:p]))
    dc.inblock[(0, 0)] = (ks.copy(), vs.copy())
    ins, osa, oca = dc.decode(0, [0], [p], [6])
    ref_sa, ref_ca = dc.oracle_decode(0, 0, p, 6, ins[0][0], ins[1][0], ins[2][0], ins[3][0])
    assert_close(out_f64(osa[0]), ref_sa, "decode osa after prefill")
    assert_close(out_f64(oca[0]), ref_ca, "decode oca after prefill")
