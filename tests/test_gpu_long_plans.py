"""Bitwise edit-path independence on the long-context split plans.

From 512 readable blocks on, the decode kernel cuts a row set into
ceil(nblk / 64) blocks per split (8 to 32 blocks, 64 or more splits), and the
one-block prefill at 16 heads cuts it into its widest plans (one cluster of 16
CTAs per head, or 16 splits without clusters). Theorem 1 and the
verification gates G7/G8 ask that the same block set read the same whatever
edit path produced it; these tests build the same block sets through
different edit paths and slot orders at 515 to about 3800 readable blocks,
require bitwise-identical outputs, and check sampled heads against the fp64
oracle.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import assert_close, f64, out_f64

pytestmark = pytest.mark.gpu
R = 64
B_TOK = 64


@pytest.fixture(params=["clusters", "no_clusters"])
def cluster_mode(request, monkeypatch):
    if request.param == "no_clusters":
        monkeypatch.setenv("SMEM_PREFILL_CLUSTERS", "0")
    else:
        monkeypatch.delenv("SMEM_PREFILL_CLUSTERS", raising=False)
    return request.param


def _append(cache, seed, seq, ids, H, D):
    """Appends blocks `ids` of `seq` in the given order, rows generated on
    the device (32 blocks per generator call)."""
    for b0 in range(0, len(ids), 32):
        chunk = [int(j) for j in ids[b0:b0 + 32]]
        K, V = synth.block_rows_torch(seed, seq, chunk, 1, H, R, D, "cuda")
        for i, j in enumerate(chunk):
            smem.smem_append_block(cache.h, seq, j, K[i], V[i])


def _build(targets, path, seed, H, D, Hkv=0, max_batch=None):
    """A cache whose sequence s holds exactly the blocks targets[s].
    path 0: ascending appends into ascending slots. path 1: another slot
    order; decoy blocks appended first, the targets in a random order, a
    random fifth of the targets deleted and appended again, the decoys
    deleted last."""
    hk = Hkv or H
    S = len(targets)
    maxidx = max(max(t) for t in targets) + 1
    decoys = [sorted(set(range(0, maxidx + 40, 3)) - set(t))[:200] for t in targets]
    cap = sum(len(t) for t in targets) + sum(len(d) for d in decoys) + 8
    perm = None if path == 0 else synth.slot_permutation(900 + seed, cap)
    cfg = smem.make_config(1, H, D, S, maxidx + 48, cap, free_order=perm, n_kv_heads=Hkv,
                           max_decode_batch=max_batch)
    cache = smem.SmemCache(cfg, device="cuda")
    rng = np.random.default_rng(seed + 17)
    for s, t in enumerate(targets):
        if path == 0:
            _append(cache, seed, s, sorted(t), hk, D)
            continue
        _append(cache, seed, s, decoys[s], hk, D)
        order = rng.permutation(sorted(t))
        _append(cache, seed, s, order, hk, D)
        again = rng.choice(order, size=len(order) // 5, replace=False)
        for j in again:
            smem.smem_delete_block(cache.h, s, int(j))
        _append(cache, seed, s, rng.permutation(again), hk, D)
        for j in decoys[s]:
            smem.smem_delete_block(cache.h, s, int(j))
    torch.cuda.synchronize()
    for s, t in enumerate(targets):
        assert smem.smem_get_table(cache.h, s)[0] == sorted(t)
    return cache


def _head_rows(seed, seq, blocks, h_kv, D):
    k, v = synth.block_head_rows_np(seed, seq, blocks, 0, h_kv, R, D)
    return f64(k)[:, None], f64(v)[:, None]


@pytest.mark.parametrize("H,D,Hkv", [(4, 64, 0), (4, 128, 0), (8, 64, 2)])
def test_decode_long_split_plan_bitwise(H, D, Hkv):
    """Four sequences reading 3771, 640, 515 and 511 blocks (the first three
    on the long plan, the last on the 16-block plan), built through two edit
    paths: identical bits, and sampled heads match the oracle."""
    seed = 31
    targets = [[j for j in range(4400) if j % 7], [j for j in range(800) if j % 5], list(range(530)),
               list(range(511))]
    qidx = [4400, 800, 515, 600]
    S, hk = len(targets), Hkv or H
    dshape, kvshape = (S, H, D), (S, hk, D)
    ins = [synth.tensor_np(seed, k, sh, 0, 2) for k, sh in
           ((synth.KIND_QDEC_S, dshape), (synth.KIND_KNEW, kvshape), (synth.KIND_VNEW, kvshape),
            (synth.KIND_QDEC_C, dshape))]
    dev = [synth.bits_to_torch_bf16(x).cuda() for x in ins]
    outs = []
    for path in (0, 1):
        cache = _build(targets, path, seed, H, D, Hkv)
        osa = torch.empty(dshape, dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_decode(cache.h, 0, np.arange(S), np.zeros(S), qidx, *dev, osa, oca)
        torch.cuda.synchronize()
        assert smem.smem_check_device_error(cache.h) == smem.OK
        outs.append((osa.view(torch.int16).clone(), oca.view(torch.int16).clone(), out_f64(oca)))
        cache.close()
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])
    G = H // hk
    for s, h in ((0, H - 1), (1, 1), (2, 2)):
        blocks = [j for j in targets[s] if j < qidx[s]]
        mk, mv = _head_rows(seed, s, blocks, h // G, D)
        q = [f64(ins[0][s, h])[None], f64(ins[1][s, h // G])[None], f64(ins[2][s, h // G])[None],
             f64(ins[3][s, h])[None]]
        _, ref_ca = oracle.reader_decode(blocks, mk, mv, qidx[s], 0, None, None, *q)
        assert_close(outs[0][2][s, h], ref_ca[0], f"decode oca seq {s} head {h} ({len(blocks)} blocks)")


@pytest.mark.parametrize("D", [64, 128])
def test_prefill_long_split_plan_bitwise(D, cluster_mode):
    """160M/1.5B head count (H = 16) with 600 readable blocks out of 700
    (and a mid-table query block reading 300), built through two edit paths:
    identical bits; sampled heads match the oracle."""
    if D == 128 and cluster_mode == "clusters":
        pytest.skip("cluster mode is the d_h = 64 prefill")
    seed, H = 37, 16
    target = [j for j in range(700) if j % 7]
    shape = (B_TOK, H, D)
    pin = [synth.tensor_np(seed, k, shape, 0, 4) for k in
           (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
    dev = [synth.bits_to_torch_bf16(x).cuda() for x in pin]
    outs = []
    for path in (0, 1):
        cache = _build([target], path, seed, H, D)
        res = []
        for q_idx in (700, 350):
            osa = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
            oca = torch.empty_like(osa)
            smem.smem_prefill_block(cache.h, 0, 0, q_idx, *dev, osa, oca)
            torch.cuda.synchronize()
            res.append((osa.view(torch.int16).clone(), oca.view(torch.int16).clone(), out_f64(oca)))
        assert smem.smem_check_device_error(cache.h) == smem.OK
        outs.append(res)
        cache.close()
    for a, b in zip(outs[0], outs[1]):
        assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    for qi, (q_idx, h) in enumerate(((700, 5), (350, 12))):
        blocks = [j for j in target if j < q_idx]
        mk, mv = _head_rows(seed, 0, blocks, h, D)
        x = [f64(t[:, h:h + 1]) for t in pin]
        _, ref_ca = oracle.reader_prefill(blocks, mk, mv, q_idx, *x)
        assert_close(outs[0][qi][2][:, h], ref_ca[:, 0], f"prefill oca head {h} ({len(blocks)} blocks)")
