"""GPU parity of grouped-query attention (key/value heads shared by groups of
query heads; arXiv 2609.32395, Sec. 3.1: it composes with the KV saving)
against the oracle with each key/value head repeated over its group:

* one-block prefill (cluster and cluster-free kernels) and ragged batched
  decode for groups of 4 and of 8 (one key/value head), with the null row;
* consecutive decode steps (the shared in-block row written once per group);
* RoPE composite together with grouped heads;
* the full reader layer with grouped key/value maps;
* bitwise edit-path independence.
"""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, assert_close, out_f64
from tests.layer_helpers import LayerModel, assert_layer_close

pytestmark = pytest.mark.gpu


@pytest.fixture(params=["clusters", "no_clusters"])
def cluster_mode(request, monkeypatch):
    if request.param == "no_clusters":
        monkeypatch.setenv("SMEM_PREFILL_CLUSTERS", "0")
    else:
        monkeypatch.delenv("SMEM_PREFILL_CLUSTERS", raising=False)
    return request.param


def _cache(Hkv, D=64, H=8, rope=0, seed=17, perm_seed=4):
    nblks = [0, 3, 37, 70]
    dc = DeviceCache(L=2, H=H, D=D, max_seqs=len(nblks), max_blocks=80, capacity=140, seed=seed, has_null=True,
                     n_kv_heads=Hkv, rope_window=rope, free_order=synth.slot_permutation(perm_seed, 140))
    rng = np.random.default_rng(seed)
    for s, n in enumerate(nblks):
        for j in rng.permutation(n):
            dc.append(s, int(j))
    return dc, nblks


@pytest.mark.parametrize("Hkv,D", [(2, 64), (1, 64), (2, 128)])
def test_gqa_prefill_matches_oracle(Hkv, D, cluster_mode):
    if D != 64 and cluster_mode == "clusters":
        pytest.skip("cluster mode is a d_h = 64 kernel")
    dc, nblks = _cache(Hkv, D=D, H=8 if D == 64 else 4)
    for s, n in enumerate(nblks):
        ins, osa, oca = dc.prefill(s, s % 2, n, tag=s)
        ref_sa, ref_ca = dc.oracle_prefill(s, s % 2, n, *ins)
        assert_close(out_f64(osa), ref_sa, f"osa seq {s}")
        assert_close(out_f64(oca), ref_ca, f"oca seq {s}")
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("Hkv,rope,D,H", [(2, 0, 64, 8), (1, 0, 64, 8), (2, 15, 64, 8), (2, 0, 128, 4),
                                          (4, 0, 128, 4), (2, 0, 32, 8), (4, 0, 64, 12), (4, 0, 64, 8)])
def test_gqa_decode_consecutive_steps(Hkv, rope, D, H):
    """Groups of 4 (one grouped unit of four queries), 8 (two units), 2 at
    d_h 128 and 64 (a unit of two in the four-query tile) and 4 at d_h 32, 3
    (one query per unit), and 1; with and without rotary phases."""
    dc, nblks = _cache(Hkv, rope=rope, D=D, H=H)
    pos0 = [0, 30, 61, 5]
    for s, p in enumerate(pos0):
        dc.write_inblock(s, 1, p, tag=s)
    for step in range(3):
        pos = [p + step for p in pos0]
        ins, osa, oca = dc.decode(1, list(range(4)), pos, nblks, step=step)
        for i in range(4):
            ref_sa, ref_ca = dc.oracle_decode(1, i, pos[i], nblks[i], *(x[i] for x in ins))
            assert_close(out_f64(osa[i]), ref_sa, f"osa seq {i} step {step}")
            assert_close(out_f64(oca[i]), ref_ca, f"oca seq {i} step {step}")
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_gqa_edit_path_independence():
    a, _ = _cache(2, seed=21, perm_seed=4)
    b, _ = _cache(2, seed=21, perm_seed=77)
    b.delete(2, 5)
    b.delete(2, 30)
    b.append(2, 30)
    b.append(2, 5)
    assert a.mirror.table(2)[1] != b.mirror.table(2)[1]
    _, sa_a, ca_a = a.prefill(2, 0, 37, tag=2)
    _, sa_b, ca_b = b.prefill(2, 0, 37, tag=2)
    assert torch.equal(sa_a, sa_b) and torch.equal(ca_a, ca_b)
    for dc in (a, b):
        dc.write_inblock(2, 0, 12)
    _, da_s, da_c = a.decode(0, [2], [12], [37], step=5)
    _, db_s, db_c = b.decode(0, [2], [12], [37], step=5)
    assert torch.equal(da_s, db_s) and torch.equal(da_c, db_c)


def test_gqa_reader_layer_matches_oracle():
    from oracle.reader_layer import reader_layer_decode, reader_layer_prefill
    from tests.test_gpu_layer import LayerCache, _np, x_rows
    H, D, Hkv = 4, 64, 2
    d = H * D
    model = LayerModel(1, d, seed=1501, kvd=Hkv * D)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=16, capacity=16, n_kv_heads=Hkv)
    for j in range(9):
        lc.append(0, j)
    x = torch.from_numpy(x_rows(model.seed, 0, 9, d)).cuda()
    x_in = _np(x)
    lc.prefill(0, 0, 9, x)
    ids, mu = lc.memory(0, 9)
    ref, ks, vs = reader_layer_prefill(x_in, ids, mu, 9, model.oracle[0], H, D, lc.nu)
    assert_layer_close(_np(x), ref, x_in, "gqa layer prefill")
    p = 20
    xd = torch.from_numpy(x_in[p:p + 1].astype(np.float32)).cuda()
    lc.decode(0, [0], [p], [9], xd)
    ref_d, _, _ = reader_layer_decode(x_in[p], ids, mu, 9, p, ks[:p], vs[:p], model.oracle[0], H, D, lc.nu)
    assert_layer_close(_np(xd)[0], ref_d, x_in[p], "gqa layer decode")
