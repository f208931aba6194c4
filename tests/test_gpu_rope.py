"""GPU parity of the SMem+RoPE composite (rotary phases inside the attention
kernels; arXiv 2609.32395, Sec. 4 and App. "Training recipes" / "Needle")
against the fp64 rotary oracle, which turns every query and key by its
absolute phase before the plain attention:

* one-block prefill (cluster and cluster-free kernels, d_h 64/128, with and
  without the null row) for query blocks beyond the window (far and near
  memory blocks) and inside it, with gaps in the block indices and window
  widths 15 and 3;
* batched decode over consecutive steps (the turned in-block keys stored by
  one step are read by the next) and after smem_write_inblock;
* bitwise edit-path independence (Theorem 1) with rotary phases;
* the full reader layer with rotary phases.
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


def _gappy_cache(D, H, W, has_null, L=1, seed=5):
    dc = DeviceCache(L=L, H=H, D=D, max_seqs=2, max_blocks=64, capacity=96, seed=seed, has_null=has_null,
                     rope_window=W, free_order=synth.slot_permutation(seed, 96))
    for j in range(40):
        if j % 7 != 3:  # gaps in the indices: deleted-looking holes, near and far
            dc.append(0, j)
    return dc


@pytest.mark.parametrize("D,H,has_null,W", [(64, 4, True, 15), (64, 4, False, 15), (64, 4, True, 3),
                                            (128, 2, True, 15), (32, 8, True, 15)])
def test_rope_prefill_matches_oracle(D, H, has_null, W, cluster_mode):
    if D != 64 and cluster_mode == "clusters":
        pytest.skip("cluster mode is a d_h = 64 kernel")
    dc = _gappy_cache(D, H, W, has_null)
    for q_idx in (40, 31, 10, 1, 0):
        ins, osa, oca = dc.prefill(0, 0, q_idx, tag=q_idx)
        ref_sa, ref_ca = dc.oracle_prefill(0, 0, q_idx, *ins)
        assert_close(out_f64(osa), ref_sa, f"osa q_idx {q_idx}")
        assert_close(out_f64(oca), ref_ca, f"oca q_idx {q_idx} W {W}")
    assert smem.smem_check_device_error(dc.h) == smem.OK


@pytest.mark.parametrize("D,H,W", [(64, 4, 15), (128, 2, 15), (64, 4, 3), (32, 8, 15)])
def test_rope_decode_consecutive_steps_match_oracle(D, H, W):
    """Two sequences (contexts 40 blocks with gaps / 2 blocks) decode three
    consecutive tokens; rows 0..p-1 came from smem_write_inblock."""
    dc = _gappy_cache(D, H, W, True)
    dc.append(1, 0)
    dc.append(1, 5)
    p0 = [20, 61]
    qidx = [40, 9]
    for s in (0, 1):
        dc.write_inblock(s, 0, p0[s], tag=s)
    for step in range(3):
        pos = [p0[0] + step, p0[1] + step]
        ins, osa, oca = dc.decode(0, [0, 1], pos, qidx, step=step)
        for i, s in enumerate((0, 1)):
            ref_sa, ref_ca = dc.oracle_decode(0, s, pos[i], qidx[i], *(x[i] for x in ins))
            assert_close(out_f64(osa[i]), ref_sa, f"osa seq {s} step {step}")
            assert_close(out_f64(oca[i]), ref_ca, f"oca seq {s} step {step}")
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_rope_outputs_are_edit_path_independent(cluster_mode):
    D, H, W = 64, 4, 15
    a = _gappy_cache(D, H, W, True, seed=5)
    b = DeviceCache(L=1, H=H, D=D, max_seqs=2, max_blocks=64, capacity=96, seed=5, has_null=True, rope_window=W,
                    free_order=synth.slot_permutation(99, 96))
    order = [j for j in range(40) if j % 7 != 3][::-1]
    b.append(0, 45, content_seq=9)
    for j in order:
        b.append(0, j)
    b.delete(0, 45)
    b.delete(0, 30)
    b.append(0, 30)
    assert a.mirror.table(0)[1] != b.mirror.table(0)[1]
    for q_idx in (40, 12):
        _, sa_a, ca_a = a.prefill(0, 0, q_idx, tag=1)
        _, sa_b, ca_b = b.prefill(0, 0, q_idx, tag=1)
        assert torch.equal(sa_a, sa_b) and torch.equal(ca_a, ca_b)
    for dc in (a, b):
        dc.write_inblock(0, 0, 9, tag=2)
    _, sa_a, ca_a = a.decode(0, [0], [9], [40], step=4)
    _, sa_b, ca_b = b.decode(0, [0], [9], [40], step=4)
    assert torch.equal(sa_a, sa_b) and torch.equal(ca_a, ca_b)


def test_rope_reader_layer_matches_oracle():
    """The full reader layer with rotary phases: prefill of a block beyond the
    window, then a decode step at offset 33 of the same block."""
    from tests.test_gpu_layer import LayerCache, _np, x_rows
    from oracle.reader_layer import reader_layer_decode, reader_layer_prefill
    H, D, W = 4, 64, 15
    d = H * D
    model = LayerModel(1, d, seed=1401)
    lc = LayerCache(model, H, D, max_seqs=1, max_blocks=32, capacity=32, rope_window=W)
    for j in range(24):
        if j != 20:
            lc.append(0, j)
    q_idx = 24
    x = torch.from_numpy(x_rows(model.seed, 0, q_idx, d)).cuda()
    x_in = _np(x)
    lc.prefill(0, 0, q_idx, x)
    ids, mu = lc.memory(0, q_idx)
    ref, ks, vs = reader_layer_prefill(x_in, ids, mu, q_idx, model.oracle[0], H, D, lc.nu, rope_window=W)
    assert_layer_close(_np(x), ref, x_in, "rope layer prefill")
    p = 33
    xd = torch.from_numpy(x_in[p:p + 1].astype(np.float32)).cuda()
    lc.decode(0, [0], [p], [q_idx], xd)
    ref_d, _, _ = reader_layer_decode(x_in[p], ids, mu, q_idx, p, ks[:p], vs[:p], model.oracle[0], H, D, lc.nu,
                                      rope_window=W)
    assert_layer_close(_np(xd)[0], ref_d, x_in[p], "rope layer decode")
