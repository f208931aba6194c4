"""The decode entry point that allocates nothing (smem_decode_static_scratch).

Some callers may not allocate device memory while serving: a plugin inside a
runtime that owns every device allocation and hands it only inputs and
outputs, or a latency-critical loop where an allocation's device-wide
synchronisation is not allowed. For them the library keeps the decode's
split-K scratch in a fixed array of its own. These tests call that entry
point through the C ABI, twice in a row (the array keeps the previous call's
contents), and require the same bits as the ordinary smem_decode on the same
cache state (same kernel instance and split plan) plus agreement with the
fp64 oracle within the decode tolerance. The cases cover full heads with and
without the null row, grouped key/value heads (grouped decode units), the
RoPE composite, head widths 32 and 128, and a batch above one launch's
item limit (several launches sharing the array). This file is collected last
so a failure here leaves every other test already run.
"""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, assert_close, out_f64, to_dev

pytestmark = pytest.mark.gpu

CASES = {
    "full": dict(H=4, D=64, has_null=False),
    "full_null": dict(H=4, D=64, has_null=True),
    "gqa": dict(H=8, D=64, n_kv_heads=2, has_null=True),
    "gqa_d128": dict(H=8, D=128, n_kv_heads=4),
    "rope": dict(H=4, D=64, rope_window=15, has_null=True),
    "d32": dict(H=8, D=32),
    "d128": dict(H=4, D=128),
}


def _run(dc, layer, seqs, pos, qidx):
    """smem_decode once (the reference), then the static-scratch entry point
    twice on the same inputs; returns the inputs and the three output pairs."""
    inputs, ref_sa, ref_ca = dc.decode(layer, seqs, pos, qidx, step=3)
    dev = [to_dev(x) for x in inputs]
    shape = ref_sa.shape
    outs = []
    for _ in range(2):
        osa = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
        oca = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
        smem.smem_decode_static_scratch(dc.h, layer, seqs, pos, qidx, *dev, osa, oca)
        torch.cuda.synchronize()
        outs.append((osa, oca))
    return inputs, (ref_sa, ref_ca), outs


@pytest.mark.parametrize("case", list(CASES))
def test_static_scratch_bitwise_and_oracle_twice(case):
    kw = CASES[case]
    nblks = [0, 1, 5, 33, 70, 130, 9, 64]
    S = len(nblks)
    dc = DeviceCache(L=2, max_seqs=S, max_blocks=160, capacity=420, seed=11,
                     free_order=synth.slot_permutation(11, 420), **kw)
    for s, n in enumerate(nblks):
        for j in range(n):
            dc.append(s, j)
    pos = [0, 63, 17, 1, 40, 5, 62, 30]
    for s, p in enumerate(pos):
        dc.write_inblock(s, 1, p)
    seqs, qidx = list(range(S)), list(nblks)
    inputs, (ref_sa, ref_ca), outs = _run(dc, 1, seqs, pos, qidx)
    for call, (osa, oca) in enumerate(outs):
        assert torch.equal(osa, ref_sa), f"{case}: osa differs from smem_decode on call {call}"
        assert torch.equal(oca, ref_ca), f"{case}: oca differs from smem_decode on call {call}"
    qs, kn, vn, qc = inputs
    osa, oca = outs[1]
    for i, s in enumerate(seqs):
        sa, ca = dc.oracle_decode(1, s, pos[i], qidx[i], qs[i], kn[i], vn[i], qc[i])
        assert_close(out_f64(osa[i]), sa, f"{case} seq {s} osa")
        if nblks[i] or kw.get("has_null"):
            assert_close(out_f64(oca[i]), ca, f"{case} seq {s} oca")
        else:
            assert float(oca[i].float().abs().max()) == 0.0
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_static_scratch_several_launches():
    """A batch above the 512-item launch limit runs as several launches that
    reuse the one array in stream order."""
    S = 600
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=S, max_blocks=8, capacity=S * 3, seed=5, max_batch=S)
    nblks = [(7 * s) % 4 for s in range(S)]
    for s, n in enumerate(nblks):
        for j in range(n):
            dc.append(s, j)
    pos = [(13 * s) % 64 for s in range(S)]
    for s, p in enumerate(pos):
        dc.write_inblock(s, 0, p)
    seqs, qidx = list(range(S)), [n + 1 for n in nblks]
    inputs, (ref_sa, ref_ca), outs = _run(dc, 0, seqs, pos, qidx)
    for osa, oca in outs:
        assert torch.equal(osa, ref_sa) and torch.equal(oca, ref_ca)
    qs, kn, vn, qc = inputs
    osa, oca = outs[1]
    for i in list(range(0, S, 37)) + [S - 1]:
        sa, ca = dc.oracle_decode(0, i, pos[i], qidx[i], qs[i], kn[i], vn[i], qc[i])
        assert_close(out_f64(osa[i]), sa, f"seq {i} osa")
        if nblks[i]:
            assert_close(out_f64(oca[i]), ca, f"seq {i} oca")
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_static_scratch_rejects_oversized_request():
    """512 single-block items at H=128 need 512*128*(64+4)*4 bytes of
    partials, more than the fixed array: refused before any launch."""
    S, H, D = 512, 128, 64
    dc = DeviceCache(L=1, H=H, D=D, max_seqs=S, max_blocks=2, capacity=S)
    z = torch.zeros((1, H, 64, D), dtype=torch.bfloat16, device="cuda")
    for s in range(S):
        smem.smem_append_block(dc.h, s, 0, z, z)
    x = torch.zeros((S, H, D), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode_static_scratch(dc.h, 0, np.arange(S), np.zeros(S), np.ones(S), x, x, x, x, x, x)
    assert e.value.code == smem.ERR_SCRATCH_LIMIT
    assert smem.smem_check_device_error(dc.h) == smem.OK
