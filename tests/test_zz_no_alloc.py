"""The decode entry point that allocates nothing (smem_decode_static_scratch).

Some callers may not allocate device memory while serving: a plugin inside a
runtime that owns every device allocation and hands it only inputs and
outputs, or a latency-critical loop where an allocation's device-wide
synchronisation is not allowed. For them the library keeps the decode's
split-K scratch in a fixed array of its own. These tests call that entry
point through the C ABI, twice in a row (the array keeps the previous call's
contents), and check it against the ordinary smem_decode; this file is
collected last so a failure here leaves every other test already run.
"""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import MAX_ABS, MEAN_ABS, DeviceCache, to_dev

pytestmark = pytest.mark.gpu


def _close(a: torch.Tensor, b: torch.Tensor, what: str):
    err = (a.float() - b.float()).abs()
    assert float(err.max()) <= MAX_ABS and float(err.mean()) <= MEAN_ABS, \
        f"{what}: max_abs {float(err.max()):.3e} mean_abs {float(err.mean()):.3e}"


@pytest.mark.parametrize("has_null", [False, True])
def test_static_scratch_matches_decode_twice(has_null):
    nblks = [0, 1, 5, 33, 70, 130, 9, 64]
    S = len(nblks)
    dc = DeviceCache(L=2, H=4, D=64, max_seqs=S, max_blocks=160, capacity=420, seed=11,
                     free_order=synth.slot_permutation(11, 420), has_null=has_null)
    for s, n in enumerate(nblks):
        for j in range(n):
            dc.append(s, j)
    pos = [0, 63, 17, 1, 40, 5, 62, 30]
    for s, p in enumerate(pos):
        dc.write_inblock(s, 1, p)
    seqs, qidx = list(range(S)), list(nblks)
    qs, kn, vn, qc = (to_dev(x) for x in dc.decode_inputs(S, 1, 0))
    shape = (S, dc.H, dc.D)
    ref_sa = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    ref_ca = torch.empty_like(ref_sa)
    smem.smem_decode(dc.h, 1, seqs, pos, qidx, qs, kn, vn, qc, ref_sa, ref_ca)
    for call in range(2):
        osa = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
        oca = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
        smem.smem_decode_static_scratch(dc.h, 1, seqs, pos, qidx, qs, kn, vn, qc, osa, oca)
        torch.cuda.synchronize()
        _close(osa, ref_sa, f"osa, call {call}")
        _close(oca, ref_ca, f"oca, call {call}")
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
