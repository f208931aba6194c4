"""The decode step with host inputs and outputs (smem_decode_host): the same
bits as smem_decode on the same cache state, over consecutive steps that
alternate between the two halves of the staging buffer, with the copies on
the compute stream or on a copy stream of their own; argument errors."""
import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, to_dev

pytestmark = pytest.mark.gpu


def _pinned(bits):
    return synth.bits_to_torch_bf16(bits).pin_memory()


@pytest.mark.parametrize("copy_stream", [False, True])
@pytest.mark.parametrize("Hkv", [0, 2])
def test_host_decode_matches_device_decode(copy_stream, Hkv):
    nblks = [3, 0, 17, 40]
    S, H, D = len(nblks), 8, 64
    dev_c = DeviceCache(L=2, H=H, D=D, max_seqs=S, max_blocks=48, capacity=80, seed=23, n_kv_heads=Hkv)
    host_c = DeviceCache(L=2, H=H, D=D, max_seqs=S, max_blocks=48, capacity=80, seed=23, n_kv_heads=Hkv)
    for dc in (dev_c, host_c):
        for s, n in enumerate(nblks):
            for j in range(n):
                dc.append(s, j)
    stage = torch.empty(smem.smem_decode_host_stage_bytes(host_c.h, S), dtype=torch.uint8, device="cuda")
    cs = torch.cuda.Stream() if copy_stream else None
    pos = [5, 0, 63, 20]
    outs = []
    for step in range(3):
        for layer in range(2):
            ins, ref_sa, ref_ca = dev_c.decode(layer, list(range(S)), [(p + step) % 64 for p in pos], nblks, step=step)
            hin = [_pinned(x) for x in ins]
            osa = torch.empty((S, H, D), dtype=torch.bfloat16).pin_memory()
            oca = torch.empty_like(osa).pin_memory()
            smem.smem_decode_host(host_c.h, layer, list(range(S)), [(p + step) % 64 for p in pos], nblks, *hin,
                                  osa, oca, stage, copy_stream=cs)
            outs.append((ref_sa.cpu(), ref_ca.cpu(), osa, oca, hin))
    torch.cuda.synchronize()
    for ref_sa, ref_ca, osa, oca, _ in outs:
        assert torch.equal(ref_sa.view(torch.int16), osa.view(torch.int16))
        assert torch.equal(ref_ca.view(torch.int16), oca.view(torch.int16))
    assert smem.smem_check_device_error(host_c.h) == smem.OK


def test_host_decode_argument_errors():
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=2, max_blocks=4, capacity=4)
    dc.append(0, 0)
    x = torch.zeros((1, 2, 64), dtype=torch.bfloat16).pin_memory()
    need = smem.smem_decode_host_stage_bytes(dc.h, 1)
    assert need > 0 and smem.smem_decode_host_stage_bytes(dc.h, 3) == 0  # above max_decode_batch
    small = torch.empty(need - 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode_host(dc.h, 0, [0], [0], [1], x, x, x, x, x, x, small)
    assert e.value.code == smem.ERR_INVALID_ARG
    big = torch.empty(need + 512, dtype=torch.uint8, device="cuda")
    with pytest.raises(smem.SmemError) as e:
        smem.smem_decode_host(dc.h, 0, [0], [0], [1], x, x, x, x, x, x, big[16:])
    assert e.value.code == smem.ERR_ALIGN
    assert np.array_equal(smem.smem_get_table(dc.h, 0)[1], dc.mirror.table(0)[1])
