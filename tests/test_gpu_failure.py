"""Failure detection on the GPU without a GPU fault.

* A slot outside the pool in the device table (written through a testing
  hook, the host state untouched) is caught by the kernels' own bounds check:
  the read is skipped, the device error word is set, the host sees
  SMEM_ERR_DEVICE_FAULT; restoring the entry gives the oracle's outputs again.
* A wait that nothing completes gives up after its limit and records the
  error; the context stays usable.
"""
import numpy as np
import pytest

from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import DeviceCache, assert_close, out_f64

pytestmark = pytest.mark.gpu


def _cache():
    dc = DeviceCache(L=1, H=2, D=64, max_seqs=1, max_blocks=16, capacity=12, seed=29)
    for j in range(6):
        dc.append(0, j)
    dc.write_inblock(0, 0, 9)
    return dc


def _decode_matches_oracle(dc):
    ins, osa, oca = dc.decode(0, [0], [9], [6])
    ref_sa, ref_ca = dc.oracle_decode(0, 0, 9, 6, ins[0][0], ins[1][0], ins[2][0], ins[3][0])
    assert_close(out_f64(osa[0]), ref_sa, "osa")
    assert_close(out_f64(oca[0]), ref_ca, "oca")


@pytest.mark.parametrize("bad", [12, 1 << 20, -1])
def test_out_of_range_slot_in_device_table_is_caught(bad):
    dc = _cache()
    _decode_matches_oracle(dc)
    assert smem.smem_check_device_error(dc.h) == smem.OK
    good = smem.smem_get_table(dc.h, 0)[1][2]
    smem.smem_debug_set_table_entry(dc.h, 0, 2, bad)
    dc.decode(0, [0], [9], [6])
    assert smem.smem_check_device_error(dc.h) == smem.ERR_DEVICE_FAULT
    assert smem.smem_check_device_error(dc.h) == smem.OK  # reading the word cleared it
    dc.prefill(0, 0, 6)
    assert smem.smem_check_device_error(dc.h) == smem.ERR_DEVICE_FAULT
    smem.smem_debug_set_table_entry(dc.h, 0, 2, good)
    _decode_matches_oracle(dc)
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_bounded_wait_gives_up_and_context_survives():
    dc = _cache()
    smem.smem_debug_wait_probe(dc.h, 1_000_000)  # 1 ms
    assert smem.smem_check_device_error(dc.h) == smem.ERR_DEVICE_FAULT
    _decode_matches_oracle(dc)
    assert smem.smem_check_device_error(dc.h) == smem.OK


def test_hooks_reject_bad_arguments():
    dc = _cache()
    with pytest.raises(smem.SmemError) as e:
        smem.smem_debug_set_table_entry(dc.h, 0, 6, 0)  # past the table's 6 entries
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:
        smem.smem_debug_wait_probe(dc.h, 0)
    assert e.value.code == smem.ERR_INVALID_ARG
    assert np.array_equal(smem.smem_get_device_table(dc.h, 0, 6), smem.smem_get_table(dc.h, 0)[1])
