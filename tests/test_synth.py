"""The seeded input generator gives the same bf16 bits from numpy and torch,
and the per-head slices agree with whole blocks."""
import numpy as np
import torch

import synth


def test_numpy_and_torch_cpu_agree():
    keys = np.array([synth.stream_key(7, 1, s, b, 0, 0) for s in range(3) for b in range(5)], dtype=np.int64)
    a = synth.normal_bf16_np(keys, 4096)
    b = synth.torch_bf16_to_bits(synth.normal_bf16_torch(torch.tensor(keys), 4096))
    assert np.array_equal(a, b)


def test_block_and_head_slices_agree():
    K, V = synth.block_rows_np(1, 2, 3, 2, 4, 64, 64)
    Kt, Vt = synth.block_rows_torch(1, 2, [3], 2, 4, 64, 64, "cpu")
    assert np.array_equal(K, synth.torch_bf16_to_bits(Kt[0])) and np.array_equal(V, synth.torch_bf16_to_bits(Vt[0]))
    for layer in range(2):
        for h in range(4):
            k, v = synth.block_head_rows_np(1, 2, [3], layer, h, 64, 64)
            assert np.array_equal(k[0], K[layer, h]) and np.array_equal(v[0], V[layer, h])


def test_distribution_is_standard_normal_like():
    x = synth.bits_to_torch_bf16(synth.tensor_np(0, 2, (64, 4096), 1)).float().numpy()
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert 3.5 < np.abs(x).max() < 4.3


def test_layer_weights_numpy_and_torch_agree():
    d = 64
    a = synth.reader_layer_weights_np(11, 2, d)
    b = synth.reader_layer_weights_torch(11, 2, d)
    for name, fi, fo in synth.LAYER_MATRICES:
        assert a[name].shape == (fi * d, fo * d)
        np.testing.assert_array_equal(a[name], synth.torch_bf16_to_bits(b[name]))
    for name in synth.LAYER_NORMS:
        for s in ("_g", "_b"):
            assert a[name + s].dtype == np.float32
            np.testing.assert_array_equal(a[name + s], b[name + s].numpy())
