"""Evidence for the reader-layer tolerance of tests/layer_helpers.py (CPU).

The device's reader layer keeps the residual stream in fp32, accumulates in
fp32 and rounds to bf16 at nine places per layer: the three LayerNorm
outputs, q/k/v, the cross-attention query, the memory keys/values stored in
the pool (and the null row's), both attention outputs and the GELU output.
This test models exactly those roundings on the CPU (torch fp32 with a bf16
round trip at each of the nine places, nothing else) on the same seeded
weights and inputs as the GPU layer tests, and measures the error the
roundings alone cause against the fp64 layer oracle. The layer tolerance must
hold that error with a margin for the GPU's different accumulation orders.

The model is first pinned to the oracle: with the nine roundings switched off
it must reproduce the fp64 layer to fp32 accuracy, so it computes the same
layer and differs only where the device rounds.
"""
import functools
import math

import numpy as np
import pytest
import torch

import synth
from oracle.reader_layer import LayerWeights, reader_layer_prefill
from tests.layer_helpers import LAYER_MAX_ABS, LAYER_MEAN_ABS, LAYER_REL_UPDATE, bits_f64, mu_bits, nu_bits, x_rows

MARGIN = 2.5  # factor between the modelled error and the tolerance


def _weights(seed, layer, d):
    hw = synth.reader_layer_weights_np(seed, layer, d)
    kw = {name: bits_f64(hw[name]) for name, _, _ in synth.LAYER_MATRICES}
    for name in synth.LAYER_NORMS:
        for s in ("_g", "_b"):
            kw[name + s] = hw[name + s].astype(np.float64)
    return LayerWeights(**kw)


def _device_rounding_model(x, mu, nu, w, H, D, rounding=True):
    """fp32 reader layer with a bf16 round trip at the device's nine
    rounding places (none when rounding is False)."""
    t = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.float32)
    r = (lambda a: a.to(torch.bfloat16).to(torch.float32)) if rounding else (lambda a: a)
    x = t(x)
    b, d = x.shape

    def ln(v, g, bb):
        m = v.mean(-1, keepdim=True)
        var = ((v - m) ** 2).mean(-1, keepdim=True)
        return r((v - m) / torch.sqrt(var + 1e-5) * t(g) + t(bb))

    def heads(a, n):
        return a.reshape(n, H, D).transpose(0, 1)

    h = ln(x, w.ln1_g, w.ln1_b)
    qkv = r(h @ t(w.w_qkv))
    q, k, v = (heads(qkv[:, i * d:(i + 1) * d], b) for i in range(3))
    s = (q @ k.transpose(1, 2)) / math.sqrt(D)
    s = s.masked_fill(~torch.tril(torch.ones(b, b, dtype=torch.bool)), -float("inf"))
    osa = r((torch.softmax(s, -1) @ v).transpose(0, 1).reshape(b, d))
    x = x + osa @ t(w.w_os)
    qc = heads(r(ln(x, w.ln2_g, w.ln2_b) @ t(w.w_qc)), b)
    rows = t(mu.reshape(-1, d))
    n = rows.shape[0]
    mk, mv = heads(r(rows @ t(w.w_kc)), n), heads(r(rows @ t(w.w_vc)), n)
    if nu is not None:
        kn, vn = r(t(nu) @ t(w.w_kc)).reshape(H, 1, D), r(t(nu) @ t(w.w_vc)).reshape(H, 1, D)
        mk, mv = torch.cat([kn, mk], 1), torch.cat([vn, mv], 1)
    s = (qc @ mk.transpose(1, 2)) / math.sqrt(D)
    oca = r((torch.softmax(s, -1) @ mv).transpose(0, 1).reshape(b, d))
    x = x + oca @ t(w.w_oc)
    f = ln(x, w.ln3_g, w.ln3_b) @ t(w.w_1)
    g = r(0.5 * f * (1 + torch.erf(f / math.sqrt(2.0))))
    return (x + g @ t(w.w_2)).double().numpy()


@functools.lru_cache(maxsize=None)
def _case(H, D, nblk, seed):
    d = H * D
    w = _weights(seed, 0, d)
    x = x_rows(seed, 0, nblk, d).astype(np.float64)
    mu = np.stack([bits_f64(mu_bits(seed, 0, j, d)) for j in range(nblk)]) if nblk else np.zeros((0, 64, d))
    nu = bits_f64(nu_bits(seed, d))
    ref, _, _ = reader_layer_prefill(x, np.arange(nblk), mu, nblk, w, H, D, nu)
    return x, mu, nu, w, ref


def _errors(got, ref, x):
    err = np.abs(got - ref)
    return float(err.max()), float(err.mean()), float(np.linalg.norm(got - ref) / np.linalg.norm(ref - x))


SHAPES = [(4, 64, 8), (16, 64, 32), (2, 128, 8), (8, 128, 16), (8, 32, 16), (12, 64, 64)]


@pytest.mark.parametrize("H,D,nblk", SHAPES)
def test_model_without_rounding_is_the_oracle(H, D, nblk):
    x, mu, nu, w, ref = _case(H, D, nblk, seed=101 + D)
    mx, mean, rel = _errors(_device_rounding_model(x, mu, nu, w, H, D, rounding=False), ref, x)
    assert mx < 2e-4 and rel < 2e-5, (mx, rel)


@pytest.mark.parametrize("H,D,nblk", SHAPES)
def test_layer_tolerance_covers_the_device_roundings(H, D, nblk):
    x, mu, nu, w, ref = _case(H, D, nblk, seed=101 + D)
    mx, mean, rel = _errors(_device_rounding_model(x, mu, nu, w, H, D), ref, x)
    assert MARGIN * mx <= LAYER_MAX_ABS, f"max-abs {mx:.3e}"
    assert MARGIN * mean <= LAYER_MEAN_ABS, f"mean-abs {mean:.3e}"
    assert MARGIN * rel <= LAYER_REL_UPDATE, f"rel-L2 of the update {rel:.3e}"
