"""GPU checks of the reader layer's projection kernel (tcgen05, through the
C ABI's testing hook) against a plain fp64 product of the same bf16 inputs:
every epilogue (bf16 store, fp32 residual add, GELU), the LayerNorm kernel,
head-scattered outputs (the pool slot layout), batched maps
with column offsets in either weight orientation (the recompute-K/V per-head
maps), one and several row tiles, split-K clusters of every size the plan
picks, and bitwise repeatability."""
import math

import numpy as np
import pytest
import torch

import synth
from paper_2609_32395_gb300 import smem

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cache():
    cfg = smem.make_config(1, 2, 64, 1, 2, 2)
    c = smem.SmemCache(cfg, device="cuda")
    yield c
    c.close()


def _bf16(seed, shape, scale=1.0, *fields):
    bits = synth.tensor_np(seed, synth.KIND_WEIGHT, shape, *fields)
    t = synth.bits_to_torch_bf16(bits).float() * scale
    return t.to(torch.bfloat16)


def _f64(t):
    return t.detach().to("cpu").to(torch.float64)


def _gelu(x):
    return 0.5 * x * (1.0 + torch.erf(x / math.sqrt(2.0)))


def _check(got, ref, what, rel=2 ** -7):
    """bf16-rounded outputs: within a few bf16 units of the reference scale."""
    got, ref = _f64(got), _f64(ref)
    scale = float(ref.abs().max()) + 1e-30
    err = float((got - ref).abs().max())
    assert err <= rel * scale, f"{what}: max err {err:.3e} vs scale {scale:.3e}"


@pytest.mark.parametrize("M,N,K", [(64, 3072, 1024), (64, 2304, 768), (1, 1024, 1024), (200, 512, 256),
                                   (64, 64, 4096), (64, 32, 32), (128, 96, 160)])
def test_plain_bf16_store(cache, M, N, K):
    A = _bf16(1, (M, K), 1.0, M, K).cuda()
    W = _bf16(2, (K, N), 1.0 / math.sqrt(K), N, K).cuda()
    out = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_gemm(cache.h, A, K, W, 0, M, N, K, out, N)
    torch.cuda.synchronize()
    _check(out, _f64(A) @ _f64(W), f"{M}x{N}x{K}")
    again = torch.empty_like(out)
    smem.smem_debug_gemm(cache.h, A, K, W, 0, M, N, K, again, N)
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), again.view(torch.int16))


@pytest.mark.parametrize("M,N,K", [(64, 1024, 4096), (64, 768, 768), (3, 1024, 1024)])
def test_residual_add(cache, M, N, K):
    A = _bf16(3, (M, K), 1.0, M).cuda()
    W = _bf16(4, (K, N), 1.0 / math.sqrt(K), N).cuda()
    x0 = _bf16(5, (M, N), 1.0, M).float().cuda()
    x = x0.clone()
    smem.smem_debug_gemm(cache.h, A, K, W, 0, M, N, K, x, N, epi=1)
    torch.cuda.synchronize()
    ref = _f64(x0) + _f64(A) @ _f64(W)
    err = float((_f64(x) - ref).abs().max())
    assert err <= 1e-4 * float(ref.abs().max()), err


def test_gelu(cache):
    M, N, K = 64, 4096, 1024
    A = _bf16(6, (M, K), 1.0, M).cuda()
    W = _bf16(7, (K, N), 1.0 / math.sqrt(K), N).cuda()
    out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_gemm(cache.h, A, K, W, 0, M, N, K, out, N, epi=2)
    torch.cuda.synchronize()
    _check(out, _gelu(_f64(A) @ _f64(W)), "gelu")


@pytest.mark.parametrize("n,d", [(64, 1024), (64, 768), (5, 2048), (130, 256)])
def test_layernorm(cache, n, d):
    """h = LayerNorm(x) * g + b per row (fp32 statistics, bf16 output)."""
    x = (_bf16(8, (n, d), 1.0, n).float() * 3.0 + 0.5).cuda()
    g = (1.0 + 0.1 * _bf16(9, (d,), 1.0).float()).cuda()
    b = (0.1 * _bf16(10, (d,), 1.0).float()).cuda()
    h = torch.empty((n, d), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_layernorm(cache.h, x, g, b, h)
    torch.cuda.synchronize()
    xd = _f64(x)
    mu = xd.mean(1, keepdim=True)
    var = ((xd - mu) ** 2).mean(1, keepdim=True)
    ref = (xd - mu) / torch.sqrt(var + 1e-5) * _f64(g) + _f64(b)
    err = float((_f64(h) - ref).abs().max())
    assert err <= 2 ** -8 * float(ref.abs().max()), err  # one bf16 rounding of values below the maximum


def test_head_scatter_into_slot_layout(cache):
    """Memory-row projection: head h of mu W goes to out + h * 2 * R * D."""
    R, d, Hkv, D = 64, 512, 8, 64
    mu = _bf16(12, (R, d), 1.0).cuda()
    W = _bf16(13, (d, Hkv * D), 1.0 / math.sqrt(d)).cuda()
    slot = torch.zeros((Hkv, 2, R, D), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_gemm(cache.h, mu, d, W, 0, R, Hkv * D, d, slot, D, col_group=D, group_stride=2 * R * D)
    torch.cuda.synchronize()
    ref = (_f64(mu) @ _f64(W)).reshape(R, Hkv, D).permute(1, 0, 2)
    _check(slot[:, 0], ref, "head scatter")
    assert float(slot[:, 1].float().abs().max()) == 0.0  # the V halves are untouched


@pytest.mark.parametrize("D", [32, 64, 128])
def test_batched_head_maps(cache, D):
    """The recompute-K/V maps: per head h, q'_h = alpha * q_h W_kc[:, hD:(h+1)D]^T
    (weights K-major, K = D) and att_h = O'_h W_vc[:, hD:(h+1)D] (N = D)."""
    H, nq = 8, 64
    d = H * D
    alpha = 0.18
    qc = _bf16(14, (nq, d), 1.0).cuda()
    wkc = _bf16(15, (d, d), 1.0 / math.sqrt(d)).cuda()
    qp = torch.empty((H, nq, d), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_gemm(cache.h, qc, d, wkc, 1, nq, d, D, qp, d, a_bs=D, w_boff=D, batch=H, alpha=alpha,
                         o_bs=nq * d)
    op = _bf16(16, (H, nq, d), 1.0).cuda()
    wvc = _bf16(17, (d, d), 1.0 / math.sqrt(d)).cuda()
    att = torch.empty((nq, d), dtype=torch.bfloat16, device="cuda")
    smem.smem_debug_gemm(cache.h, op, d, wvc, 0, nq, D, d, att, d, a_bs=nq * d, w_boff=D, batch=H, o_bs=D)
    torch.cuda.synchronize()
    q64, wk64, o64, wv64 = _f64(qc), _f64(wkc), _f64(op), _f64(wvc)
    for h in range(H):
        ref_q = alpha * q64[:, h * D:(h + 1) * D] @ wk64[:, h * D:(h + 1) * D].T
        _check(qp[h], ref_q, f"q' map head {h}")
        ref_a = o64[h] @ wv64[:, h * D:(h + 1) * D]
        _check(att[:, h * D:(h + 1) * D], ref_a, f"value map head {h}")


def test_argument_errors(cache):
    A = torch.zeros((64, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(smem.SmemError) as e:
        smem.smem_debug_gemm(cache.h, A, 64, A, 0, 64, 48, 64, A, 64)  # N not a multiple of 32
    assert e.value.code == smem.ERR_INVALID_ARG
    with pytest.raises(smem.SmemError) as e:
        smem.smem_debug_gemm(cache.h, A[:, 1:], 64, A, 0, 64, 64, 32, A, 64)  # misaligned A
    assert e.value.code in (smem.ERR_ALIGN, smem.ERR_INVALID_ARG)
    assert smem.smem_check_device_error(cache.h) == smem.OK
