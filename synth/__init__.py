"""Seeded synthetic inputs for the SMem reader path.

This module holds no arithmetic of the method. It only produces inputs:
memory-block rows, query vectors, in-block K/V rows, free-slot orders and
edit-op streams, all from integer seeds. Both the CPU oracle (via numpy) and
the device path (via torch, on any device) draw from the functions here, and
the two backends give bitwise-identical bf16 bit patterns for the same keys.

Value recipe (stands in for the projected encoder rows and reader queries of
the paper's FineWeb-Edu workloads, which are not available here):

* every element is keyed by a 32-bit stream key and a 0-based element counter;
* three 32-bit hashes (the MurmurHash3 32-bit finaliser, Austin
  Appleby's published ``fmix32``) of ``key + (3*i + j) * 0x9E3779B9`` give six 16-bit
  uniforms; their centred, scaled sum (Irwin--Hall, n = 6) is an approximately
  N(0, 1) float32, range about +-4.24;
* that float32 is rounded to bf16 with round-to-nearest-even.

All arithmetic is on int64 values below 2**50, so numpy and torch (CPU or
CUDA) agree bit for bit; the single float step is one correctly rounded
float32 multiply of an exactly representable integer.
"""
from __future__ import annotations

import numpy as np

M32 = 0xFFFFFFFF
_GOLDEN = 0x9E3779B9
_C1 = 0x85EBCA6B
_C2 = 0xC2B2AE35
_N_UNIF = 6
_MEAN = _N_UNIF * 65535 // 2  # 196605: the sum's mean (6 * 65535 is even)
# std of the sum of 6 discrete uniforms on {0..65535}
_STD = float(np.sqrt(_N_UNIF * (65536.0 ** 2 - 1.0) / 12.0))
_SCALE_F32 = np.float32(1.0 / _STD)

# stream kinds
KIND_K, KIND_V = 0, 1
KIND_QS, KIND_QC, KIND_KS, KIND_VS = 2, 3, 4, 5
KIND_KNULL, KIND_VNULL = 6, 7
KIND_KIN, KIND_VIN = 8, 9
KIND_QDEC_S, KIND_QDEC_C, KIND_KNEW, KIND_VNEW = 10, 11, 12, 13
KIND_MU, KIND_NU, KIND_X = 14, 15, 16
KIND_WEIGHT, KIND_LN = 17, 18


# ---------------------------------------------------------------------------
# scalar key derivation (pure Python ints; identical everywhere)
# ---------------------------------------------------------------------------
def _fmix32_int(h: int) -> int:
    h &= M32
    h ^= h >> 16
    h = (h * _C1) & M32
    h ^= h >> 13
    h = (h * _C2) & M32
    h ^= h >> 16
    return h


def stream_key(seed: int, *fields: int) -> int:
    """32-bit key for one stream, folded from a seed and integer fields."""
    k = _fmix32_int((seed & M32) ^ _fmix32_int((seed >> 32) & M32))
    for f in fields:
        k = _fmix32_int(k ^ _fmix32_int((f + 0x632BE5AB) & M32))
    return k


# ---------------------------------------------------------------------------
# vectorised generator, backend-generic (numpy int64 arrays or torch int64)
# ---------------------------------------------------------------------------
def _mul32(h, c: int):
    """(h * c) mod 2**32 for 0 <= h < 2**32 without exceeding 2**49."""
    lo = h * (c & 0xFFFF)
    hi = ((h * (c >> 16)) & 0xFFFF) << 16
    return (lo + hi) & M32


def _fmix32(h):
    h = h ^ (h >> 16)
    h = _mul32(h, _C1)
    h = h ^ (h >> 13)
    h = _mul32(h, _C2)
    h = h ^ (h >> 16)
    return h


def _unif_sum(keys, ctr):
    """Sum of six 16-bit uniforms for each (key, counter) pair (broadcast)."""
    s = None
    for j in range(3):
        x = _fmix32((keys + _mul32((ctr * 3 + j) & M32, _GOLDEN)) & M32)
        t = (x & 0xFFFF) + (x >> 16)
        s = t if s is None else s + t
    return s


def _round_f32_bits_to_bf16(bits):
    """float32 bit pattern (as int64 in [0, 2**32)) -> bf16 bits, RNE."""
    return ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) & 0xFFFF


def normal_bf16_np(keys: np.ndarray, n: int, start: int = 0) -> np.ndarray:
    """bf16 bit patterns (uint16), shape keys.shape + (n,), element counters
    start .. start+n-1 of each stream."""
    keys = np.asarray(keys, dtype=np.int64)[..., None]
    ctr = np.arange(start, start + n, dtype=np.int64)
    s = _unif_sum(keys, ctr)
    z = (s - _MEAN).astype(np.float32) * _SCALE_F32
    bits = z.view(np.uint32).astype(np.int64)
    return _round_f32_bits_to_bf16(bits).astype(np.uint16)


def normal_bf16_torch(keys, n: int, device=None):
    """Same values as :func:`normal_bf16_np`, as a torch.bfloat16 tensor."""
    import torch

    keys = torch.as_tensor(keys, dtype=torch.int64, device=device)[..., None]
    ctr = torch.arange(n, dtype=torch.int64, device=keys.device)
    s = _unif_sum(keys, ctr)
    scale = torch.tensor(float(_SCALE_F32), dtype=torch.float32, device=keys.device)
    z = (s - _MEAN).to(torch.float32) * scale
    bits = z.view(torch.int32).to(torch.int64) & M32
    r = _round_f32_bits_to_bf16(bits)
    r = r - ((r >> 15) << 16)  # to signed 16-bit range
    return r.to(torch.int16).view(torch.bfloat16)


# ---------------------------------------------------------------------------
# workload-shaped helpers
# ---------------------------------------------------------------------------
def block_keys(seed: int, seq: int, block_idx: int, n_layers: int, kind: int):
    """Per-layer stream keys of one memory block's K (kind 0) or V (kind 1)."""
    return [stream_key(seed, 1, seq, block_idx, layer, kind) for layer in range(n_layers)]


def block_rows_np(seed, seq, block_idx, L, H, R, D):
    """(K, V) uint16 arrays [L][H][R][D] of one memory block."""
    out = []
    for kind in (KIND_K, KIND_V):
        keys = np.array(block_keys(seed, seq, block_idx, L, kind), dtype=np.int64)
        out.append(normal_bf16_np(keys, H * R * D).reshape(L, H, R, D))
    return out[0], out[1]


def block_head_rows_np(seed, seq, block_ids, layer, head, R, D):
    """(K, V) uint16 arrays [n_blocks][R][D]: one head of one layer of many
    blocks (the same values as the matching slice of :func:`block_rows_np`)."""
    out = []
    for kind in (KIND_K, KIND_V):
        keys = np.array([stream_key(seed, 1, seq, b, layer, kind) for b in block_ids], dtype=np.int64)
        out.append(normal_bf16_np(keys, R * D, start=head * R * D).reshape(len(block_ids), R, D))
    return out[0], out[1]


def block_rows_torch(seed, seq, block_ids, L, H, R, D, device, layers=None):
    """(K, V) bf16 tensors [n_blocks][L][H][R][D] for several blocks at once."""
    import torch

    layers = list(range(L)) if layers is None else list(layers)
    res = []
    for kind in (KIND_K, KIND_V):
        keys = [[stream_key(seed, 1, seq, bi, layer, kind) for layer in layers] for bi in block_ids]
        t = normal_bf16_torch(torch.tensor(keys, dtype=torch.int64), H * R * D, device=device)
        res.append(t.reshape(len(block_ids), len(layers), H, R, D))
    return res[0], res[1]


def tensor_np(seed: int, kind: int, shape, *fields: int) -> np.ndarray:
    """A generic seeded bf16 tensor (uint16 bits) of the given shape."""
    n = int(np.prod(shape[-1:])) if len(shape) else 1
    lead = shape[:-1]
    nlead = int(np.prod(lead)) if len(lead) else 1
    keys = np.array([stream_key(seed, 2, kind, *fields, r) for r in range(nlead)], dtype=np.int64)
    return normal_bf16_np(keys, n).reshape(shape)


def tensor_torch(seed: int, kind: int, shape, *fields: int, device=None):
    """Same values as :func:`tensor_np`, as a torch.bfloat16 tensor."""
    import torch

    n = int(shape[-1])
    lead = tuple(shape[:-1])
    nlead = int(np.prod(lead)) if len(lead) else 1
    keys = torch.tensor([stream_key(seed, 2, kind, *fields, r) for r in range(nlead)], dtype=torch.int64)
    return normal_bf16_torch(keys, n, device=device).reshape(tuple(shape))


def bits_to_torch_bf16(bits: np.ndarray):
    """uint16 bf16 bit patterns -> torch.bfloat16 CPU tensor (no rounding)."""
    import torch

    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def torch_bf16_to_bits(t) -> np.ndarray:
    import torch

    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


def slot_permutation(seed: int, capacity: int) -> np.ndarray:
    """A seeded permutation of 0..capacity-1 (initial free-slot order)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.permutation(capacity).astype(np.int32)


def ragged_contexts(seed: int, n_seqs: int, lo: int, hi: int) -> np.ndarray:
    """Per-sequence block counts uniform in [lo, hi]."""
    rng = np.random.Generator(np.random.PCG64(seed ^ 0x5EED))
    return rng.integers(lo, hi + 1, size=n_seqs).astype(np.int32)


def inblock_positions(seed: int, n_seqs: int, b: int) -> np.ndarray:
    """Per-sequence in-block decode offsets uniform in [0, b-1]."""
    rng = np.random.Generator(np.random.PCG64(seed ^ 0xB10C))
    return rng.integers(0, b, size=n_seqs).astype(np.int32)


# ---------------------------------------------------------------------------
# random-init reader-layer weights (the recipe: matrices N(0, 1/fan_in) as
# bf16, LayerNorm gains 1 + 0.1 N(0,1) and biases 0.1 N(0,1) as float32;
# every scaling is one float32 multiply, then round-to-nearest-even)
# ---------------------------------------------------------------------------
# (name, fan_in / d, fan_out / d), stored [fan_in][fan_out] row-major
LAYER_MATRICES = (("w_qkv", 1, 3), ("w_os", 1, 1), ("w_qc", 1, 1), ("w_oc", 1, 1), ("w_kc", 1, 1),
                  ("w_vc", 1, 1), ("w_1", 1, 4), ("w_2", 4, 1))
LAYER_NORMS = ("ln1", "ln2", "ln3")


def _matrix_scale(fan_in: int) -> np.float32:
    return np.float32(1.0 / np.sqrt(fan_in))


def _fan_out(name: str, fo: int, d: int, kvd) -> int:
    """Columns of a matrix; with grouped key/value heads (kvd = their width)
    W_qkv is [d][d + 2 kvd] and W_kc, W_vc are [d][kvd]."""
    if kvd is None:
        return fo * d
    return d + 2 * kvd if name == "w_qkv" else (kvd if name in ("w_kc", "w_vc") else fo * d)


def reader_layer_weights_np(seed: int, layer: int, d: int, kvd=None) -> dict:
    """One layer's weights: matrices as bf16 bits (uint16 [fan_in][fan_out]),
    LayerNorm parameters as float32 [d]."""
    out = {}
    for i, (name, fi, fo) in enumerate(LAYER_MATRICES):
        z = tensor_np(seed, KIND_WEIGHT, (fi * d, _fan_out(name, fo, d, kvd)), layer, i)
        f = (z.astype(np.uint32) << 16).view(np.float32) * _matrix_scale(fi * d)
        out[name] = _round_f32_bits_to_bf16(f.view(np.uint32).astype(np.int64)).astype(np.uint16)
    for i, name in enumerate(LAYER_NORMS):
        z = tensor_np(seed, KIND_LN, (2, d), layer, i)
        zf = (z.astype(np.uint32) << 16).view(np.float32)
        out[name + "_g"] = np.float32(1.0) + np.float32(0.1) * zf[0]
        out[name + "_b"] = np.float32(0.1) * zf[1]
    return out


def reader_layer_weights_torch(seed: int, layer: int, d: int, device=None, kvd=None) -> dict:
    """Same values as :func:`reader_layer_weights_np`, as torch tensors
    (bfloat16 matrices, float32 LayerNorm parameters) on `device`."""
    import torch

    out = {}
    for i, (name, fi, fo) in enumerate(LAYER_MATRICES):
        z = tensor_torch(seed, KIND_WEIGHT, (fi * d, _fan_out(name, fo, d, kvd)), layer, i, device=device)
        f = z.to(torch.float32) * torch.tensor(float(_matrix_scale(fi * d)), dtype=torch.float32, device=z.device)
        bits = f.view(torch.int32).to(torch.int64) & M32
        r = _round_f32_bits_to_bf16(bits)
        r = r - ((r >> 15) << 16)
        out[name] = r.to(torch.int16).view(torch.bfloat16)
    for i, name in enumerate(LAYER_NORMS):
        zf = tensor_torch(seed, KIND_LN, (2, d), layer, i, device=device).to(torch.float32)
        one = torch.tensor(1.0, dtype=torch.float32, device=zf.device)
        tenth = torch.tensor(float(np.float32(0.1)), dtype=torch.float32, device=zf.device)
        out[name + "_g"] = (one + tenth * zf[0]).contiguous()
        out[name + "_b"] = (tenth * zf[1]).contiguous()
    return out
