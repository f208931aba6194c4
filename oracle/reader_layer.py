"""fp64 oracle of one full SMem reader layer around the attention path.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The reader layer (arXiv 2609.32395, Sec. 2 "Model", App. A "Reader"): three
sequential pre-LN residual branches -- block-local causal self-attention,
cross-attention into the memory rows of strictly earlier blocks (with the null
row), and an FFN of hidden width 4d with GELU:

    x1 = x  + SA(LN1(x)) W_os          SA queries/keys/values: LN1(x) W_qkv
    x2 = x1 + CA(LN2(x1)) W_oc         CA query: LN2(x1) W_qc
    x3 = x2 + GELU(LN3(x2) W_1) W_2

The memory rows mu_j (d wide, shared by all reader layers) are projected by
each layer's key/value maps: K = mu W_kc, V = mu W_vc; the null row is one
d-vector nu projected the same way (App. A "Positions and memory").

Readings (the paper does not fix them): LayerNorm with biased variance and
eps = 1e-5, affine gain and bias; GELU(x) = x * Phi(x) (the exact form);
no biases in the projections. Matrix products use numpy's matmul (a library
primitive); the attentions are the C oracle's.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

from . import reader_decode, reader_prefill

LN_EPS = 1e-5


def layer_norm(x, g, b, eps=LN_EPS):
    """Per row: (x - mean) / sqrt(biased variance + eps) * g + b."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


_erf = np.vectorize(math.erf, otypes=[np.float64])


def gelu(x):
    """x * Phi(x), Phi the standard normal CDF: 0.5 (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))


@dataclass
class LayerWeights:
    """One reader layer's parameters (fp64 arrays). d = H * d_h.
    w_qkv: [d][3d] columns Q | K | V, each laid out [H][d_h];
    w_os, w_qc, w_oc: [d][d]; w_kc, w_vc: [d][d] (memory key/value maps);
    w_1: [d][4d]; w_2: [4d][d]; ln*_g, ln*_b: [d]."""
    ln1_g: np.ndarray
    ln1_b: np.ndarray
    w_qkv: np.ndarray
    w_os: np.ndarray
    ln2_g: np.ndarray
    ln2_b: np.ndarray
    w_qc: np.ndarray
    w_oc: np.ndarray
    w_kc: np.ndarray
    w_vc: np.ndarray
    ln3_g: np.ndarray
    ln3_b: np.ndarray
    w_1: np.ndarray
    w_2: np.ndarray


def _group(w: LayerWeights, H: int, D: int) -> int:
    """Query heads per key/value head (grouped-query attention: W_kc has
    H_kv * D columns and query head h reads key/value head h // G)."""
    return H // (w.w_kc.shape[1] // D)


def memory_kv(mu, w: LayerWeights, H: int, D: int):
    """Per-layer cross-attention K/V of memory rows mu [..][R][d] ->
    ([..][H][R][D], [..][H][R][D]), key/value heads repeated over their group."""
    G = _group(w, H, D)
    k = mu @ w.w_kc
    v = mu @ w.w_vc
    shp = mu.shape[:-1] + (H // G, D)
    k = np.repeat(np.moveaxis(k.reshape(shp), -2, -3), G, axis=-3)
    v = np.repeat(np.moveaxis(v.reshape(shp), -2, -3), G, axis=-3)
    return k, v


def null_kv(nu, w: LayerWeights, H: int, D: int):
    G = _group(w, H, D)
    return (np.repeat((nu @ w.w_kc).reshape(H // G, D), G, axis=0),
            np.repeat((nu @ w.w_vc).reshape(H // G, D), G, axis=0))


def _attn_prefill(rope_window):
    if rope_window:
        from .rope import reader_prefill_rope
        return lambda *a: reader_prefill_rope(*a, window=rope_window)
    return reader_prefill


def _attn_decode(rope_window):
    if rope_window:
        from .rope import reader_decode_rope
        return lambda *a: reader_decode_rope(*a, window=rope_window)
    return reader_decode


def reader_layer_prefill(x, block_idx, mu_blocks, q_idx, w: LayerWeights, H: int, D: int, nu=None, rope_window=0):
    """One-block pass of one reader layer.
    x: [b][d] residual stream of the query block; block_idx: [n] memory block
    indices (any order); mu_blocks: [n][R][d] their memory rows. rope_window
    W > 0: the SMem+RoPE composite's rotary phases (oracle.rope).
    Returns (x_out [b][d], k_s [b][H_kv][D], v_s [b][H_kv][D]); k_s unrotated."""
    attn = _attn_prefill(rope_window)
    b, d = x.shape
    G = _group(w, H, D)
    kvd = d // G
    h1 = layer_norm(x, w.ln1_g, w.ln1_b)
    qkv = h1 @ w.w_qkv
    qs = qkv[:, :d].reshape(b, H, D)
    ks = qkv[:, d:d + kvd].reshape(b, H // G, D)
    vs = qkv[:, d + kvd:].reshape(b, H // G, D)
    zero = np.zeros((b, H, D))
    osa, _ = attn([], None, None, 0, qs, np.repeat(ks, G, axis=1), np.repeat(vs, G, axis=1), zero)
    x1 = x + osa.reshape(b, d) @ w.w_os
    h2 = layer_norm(x1, w.ln2_g, w.ln2_b)
    qc = (h2 @ w.w_qc).reshape(b, H, D)
    n = len(block_idx)
    mk, mv = memory_kv(np.asarray(mu_blocks), w, H, D) if n else (None, None)
    kn, vn = null_kv(nu, w, H, D) if nu is not None else (None, None)
    _, oca = attn(block_idx, mk, mv, q_idx, zero, zero, zero, qc, kn, vn)
    x2 = x1 + oca.reshape(b, d) @ w.w_oc
    h3 = layer_norm(x2, w.ln3_g, w.ln3_b)
    x3 = x2 + gelu(h3 @ w.w_1) @ w.w_2
    return x3, ks, vs


def reader_layer_decode(x, block_idx, mu_blocks, q_idx, p, kin, vin, w: LayerWeights, H: int, D: int, nu=None,
                        rope_window=0):
    """One decode step of one reader layer for one sequence.
    x: [d]; kin/vin: [p][H_kv][D] in-block rows of earlier tokens (unrotated).
    Returns (x_out [d], k_new [H_kv][D], v_new [H_kv][D])."""
    attn = _attn_decode(rope_window)
    d = x.shape[0]
    G = _group(w, H, D)
    kvd = d // G
    h1 = layer_norm(x[None], w.ln1_g, w.ln1_b)[0]
    qkv = h1 @ w.w_qkv
    qs = qkv[:d].reshape(H, D)
    kn_, vn_ = qkv[d:d + kvd].reshape(H // G, D), qkv[d + kvd:].reshape(H // G, D)
    zero = np.zeros((H, D))
    rep = lambda a, ax: np.repeat(a, G, axis=ax) if a is not None and len(a) else a  # noqa: E731
    osa, _ = attn([], None, None, 0, p, rep(kin, 1), rep(vin, 1), qs, rep(kn_, 0), rep(vn_, 0), zero)
    x1 = x + osa.reshape(d) @ w.w_os
    h2 = layer_norm(x1[None], w.ln2_g, w.ln2_b)[0]
    qc = (h2 @ w.w_qc).reshape(H, D)
    n = len(block_idx)
    mk, mv = memory_kv(np.asarray(mu_blocks), w, H, D) if n else (None, None)
    knull, vnull = null_kv(nu, w, H, D) if nu is not None else (None, None)
    _, oca = attn(block_idx, mk, mv, q_idx, 0, None, None, zero, zero, zero, qc, knull, vnull)
    x2 = x1 + oca.reshape(d) @ w.w_oc
    h3 = layer_norm(x2[None], w.ln3_g, w.ln3_b)[0]
    x3 = x2 + gelu(h3 @ w.w_1) @ w.w_2
    return x3, kn_, vn_
