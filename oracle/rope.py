"""fp64 oracle of the SMem+RoPE composite ("v2") reader attention.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The composite (arXiv 2609.32395, Sec. 4 "SMem composes with RoPE", App.
"Training recipes", paragraph "SMem+RoPE composite"; App. "Needle" for the
saturating extension) drops the position table and applies rotary phases:

* within-block self-attention: queries and keys rotated by their in-block
  offset t in [0, b);
* cross-attention: the query rotated by its block index i, a memory row's
  key by its block index j, the null row's key by index 0; with the
  saturating extension of window W (the trained range minus one, 15 in the
  paper) every key phase is clamped to max(j, i - W) -- the null row like
  any other row -- while the query phase stays i;
* values are never rotated.

Rotary phases (Su et al., RoFormer, Eq. 34): the feature pairs (2m, 2m+1)
of a d_h-vector turn by the angle phi * theta_m, theta_m = base^(-2m/d_h).

This module rotates every query and key by its absolute phase and then calls
the plain attention of the C oracle -- the definition written out, with no
relative-phase shortcut.

Readings (the paper does not fix them): the interleaved pair convention of
RoFormer; phases in units of blocks for cross-attention and of tokens for
self-attention, both with the same base; window W >= 1, W = None for the
unsaturated reading (phases carried on past the trained range).
"""
from __future__ import annotations

import numpy as np

from . import reader_decode, reader_prefill

BASE = 1e4


def rope(x, phi, base=BASE):
    """Rotate the last axis of x (even length) by phase phi (scalar or array
    broadcasting against x's leading axes)."""
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    theta = base ** (-2.0 * np.arange(D // 2) / D)
    ang = np.asarray(phi, dtype=np.float64)[..., None] * theta
    c, s = np.cos(ang), np.sin(ang)
    xe, xo = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = xe * c - xo * s
    out[..., 1::2] = xe * s + xo * c
    return out


def key_phase(j, i, window):
    """Cross-attention key phase of a row of block j read from query block i."""
    return j if window is None else max(j, i - window)


def reader_prefill_rope(block_idx, blocks_k, blocks_v, q_idx, qs, ks, vs, qc, k_null=None, v_null=None,
                        window=15, base=BASE):
    """One-block reader attention with the composite's rotary phases.
    Shapes as oracle.reader_prefill (qs/ks/vs/qc: [b][H][D]; blocks: [n][H][R][D])."""
    qs, ks, qc = (np.asarray(a, dtype=np.float64) for a in (qs, ks, qc))
    b = qs.shape[0]
    t = np.arange(b, dtype=np.float64)[:, None]          # in-block offset per token (broadcast over heads)
    qs_r = rope(qs, t, base)
    ks_r = rope(ks, t, base)
    qc_r = rope(qc, np.full((b, 1), float(q_idx)), base)
    n = len(block_idx)
    bk = None
    if n:
        bk = np.asarray(blocks_k, dtype=np.float64)
        ph = np.array([key_phase(int(j), int(q_idx), window) for j in block_idx], dtype=np.float64)
        bk = rope(bk, ph[:, None, None], base)               # [n][H][R][D], one phase per block
    kn = None
    if k_null is not None:
        kn = rope(np.asarray(k_null, dtype=np.float64), np.full((k_null.shape[0],), float(key_phase(0, q_idx, window))),
                  base)
    return reader_prefill(block_idx, bk, blocks_v, q_idx, qs_r, ks_r, vs, qc_r, kn, v_null)


def reader_decode_rope(block_idx, blocks_k, blocks_v, q_idx, p, kin, vin, qs, k_new, v_new, qc, k_null=None,
                       v_null=None, window=15, base=BASE):
    """One decode step with the composite's rotary phases (kin/vin: [p][H][D]
    UNROTATED in-block rows of offsets 0..p-1; the new token sits at p)."""
    H = np.asarray(qs).shape[0]
    qs_r = rope(qs, np.full((H,), float(p)), base)
    kn_r = rope(k_new, np.full((H,), float(p)), base)
    kin_r = rope(kin, np.arange(p, dtype=np.float64)[:, None], base) if p > 0 else kin
    qc_r = rope(qc, np.full((H,), float(q_idx)), base)
    n = len(block_idx)
    bk = None
    if n:
        bk = np.asarray(blocks_k, dtype=np.float64)
        ph = np.array([key_phase(int(j), int(q_idx), window) for j in block_idx], dtype=np.float64)
        bk = rope(bk, ph[:, None, None], base)
    knull = None
    if k_null is not None:
        knull = rope(np.asarray(k_null, dtype=np.float64), np.full((H,), float(key_phase(0, q_idx, window))), base)
    return reader_decode(block_idx, bk, blocks_v, q_idx, p, kin_r, vin, qs_r, kn_r, v_new, qc_r, knull, v_null)
