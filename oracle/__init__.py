"""fp64 CPU oracle of the SMem reader's attention, and an independent mirror
of the cache bookkeeping.

TEST INFRASTRUCTURE ONLY: only tests/, ``__graft_entry__.smoke()`` and the
cpu-baseline / reference legs of ``bench.py`` may import this package. It
shares no code with the CUDA path and never imports it.

* :func:`reader_prefill` and :func:`reader_decode` wrap the C oracle in
  ``smem_oracle.c`` (plain definitions of block-local causal self-attention
  and block-causal cross-attention over the canonical memory, arXiv
  2609.32395 Sec. 2 "Model", App. A "Reader", Sec. 3.1).
* :mod:`oracle.bookkeeping` mirrors the block table and free-slot FIFO.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

_lib = None
_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int32)


def _load():
    global _lib
    if _lib is None:
        path = _build.build()
        lib = ctypes.CDLL(path)
        lib.oracle_rowset.argtypes = [ctypes.c_int, _ip, ctypes.c_int32, _ip]
        lib.oracle_rowset.restype = ctypes.c_int
        lib.oracle_reader_prefill.argtypes = [ctypes.c_int] * 5 + [_ip, _dp, _dp, ctypes.c_int, _dp, _dp,
                                                                    ctypes.c_int32] + [_dp] * 6
        lib.oracle_reader_prefill.restype = ctypes.c_int
        lib.oracle_reader_decode.argtypes = [ctypes.c_int] * 4 + [_ip, _dp, _dp, ctypes.c_int, _dp, _dp,
                                                                   ctypes.c_int32, ctypes.c_int] + [_dp] * 8
        lib.oracle_reader_decode.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        lib.oracle_set_threads.restype = ctypes.c_int
        _lib = lib
    return _lib


def set_threads(n: int) -> int:
    """Threads the oracle's per-head loops use (OpenMP); 0 keeps the current
    setting. Returns the count in effect (1 when built without OpenMP)."""
    return int(_load().oracle_set_threads(int(n)))


def bf16_bits_to_f64(bits) -> np.ndarray:
    """bf16 bit patterns (uint16) -> exact fp64 values."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    if a is None:
        return None
    if a.dtype == np.float64:
        return a.ctypes.data_as(_dp)
    return a.ctypes.data_as(_ip)


class OracleError(RuntimeError):
    pass


def rowset(block_idx, q_idx: int) -> np.ndarray:
    """Positions (into ``block_idx``) of the blocks a query block ``q_idx``
    cross-attends to, in canonical (ascending block index) order."""
    lib = _load()
    bi = np.ascontiguousarray(block_idx, dtype=np.int32)
    out = np.zeros(max(len(bi), 1), dtype=np.int32)
    n = lib.oracle_rowset(len(bi), _ptr(bi), int(q_idx), _ptr(out))
    if n < 0:
        raise OracleError(f"oracle_rowset failed ({n})")
    return out[:n].copy()


def reader_prefill(block_idx, blocks_k, blocks_v, q_idx, qs, ks, vs, qc, k_null=None, v_null=None):
    """One-block reader attention for one layer.

    block_idx: [n]; blocks_k/v: [n][H][R][D] (any block order);
    qs/ks/vs/qc: [b][H][D]; k_null/v_null: [H][D] or None.
    Returns (osa, oca), each [b][H][D] fp64.
    """
    lib = _load()
    bi = np.ascontiguousarray(block_idx, dtype=np.int32).reshape(-1)
    qs, ks, vs, qc = (_f64(x) for x in (qs, ks, vs, qc))
    b, H, D = qs.shape
    n = len(bi)
    if n:
        bk, bv = _f64(blocks_k), _f64(blocks_v)
        R = bk.shape[2]
    else:
        R = 64
        bk = bv = np.zeros(1, dtype=np.float64)
    has_null = k_null is not None
    kn = _f64(k_null) if has_null else np.zeros(1)
    vn = _f64(v_null) if has_null else np.zeros(1)
    osa = np.zeros((b, H, D))
    oca = np.zeros((b, H, D))
    rc = lib.oracle_reader_prefill(H, D, b, R, n, _ptr(bi) if n else None, _ptr(bk), _ptr(bv), int(has_null),
                                   _ptr(kn), _ptr(vn), int(q_idx), _ptr(qs), _ptr(ks), _ptr(vs), _ptr(qc),
                                   _ptr(osa), _ptr(oca))
    if rc:
        raise OracleError(f"oracle_reader_prefill failed ({rc})")
    return osa, oca


def reader_decode(block_idx, blocks_k, blocks_v, q_idx, p, kin, vin, qs, k_new, v_new, qc,
                  k_null=None, v_null=None):
    """One decode step of one sequence for one layer.

    kin/vin: [p][H][D] earlier in-block rows; qs/k_new/v_new/qc: [H][D].
    Returns (osa, oca), each [H][D] fp64.
    """
    lib = _load()
    bi = np.ascontiguousarray(block_idx, dtype=np.int32).reshape(-1)
    qs, k_new, v_new, qc = (_f64(x) for x in (qs, k_new, v_new, qc))
    H, D = qs.shape
    n = len(bi)
    if n:
        bk, bv = _f64(blocks_k), _f64(blocks_v)
        R = bk.shape[2]
    else:
        R = 64
        bk = bv = np.zeros(1, dtype=np.float64)
    kin = _f64(kin).reshape(-1) if p > 0 else np.zeros(1)
    vin = _f64(vin).reshape(-1) if p > 0 else np.zeros(1)
    has_null = k_null is not None
    kn = _f64(k_null) if has_null else np.zeros(1)
    vn = _f64(v_null) if has_null else np.zeros(1)
    osa = np.zeros((H, D))
    oca = np.zeros((H, D))
    rc = lib.oracle_reader_decode(H, D, R, n, _ptr(bi) if n else None, _ptr(bk), _ptr(bv), int(has_null),
                                  _ptr(kn), _ptr(vn), int(q_idx), int(p), _ptr(kin), _ptr(vin), _ptr(qs),
                                  _ptr(k_new), _ptr(v_new), _ptr(qc), _ptr(osa), _ptr(oca))
    if rc:
        raise OracleError(f"oracle_reader_decode failed ({rc})")
    return osa, oca
