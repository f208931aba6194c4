"""Python binding of the C ABI in include/smem.h (argument marshalling only).

Every function keeps the C name and forwards to ``libsmem.so``; all work of
the reader path runs in the library's CUDA kernels. Device buffers are torch
tensors (bf16, contiguous, on the cache's device); the stream is torch's
current CUDA stream unless one is given. A negative return code raises
:class:`SmemError`. There is no CPU fallback: if the library is missing or
fails to load, :func:`lib` raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import _build

OK = 0
ERR_INVALID_ARG = -1
ERR_ALIGN = -2
ERR_NO_SUCH_SEQ = -3
ERR_DUPLICATE_BLOCK = -4
ERR_NO_SUCH_BLOCK = -5
ERR_POOL_FULL = -6
ERR_TABLE_FULL = -7
ERR_CUDA = -8
ERR_DEVICE_FAULT = -9
ERR_UNSUPPORTED = -10
ERR_NO_DEVICE = -11
ERR_SCRATCH_LIMIT = -12
STATIC_SCRATCH_BYTES = 16 << 20

EXPORTED = [
    "smem_cache_required_bytes", "smem_cache_create", "smem_cache_destroy", "smem_set_null_row",
    "smem_append_block", "smem_delete_block", "smem_release_seq", "smem_write_inblock", "smem_prefill_block",
    "smem_decode", "smem_decode_static_scratch", "smem_decode_host", "smem_decode_host_stage_bytes", "smem_get_table", "smem_get_free_fifo", "smem_get_device_table",
    "smem_check_device_error", "smem_debug_gemm", "smem_debug_layernorm", "smem_debug_set_table_entry",
    "smem_debug_wait_probe",
    "smem_free_slots", "smem_last_error_detail", "smem_debug_fail_after", "smem_strerror", "smem_abi_version",
    "smem_layer_workspace_bytes", "smem_append_block_rows", "smem_set_null_vector", "smem_reader_layer_prefill",
    "smem_reader_layer_decode", "smem_mu_decode", "smem_mu_prefill", "smem_share_block", "smem_slot_refs",
    "smem_mu_decode_plan",
]


class SmemError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        detail = ""
        if code in (ERR_CUDA, ERR_DEVICE_FAULT):
            detail = " (" + lib().smem_last_error_detail().decode() + ")"
        super().__init__(f"{where}: {lib().smem_strerror(code).decode()} [{code}]{detail}")


class SmemConfig(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("block_tokens", ctypes.c_int32), ("rows_per_block", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
        ("max_blocks_per_seq", ctypes.c_int32), ("capacity_slots", ctypes.c_int32),
        ("has_null_row", ctypes.c_int32), ("max_decode_batch", ctypes.c_int32),
        ("free_order", ctypes.POINTER(ctypes.c_int32)), ("recompute_kv", ctypes.c_int32),
        ("rope_window", ctypes.c_int32), ("rope_base", ctypes.c_float), ("n_kv_heads", ctypes.c_int32),
    ]


class SmemLayerWeights(ctypes.Structure):
    """struct smem_layer_weights: device pointers of one reader layer."""
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "ln1_g", "ln1_b", "w_qkv", "w_os", "ln2_g", "ln2_b", "w_qc", "w_oc", "w_kc", "w_vc", "ln3_g", "ln3_b",
        "w_1", "w_2")]


LAYER_FIELDS = [f for f, _ in SmemLayerWeights._fields_]


_lib = None
_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_i32p = ctypes.POINTER(ctypes.c_int32)
_wp = ctypes.POINTER(SmemLayerWeights)


def lib():
    """The loaded libsmem.so (built in-tree on first use)."""
    global _lib
    if _lib is None:
        import torch  # noqa: F401  (load PyTorch's CUDA runtime first, so both share it)

        path = _build.build()
        L = ctypes.CDLL(path, mode=ctypes.RTLD_GLOBAL)
        cfgp = ctypes.POINTER(SmemConfig)
        sig = {
            "smem_cache_required_bytes": (ctypes.c_size_t, [cfgp]),
            "smem_cache_create": (ctypes.c_int, [cfgp, _vp, ctypes.c_size_t, ctypes.POINTER(_vp)]),
            "smem_cache_destroy": (ctypes.c_int, [_vp]),
            "smem_set_null_row": (ctypes.c_int, [_vp, _vp, _vp, _vp]),
            "smem_append_block": (ctypes.c_int, [_vp, _i32, _i32, _vp, _vp, _vp, _i32p]),
            "smem_delete_block": (ctypes.c_int, [_vp, _i32, _i32, _vp]),
            "smem_release_seq": (ctypes.c_int, [_vp, _i32, _vp]),
            "smem_write_inblock": (ctypes.c_int, [_vp, _i32, _i32, _i32, _vp, _vp, _vp]),
            "smem_prefill_block": (ctypes.c_int, [_vp, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
            "smem_decode": (ctypes.c_int, [_vp, _i32, _i32, _i32p, _i32p, _i32p, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
            "smem_decode_static_scratch": (ctypes.c_int, [_vp, _i32, _i32, _i32p, _i32p, _i32p, _vp, _vp, _vp, _vp,
                                                          _vp, _vp, _vp]),
            "smem_get_table": (ctypes.c_int, [_vp, _i32, _i32p, _i32p, _i32, _i32p]),
            "smem_get_free_fifo": (ctypes.c_int, [_vp, _i32p, _i32, _i32p]),
            "smem_get_device_table": (ctypes.c_int, [_vp, _i32, _i32p, _i32, _i32p, _vp]),
            "smem_check_device_error": (ctypes.c_int, [_vp, _vp]),
            "smem_free_slots": (ctypes.c_int, [_vp, _i32p]),
            "smem_last_error_detail": (ctypes.c_char_p, []),
            "smem_debug_fail_after": (ctypes.c_int, [_vp, _i32]),
            "smem_strerror": (ctypes.c_char_p, [ctypes.c_int]),
            "smem_abi_version": (ctypes.c_int, []),
            "smem_layer_workspace_bytes": (ctypes.c_size_t, [_vp, _i32]),
            "smem_append_block_rows": (ctypes.c_int, [_vp, _i32, _i32, _vp, _wp, _vp, ctypes.c_size_t, _vp, _i32p]),
            "smem_set_null_vector": (ctypes.c_int, [_vp, _vp, _wp, _vp, ctypes.c_size_t, _vp]),
            "smem_reader_layer_prefill": (ctypes.c_int, [_vp, _i32, _i32, _i32, _wp, _vp, _vp, ctypes.c_size_t,
                                                         _vp]),
            "smem_reader_layer_decode": (ctypes.c_int, [_vp, _i32, _i32, _i32p, _i32p, _i32p, _wp, _vp, _vp,
                                                        ctypes.c_size_t, _vp]),
            "smem_mu_decode": (ctypes.c_int, [_vp, _i32, _i32p, _i32p, _vp, _vp, _vp, ctypes.c_size_t, _vp]),
            "smem_mu_prefill": (ctypes.c_int, [_vp, _i32, _i32, _vp, _vp, _vp, ctypes.c_size_t, _vp]),
            "smem_share_block": (ctypes.c_int, [_vp, _i32, _i32, _i32, _i32, _vp, _i32p]),
            "smem_slot_refs": (ctypes.c_int, [_vp, _i32, _i32p]),
            "smem_mu_decode_plan": (ctypes.c_int, [_vp, _i32p, _i32p, _i32p]),
            "smem_decode_host_stage_bytes": (ctypes.c_size_t, [_vp, _i32]),
            "smem_decode_host": (ctypes.c_int, [_vp, _i32, _i32, _i32p, _i32p, _i32p, _vp, _vp, _vp, _vp, _vp, _vp,
                                                _vp, ctypes.c_size_t, _vp, _vp]),
            "smem_debug_set_table_entry": (ctypes.c_int, [_vp, _i32, _i32, _i32, _vp]),
            "smem_debug_wait_probe": (ctypes.c_int, [_vp, ctypes.c_longlong, _vp]),
            "smem_debug_gemm": (ctypes.c_int, [_vp, _vp, _i32, ctypes.c_longlong, _vp, _i32, _i32, _i32, _i32, _i32,
                                               _i32, _i32, _i32, _i32, ctypes.c_float, _vp, _i32, ctypes.c_longlong,
                                               _i32, ctypes.c_longlong, _vp]),
            "smem_debug_layernorm": (ctypes.c_int, [_vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(rc: int, where: str) -> int:
    if rc != OK:
        raise SmemError(rc, where)
    return rc


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch

        if not torch.cuda.is_available():
            return None
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _i32arr(a):
    arr = np.ascontiguousarray(a, dtype=np.int32)
    return arr, arr.ctypes.data_as(_i32p)


def make_config(n_layers, n_heads, head_dim, max_seqs, max_blocks_per_seq, capacity_slots, has_null_row=False,
                max_decode_batch=None, free_order=None, block_tokens=64, rows_per_block=64,
                recompute_kv=False, rope_window=0, rope_base=1e4, n_kv_heads=0) -> SmemConfig:
    cfg = SmemConfig(n_layers, n_heads, head_dim, block_tokens, rows_per_block, max_seqs, max_blocks_per_seq,
                     capacity_slots, int(bool(has_null_row)),
                     max_seqs if max_decode_batch is None else max_decode_batch, None, int(bool(recompute_kv)),
                     int(rope_window), float(rope_base), int(n_kv_heads))
    if free_order is not None:
        arr, p = _i32arr(free_order)
        cfg._free_order_keep = arr
        cfg.free_order = p
    return cfg


def smem_cache_required_bytes(cfg: SmemConfig) -> int:
    return int(lib().smem_cache_required_bytes(ctypes.byref(cfg)))


def smem_cache_create(cfg: SmemConfig, dev_buf=None):
    """dev_buf: a torch uint8 CUDA tensor of >= required bytes, or None for a
    bookkeeping-only cache. Returns the opaque handle (c_void_p)."""
    h = ctypes.c_void_p()
    nbytes = 0 if dev_buf is None else dev_buf.numel() * dev_buf.element_size()
    _check(lib().smem_cache_create(ctypes.byref(cfg), _ptr(dev_buf), nbytes, ctypes.byref(h)), "smem_cache_create")
    return h


def smem_cache_destroy(h):
    return _check(lib().smem_cache_destroy(h), "smem_cache_destroy")


def smem_set_null_row(h, k_null, v_null, stream=None):
    return _check(lib().smem_set_null_row(h, _ptr(k_null), _ptr(v_null), _stream(stream)), "smem_set_null_row")


def smem_append_block(h, seq, block_idx, K=None, V=None, stream=None) -> int:
    slot = ctypes.c_int32(-1)
    st = _stream(stream) if K is not None else None
    _check(lib().smem_append_block(h, seq, block_idx, _ptr(K), _ptr(V), st, ctypes.byref(slot)), "smem_append_block")
    return slot.value


def smem_share_block(h, src_seq, src_idx, dst_seq, dst_idx, stream=None, device=True) -> int:
    """dst_seq's table gains (dst_idx -> the slot of src_seq's src_idx); returns the slot."""
    slot = ctypes.c_int32(-1)
    st = _stream(stream) if device else None
    _check(lib().smem_share_block(h, src_seq, src_idx, dst_seq, dst_idx, st, ctypes.byref(slot)), "smem_share_block")
    return slot.value


def smem_slot_refs(h, slot) -> int:
    n = ctypes.c_int32(0)
    _check(lib().smem_slot_refs(h, slot, ctypes.byref(n)), "smem_slot_refs")
    return n.value


def smem_mu_decode_plan(h):
    """(nq, cluster, slice_cols) of a recompute cache's decode kernel; cluster 0: two-pass form."""
    v = [ctypes.c_int32(0) for _ in range(3)]
    _check(lib().smem_mu_decode_plan(h, *[ctypes.byref(x) for x in v]), "smem_mu_decode_plan")
    return tuple(x.value for x in v)


def smem_delete_block(h, seq, block_idx, stream=None, device=True):
    st = _stream(stream) if device else None
    return _check(lib().smem_delete_block(h, seq, block_idx, st), "smem_delete_block")


def smem_release_seq(h, seq, stream=None):
    return _check(lib().smem_release_seq(h, seq, None), "smem_release_seq")


def smem_write_inblock(h, seq, layer, n_rows, K, V, stream=None):
    return _check(lib().smem_write_inblock(h, seq, layer, n_rows, _ptr(K), _ptr(V), _stream(stream)),
                  "smem_write_inblock")


def smem_prefill_block(h, seq, layer, q_block_idx, Qs, Ks, Vs, Qc, Osa, Oca, stream=None):
    return _check(lib().smem_prefill_block(h, seq, layer, q_block_idx, _ptr(Qs), _ptr(Ks), _ptr(Vs), _ptr(Qc),
                                           _ptr(Osa), _ptr(Oca), _stream(stream)), "smem_prefill_block")


def smem_decode(h, layer, seq_ids, pos, q_block_idx, qs, k_new, v_new, qc, osa, oca, stream=None):
    s, sp = _i32arr(seq_ids)
    p, pp = _i32arr(pos)
    q, qp = _i32arr(q_block_idx)
    return _check(lib().smem_decode(h, layer, len(s), sp, pp, qp, _ptr(qs), _ptr(k_new), _ptr(v_new), _ptr(qc),
                                    _ptr(osa), _ptr(oca), _stream(stream)), "smem_decode")


def smem_decode_static_scratch(h, layer, seq_ids, pos, q_block_idx, qs, k_new, v_new, qc, osa, oca, stream=None):
    """smem_decode with the library's fixed scratch array (allocates nothing)."""
    s, sp = _i32arr(seq_ids)
    p, pp = _i32arr(pos)
    q, qp = _i32arr(q_block_idx)
    return _check(lib().smem_decode_static_scratch(h, layer, len(s), sp, pp, qp, _ptr(qs), _ptr(k_new), _ptr(v_new),
                                                   _ptr(qc), _ptr(osa), _ptr(oca), _stream(stream)),
                  "smem_decode_static_scratch")


def smem_decode_host_stage_bytes(h, nb) -> int:
    return int(lib().smem_decode_host_stage_bytes(h, nb))


def smem_decode_host(h, layer, seq_ids, pos, q_block_idx, qs, k_new, v_new, qc, osa, oca, stage, stream=None,
                     copy_stream=None):
    """smem_decode with host (pinned) input/output tensors and a device
    staging buffer; asynchronous (see include/smem.h)."""
    s, sp = _i32arr(seq_ids)
    p_, pp = _i32arr(pos)
    q, qp = _i32arr(q_block_idx)
    cs = None if copy_stream is None else _stream(copy_stream)
    return _check(lib().smem_decode_host(h, layer, len(s), sp, pp, qp, _ptr(qs), _ptr(k_new), _ptr(v_new), _ptr(qc),
                                         _ptr(osa), _ptr(oca), _ptr(stage), stage.numel() * stage.element_size(),
                                         _stream(stream), cs), "smem_decode_host")


def smem_get_table(h, seq):
    n = ctypes.c_int32(0)
    _check(lib().smem_get_table(h, seq, None, None, 0, ctypes.byref(n)), "smem_get_table")
    idx = np.zeros(max(n.value, 1), dtype=np.int32)
    slot = np.zeros(max(n.value, 1), dtype=np.int32)
    _check(lib().smem_get_table(h, seq, idx.ctypes.data_as(_i32p), slot.ctypes.data_as(_i32p), n.value,
                                ctypes.byref(n)), "smem_get_table")
    return idx[: n.value].tolist(), slot[: n.value].tolist()


def smem_get_free_fifo(h):
    n = ctypes.c_int32(0)
    _check(lib().smem_get_free_fifo(h, None, 0, ctypes.byref(n)), "smem_get_free_fifo")
    out = np.zeros(max(n.value, 1), dtype=np.int32)
    _check(lib().smem_get_free_fifo(h, out.ctypes.data_as(_i32p), n.value, ctypes.byref(n)), "smem_get_free_fifo")
    return out[: n.value].tolist()


def smem_get_device_table(h, seq, cap, stream=None):
    n = ctypes.c_int32(0)
    out = np.zeros(max(cap, 1), dtype=np.int32)
    _check(lib().smem_get_device_table(h, seq, out.ctypes.data_as(_i32p), cap, ctypes.byref(n), _stream(stream)),
           "smem_get_device_table")
    return out[: min(n.value, cap)].tolist()


def smem_check_device_error(h, stream=None) -> int:
    """Returns OK or ERR_DEVICE_FAULT (does not raise for the latter)."""
    rc = lib().smem_check_device_error(h, _stream(stream))
    if rc not in (OK, ERR_DEVICE_FAULT):
        raise SmemError(rc, "smem_check_device_error")
    return rc


def smem_free_slots(h) -> int:
    n = ctypes.c_int32(0)
    _check(lib().smem_free_slots(h, ctypes.byref(n)), "smem_free_slots")
    return n.value


def smem_debug_fail_after(h, n: int):
    return _check(lib().smem_debug_fail_after(h, n), "smem_debug_fail_after")


def smem_debug_set_table_entry(h, seq, pos, slot, stream=None):
    """Testing hook: overwrite one entry of the device copy of a table."""
    _check(lib().smem_debug_set_table_entry(h, seq, pos, slot, _stream(stream)), "smem_debug_set_table_entry")


def smem_debug_wait_probe(h, limit_ns, stream=None):
    """Testing hook: a kernel whose one bounded wait must give up."""
    _check(lib().smem_debug_wait_probe(h, int(limit_ns), _stream(stream)), "smem_debug_wait_probe")


def smem_debug_gemm(h, A, lda, W, b_kmajor, M, N, K, out, ldo, a_bs=0, w_boff=0, batch=1, epi=0, alpha=1.0,
                    o_bs=0, col_group=0, group_stride=0, stream=None):
    """Testing hook: one projection on the reader layer's tensor-core kernel
    (see include/smem.h); W's shape is taken from the tensor."""
    w_rows, w_cols = int(W.shape[0]), int(W.shape[1])
    return _check(lib().smem_debug_gemm(h, _ptr(A), lda, a_bs, _ptr(W), w_rows, w_cols, b_kmajor, w_boff, M, N, K,
                                        batch, epi, float(alpha), _ptr(out), ldo, o_bs, col_group, group_stride,
                                        _stream(stream)), "smem_debug_gemm")


def smem_debug_layernorm(h, x, gain, bias, out, stream=None):
    """Testing hook: the reader layer's LayerNorm kernel on x [n][d] fp32."""
    n, d = int(x.shape[0]), int(x.shape[1])
    return _check(lib().smem_debug_layernorm(h, _ptr(x), n, d, _ptr(gain), _ptr(bias), _ptr(out), _stream(stream)),
                  "smem_debug_layernorm")


def smem_abi_version() -> int:
    return int(lib().smem_abi_version())


def layer_weights(tensors: dict) -> SmemLayerWeights:
    """A SmemLayerWeights from a dict of device tensors keyed by field name
    (LayerNorm gains/biases fp32 [d], matrices bf16 row-major). The caller
    keeps the tensors alive."""
    return SmemLayerWeights(*[tensors[f].data_ptr() if tensors.get(f) is not None else None for f in LAYER_FIELDS])


def _warr(weights):
    if isinstance(weights, SmemLayerWeights):
        weights = [weights]
    arr = (SmemLayerWeights * len(weights))(*weights)
    return arr


def _ws(ws):
    return _ptr(ws), (0 if ws is None else ws.numel() * ws.element_size())


def smem_layer_workspace_bytes(h, n_rows) -> int:
    return int(lib().smem_layer_workspace_bytes(h, n_rows))


def smem_append_block_rows(h, seq, block_idx, mu, weights, ws, stream=None) -> int:
    """weights: a list of SmemLayerWeights, one per layer."""
    slot = ctypes.c_int32(-1)
    arr = _warr(weights)
    wp, wn = _ws(ws)
    _check(lib().smem_append_block_rows(h, seq, block_idx, _ptr(mu), arr, wp, wn, _stream(stream),
                                        ctypes.byref(slot)), "smem_append_block_rows")
    return slot.value


def smem_set_null_vector(h, nu, weights, ws, stream=None):
    arr = _warr(weights)
    wp, wn = _ws(ws)
    return _check(lib().smem_set_null_vector(h, _ptr(nu), arr, wp, wn, _stream(stream)), "smem_set_null_vector")


def smem_reader_layer_prefill(h, seq, layer, q_block_idx, weights, x, ws, stream=None):
    """weights: this layer's SmemLayerWeights; x: fp32 [b][d], updated in place."""
    arr = _warr(weights)
    wp, wn = _ws(ws)
    return _check(lib().smem_reader_layer_prefill(h, seq, layer, q_block_idx, arr, _ptr(x), wp, wn, _stream(stream)),
                  "smem_reader_layer_prefill")


def smem_reader_layer_decode(h, layer, seq_ids, pos, q_block_idx, weights, x, ws, stream=None):
    """x: fp32 [nb][d], updated in place."""
    s, sp = _i32arr(seq_ids)
    p, pp = _i32arr(pos)
    q, qp = _i32arr(q_block_idx)
    arr = _warr(weights)
    wp, wn = _ws(ws)
    return _check(lib().smem_reader_layer_decode(h, layer, len(s), sp, pp, qp, arr, _ptr(x), wp, wn,
                                                 _stream(stream)), "smem_reader_layer_decode")


def smem_mu_decode(h, seq_ids, q_block_idx, qp, op, ws, stream=None):
    """Memory-row cross-attention of a recompute cache: qp, op [nb][H][d]."""
    s, sp = _i32arr(seq_ids)
    q, qptr = _i32arr(q_block_idx)
    wp, wn = _ws(ws)
    return _check(lib().smem_mu_decode(h, len(s), sp, qptr, _ptr(qp), _ptr(op), wp, wn, _stream(stream)),
                  "smem_mu_decode")


def smem_mu_prefill(h, seq, q_block_idx, qp, op, ws, stream=None):
    """Memory-row cross-attention of one block's queries: qp, op [H][b][d]."""
    wp, wn = _ws(ws)
    return _check(lib().smem_mu_prefill(h, seq, q_block_idx, _ptr(qp), _ptr(op), wp, wn, _stream(stream)),
                  "smem_mu_prefill")


class SmemCache:
    """Owns a cache handle and (for device caches) its device buffer."""

    def __init__(self, cfg: SmemConfig, device=None):
        import torch

        self.cfg = cfg
        self.nbytes = smem_cache_required_bytes(cfg)
        if self.nbytes == 0:
            raise SmemError(ERR_INVALID_ARG, "smem_cache_required_bytes")
        self.buf = None
        if device is not None:
            self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        self.h = smem_cache_create(cfg, self.buf)

    def close(self):
        if self.h is not None:
            smem_cache_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
