"""Shared helpers for the GPU parity tests: a device cache driven through the
C ABI, seeded inputs from ``synth`` and the fp64 oracle on the same inputs."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import synth
from oracle.bookkeeping import CacheMirror
from paper_2609_32395_gb300 import smem

R = 64
B_TOK = 64
# tolerance on bf16 outputs (fp32 accumulation) against the fp64 oracle
MAX_ABS = 2e-2
MEAN_ABS = 2e-3
REL_L2 = 1e-2  # internal gate: cross-attention outputs shrink like 1/sqrt(N)


def to_dev(bits: np.ndarray, device="cuda"):
    return synth.bits_to_torch_bf16(bits).to(device)


def f64(bits):
    return oracle.bf16_bits_to_f64(bits)


def out_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close(got: np.ndarray, ref: np.ndarray, what: str):
    err = np.abs(got - ref)
    mx, mean = float(err.max()), float(err.mean())
    rel = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))
    assert mx <= MAX_ABS and mean <= MEAN_ABS and rel <= REL_L2, \
        f"{what}: max_abs {mx:.3e} mean_abs {mean:.3e} rel_l2 {rel:.3e}"
    return mx, mean, rel


class DeviceCache:
    """A device cache plus a host record of what each slot holds."""

    def __init__(self, L, H, D, max_seqs, max_blocks, capacity, seed=0, free_order=None, has_null=False,
                 max_batch=None, rope_window=0, n_kv_heads=0):
        self.L, self.H, self.D = L, H, D
        self.Hkv = n_kv_heads or H          # key/value heads (grouped-query attention)
        self.G = H // self.Hkv
        self.seed = seed
        self.rope_window = rope_window
        self.cfg = smem.make_config(L, H, D, max_seqs, max_blocks, capacity, has_null_row=has_null,
                                    max_decode_batch=max_batch, free_order=free_order, rope_window=rope_window,
                                    n_kv_heads=n_kv_heads)
        self.cache = smem.SmemCache(self.cfg, device="cuda")
        self.h = self.cache.h
        self.mirror = CacheMirror(capacity, max_seqs, max_blocks, free_order=free_order)
        self.blocks = {}  # (seq, block_idx) -> (K bits, V bits) [L][H][R][D]
        self.inblock = {}  # (seq, layer) -> (K bits, V bits) [b][H][D], rows written so far
        self.k_null = self.v_null = None
        if has_null:
            self.k_null = synth.tensor_np(seed, synth.KIND_KNULL, (L, self.Hkv, D))
            self.v_null = synth.tensor_np(seed, synth.KIND_VNULL, (L, self.Hkv, D))
            smem.smem_set_null_row(self.h, to_dev(self.k_null), to_dev(self.v_null))

    def block_bits(self, seq, idx, content_seq=None):
        cs = seq if content_seq is None else content_seq
        return synth.block_rows_np(self.seed, cs, idx, self.L, self.Hkv, R, self.D)

    def append(self, seq, idx, content_seq=None):
        K, V = self.block_bits(seq, idx, content_seq)
        slot = smem.smem_append_block(self.h, seq, idx, to_dev(K), to_dev(V))
        rc, s_m = self.mirror.append(seq, idx)
        assert rc == 0 and s_m == slot
        self.blocks[(seq, idx)] = (K, V)
        return slot

    def delete(self, seq, idx):
        smem.smem_delete_block(self.h, seq, idx)
        assert self.mirror.delete(seq, idx) == 0
        del self.blocks[(seq, idx)]

    def write_inblock(self, seq, layer, n, tag=0):
        Kb = synth.tensor_np(self.seed, synth.KIND_KIN, (B_TOK, self.Hkv, self.D), seq, layer, tag)
        Vb = synth.tensor_np(self.seed, synth.KIND_VIN, (B_TOK, self.Hkv, self.D), seq, layer, tag)
        smem.smem_write_inblock(self.h, seq, layer, n, to_dev(Kb[:n]), to_dev(Vb[:n]))
        self.inblock[(seq, layer)] = (Kb.copy(), Vb.copy())

    def check_tables(self, seqs):
        torch.cuda.synchronize()
        for s in seqs:
            idx, slots = smem.smem_get_table(self.h, s)
            assert (idx, slots) == self.mirror.table(s)
            dev = smem.smem_get_device_table(self.h, s, len(slots))
            assert dev == slots
        assert smem.smem_get_free_fifo(self.h) == self.mirror.free_list()

    def oracle_memory(self, seq, layer):
        """Oracle inputs of one layer: block indices and fp64 rows, in an
        arbitrary (insertion) order; the oracle canonicalises."""
        keys = [k for k in self.blocks if k[0] == seq]
        idx = [k[1] for k in keys]
        if not keys:
            return idx, None, None
        mk = np.stack([f64(self.blocks[k][0][layer]) for k in keys])
        mv = np.stack([f64(self.blocks[k][1][layer]) for k in keys])
        # query head h reads key/value head h // G
        return idx, np.repeat(mk, self.G, axis=1), np.repeat(mv, self.G, axis=1)

    def null(self, layer):
        if self.k_null is None:
            return None, None
        return np.repeat(f64(self.k_null[layer]), self.G, axis=0), np.repeat(f64(self.v_null[layer]), self.G, axis=0)

    # -------------------------------------------------------------- prefill
    def prefill_inputs(self, layer, tag=0):
        shape, kvs = (B_TOK, self.H, self.D), (B_TOK, self.Hkv, self.D)
        return [synth.tensor_np(self.seed, k, sh, layer, tag)
                for k, sh in ((synth.KIND_QS, shape), (synth.KIND_KS, kvs), (synth.KIND_VS, kvs),
                              (synth.KIND_QC, shape))]

    def prefill(self, seq, layer, q_idx, tag=0):
        qs, ks, vs, qc = self.prefill_inputs(layer, tag)
        osa = torch.empty((B_TOK, self.H, self.D), dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_prefill_block(self.h, seq, layer, q_idx, to_dev(qs), to_dev(ks), to_dev(vs), to_dev(qc), osa, oca)
        torch.cuda.synchronize()
        return (qs, ks, vs, qc), osa, oca

    def oracle_prefill(self, seq, layer, q_idx, qs, ks, vs, qc):
        idx, mk, mv = self.oracle_memory(seq, layer)
        kn0, vn0 = self.null(layer)
        ks, vs = (np.repeat(f64(a), self.G, axis=1) for a in (ks, vs))
        if self.rope_window:
            from oracle.rope import reader_prefill_rope
            return reader_prefill_rope(idx, mk, mv, q_idx, f64(qs), ks, vs, f64(qc), kn0, vn0,
                                       window=self.rope_window)
        return oracle.reader_prefill(idx, mk, mv, q_idx, f64(qs), ks, vs, f64(qc), kn0, vn0)

    # -------------------------------------------------------------- decode
    def decode_inputs(self, nb, layer, step):
        H, D, Hk = self.H, self.D, self.Hkv
        t = [synth.tensor_np(self.seed, k, (nb, h, D), layer, step)
             for k, h in ((synth.KIND_QDEC_S, H), (synth.KIND_KNEW, Hk), (synth.KIND_VNEW, Hk), (synth.KIND_QDEC_C, H))]
        return t  # qs, k_new, v_new, qc bits

    def decode(self, layer, seqs, pos, qidx, step=0):
        nb = len(seqs)
        qs, kn, vn, qc = self.decode_inputs(nb, layer, step)
        osa = torch.empty((nb, self.H, self.D), dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_decode(self.h, layer, seqs, pos, qidx, to_dev(qs), to_dev(kn), to_dev(vn), to_dev(qc), osa, oca)
        torch.cuda.synchronize()
        # the step stored the new token's k, v at in-block row pos
        for i, (s, p) in enumerate(zip(seqs, pos)):
            Kb, Vb = self.inblock.setdefault((s, layer), (np.zeros((B_TOK, self.Hkv, self.D), np.uint16),
                                                          np.zeros((B_TOK, self.Hkv, self.D), np.uint16)))
            Kb[p] = kn[i]
            Vb[p] = vn[i]
        return (qs, kn, vn, qc), osa, oca

    def oracle_decode(self, layer, seq, p, qidx, qs, kn, vn, qc):
        idx, mk, mv = self.oracle_memory(seq, layer)
        Kb, Vb = self.inblock[(seq, layer)]
        kin = np.repeat(f64(Kb[:p]), self.G, axis=1) if p else None
        vin = np.repeat(f64(Vb[:p]), self.G, axis=1) if p else None
        kn0, vn0 = self.null(layer)
        kn, vn = (np.repeat(f64(a), self.G, axis=0) for a in (kn, vn))
        if self.rope_window:
            from oracle.rope import reader_decode_rope
            return reader_decode_rope(idx, mk, mv, qidx, p, kin, vin, f64(qs), kn, vn, f64(qc), kn0, vn0,
                                      window=self.rope_window)
        return oracle.reader_decode(idx, mk, mv, qidx, p, kin, vin, f64(qs), kn, vn, f64(qc), kn0, vn0)
