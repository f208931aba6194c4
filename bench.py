"""Benchmark of the SMem reader hot path on GB300.

Default workload (one GPU): 410M-shaped batched decode -- L = 24 reader
layers, H = 16 heads, d_h = 64, blocks of b = R = 64, 64 sequences with
contexts uniform in [64, 256] memory blocks and in-block offsets uniform in
[0, 63], pool slots in a seeded shuffled order. A step is one decode token
for all 64 sequences through all 24 layers (24 decode launches); whenever a
sequence's in-block offset wraps 63 -> 0 the finished block is appended to
its memory (synthetic rows) inside the step. The pool (~66 GB) is far
larger than L2, so no flush is needed between steps.

Prints one JSON line. ``--impl reference`` times the fp64 CPU oracle on the
same workload (a bounded sample) instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "decode tok/s + cross-attn HBM GB/s (% peak); one-block cached-serve latency ms"
WORKLOAD = dict(name="410M-shaped batched decode", L=24, H=16, D=64, seqs=64, ctx_lo=64, ctx_hi=256, seed=0)
R = 64
B_TOK = 64
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0  # the nominal HBM3e bandwidth (context beside the measured copy peak)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-serve", action="store_true")
    ap.add_argument("--no-layer", action="store_true", help="skip the full-reader-layer cells")
    ap.add_argument("--no-recompute", action="store_true", help="skip the recompute-K/V cells")
    ap.add_argument("--no-rope", action="store_true", help="skip the rotary-phase (RoPE composite) cells")
    ap.add_argument("--no-d32", action="store_true", help="skip the d_h = 32 decode cell")
    ap.add_argument("--no-gqa", action="store_true", help="skip the grouped-query decode cell")
    ap.add_argument("--no-long", action="store_true", help="skip the bounded 1.5B long-context cells")
    ap.add_argument("--workload", default="decode", choices=["decode", "long"],
                    help="long: the 1.5B-shaped long-context cells (prefill latency, decode tok/s)")
    ap.add_argument("--long-batches", default="1,16", help="batches of the long-context cells")
    ap.add_argument("--long-layers", type=int, default=None,
                    help="physical layers of the long-context cache (profiling captures)")
    ap.add_argument("--long-contexts", default="512,1024,4096")
    ap.add_argument("--only-serve", action="store_true",
                    help="time only the one-block cached-serve cells (profiling)")
    ap.add_argument("--seqs", type=int, default=WORKLOAD["seqs"])
    ap.add_argument("--layers", type=int, default=WORKLOAD["L"],
                    help="fewer layers: same per-launch work, smaller pool (profiling captures)")
    return ap.parse_args()


# ----------------------------------------------------------------------------- helpers
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def source_sha(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def profiled_traffic(profile_name, units_now, exact=False):
    """DRAM bytes per launch from a committed ncu summary, scaled to this
    launch's units; None if any source the summary lists changed since the
    capture (so a stale count is never reported)."""
    path = os.path.join(ROOT, "profiles", profile_name)
    if not os.path.exists(path):
        return None
    kv, shas = {}, []
    for line in open(path):
        if line.startswith("#") or ":" not in line:
            continue
        k, v = line.split(":", 1)
        k, v = k.strip(), v.strip()
        if k == "source_sha256":
            name, digest = v.split()
            shas.append((name, digest))
        else:
            kv[k] = v
    try:
        if not shas or any(source_sha(os.path.join(ROOT, n)) != d for n, d in shas):
            return None
        if exact:  # traffic with a fixed part: only the captured size is known
            return float(kv["dram_bytes_per_launch"]) if float(kv["units_per_launch"]) == units_now else None
        per_unit = float(kv["dram_bytes_per_launch"]) / float(kv["units_per_launch"])
        return per_unit * units_now
    except (KeyError, ValueError, OSError):
        return None


def max_over_ranks(x: float, device=None) -> float:
    """Max of a per-rank float over the process group (identity without one)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def rank_seed(seed: int, rank: int) -> int:
    """Each rank serves its own sequences: the seed is offset by the rank."""
    return seed + 1000 * rank


# ----------------------------------------------------------------------------- decode workload
class DecodeWorkload:
    """Device state of the 410M-shaped batched-decode workload."""

    def __init__(self, seqs, steps_total, seed, device, rank=0, layers=None, rope_window=0, heads=None, kv_heads=0):
        import torch

        import synth
        from paper_2609_32395_gb300 import smem

        W = WORKLOAD
        self.L, self.H, self.D = (layers or W["L"]), W["H"], W["D"]
        if heads is not None:  # same width d = H * d_h, other head count
            self.H, self.D = heads, W["H"] * W["D"] // heads
        self.Hkv = kv_heads or self.H  # key/value heads (grouped-query attention)
        self.S = seqs
        self.seed = rank_seed(seed, rank)
        self.device = device
        self.nblk = synth.ragged_contexts(self.seed, seqs, W["ctx_lo"], W["ctx_hi"]).astype(np.int64)
        self.pos = synth.inblock_positions(self.seed, seqs, B_TOK).astype(np.int64)
        # appends each sequence will need over all steps
        self.n_new = [(int(p) + steps_total) // B_TOK + 1 for p in self.pos]
        capacity = int(self.nblk.sum()) + sum(self.n_new)
        max_blocks = int(self.nblk.max()) + max(self.n_new) + 1
        perm = synth.slot_permutation(self.seed, capacity)
        self.cfg = smem.make_config(self.L, self.H, self.D, seqs, max_blocks, capacity, free_order=perm,
                                    rope_window=rope_window, n_kv_heads=kv_heads)
        self.cache = smem.SmemCache(self.cfg, device=device)
        self.h = self.cache.h
        torch.cuda.synchronize()
        # memory blocks 0..nblk-1 of every sequence
        chunk = 16
        for s in range(seqs):
            n = int(self.nblk[s])
            for b0 in range(0, n, chunk):
                ids = list(range(b0, min(n, b0 + chunk)))
                K, V = synth.block_rows_torch(self.seed, s, ids, self.L, self.Hkv, R, self.D, device)
                for i, j in enumerate(ids):
                    smem.smem_append_block(self.h, s, j, K[i], V[i])
                del K, V
        # blocks that will be appended when a sequence's block completes
        self.new_K, self.new_V = [], []
        for s in range(seqs):
            ids = [int(self.nblk[s]) + k for k in range(self.n_new[s])]
            K, V = synth.block_rows_torch(self.seed, s, ids, self.L, self.Hkv, R, self.D, device)
            self.new_K.append(K)
            self.new_V.append(V)
        self.new_used = [0] * seqs
        # in-block rows 0..p-1 of every sequence and layer
        for s in range(seqs):
            p = int(self.pos[s])
            for layer in range(self.L):
                if p:
                    Kb = synth.tensor_torch(self.seed, synth.KIND_KIN, (p, self.Hkv, self.D), s, layer, 0,
                                            device=device)
                    Vb = synth.tensor_torch(self.seed, synth.KIND_VIN, (p, self.Hkv, self.D), s, layer, 0,
                                            device=device)
                    smem.smem_write_inblock(self.h, s, layer, p, Kb, Vb)
        # per-layer decode inputs (a few distinct sets, cycled)
        self.n_sets = 2
        shape = (seqs, self.H, self.D)
        self.inputs = []
        for k in range(self.n_sets):
            per_layer = []
            for layer in range(self.L):
                kv_shape = (seqs, self.Hkv, self.D)
                per_layer.append([synth.tensor_torch(self.seed, kind, sh, layer, k, device=device)
                                  for kind, sh in ((synth.KIND_QDEC_S, shape), (synth.KIND_KNEW, kv_shape),
                                                   (synth.KIND_VNEW, kv_shape), (synth.KIND_QDEC_C, shape))])
            self.inputs.append(per_layer)
        self.osa = torch.empty(shape, dtype=torch.bfloat16, device=device)
        self.oca = torch.empty(shape, dtype=torch.bfloat16, device=device)
        self.seq_ids = np.arange(seqs, dtype=np.int32)
        self.step_no = 0
        torch.cuda.synchronize()

    def rows_read(self):
        """Memory rows + in-block rows one decode launch reads (all sequences)."""
        return int(self.nblk.sum()) * R + int((self.pos + 1).sum())

    def step(self, events=None, host_inputs=None, host_outputs=None, host_blocks=None):
        """One decode token for every sequence through all layers. Returns the
        number of this library's kernel launches."""
        import torch

        from paper_2609_32395_gb300 import smem

        if host_inputs is not None and host_outputs is not None:
            return self._step_host(host_inputs, host_outputs, host_blocks)
        launches = 0
        st = torch.cuda.current_stream()
        k = self.step_no % self.n_sets
        for layer in range(self.L):
            qs, kn, vn, qc = self.inputs[k][layer]
            if host_inputs is not None:
                hq = host_inputs[k][layer]
                for dst, src in zip((qs, kn, vn, qc), hq):
                    dst.copy_(src, non_blocking=True)
            if events is not None:
                events[0][layer].record(st)
            smem.smem_decode(self.h, layer, self.seq_ids, self.pos.astype(np.int32), self.nblk.astype(np.int32),
                             qs, kn, vn, qc, self.osa, self.oca)
            if events is not None:
                events[1][layer].record(st)
            launches += 1
            if host_outputs is not None:
                host_outputs[0][layer].copy_(self.osa, non_blocking=True)
                host_outputs[1][layer].copy_(self.oca, non_blocking=True)
        return launches + self._advance(host_blocks)

    def _advance(self, host_blocks):
        """Moves every sequence one token on; a block that completes is
        appended (its rows from the host when host_blocks is given)."""
        from paper_2609_32395_gb300 import smem

        launches = 0
        self.pos += 1
        for s in np.nonzero(self.pos == B_TOK)[0]:
            u = self.new_used[s]
            K, V = self.new_K[s][u], self.new_V[s][u]
            if host_blocks is not None:
                K.copy_(host_blocks[0], non_blocking=True)
                V.copy_(host_blocks[1], non_blocking=True)
            smem.smem_append_block(self.h, int(s), int(self.nblk[s]), K, V)
            launches += 1
            self.new_used[s] += 1
            self.nblk[s] += 1
            self.pos[s] = 0
        self.step_no += 1
        return launches

    def _step_host(self, host_inputs, host_outputs, host_blocks):
        """One step through the library's host-buffer decode call: every
        layer's inputs come from pinned host memory and its outputs go back
        to it through smem_decode_host, the copies on a copy stream of their
        own, ordered by the library against the decode of the neighbouring
        layers (two staging halves). The rows of a block that completes with
        this step's token come from the host on the same copy stream while
        the step's layers decode (they do not depend on them); the append
        follows the step. The step ends when its last copy has landed."""
        import torch

        from paper_2609_32395_gb300 import smem

        if not hasattr(self, "copy_stream"):
            self.copy_stream = torch.cuda.Stream()
            self.stage = torch.empty(smem.smem_decode_host_stage_bytes(self.h, self.S), dtype=torch.uint8,
                                     device=self.osa.device)
        st = torch.cuda.current_stream()
        cs = self.copy_stream
        k = self.step_no % self.n_sets
        pos, nblk = self.pos.astype(np.int32), self.nblk.astype(np.int32)
        completing = np.nonzero(self.pos + 1 == B_TOK)[0] if host_blocks is not None else []
        for layer in range(self.L):
            qs, kn, vn, qc = host_inputs[k][layer]
            smem.smem_decode_host(self.h, layer, self.seq_ids, pos, nblk, qs, kn, vn, qc, host_outputs[0][layer],
                                  host_outputs[1][layer], self.stage, stream=st, copy_stream=cs)
            if layer == min(2, self.L - 1) and len(completing):
                with torch.cuda.stream(cs):  # after the first layers' input copies
                    for s in completing:
                        u = self.new_used[s]
                        self.new_K[s][u].copy_(host_blocks[0], non_blocking=True)
                        self.new_V[s][u].copy_(host_blocks[1], non_blocking=True)
        st.wait_stream(cs)
        return self.L + self._advance(None)


class LayerStack:
    """Random-init weights of L reader layers of width d on the device (the
    seeded recipe of ``synth.reader_layer_weights_torch``)."""

    def __init__(self, L, d, seed, device):
        import synth
        from paper_2609_32395_gb300 import smem

        self.L, self.d = L, d
        self.tensors = [synth.reader_layer_weights_torch(seed, l, d, device=device) for l in range(L)]
        self.sw = [smem.layer_weights(t) for t in self.tensors]

    def bytes_per_layer(self):
        # every weight matrix read once (bf16) + LayerNorm parameters (fp32)
        return 14 * self.d * self.d * 2 + 6 * self.d * 4

    def flops_per_layer(self, rows):
        # the six token projections (memory-row projections happen at append)
        return 2 * rows * (3 + 1 + 1 + 1 + 4 + 4) * self.d * self.d


def layer_decode_step(wl, stack, x, ws, mu, events=None):
    """One decode token for every sequence through all layers of the full
    reader layer (LayerNorm, projections, attention, FFN); a finished block
    is appended from synthetic memory rows through the layer's key/value
    maps. Returns the number of kernel launches."""
    import torch

    from paper_2609_32395_gb300 import smem

    st = torch.cuda.current_stream()
    if events is not None:
        events[0].record(st)
    for layer in range(wl.L):
        smem.smem_reader_layer_decode(wl.h, layer, wl.seq_ids, wl.pos.astype(np.int32), wl.nblk.astype(np.int32),
                                      stack.sw[layer], x, ws)
    if events is not None:
        events[1].record(st)
    ours = 11 * wl.L  # per layer: 3 LayerNorm, 6 projections (GELU, residual fused) and 2 attention launches
    wl.pos += 1
    for s in np.nonzero(wl.pos == B_TOK)[0]:
        smem.smem_append_block_rows(wl.h, int(s), int(wl.nblk[s]), mu, stack.sw, ws)
        ours += 1 + 2 * wl.L  # key and value projections of every layer, then the table insert
        wl.new_used[s] += 1
        wl.nblk[s] += 1
        wl.pos[s] = 0
    wl.step_no += 1
    return ours


def measure_layer_decode(wl, steps, warmup, device):
    """Full-reader-layer decode on the decode workload's cache (its memory
    rows stand in for projected ones): tok/s, and the HBM roofline of a step
    (weights of every layer + the K/V rows the attention reads)."""
    import torch

    import synth
    from paper_2609_32395_gb300 import smem

    d = wl.H * wl.D
    stack = LayerStack(wl.L, d, 5, device)
    ws = torch.empty(smem.smem_layer_workspace_bytes(wl.h, wl.S), dtype=torch.uint8, device=device)
    x0 = synth.tensor_torch(wl.seed, synth.KIND_X, (wl.S, d), 0, device=device).float()
    x = x0.clone()
    mu = synth.tensor_torch(wl.seed, synth.KIND_MU, (R, d), 0, device=device)
    for _ in range(warmup):
        layer_decode_step(wl, stack, x, ws, mu)
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
    rows, ours = [], 0
    for i in range(steps):
        x.copy_(x0)
        rows.append(wl.rows_read())
        ours += layer_decode_step(wl, stack, x, ws, mu, events=ev[i])
    torch.cuda.synchronize()
    if smem.smem_check_device_error(wl.h) != smem.OK:
        raise RuntimeError("device error recorded during the full-layer decode")
    ms = [a.elapsed_time(b) for a, b in ev]
    step_ms = float(np.mean(ms))
    kv = float(np.mean(rows)) * 4 * d * wl.L  # K + V bf16 per row per layer
    w = stack.bytes_per_layer() * wl.L
    act = wl.L * wl.S * d * 4 * 2 * 3  # residual stream read + written per branch (fp32)
    alg = kv + w + act
    return {"tok_per_s": wl.S / (step_ms / 1e3), "step_ms": step_ms, "step_ms_p50": float(np.median(ms)),
            "alg_bytes_per_step": alg, "weight_bytes_per_step": w, "kv_bytes_per_step": kv,
            "achieved_gbs": alg / (step_ms / 1e3) / 1e9, "launches": ours,
            "timing": "CUDA events around the layer calls of each step (appends excluded), inputs resident"}


ROPE_WINDOW = 15  # the paper's saturating window (trained range of 16 blocks)


def measure_decode_variant(steps, warmup, device, seqs, layers=None, window=None, heads=None, kv_heads=0):
    """The headline decode workload on a cache variant -- the SMem+RoPE
    composite's rotary phases (window 15 by default; 0: none) and/or another
    head count at the same width (heads=32: d_h = 32): decode tok/s and the
    decode kernel's HBM fraction, timed like the headline (CUDA events per
    launch)."""
    import torch

    from paper_2609_32395_gb300 import smem

    win = ROPE_WINDOW if window is None else window
    wl = DecodeWorkload(seqs, warmup + steps + 2, WORKLOAD["seed"], device, layers=layers, rope_window=win,
                        heads=heads, kv_heads=kv_heads)
    for _ in range(warmup):
        wl.step()
    torch.cuda.synchronize()
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(wl.L)] for _ in range(2)] for _ in range(steps)]
    st = torch.cuda.current_stream()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    rows = []
    start.record(st)
    for i in range(steps):
        rows.append(wl.rows_read())
        wl.step(events=ev[i])
    end.record(st)
    torch.cuda.synchronize()
    if smem.smem_check_device_error(wl.h) != smem.OK:
        raise RuntimeError("device error recorded during the rotary decode")
    elapsed = start.elapsed_time(end) / 1e3
    kern_ms = [ev[i][0][l].elapsed_time(ev[i][1][l]) for i in range(steps) for l in range(wl.L)]
    alg = [r * 4 * wl.Hkv * wl.D for r in rows for _ in range(wl.L)]  # each key/value row once
    out = {"window": win, "heads": wl.H, "kv_heads": wl.Hkv, "head_dim": wl.D, "pool_bytes": int(wl.cache.nbytes),
           "tok_per_s": steps * seqs / elapsed, "steps": steps,
           "kernel_ms_mean": float(np.mean(kern_ms)), "rows_per_launch": float(np.mean(rows)),
           "achieved_gbs": sum(alg) / (sum(kern_ms) / 1e3) / 1e9}
    wl.cache.close()
    return out


class RecomputeDecode:
    """The 410M-shaped decode workload on a recompute-K/V cache: the pool
    holds only each block's memory rows mu [R][d] (d = H*d_h, shared by the
    24 layers); every layer re-derives its cross-attention from them. Same
    sequences, contexts and in-block offsets as the materialized workload."""

    def __init__(self, seqs, steps_total, seed, device, rank=0, layers=None):
        import torch

        import synth
        from paper_2609_32395_gb300 import smem

        W = WORKLOAD
        self.L, self.H, self.D = (layers or W["L"]), W["H"], W["D"]
        self.d = self.H * self.D
        self.S = seqs
        self.seed = rank_seed(seed, rank)
        self.nblk = synth.ragged_contexts(self.seed, seqs, W["ctx_lo"], W["ctx_hi"]).astype(np.int64)
        self.pos = synth.inblock_positions(self.seed, seqs, B_TOK).astype(np.int64)
        n_new = [(int(p) + steps_total) // B_TOK + 1 for p in self.pos]
        capacity = int(self.nblk.sum()) + sum(n_new)
        max_blocks = int(self.nblk.max()) + max(n_new) + 1
        perm = synth.slot_permutation(self.seed, capacity)
        self.cfg = smem.make_config(self.L, self.H, self.D, seqs, max_blocks, capacity, free_order=perm,
                                    recompute_kv=True)
        self.cache = smem.SmemCache(self.cfg, device=device)
        self.h = self.cache.h
        self.ws = torch.empty(smem.smem_layer_workspace_bytes(self.h, seqs), dtype=torch.uint8, device=device)
        for s in range(seqs):
            n = int(self.nblk[s])
            mu = synth.tensor_torch(self.seed, synth.KIND_MU, (n * R, self.d), s, device=device)
            for j in range(n):
                smem.smem_append_block_rows(self.h, s, j, mu[j * R:(j + 1) * R], [], self.ws)
            del mu
        for s in range(seqs):
            p = int(self.pos[s])
            for layer in range(self.L):
                if p:
                    Kb = synth.tensor_torch(self.seed, synth.KIND_KIN, (p, self.H, self.D), s, layer, 0,
                                            device=device)
                    Vb = synth.tensor_torch(self.seed, synth.KIND_VIN, (p, self.H, self.D), s, layer, 0,
                                            device=device)
                    smem.smem_write_inblock(self.h, s, layer, p, Kb, Vb)
        self.seq_ids = np.arange(seqs, dtype=np.int32)
        self.new_used = [0] * seqs
        self.step_no = 0
        torch.cuda.synchronize()

    def rows_read(self):
        return int(self.nblk.sum()) * R


def measure_recompute(steps, warmup, device, seqs, layers=None):
    """Recompute-K/V regime at the 410M decode shape: the memory-row
    attention kernel alone (CUDA events per launch; algorithmic bytes = 2d
    per memory row read + the folded queries and outputs) and the full
    reader layer's decode tok/s on the same cache."""
    import torch

    import synth
    from paper_2609_32395_gb300 import smem

    rw = RecomputeDecode(seqs, warmup + steps + 4 + (warmup + steps), WORKLOAD["seed"], device, layers=layers)
    d, H = rw.d, rw.H
    qp = (synth.tensor_torch(rw.seed, synth.KIND_QDEC_C, (seqs, H, d), 7, device=device).float() / math.sqrt(d)
          ).to(torch.bfloat16)
    op = torch.empty(seqs, H, d, dtype=torch.bfloat16, device=device)
    st = torch.cuda.current_stream()
    ctx = rw.nblk.astype(np.int32)
    for _ in range(warmup):
        smem.smem_mu_decode(rw.h, rw.seq_ids, ctx, qp, op, rw.ws)
    torch.cuda.synchronize()
    n_launch = steps * 2
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(n_launch)]
    for i in range(n_launch):
        ev[i][0].record(st)
        smem.smem_mu_decode(rw.h, rw.seq_ids, ctx, qp, op, rw.ws)
        ev[i][1].record(st)
    torch.cuda.synchronize()
    if smem.smem_check_device_error(rw.h) != smem.OK:
        raise RuntimeError("device error recorded during the memory-row attention")
    kern_ms = float(np.mean([a.elapsed_time(b) for a, b in ev]))
    rows = rw.rows_read()
    alg = rows * 2 * d + 2 * seqs * H * d * 2
    nq, cl, wsl = smem.smem_mu_decode_plan(rw.h)
    name = (f"mu_slice_kernel<{nq}> (memory-row cross-attention, tcgen05; clusters of {cl} CTAs x {wsl} columns)"
            if cl else f"mu_attention_kernel<{nq}> (memory-row cross-attention, tcgen05; two-pass)")
    kernel = {"kernel": name, "launches": n_launch,
              "kernel_ms_mean": kern_ms, "rows_per_launch": rows, "alg_bytes_per_launch": alg,
              "achieved_gbs": alg / (kern_ms / 1e3) / 1e9,
              "materialized_bytes_per_launch": rows * 4 * H * rw.D}
    # full reader layer on the recompute cache (appends take memory rows)
    stack = LayerStack(rw.L, d, 5, device)
    x0 = synth.tensor_torch(rw.seed, synth.KIND_X, (seqs, d), 0, device=device).float()
    x = x0.clone()
    mu = synth.tensor_torch(rw.seed, synth.KIND_MU, (R, d), 1 << 20, device=device)
    for _ in range(warmup):
        layer_decode_step(rw, stack, x, rw.ws, mu)
    torch.cuda.synchronize()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
    for i in range(steps):
        x.copy_(x0)
        layer_decode_step(rw, stack, x, rw.ws, mu, events=evs[i])
    torch.cuda.synchronize()
    if smem.smem_check_device_error(rw.h) != smem.OK:
        raise RuntimeError("device error recorded during the recompute decode")
    step_ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
    out = {"workload": WORKLOAD["name"] + ", recompute-K/V cache", "pool_bytes": int(rw.cache.nbytes),
           "memory_row_kernel": kernel,
           "layer_decode": {"tok_per_s": seqs / (step_ms / 1e3), "step_ms": step_ms, "steps": steps,
                            "timing": "CUDA events around each step's layer calls (appends excluded)"}}
    rw.cache.close()
    return out


# ----------------------------------------------------------------------------- prefill workload
SERVE = dict(name="160M-shaped one-block cached-context prefill", L=12, H=12, D=64, contexts=(16, 64, 256), seed=1)


class PrefillWorkload:
    """A fully cached context of `nblk` memory blocks (160M reader shape,
    shuffled slots) served by running the reader's attention on the final
    block alone: 12 one-block prefill launches, one per layer."""

    def __init__(self, nblk, device, L=None, H=None, D=None, seed=None, recompute=False, rope_window=0):
        import torch

        import synth
        from paper_2609_32395_gb300 import smem

        self.L = L or SERVE["L"]
        self.H = H or SERVE["H"]
        self.D = D or SERVE["D"]
        self.nblk = nblk
        seed = SERVE["seed"] if seed is None else seed
        cap = nblk + 2
        self.cfg = smem.make_config(self.L, self.H, self.D, 1, nblk + 1, cap,
                                    free_order=synth.slot_permutation(seed + nblk, cap), recompute_kv=recompute,
                                    rope_window=rope_window)
        self.cache = smem.SmemCache(self.cfg, device=device)
        self.h = self.cache.h
        if recompute:  # the pool keeps memory rows only; attention-only launches do not apply
            import torch

            d = self.H * self.D
            ws = torch.empty(smem.smem_layer_workspace_bytes(self.h, 0), dtype=torch.uint8, device=device)
            mu = synth.tensor_torch(seed, synth.KIND_MU, (max(nblk, 1) * R, d), 0, device=device)
            for j in range(nblk):
                smem.smem_append_block_rows(self.h, 0, j, mu[j * R:(j + 1) * R], [], ws)
            torch.cuda.synchronize()
            return
        for b0 in range(0, nblk, 16):
            ids = list(range(b0, min(nblk, b0 + 16)))
            K, V = synth.block_rows_torch(seed, 0, ids, self.L, self.H, R, self.D, device)
            for i, j in enumerate(ids):
                smem.smem_append_block(self.h, 0, j, K[i], V[i])
        shape = (B_TOK, self.H, self.D)
        self.inputs = [[synth.tensor_torch(seed, k, shape, layer, 0, device=device)
                        for k in (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
                       for layer in range(self.L)]
        self.outputs = [(torch.empty(shape, dtype=torch.bfloat16, device=device),
                         torch.empty(shape, dtype=torch.bfloat16, device=device)) for _ in range(self.L)]
        torch.cuda.synchronize()

    def layer(self, layer):
        from paper_2609_32395_gb300 import smem

        qs, ks, vs, qc = self.inputs[layer]
        osa, oca = self.outputs[layer]
        smem.smem_prefill_block(self.h, 0, layer, self.nblk, qs, ks, vs, qc, osa, oca)

    def serve(self):
        for layer in range(self.L):
            self.layer(layer)

    def bytes_per_launch(self):
        # K/V of every memory row read (4*H*d_h bytes per row) + Qs, Ks, Vs, Qc read and Osa, Oca written
        return self.nblk * R * 4 * self.H * self.D + 6 * B_TOK * self.H * self.D * 2

    def flops_per_launch(self):
        # CA: QK^T and P.V over all memory rows; SA: the causal half of the 64 x 64 block
        ca = 4 * B_TOK * self.nblk * R * self.H * self.D
        sa = 4 * (B_TOK * (B_TOK + 1) // 2) * self.H * self.D
        return ca + sa


def measure_serve(nblk, device, iters=30, flush_bytes=512 << 20, rope_window=0):
    """Latency of one cached-context serve (12 layers) replayed from a CUDA
    graph, and the mean duration of one prefill launch; L2 is flushed before
    each timed iteration (the flush also keeps the stream busy while the
    timed work is enqueued)."""
    import torch

    wl = PrefillWorkload(nblk, device, rope_window=rope_window)
    flush = torch.empty(flush_bytes, dtype=torch.uint8, device=device)
    st = torch.cuda.current_stream()
    for _ in range(3):
        wl.serve()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        wl.serve()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    k0 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    k1 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    for i in range(iters):
        flush.zero_()
        e0[i].record(st)
        g.replay()
        e1[i].record(st)
    for i in range(iters):
        flush.zero_()
        k0[i].record(st)
        wl.layer(i % wl.L)
        k1[i].record(st)
    torch.cuda.synchronize()
    serve_ms = sorted(a.elapsed_time(b) for a, b in zip(e0, e1))
    kern_ms = [a.elapsed_time(b) for a, b in zip(k0, k1)]
    del g
    out = {"context_blocks": nblk, "memory_rows": nblk * R, "latency_ms": serve_ms[len(serve_ms) // 2],
           "latency_ms_min": serve_ms[0], "kernel_ms_mean": float(np.mean(kern_ms)),
           "bytes_per_launch": wl.bytes_per_launch(), "flops_per_launch": wl.flops_per_launch()}
    wl.cache.close()
    return out


def measure_layer_serve(nblk, device, iters=30, flush_bytes=512 << 20, recompute=False):
    """Latency of one cached-context serve through the full reader layer
    (12 layers of LayerNorm, projections, attention and FFN over the final
    block's 64 tokens), replayed from a CUDA graph with L2 flushed before
    each replay."""
    import torch

    import synth
    from paper_2609_32395_gb300 import smem

    wl = PrefillWorkload(nblk, device, recompute=recompute)
    d = wl.H * wl.D
    stack = LayerStack(wl.L, d, 6, device)
    ws = torch.empty(smem.smem_layer_workspace_bytes(wl.h, B_TOK), dtype=torch.uint8, device=device)
    x0 = synth.tensor_torch(SERVE["seed"], synth.KIND_X, (B_TOK, d), 0, nblk, device=device).float()
    x = x0.clone()
    flush = torch.empty(flush_bytes, dtype=torch.uint8, device=device)
    st = torch.cuda.current_stream()

    def serve():
        x.copy_(x0)
        for layer in range(wl.L):
            smem.smem_reader_layer_prefill(wl.h, 0, layer, nblk, stack.sw[layer], x, ws)

    for _ in range(3):
        serve()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        serve()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(iters)]
    for i in range(iters):
        flush.zero_()
        e0[i].record(st)
        g.replay()
        e1[i].record(st)
    torch.cuda.synchronize()
    if smem.smem_check_device_error(wl.h) != smem.OK:
        raise RuntimeError("device error recorded during the full-layer serve")
    lat = sorted(a.elapsed_time(b) for a, b in zip(e0, e1))
    del g
    kv = nblk * R * (2 * d if recompute else 4 * d) * wl.L  # memory rows (recompute) or K/V read per layer
    w = stack.bytes_per_layer() * wl.L
    alg = kv + w
    med = lat[len(lat) // 2]
    out = {"context_blocks": nblk, "latency_ms": med, "latency_ms_min": lat[0], "alg_bytes": alg,
           "weight_bytes": w, "kv_bytes": kv, "achieved_gbs": alg / (med / 1e3) / 1e9,
           "flops": stack.flops_per_layer(B_TOK) * wl.L + wl.flops_per_launch() * wl.L,
           "launches_per_serve": (14 if recompute else 11) * wl.L}
    wl.cache.close()
    return out


# ----------------------------------------------------------------------------- long-context workload
LONG = dict(name="1.5B-shaped long cached context", L=24, H=16, D=128, contexts=(512, 1024, 4096), batches=(1, 16),
            seed=2)


def long_batch_cells(batch, contexts, device, peak, bf16_peak, layers_cap=None, serve_iters=6, n_steps=8):
    """Cells of one batch size: a cache at the longest context (1.5B reader
    shape, shuffled slots) whose shorter contexts read its block prefix
    (block-causal mask); decode tok/s and kernel HBM fraction per context and,
    at batch 1, the 24-layer one-block serve latency and the prefill kernel's
    HBM and tensor fractions. Layers that do not fit (or above `layers_cap`)
    are emulated: the 24 logical layers cycle over the physical ones (each
    physical layer's working set is far above L2)."""
    import torch

    import synth
    from paper_2609_32395_gb300 import smem

    W = LONG
    H, D, L = W["H"], W["D"], W["L"]
    nmax = max(contexts)
    block_bytes = 2 * H * R * D * 2  # K and V of one layer
    free, _ = torch.cuda.mem_get_info()
    budget = free - (16 << 30)
    l_phys = max(1, min(L, budget // (batch * (nmax + 8) * block_bytes)))
    if layers_cap:
        l_phys = min(l_phys, layers_cap)
    l_phys = int(l_phys)
    cap = batch * (nmax + 4)
    cfg = smem.make_config(l_phys, H, D, batch, nmax + 4, cap,
                           free_order=synth.slot_permutation(W["seed"] + batch, cap))
    cache = smem.SmemCache(cfg, device=device)
    for s in range(batch):
        for b0 in range(0, nmax, 16):
            ids = list(range(b0, min(nmax, b0 + 16)))
            K, V = synth.block_rows_torch(W["seed"], s, ids, l_phys, H, R, D, device)
            for i, j in enumerate(ids):
                smem.smem_append_block(cache.h, s, j, K[i], V[i])
            del K, V
    shape = (batch, H, D)
    dins = [synth.tensor_torch(W["seed"], k, shape, 0, 0, device=device)
            for k in (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    osa = torch.empty(shape, dtype=torch.bfloat16, device=device)
    oca = torch.empty_like(osa)
    pshape = (B_TOK, H, D)
    pins = [synth.tensor_torch(W["seed"], k, pshape, 0, 0, device=device)
            for k in (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
    posa = torch.empty(pshape, dtype=torch.bfloat16, device=device)
    poca = torch.empty_like(posa)
    seqs = np.arange(batch, dtype=np.int32)
    st = torch.cuda.current_stream()
    cells = []
    for ctx in contexts:
        qidx = np.full(batch, ctx, dtype=np.int32)
        pos = np.zeros(batch, dtype=np.int32)
        for _ in range(2):
            for layer in range(L):
                smem.smem_decode(cache.h, layer % l_phys, seqs, pos, qidx, *dins, osa, oca)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * L * n_steps)]
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        t0.record(st)
        for i in range(n_steps):
            for layer in range(L):
                ev[2 * (i * L + layer)].record(st)
                smem.smem_decode(cache.h, layer % l_phys, seqs, pos, qidx, *dins, osa, oca)
                ev[2 * (i * L + layer) + 1].record(st)
        t1.record(st)
        torch.cuda.synchronize()
        step_ms = t0.elapsed_time(t1) / n_steps
        kms = float(np.mean([ev[2 * k].elapsed_time(ev[2 * k + 1]) for k in range(L * n_steps)]))
        dec_bytes = batch * (ctx * R + 1) * 4 * H * D
        cell = {"batch": batch, "context_blocks": ctx, "memory_rows": ctx * R,
                "layers_physical": l_phys, "layers_logical": L,
                "emulated": bool(l_phys < L),
                "decode_tok_s": batch / (step_ms / 1e3), "decode_ms_per_step": step_ms,
                "decode_kernel_ms": kms, "decode_gbs": dec_bytes / (kms / 1e3) / 1e9,
                "decode_hbm_frac": dec_bytes / (kms / 1e3) / 1e9 / peak,
                "decode_hbm_frac_nominal_8tbs": dec_bytes / (kms / 1e3) / 1e9 / NOMINAL_HBM_GBS}
        if batch == 1:
            # one-block cached serve: 24 prefill launches, graph-replayed, L2 flushed
            def serve():
                for layer in range(L):
                    smem.smem_prefill_block(cache.h, 0, layer % l_phys, ctx, *pins, posa, poca)

            serve()
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                serve()
            flush = torch.empty(512 << 20, dtype=torch.uint8, device=device)
            lat, kern = [], []
            for i in range(serve_iters):
                flush.zero_()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(st)
                g.replay()
                b.record(st)
                torch.cuda.synchronize()
                lat.append(a.elapsed_time(b))
            for i in range(serve_iters):
                flush.zero_()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(st)
                smem.smem_prefill_block(cache.h, 0, i % l_phys, ctx, *pins, posa, poca)
                b.record(st)
                torch.cuda.synchronize()
                kern.append(a.elapsed_time(b))
            del g, flush
            pf_bytes = ctx * R * 4 * H * D + 6 * B_TOK * H * D * 2
            pf_flops = 4 * B_TOK * ctx * R * H * D + 4 * (B_TOK * (B_TOK + 1) // 2) * H * D
            km = float(np.median(kern))
            cell.update({"serve_latency_ms": float(np.median(lat)), "prefill_kernel_ms": km,
                         "prefill_gbs": pf_bytes / (km / 1e3) / 1e9,
                         "prefill_hbm_frac": pf_bytes / (km / 1e3) / 1e9 / peak,
                         "prefill_tflops": pf_flops / (km / 1e3) / 1e12,
                         "prefill_tensor_frac": pf_flops / (km / 1e3) / 1e12 / bf16_peak})
        cells.append(cell)
    if smem.smem_check_device_error(cache.h) != smem.OK:
        raise RuntimeError("device error recorded")
    cache.close()
    cache.buf = None
    torch.cuda.empty_cache()
    return cells


def run_long(args):
    """One-block prefill latency and decode tok/s per context length at the
    1.5B reader shape, every batch and context of the workload."""
    import torch

    from paper_2609_32395_gb300 import smem

    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    smem.lib()
    W = LONG
    contexts = [int(x) for x in args.long_contexts.split(",")]
    batches = [int(x) for x in args.long_batches.split(",")]
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    bf16_peak = float(peaks.get("bf16_tflops", 1900.0))
    cells = []
    for batch in batches:
        for cell in long_batch_cells(batch, contexts, device, peak, bf16_peak, layers_cap=args.long_layers):
            cells.append(cell)
            print(json.dumps(cell), file=sys.stderr, flush=True)
    print(json.dumps({"workload": W["name"], "heads": W["H"], "head_dim": W["D"], "layers": W["L"],
                      "peak_hbm_gbs": peak, "peak_source": peak_src, "cells": cells}), flush=True)


# ----------------------------------------------------------------------------- edit latency
EDIT = dict(name="410M-shaped edit churn, 32 sequences", H=16, D=64, seqs=32, contexts=(512, 4096), seed=4)


def measure_edit_latency(ctx, device, n_ops=400):
    """Per-delete and per-append latency with every sequence holding `ctx`
    blocks (block contents do not affect an edit, so every block is filled
    from one zero block). Host time is the whole C ABI call (bookkeeping,
    validation and the launch of the table-edit kernel); device time is the
    table-edit kernel alone."""
    import torch

    from paper_2609_32395_gb300 import smem

    W = EDIT
    S, H, D = W["seqs"], W["H"], W["D"]
    cap = S * ctx + 8
    cfg = smem.make_config(1, H, D, S, ctx + 8, cap)
    cache = smem.SmemCache(cfg, device=device)
    z = torch.zeros((1, H, R, D), dtype=torch.bfloat16, device=device)
    for s in range(S):
        for j in range(ctx):
            smem.smem_append_block(cache.h, s, j, z, z)
    torch.cuda.synchronize()
    rng = np.random.default_rng(W["seed"] + ctx)
    st = torch.cuda.current_stream()
    host_del, host_app, dev_del = [], [], []
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_ops)]
    for i in range(n_ops):
        s = int(rng.integers(0, S))
        j = int(rng.integers(0, ctx))
        ev[i][0].record(st)
        t0 = time.perf_counter()
        smem.smem_delete_block(cache.h, s, j)
        t1 = time.perf_counter()
        ev[i][1].record(st)
        smem.smem_append_block(cache.h, s, j, z, z)
        t2 = time.perf_counter()
        host_del.append(t1 - t0)
        host_app.append(t2 - t1)
        if i % 50 == 49:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    dev_del = [a.elapsed_time(b) * 1e3 for a, b in ev]
    err = smem.smem_check_device_error(cache.h)
    cache.close()
    cache.buf = None
    torch.cuda.empty_cache()
    if err != smem.OK:
        raise RuntimeError("device error recorded during the edit measurement")
    us = lambda v, q: float(np.percentile(np.array(v) * 1e6, q))  # noqa: E731
    return {"context_blocks": ctx, "sequences": S, "delete_host_us_p50": us(host_del, 50),
            "delete_host_us_p99": us(host_del, 99), "append_host_us_p50": us(host_app, 50),
            "delete_device_us_p50": float(np.percentile(dev_del, 50)),
            "append_bytes": 2 * H * R * D * 2}


# ----------------------------------------------------------------------------- oracle (cpu) timing
class OracleDecodeSample:
    """A bounded sample of the default workload for the fp64 CPU oracle: the
    first `n_seqs` sequences at `layers`, inputs generated once. `call(i)`
    runs and times one (sequence, layer) decode call of the oracle."""

    def __init__(self, seqs, n_seqs=3, layers=(0, 13), rank=0):
        import oracle
        import synth

        W = WORKLOAD
        self.L, self.H, self.D = W["L"], W["H"], W["D"]
        s_seed = rank_seed(W["seed"], rank)
        nblk = synth.ragged_contexts(s_seed, seqs, W["ctx_lo"], W["ctx_hi"])
        pos = synth.inblock_positions(s_seed, seqs, B_TOK)
        self.mean_rows = float(nblk.mean()) * R + float(pos.mean()) + 1
        f = oracle.bf16_bits_to_f64
        H, D = self.H, self.D
        self.calls = []
        for s in range(min(n_seqs, seqs)):
            n, p = int(nblk[s]), int(pos[s])
            for layer in layers:
                keys = np.array([synth.stream_key(s_seed, 1, s, j, layer, kind)
                                 for kind in (synth.KIND_K, synth.KIND_V) for j in range(n)], dtype=np.int64)
                rows = synth.normal_bf16_np(keys, H * R * D).reshape(2, n, H, R, D)
                kin = synth.tensor_np(s_seed, synth.KIND_KIN, (B_TOK, H, D), s, layer, 0)[:p]
                vin = synth.tensor_np(s_seed, synth.KIND_VIN, (B_TOK, H, D), s, layer, 0)[:p]
                q = [synth.tensor_np(s_seed, kind, (seqs, H, D), layer, 0)[s]
                     for kind in (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
                self.calls.append(dict(idx=np.arange(n), mk=f(rows[0]), mv=f(rows[1]), n=n, p=p, kin=f(kin),
                                       vin=f(vin), q=[f(x) for x in q], rows=n * R + p + 1))
        self.desc = (f"fp64 C oracle: decode calls (all {H} heads, full contexts) of sequences "
                     f"0..{min(n_seqs, seqs) - 1} at layers {list(layers)}, repeated; time per memory row "
                     f"extrapolated to the workload's mean context and {self.L} layers per token")

    def call(self, i):
        import oracle

        c = self.calls[i % len(self.calls)]
        t0 = time.perf_counter()
        oracle.reader_decode(c["idx"], c["mk"], c["mv"], c["n"], c["p"], c["kin"], c["vin"], *c["q"])
        return time.perf_counter() - t0, c["rows"]

    def tok_per_s(self, secs, rows):
        """Tokens/s of the oracle on the workload, from time spent on rows."""
        per_row = secs / rows
        return 1.0 / (per_row * self.mean_rows * self.L)


def _time_threads(fn, threads):
    """Wall time of fn() with the oracle's per-head loops on `threads`."""
    import oracle

    used = oracle.set_threads(threads)
    t0 = time.perf_counter()
    fn()
    return time.perf_counter() - t0, used


def _oracle_block_rows(seed, seq, ids, layer, H, D, device):
    """fp64 host copies [n][H][R][D] of memory rows from the seeded
    generator (run on the device for speed; the values are the generator's,
    bit for bit the numpy ones)."""
    import synth

    K, V = synth.block_rows_torch(seed, seq, list(ids), 1, H, R, D, device, layers=[layer])
    return K[:, 0].double().cpu().numpy(), V[:, 0].double().cpu().numpy()


def oracle_config_baselines(device, ncores):
    """The fp64 oracle on every workload of the benchmark's configuration
    list, single-threaded and with OpenMP over heads on `ncores` threads.
    Configs 1 and 2 run in full; configs 3-5 on a stated sample, extrapolated
    linearly in memory rows, heads and layers (labelled)."""
    import oracle
    import synth
    from oracle.bookkeeping import CacheMirror

    f = oracle.bf16_bits_to_f64
    out = {}

    def both(fn):
        t1, _ = _time_threads(fn, 1)
        tn, used = _time_threads(fn, ncores)
        return t1, tn, used

    # config 1: tiny reader (H 4, d_h 64, 8 blocks): one-block pass and a decode, in full
    H, D, n = 4, 64, 8
    mk, mv = _oracle_block_rows(0, 0, range(n), 0, H, D, device)
    pin = [f(synth.tensor_np(0, k, (B_TOK, H, D), 0, 1)) for k in
           (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
    t1, tn, used = both(lambda: oracle.reader_prefill(np.arange(n), mk, mv, n, *pin))
    out["tiny"] = {"what": "one-block pass, H 4, d_h 64, 8 blocks (full)", "unit": "ms",
                   "single_thread": 1e3 * t1, "openmp": 1e3 * tn, "threads": used}

    # config 2: 160M one-block serve, 12 layers, 16 / 64 / 256 blocks; OpenMP
    # in full, single thread in full at 16 / 64 blocks and on layers {0, 11}
    # at 256 blocks (x6, labelled)
    H, D, L = SERVE["H"], SERVE["D"], SERVE["L"]
    cells = []
    for nblk in SERVE["contexts"]:
        t1 = tn = 0.0
        single_layers = range(L) if nblk <= 64 else (0, L - 1)
        for layer in range(L):
            mk, mv = _oracle_block_rows(SERVE["seed"], 0, range(nblk), layer, H, D, device)
            pin = [f(synth.tensor_np(SERVE["seed"], k, (B_TOK, H, D), layer, 0)) for k in
                   (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
            fn = lambda: oracle.reader_prefill(np.arange(nblk), mk, mv, nblk, *pin)  # noqa: E731
            if layer in single_layers:
                t1 += _time_threads(fn, 1)[0]
            b, used = _time_threads(fn, ncores)
            tn += b
        cell = {"context_blocks": nblk, "single_thread_ms": 1e3 * t1 * L / len(single_layers), "openmp_ms": 1e3 * tn}
        if len(single_layers) < L:
            cell["single_thread_extrapolated"] = f"layers {list(single_layers)} x {L / len(single_layers):g}"
        cells.append(cell)
    out["serve_160m"] = {"what": f"one-block serve, {L} layers, H {H}, d_h {D} (OpenMP: full)", "threads": used,
                         "unit": "ms", "cells": cells}

    # config 4: 1.5B long context; sample: layer 0 at 512 blocks (one-block
    # pass: every head with OpenMP, heads 0-1 single-threaded; batch-1 decode:
    # every head), extrapolated per memory row, head and layer to 24 layers
    H, D, L, n = LONG["H"], LONG["D"], LONG["L"], 512
    mk, mv = _oracle_block_rows(LONG["seed"], 0, range(n), 0, H, D, device)
    pin = [f(synth.tensor_np(LONG["seed"], k, (B_TOK, H, D), 0, 0)) for k in
           (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
    dq = [f(synth.tensor_np(LONG["seed"], k, (1, H, D), 0, 0))[0] for k in
          (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    mk2, mv2 = np.ascontiguousarray(mk[:, :2]), np.ascontiguousarray(mv[:, :2])
    pin2 = [np.ascontiguousarray(x[:, :2]) for x in pin]
    p1 = _time_threads(lambda: oracle.reader_prefill(np.arange(n), mk2, mv2, n, *pin2), 1)[0] * H / 2
    pn, used = _time_threads(lambda: oracle.reader_prefill(np.arange(n), mk, mv, n, *pin), ncores)
    d1, dn, _ = both(lambda: oracle.reader_decode(np.arange(n), mk, mv, n, 0, None, None, *dq))
    cells = []
    for ctx in LONG["contexts"]:
        k = ctx / n * L
        cells.append({"context_blocks": ctx, "serve_single_thread_ms": 1e3 * p1 * k, "serve_openmp_ms": 1e3 * pn * k,
                      "decode_single_thread_tok_s": 1.0 / (d1 * k), "decode_openmp_tok_s": 1.0 / (dn * k)})
    out["long_1p5b"] = {"what": f"H {H}, d_h {D}, {L} layers; sample: layer 0 at {n} blocks, one-block pass "
                                f"(single thread: heads 0-1) and batch-1 decode; extrapolated per memory row, head "
                                f"and layer", "extrapolated": True, "threads": used, "cells": cells}

    # config 5: churn at the 410M shape; the oracle's bookkeeping mirror times its
    # deletes, the attention oracle one sequence's decode at 4096 blocks (layer 0)
    H, D = EDIT["H"], EDIT["D"]
    cells = []
    for ctx in EDIT["contexts"]:
        m = CacheMirror(EDIT["seqs"] * (ctx + 8), EDIT["seqs"], ctx + 8)
        for sq in range(EDIT["seqs"]):
            for j in range(ctx):
                m.append(sq, j)
        rng = np.random.default_rng(ctx)
        victims = [(int(rng.integers(0, EDIT["seqs"])), int(j)) for j in rng.choice(ctx, 200, replace=False)]
        t0 = time.perf_counter()
        for sq, j in victims:
            m.delete(sq, j)
        cells.append({"context_blocks": ctx, "mirror_delete_us": 1e6 * (time.perf_counter() - t0) / len(victims)})
    n = max(EDIT["contexts"])
    mk, mv = _oracle_block_rows(EDIT["seed"], 0, range(n), 0, H, D, device)
    dq = [f(synth.tensor_np(EDIT["seed"], k, (1, H, D), 0, 0))[0] for k in
          (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    d1, dn, used = both(lambda: oracle.reader_decode(np.arange(n), mk, mv, n, 0, None, None, *dq))
    out["churn_410m"] = {"what": f"bookkeeping mirror deletes (32 sequences); decode of one sequence at {n} blocks, "
                                 "one layer, all heads", "threads": used, "cells": cells,
                         "decode_ms_single_thread": 1e3 * d1, "decode_ms_openmp": 1e3 * dn}
    return out


def oracle_baseline(seqs, device=None, budget_s=10.0, configs=True):
    """The headline (config 3) oracle time, single-threaded and with OpenMP
    over heads on every host core, plus the per-config table."""
    import oracle

    ncores = os.cpu_count() or 1
    samp = OracleDecodeSample(seqs)

    def timed(threads, budget):
        used = oracle.set_threads(threads)
        secs = rows = 0.0
        n = 0
        while secs < budget or n < len(samp.calls):
            t, r = samp.call(n)
            secs += t
            rows += r
            n += 1
        return samp.tok_per_s(secs, rows), used, n, secs

    v1, _, n1, s1 = timed(1, budget_s)
    vn, used, nn, sn = timed(ncores, budget_s / 2)
    desc = samp.desc.replace("single thread: ", "")
    res = {"value": vn, "unit": "tok/s", "cores": used, "kind": "oracle",
           "sample": f"{desc}; OpenMP over heads on {used} threads ({ncores} host cores); {nn} calls, "
                     f"{sn:.1f} s; extrapolated",
           "single_thread": {"value": v1, "unit": "tok/s", "cores": 1, "calls": n1, "seconds": s1},
           "host_cores": ncores}
    if configs and device is not None:
        res["configs"] = oracle_config_baselines(device, ncores)
    oracle.set_threads(ncores)
    return res


# ----------------------------------------------------------------------------- arms
def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle

    W = WORKLOAD
    samp = OracleDecodeSample(args.seqs)
    used = oracle.set_threads(os.cpu_count() or 1)
    secs = rows = 0.0
    for i in range(args.warmup + args.steps):
        t, r = samp.call(i)
        if i >= args.warmup:
            secs += t
            rows += r
    value = samp.tok_per_s(secs, rows)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tok/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": W["name"], "layers": W["L"], "heads": W["H"], "head_dim": W["D"],
                   "sequences": args.seqs, "context_blocks": [W["ctx_lo"], W["ctx_hi"]], "block": B_TOK},
        "cpu_baseline": {"value": value, "unit": "tok/s", "cores": used, "kind": "oracle",
                         "sample": f"each step one call; OpenMP over heads on {used} threads; {samp.desc}"},
        "e2e": {"value": value, "unit": "tok/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch

    from paper_2609_32395_gb300 import smem

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    smem.lib()  # fails loudly without the CUDA library

    e2e_steps = 0 if args.no_e2e else min(args.steps, 64)
    layer_steps = 0 if args.no_layer else min(args.steps, 64)
    wl = DecodeWorkload(args.seqs, args.warmup + args.steps + e2e_steps + 2 + (layer_steps + args.warmup),
                        WORKLOAD["seed"], device, rank, layers=args.layers)

    def barrier():
        if ws > 1:
            import torch.distributed as dist

            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        wl.step()
    barrier()

    # --- timed region (device-resident inputs)
    rows, bytes_alg = [], []
    st = torch.cuda.current_stream()
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(wl.L)] for _ in range(2)]
          for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches = 0
    with ClockSampler(local) as clk:
        barrier()
        torch.cuda.nvtx.range_push("timed")
        start.record(st)
        for i in range(args.steps):
            r = wl.rows_read()
            rows.append(r)
            launches += wl.step(events=ev[i])
        end.record(st)
        torch.cuda.nvtx.range_pop()
        barrier()
    elapsed = start.elapsed_time(end) / 1e3
    # per-launch durations of the decode kernel
    kern_ms = [ev[i][0][l].elapsed_time(ev[i][1][l]) for i in range(args.steps) for l in range(wl.L)]
    row_bytes = 4 * wl.H * wl.D  # K + V bf16 per row per layer
    alg_bytes = [r * row_bytes for r in rows for _ in range(wl.L)]
    achieved = sum(alg_bytes) / (sum(kern_ms) / 1e3) / 1e9

    tokens = args.steps * args.seqs
    elapsed = max_over_ranks(elapsed, device)
    value = tokens * ws / elapsed

    # --- end to end: host inputs / outputs / appended rows through the C ABI
    e2e = None
    if e2e_steps:
        pin = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True).copy_(t.cpu())  # noqa: E731
        host_in = [[[pin(x) for x in wl.inputs[k][l]] for l in range(wl.L)] for k in range(wl.n_sets)]
        host_out = [[torch.empty(wl.osa.shape, dtype=torch.bfloat16, pin_memory=True) for _ in range(wl.L)]
                    for _ in range(2)]
        host_blk = (pin(wl.new_K[0][0]), pin(wl.new_V[0][0]))
        appends_before = sum(wl.new_used)
        barrier()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            wl.step(host_inputs=host_in, host_outputs=host_out, host_blocks=host_blk)
            torch.cuda.current_stream().synchronize()  # the step's outputs are on the host
        barrier()
        e2e_el = time.perf_counter() - t0
        n_app = sum(wl.new_used) - appends_before
        h2d = wl.L * 4 * args.seqs * wl.H * wl.D * 2 + n_app / e2e_steps * 2 * host_blk[0].numel() * 2
        d2h = wl.L * 2 * args.seqs * wl.H * wl.D * 2
        e2e_el = max_over_ranks(e2e_el, device)
        e2e = {"value": e2e_steps * args.seqs * ws / e2e_el, "unit": "tok/s",
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)}

    err = smem.smem_check_device_error(wl.h)
    if err != smem.OK:
        raise RuntimeError("device error recorded during the benchmark")

    # --- the full reader layer around the attention (projections, LayerNorm, FFN)
    layer_dec = measure_layer_decode(wl, layer_steps, args.warmup, device) if layer_steps else None

    # --- one-block cached-context serve (prefill), the metric's second half
    serve = layer_serve = rec_serve = None
    recompute = None
    if not args.no_recompute and rank == 0:
        recompute = measure_recompute(min(args.steps, 64), args.warmup, device, args.seqs, layers=args.layers)
    rope = None
    if not args.no_rope and rank == 0:
        wl.cache.close()
        wl.cache.buf = None
        torch.cuda.empty_cache()
        rope = {"decode": measure_decode_variant(min(args.steps, 64), args.warmup, device, args.seqs, layers=args.layers)}
    gqa = None
    if not args.no_gqa and rank == 0:
        gqa = measure_decode_variant(min(args.steps, 32), args.warmup, device, args.seqs, layers=args.layers, window=0,
                                     kv_heads=WORKLOAD["H"] // 4)
    d32 = None
    if not args.no_d32 and rank == 0:
        # the paper's head width: 32 heads of d_h = 32 at the same d = 1024
        d32 = measure_decode_variant(min(args.steps, 32), args.warmup, device, args.seqs, layers=args.layers, window=0,
                                  heads=WORKLOAD["H"] * WORKLOAD["D"] // 32)
    if not args.no_serve:
        wl.cache.close()
        wl.cache.buf = None
        del wl.new_K, wl.new_V
        torch.cuda.empty_cache()
        serve = [measure_serve(n, device) for n in SERVE["contexts"]]
        layer_serve = None if args.no_layer else [measure_layer_serve(n, device) for n in SERVE["contexts"]]
        if not args.no_layer and not args.no_recompute:
            rec_serve = [measure_layer_serve(n, device, recompute=True) for n in SERVE["contexts"]]
        if rope is not None:
            rope["serve"] = [measure_serve(n, device, rope_window=ROPE_WINDOW) for n in SERVE["contexts"]]
    edit = None if args.no_serve else [measure_edit_latency(n, device) for n in EDIT["contexts"]]
    long_cells = None
    if not args.no_long and rank == 0:
        # the 1.5B long-context cells, bounded: batch 1 at 1024 and 4096 blocks
        # and batch 16 at 1024, on two physical layers (24-layer emulated)
        wl.cache.close()
        wl.cache.buf = None
        torch.cuda.empty_cache()
        pk, _ = measured_peaks()
        hbm, tf = float(pk.get("hbm_gbs", FALLBACK_HBM_GBS)), float(pk.get("bf16_tflops", 1900.0))
        long_cells = long_batch_cells(1, [1024, 4096], device, hbm, tf, layers_cap=2)
        long_cells += long_batch_cells(16, [1024], device, hbm, tf, layers_cap=2)

    if rank != 0:
        if ws > 1:
            import torch.distributed as dist

            dist.destroy_process_group()
        return

    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    units_launch = float(np.mean(rows))
    traffic = profiled_traffic("decode_410m.txt", units_launch)
    cpu = None if args.no_cpu_baseline else oracle_baseline(args.seqs, device)
    line = {
        "metric": METRIC, "value": value, "unit": "tok/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOAD["name"], "layers": wl.L, "heads": wl.H, "head_dim": wl.D,
                   "sequences": args.seqs, "context_blocks": [WORKLOAD["ctx_lo"], WORKLOAD["ctx_hi"]],
                   "block": B_TOK, "rows_per_block": R, "pool_bytes": int(wl.cache.nbytes),
                   "l2": "inputs larger than L2 (pool of memory rows >> 129 MB); no flush",
                   "parallelism": f"independent sequences per GPU x{ws}"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "frac_nominal_8tbs": achieved / NOMINAL_HBM_GBS, "traffic": traffic,
                     "kernel": "decode_kernel<64> (split-K paged cross-attention + in-block self-attention)",
                     "peak_source": f"{peak_src} hbm_gbs", "kernel_ms_mean": float(np.mean(kern_ms)),
                     "alg_bytes_per_launch": float(np.mean(alg_bytes))},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    if serve:
        bf16_peak = float(peaks.get("bf16_tflops", 1900.0))
        for sv in serve:
            gbs = sv["bytes_per_launch"] / (sv["kernel_ms_mean"] / 1e3) / 1e9
            tfs = sv["flops_per_launch"] / (sv["kernel_ms_mean"] / 1e3) / 1e12
            tr = profiled_traffic("prefill_160m.txt", sv["memory_rows"], exact=True)
            sv["roofline"] = {"bound": "hbm", "achieved_gbs": gbs, "hbm_frac": gbs / peak, "traffic": tr,
                              "achieved_tflops": tfs, "tensor_frac": tfs / bf16_peak,
                              "peak_tflops_bf16": bf16_peak}
        line["serve"] = {"workload": SERVE["name"], "layers": SERVE["L"], "heads": SERVE["H"],
                         "head_dim": SERVE["D"], "metric": "one-block cached-serve latency (12 layers)",
                         "unit": "ms", "timing": "CUDA graph of the 12 per-layer launches, L2 flushed before each",
                         "cells": serve}
    if layer_dec or layer_serve:
        layer = {"what": "full reader layer: pre-LN self-attention, cross-attention and 4d GELU FFN "
                         "branches with random-init bf16 weights (projections on the library's tcgen05 "
                         "kernel, LayerNorm / residual / GELU fused)"}
        if layer_dec:
            layer_dec["hbm_frac"] = layer_dec["achieved_gbs"] / peak
            layer["decode"] = dict(workload=WORKLOAD["name"], unit="tok/s", steps=layer_steps, **layer_dec)
        if layer_serve:
            for c in layer_serve:
                c["hbm_frac"] = c["achieved_gbs"] / peak
            layer["serve"] = {"workload": SERVE["name"], "unit": "ms", "cells": layer_serve,
                              "timing": "CUDA graph of the 12 layer calls, L2 flushed before each"}
        line["layer"] = layer
    if gqa:
        gqa["hbm_frac"] = gqa["achieved_gbs"] / peak
        gqa["workload"] = WORKLOAD["name"] + " with 4 key/value heads shared by groups of 4 query heads"
        # DRAM bytes per launch from the committed ncu summary (32-sequence
        # capture, scaled by the rows read; null once the kernel changed)
        gqa["traffic"] = profiled_traffic("decode_gqa_410m.txt", gqa["rows_per_launch"])
        line["gqa"] = gqa
    if d32:
        d32["hbm_frac"] = d32["achieved_gbs"] / peak
        d32["workload"] = WORKLOAD["name"] + " with 32 heads of d_h = 32 (the same d)"
        line["d32"] = d32
    if rope:
        rope["decode"]["hbm_frac"] = rope["decode"]["achieved_gbs"] / peak
        rope["workload"] = WORKLOAD["name"] + " and " + SERVE["name"] + ", SMem+RoPE composite (window 15)"
        line["rope"] = rope
    if recompute:
        k = recompute["memory_row_kernel"]
        k["hbm_frac"] = k["achieved_gbs"] / peak
        # DRAM bytes of one launch from the committed ncu summary (16-sequence
        # capture, scaled by the memory rows read; null once the kernel changed)
        k["traffic"] = profiled_traffic("mu_decode_410m.txt", k["rows_per_launch"])
        if rec_serve:
            for c in rec_serve:
                c["hbm_frac"] = c["achieved_gbs"] / peak
            recompute["layer_serve"] = {"workload": SERVE["name"] + ", recompute-K/V cache", "unit": "ms",
                                        "cells": rec_serve}
        line["recompute"] = recompute
    if edit:
        line["edit"] = {"workload": EDIT["name"], "unit": "us",
                        "note": "host = whole C ABI call; device = table-edit kernel; no row moves", "cells": edit}
    if long_cells:
        line["long"] = {"workload": LONG["name"], "heads": LONG["H"], "head_dim": LONG["D"], "layers": LONG["L"],
                        "note": "24 logical layers cycled over 2 physical layers (24-layer emulated; each "
                                "physical layer's K/V far above L2); fractions of the measured HBM copy peak and "
                                "of the measured bf16 burst peak",
                        "cells": long_cells}
    if e2e:
        line["e2e"] = e2e
    if cpu:
        line["cpu_baseline"] = cpu
    print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def run_serve_only(args):
    import torch

    from paper_2609_32395_gb300 import smem

    torch.cuda.set_device(0)
    smem.lib()
    cells = [measure_serve(n, torch.device("cuda", 0)) for n in SERVE["contexts"]]
    out = {"serve_only": True, "workload": SERVE["name"], "cells": cells}
    if not args.no_recompute:  # the full reader layer on a recompute-K/V cache
        out["recompute_layer_cells"] = [measure_layer_serve(n, torch.device("cuda", 0), recompute=True)
                                        for n in SERVE["contexts"]]
    print(json.dumps(out), flush=True)


def main():
    args = parse_args()
    if args.only_serve:
        run_serve_only(args)
        return
    if args.workload == "long":
        run_long(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
