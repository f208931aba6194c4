"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times, on outputs the fp64 oracle computes one (sequence, head) at
a time; plus the edit-churn workload's bitwise replay.

A launch handles one layer; its grid and split plan depend only on the block
counts, the head count and the head dimension, so one physical layer gives
the benchmark's per-layer launch."""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2609_32395_gb300 import smem
from tests.gpu_helpers import MAX_ABS, MEAN_ABS, REL_L2, assert_close, f64, out_f64

pytestmark = pytest.mark.gpu
R = 64
B_TOK = 64


def build_cache(seed, nblks, H, D, L=1, extra=8, perm_seed=None):
    S = len(nblks)
    cap = int(sum(nblks)) + extra
    perm = synth.slot_permutation(seed if perm_seed is None else perm_seed, cap)
    cfg = smem.make_config(L, H, D, S, int(max(nblks)) + extra, cap, free_order=perm)
    cache = smem.SmemCache(cfg, device="cuda")
    for s, n in enumerate(nblks):
        for b0 in range(0, n, 32):
            ids = list(range(b0, min(n, b0 + 32)))
            K, V = synth.block_rows_torch(seed, s, ids, L, H, R, D, "cuda")
            for i, j in enumerate(ids):
                smem.smem_append_block(cache.h, s, j, K[i], V[i])
    torch.cuda.synchronize()
    return cache


def head_memory(seed, seq, nblk, layer, h, D):
    k, v = synth.block_head_rows_np(seed, seq, list(range(nblk)), layer, h, R, D)
    return f64(k)[:, None], f64(v)[:, None]  # [n][1][R][D]


def test_decode_410m_launch_sampled():
    """64 sequences, contexts uniform in [64, 256] blocks, in-block offsets
    uniform in [0, 63], H = 16, d_h = 64, shuffled slots: the bench's decode
    launch. Six sequences x two heads checked against the oracle."""
    seed, H, D = 0, 16, 64
    nblk = synth.ragged_contexts(seed, 64, 64, 256)
    pos = synth.inblock_positions(seed, 64, B_TOK)
    cache = build_cache(seed, nblk, H, D)
    for s in range(64):
        p = int(pos[s])
        if p:
            Kb = synth.tensor_torch(seed, synth.KIND_KIN, (p, H, D), s, 0, 0, device="cuda")
            Vb = synth.tensor_torch(seed, synth.KIND_VIN, (p, H, D), s, 0, 0, device="cuda")
            smem.smem_write_inblock(cache.h, s, 0, p, Kb, Vb)
    shape = (64, H, D)
    ins = [synth.tensor_np(seed, k, shape, 0, 0) for k in
           (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    dev = [synth.bits_to_torch_bf16(x).cuda() for x in ins]
    osa = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    oca = torch.empty_like(osa)
    smem.smem_decode(cache.h, 0, np.arange(64), pos, nblk, *dev, osa, oca)
    torch.cuda.synchronize()
    got_sa, got_ca = out_f64(osa), out_f64(oca)
    for s in (0, 9, 23, 40, 51, 63):
        p, n = int(pos[s]), int(nblk[s])
        kin_all = synth.tensor_np(seed, synth.KIND_KIN, (max(p, 1), H, D), s, 0, 0)[:p]
        vin_all = synth.tensor_np(seed, synth.KIND_VIN, (max(p, 1), H, D), s, 0, 0)[:p]
        for h in (3, 14):
            mk, mv = head_memory(seed, s, n, 0, h, D)
            q = [f64(x[s, h])[None] for x in ins]
            ref_sa, ref_ca = oracle.reader_decode(np.arange(n), mk, mv, n, p, f64(kin_all[:, h:h + 1]),
                                                  f64(vin_all[:, h:h + 1]), *q)
            assert_close(got_sa[s, h], ref_sa[0], f"osa seq {s} head {h}")
            assert_close(got_ca[s, h], ref_ca[0], f"oca seq {s} head {h}")
    assert smem.smem_check_device_error(cache.h) == smem.OK


def test_long_context_1p5b_sampled():
    """1.5B reader shape (H = 16, d_h = 128) with 4096 cached blocks (262144
    memory rows): one-block prefill at 4096 and at the 512 / 1024 prefixes, and
    a batch-1 decode at 4096, checked on sampled heads."""
    seed, H, D, N = 2, 16, 128, 4096
    cache = build_cache(seed, [N], H, D)
    shape = (B_TOK, H, D)
    pin = [synth.tensor_np(seed, k, shape, 0, 7) for k in
           (synth.KIND_QS, synth.KIND_KS, synth.KIND_VS, synth.KIND_QC)]
    dev = [synth.bits_to_torch_bf16(x).cuda() for x in pin]
    mem = {}
    for q_idx, heads in ((N, (0, 11)), (1024, (6,)), (512, (15,))):
        osa = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_prefill_block(cache.h, 0, 0, q_idx, *dev, osa, oca)
        torch.cuda.synchronize()
        got_sa, got_ca = out_f64(osa), out_f64(oca)
        for h in heads:
            if h not in mem:
                mem[h] = head_memory(seed, 0, q_idx, 0, h, D)
            mk, mv = mem[h]
            x = [f64(t[:, h:h + 1]) for t in pin]
            ref_sa, ref_ca = oracle.reader_prefill(np.arange(q_idx), mk[:q_idx], mv[:q_idx], q_idx, *x)
            assert_close(got_sa[:, h], ref_sa[:, 0], f"prefill osa head {h} ctx {q_idx}")
            assert_close(got_ca[:, h], ref_ca[:, 0], f"prefill oca head {h} ctx {q_idx}")
    # batch-1 decode at the full context, new token at offset 0
    dshape = (1, H, D)
    din = [synth.tensor_np(seed, k, dshape, 0, 3) for k in
           (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    ddev = [synth.bits_to_torch_bf16(x).cuda() for x in din]
    osa = torch.empty(dshape, dtype=torch.bfloat16, device="cuda")
    oca = torch.empty_like(osa)
    smem.smem_decode(cache.h, 0, [0], [0], [N], *ddev, osa, oca)
    torch.cuda.synchronize()
    for h in (0, 11):
        mk, mv = mem[h]
        q = [f64(x[0, h])[None] for x in din]
        ref_sa, ref_ca = oracle.reader_decode(np.arange(N), mk, mv, N, 0, None, None, *q)
        assert_close(out_f64(osa[0, h]), ref_sa[0], f"decode osa head {h}")
        assert_close(out_f64(oca[0, h]), ref_ca[0], f"decode oca head {h}")
    assert smem.smem_check_device_error(cache.h) == smem.OK


def test_decode_batch_above_one_launch():
    """600 sequences (more than one launch's 512 items) with one block each."""
    S, H, D = 600, 2, 64
    cache = build_cache(5, [1] * S, H, D)
    shape = (S, H, D)
    ins = [synth.tensor_np(5, k, shape, 0, 0) for k in
           (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    dev = [synth.bits_to_torch_bf16(x).cuda() for x in ins]
    osa = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    oca = torch.empty_like(osa)
    smem.smem_decode(cache.h, 0, np.arange(S), np.zeros(S), np.ones(S), *dev, osa, oca)
    torch.cuda.synchronize()
    got_sa, got_ca = out_f64(osa), out_f64(oca)
    for s in (0, 311, 511, 512, 599):
        mk, mv = synth.block_rows_np(5, s, 0, 1, H, R, D)
        q = [f64(x[s]) for x in ins]
        ref_sa, ref_ca = oracle.reader_decode([0], f64(mk[0])[None], f64(mv[0])[None], 1, 0, None, None, *q)
        assert_close(got_sa[s], ref_sa, f"osa seq {s}")
        assert_close(got_ca[s], ref_ca, f"oca seq {s}")


def _churn_ops(seed, S, nblk0, n_ops):
    """Seeded op stream: 40% delete of a random live block, 40% append of a
    sequence's next fresh block index, 20% decode steps."""
    rng = np.random.default_rng(seed)
    live = [set(range(nblk0)) for _ in range(S)]
    fresh = [nblk0] * S
    ops = []
    for _ in range(n_ops):
        u = rng.random()
        if u < 0.4:
            s = int(rng.integers(0, S))
            if not live[s]:
                continue
            j = int(rng.choice(sorted(live[s])))
            live[s].discard(j)
            ops.append(("del", s, j))
        elif u < 0.8:
            s = int(rng.integers(0, S))
            j = fresh[s]
            fresh[s] += 1
            live[s].add(j)
            ops.append(("app", s, j))
        else:
            ops.append(("dec",))
    return ops, live, fresh


def _replay_order(ops, seed):
    """A different order of the same ops reaching the same block set: edits
    in a random topological order (a block appended in the stream is deleted
    only after its append), decode steps in their original relative order at
    random positions."""
    rng = np.random.default_rng(seed)
    edits = [o for o in ops if o[0] != "dec"]
    decs = [o for o in ops if o[0] == "dec"]
    appended = {(o[1], o[2]) for o in edits if o[0] == "app"}
    placed = set()
    remaining = list(edits)
    order = []
    while remaining:
        avail = [i for i, o in enumerate(remaining)
                 if o[0] == "app" or (o[1], o[2]) not in appended or (o[1], o[2]) in placed]
        o = remaining.pop(avail[int(rng.integers(0, len(avail)))])
        if o[0] == "app":
            placed.add((o[1], o[2]))
        order.append(o)
    slots = sorted(rng.choice(len(order) + len(decs), size=len(decs), replace=False).tolist())
    out, ei, di = [], 0, 0
    for k in range(len(order) + len(decs)):
        if di < len(decs) and k == slots[di]:
            out.append(decs[di])
            di += 1
        else:
            out.append(order[ei])
            ei += 1
    return out


@pytest.mark.parametrize("N0", [512, 4096])
def test_churn_410m_replay_bitwise(N0):
    """32 sequences x 512 or 4096 blocks (H = 16, d_h = 64, one physical
    layer: 34 GB per cache at 4096): a seeded stream of 2000 edit / decode
    ops, a permuted replay reaching the same block set, and a cache built
    directly from that set give bitwise-identical probe decodes; the probe
    matches the oracle on sampled heads. At 4096 blocks every probe item
    reads on the long-context split plan."""
    seed, S, H, D = 4, 32, 16, 64
    ops, live, fresh = _churn_ops(seed, S, N0, 2000)
    n_new = sum(1 for o in ops if o[0] == "app")  # slot headroom for every append
    pool_new = {}

    def new_block(s, j):
        if (s, j) not in pool_new:
            K, V = synth.block_rows_torch(seed, s, [j], 1, H, R, D, "cuda")
            pool_new[(s, j)] = (K[0], V[0])
        return pool_new[(s, j)]

    dshape = (S, H, D)
    dec_in = [synth.bits_to_torch_bf16(synth.tensor_np(seed, k, dshape, 0, 1)).cuda() for k in
              (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    scratch = (torch.empty(dshape, dtype=torch.bfloat16, device="cuda"),
               torch.empty(dshape, dtype=torch.bfloat16, device="cuda"))

    def run(op_list, perm_seed):
        cache = build_cache(seed, [N0] * S, H, D, extra=n_new + 8, perm_seed=perm_seed)
        cap = S * N0 + n_new + 8
        # enough slots for every append (the extra covers the largest per-seq growth only)
        step = 0
        for o in op_list:
            if o[0] == "del":
                smem.smem_delete_block(cache.h, o[1], o[2])
            elif o[0] == "app":
                K, V = new_block(o[1], o[2])
                smem.smem_append_block(cache.h, o[1], o[2], K, V)
            else:
                qidx = [fresh[s] + 1 for s in range(S)]
                smem.smem_decode(cache.h, 0, np.arange(S), np.full(S, step % B_TOK), qidx, *dec_in, *scratch)
                step += 1
        return cache, cap

    c1, _ = run(ops, 100)
    c2, _ = run(_replay_order(ops, 7), 200)
    qidx = [fresh[s] + 1 for s in range(S)]
    probes = []
    for c in (c1, c2):
        osa = torch.empty(dshape, dtype=torch.bfloat16, device="cuda")
        oca = torch.empty_like(osa)
        smem.smem_decode(c.h, 0, np.arange(S), np.zeros(S), qidx, *dec_in, osa, oca)
        torch.cuda.synchronize()
        probes.append(oca.view(torch.int16).clone())
        assert smem.smem_check_device_error(c.h) == smem.OK
    for s in range(S):
        assert smem.smem_get_table(c1.h, s)[0] == sorted(live[s])
        assert smem.smem_get_table(c2.h, s)[0] == sorted(live[s])
    assert torch.equal(probes[0], probes[1])
    # a cache built directly from the final block set
    c1.close()
    c2.close()
    del c1, c2
    torch.cuda.empty_cache()
    total = sum(len(x) for x in live)
    cfg = smem.make_config(1, H, D, S, max(fresh) + 8, total + 8, free_order=synth.slot_permutation(300, total + 8))
    c3 = smem.SmemCache(cfg, device="cuda")
    for s in range(S):
        old = [j for j in sorted(live[s]) if j < N0]
        for b0 in range(0, len(old), 64):  # original blocks, generated 64 at a time
            ids = old[b0:b0 + 64]
            K, V = synth.block_rows_torch(seed, s, ids, 1, H, R, D, "cuda")
            for i, j in enumerate(ids):
                smem.smem_append_block(c3.h, s, j, K[i], V[i])
        for j in sorted(live[s]):
            if j >= N0:
                K, V = new_block(s, j)
                smem.smem_append_block(c3.h, s, j, K, V)
    osa = torch.empty(dshape, dtype=torch.bfloat16, device="cuda")
    oca = torch.empty_like(osa)
    smem.smem_decode(c3.h, 0, np.arange(S), np.zeros(S), qidx, *dec_in, osa, oca)
    torch.cuda.synchronize()
    assert torch.equal(oca.view(torch.int16), probes[0])
    # oracle on two sequences x one head
    got = out_f64(oca)
    ins = [synth.tensor_np(seed, k, dshape, 0, 1) for k in
           (synth.KIND_QDEC_S, synth.KIND_KNEW, synth.KIND_VNEW, synth.KIND_QDEC_C)]
    for s, h in ((3, 5), (30, 12)):
        blocks = sorted(live[s])
        k, v = synth.block_head_rows_np(seed, s, blocks, 0, h, R, D)
        q = [f64(x[s, h])[None] for x in ins]
        ref_sa, ref_ca = oracle.reader_decode(blocks, f64(k)[:, None], f64(v)[:, None], qidx[s], 0, None, None, *q)
        assert_close(got[s, h], ref_ca[0], f"churn probe oca seq {s} head {h}")
