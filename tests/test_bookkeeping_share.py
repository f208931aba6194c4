"""Block sharing with reference-counted slots (exact reuse of a cached block
by other tables; arXiv 2609.32395, Sec. 2 "Exact composition", Theorem 1):

* the independent mirror against a hand-worked golden example;
* the C ABI (bookkeeping-only caches, no CUDA) against the mirror, bit for
  bit, on the golden example and on seeded random streams of appends,
  shares, deletes and releases -- tables, slots, FIFO order, reference counts
  and error codes;
* invariants: a slot is free exactly when no entry names it; every live slot
  is named as many times as its count says.
"""
import os
import random

import pytest

from oracle import bookkeeping as bk
from oracle.bookkeeping import CacheMirror
from paper_2609_32395_gb300 import smem

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "bookkeeping_share.txt")
RC = {"OK": bk.OK, "INVALID_ARG": bk.ERR_INVALID_ARG, "NO_SUCH_SEQ": bk.ERR_NO_SUCH_SEQ,
      "DUPLICATE_BLOCK": bk.ERR_DUPLICATE_BLOCK, "NO_SUCH_BLOCK": bk.ERR_NO_SUCH_BLOCK,
      "POOL_FULL": bk.ERR_POOL_FULL, "TABLE_FULL": bk.ERR_TABLE_FULL}


def parse(path=GOLDEN):
    steps = []
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        lhs, rhs = line.split("->")
        op, *args = lhs.split()
        parts = [p.strip() for p in rhs.split("|")]
        rc, slot = parts[0].split()
        tables = [[] if t == "-" else [tuple(int(x) for x in e.split(":")) for e in t.split()] for t in parts[1:3]]
        fifo = [] if parts[3] == "-" else [int(x) for x in parts[3].split()]
        refs = [int(x) for x in parts[4].split()]
        steps.append(dict(op=op, args=[int(a) for a in args], rc=RC[rc], slot=None if slot == "-" else int(slot),
                          tables=tables, fifo=fifo, refs=refs))
    return steps


def mirror_step(m, st):
    a = st["args"]
    if st["op"] == "append":
        rc, s = m.append(*a)
        return rc, (s if rc == 0 else None)
    if st["op"] == "share":
        rc, s = m.share(*a)
        return rc, (s if rc == 0 else None)
    if st["op"] == "delete":
        return m.delete(*a), None
    return m.release(*a), None


def abi_step(h, st):
    import ctypes
    a = st["args"]
    L = smem.lib()
    slot = ctypes.c_int32(-1)
    if st["op"] == "append":
        rc = L.smem_append_block(h, a[0], a[1], None, None, None, ctypes.byref(slot))
    elif st["op"] == "share":
        rc = L.smem_share_block(h, a[0], a[1], a[2], a[3], None, ctypes.byref(slot))
    elif st["op"] == "delete":
        rc = L.smem_delete_block(h, a[0], a[1], None)
    else:
        rc = L.smem_release_seq(h, a[0], None)
    return rc, (slot.value if rc == 0 and st["op"] in ("append", "share") else None)


def check_invariants(m):
    named = {}
    for sl in m.slot:
        for s in sl:
            named[s] = named.get(s, 0) + 1
    for s in range(m.capacity):
        assert m.refs[s] == named.get(s, 0)
        assert (s in m.fifo) == (m.refs[s] == 0)
    assert len(set(m.fifo)) == len(m.fifo)


def test_mirror_matches_golden():
    m = CacheMirror(3, 2, 3)
    for st in parse():
        rc, slot = mirror_step(m, st)
        assert (rc, slot) == (st["rc"], st["slot"]), st
        assert [list(zip(*m.table(s))) for s in (0, 1)] == st["tables"], st
        assert m.free_list() == st["fifo"], st
        assert m.refs == st["refs"], st
        check_invariants(m)


def abi_state(h, cap):
    tabs = []
    for s in (0, 1):
        idx, slots = smem.smem_get_table(h, s)
        tabs.append(list(zip(idx, slots)))
    return tabs, smem.smem_get_free_fifo(h), [smem.smem_slot_refs(h, s) for s in range(cap)]


def test_abi_matches_golden():
    h = smem.smem_cache_create(smem.make_config(1, 1, 64, 2, 3, 3), None)
    try:
        for st in parse():
            rc, slot = abi_step(h, st)
            assert (rc, slot) == (st["rc"], st["slot"]), st
            tabs, fifo, refs = abi_state(h, 3)
            assert tabs == st["tables"] and fifo == st["fifo"] and refs == st["refs"], st
    finally:
        smem.smem_cache_destroy(h)


@pytest.mark.parametrize("rope", [0, 15])
@pytest.mark.parametrize("seed", range(4))
def test_abi_matches_mirror_on_random_streams(seed, rope):
    rng = random.Random(seed * 7 + rope)
    cap, seqs, maxb = 12, 4, 6
    m = CacheMirror(cap, seqs, maxb)
    h = smem.smem_cache_create(smem.make_config(1, 1, 64, seqs, maxb, cap, rope_window=rope), None)
    import ctypes
    L = smem.lib()
    try:
        for _ in range(600):
            r = rng.random()
            s, t = rng.randrange(-1, seqs + 1), rng.randrange(seqs)
            i, j = rng.randrange(-1, 9), rng.randrange(9)
            if r < 0.35:
                st = dict(op="append", args=[s, i])
                rc_m, slot_m = m.append(s, i)
            elif r < 0.65:
                jj = j if rope else i
                st = dict(op="share", args=[s, i, t, jj])
                rc_m, slot_m = m.share(s, i, t, jj, any_index=bool(rope))
            elif r < 0.95:
                st = dict(op="delete", args=[s, i])
                rc_m, slot_m = m.delete(s, i), -1
            else:
                st = dict(op="release", args=[max(s, 0) if s < seqs else s])
                rc_m, slot_m = m.release(st["args"][0]), -1
            rc_a, slot_a = abi_step(h, st)
            assert rc_a == rc_m, (st, rc_a, rc_m)
            if rc_m == 0 and st["op"] in ("append", "share"):
                assert slot_a == slot_m
            check_invariants(m)
        for q in range(seqs):
            assert smem.smem_get_table(h, q) == m.table(q)
        assert smem.smem_get_free_fifo(h) == m.free_list()
        assert [smem.smem_slot_refs(h, x) for x in range(cap)] == m.refs
    finally:
        smem.smem_cache_destroy(h)
