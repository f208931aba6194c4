"""Pins of the bookkeeping mirror: a hand-worked example and invariants."""
import os

import numpy as np

from oracle import bookkeeping as bk
from oracle.bookkeeping import CacheMirror

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "bookkeeping_fifo.txt")
RC = {"OK": bk.OK, "INVALID_ARG": bk.ERR_INVALID_ARG, "NO_SUCH_SEQ": bk.ERR_NO_SUCH_SEQ,
      "DUPLICATE_BLOCK": bk.ERR_DUPLICATE_BLOCK, "NO_SUCH_BLOCK": bk.ERR_NO_SUCH_BLOCK,
      "POOL_FULL": bk.ERR_POOL_FULL, "TABLE_FULL": bk.ERR_TABLE_FULL}


def parse_golden(path=GOLDEN):
    steps = []
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        lhs, rhs = line.split("->")
        op, seq, blk = lhs.split()
        parts = [p.strip() for p in rhs.split("|")]
        rc, slot = parts[0].split()
        tables = []
        for tpart in parts[1:3]:
            ent = [] if tpart == "-" else [tuple(int(x) for x in e.split(":")) for e in tpart.split()]
            tables.append(ent)
        fifo = [] if parts[3] == "-" else [int(x) for x in parts[3].split()]
        steps.append(dict(op=op, seq=int(seq), blk=None if blk == "-" else int(blk), rc=RC[rc],
                          slot=None if slot == "-" else int(slot), tables=tables, fifo=fifo))
    return steps


def run_step(m, st):
    if st["op"] == "append":
        rc, slot = m.append(st["seq"], st["blk"])
        return rc, (slot if rc == 0 else None)
    if st["op"] == "delete":
        return m.delete(st["seq"], st["blk"]), None
    return m.release(st["seq"]), None


def test_golden_fifo_example():
    m = CacheMirror(4, 2, 3)
    for st in parse_golden():
        rc, slot = run_step(m, st)
        assert rc == st["rc"], st
        assert slot == st["slot"], st
        for seq in range(2):
            idx, slots = m.table(seq)
            assert list(zip(idx, slots)) == st["tables"][seq], st
        assert m.free_list() == st["fifo"], st


def test_random_stream_invariants():
    rng = np.random.default_rng(21)
    C, S, MB = 40, 4, 16
    m = CacheMirror(C, S, MB, free_order=rng.permutation(C))
    for _ in range(3000):
        seq = int(rng.integers(-1, S + 1))
        blk = int(rng.integers(-1, 24))
        u = rng.random()
        if u < 0.5:
            m.append(seq, blk)
        elif u < 0.95:
            m.delete(seq, blk)
        else:
            m.release(seq)
        live = m.live_slots()
        free = m.free_list()
        assert sorted(live + free) == list(range(C))  # every slot exactly once
        for s in range(S):
            idx, slots = m.table(s)
            assert idx == sorted(set(idx)) and len(idx) <= MB


def test_delete_then_reappend_moves_slot():
    """The tiny-cache edit: delete block 3 of 8, re-append it -> a different slot."""
    m = CacheMirror(16, 1, 16)
    for j in range(8):
        assert m.append(0, j) == (0, j)
    assert m.delete(0, 3) == 0
    rc, s = m.append(0, 3)
    assert rc == 0 and s == 8
    assert m.table(0) == (list(range(8)), [0, 1, 2, 8, 4, 5, 6, 7])
    assert m.free_list() == list(range(9, 16)) + [3]
