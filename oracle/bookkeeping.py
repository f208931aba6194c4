"""Independent mirror of the memory-cache bookkeeping (test infrastructure).

The paper stores the memory as a multiset ordered canonically by block index
(arXiv 2609.32395, Sec. 2 "Model") and makes deletion an O(b) update that
yields exactly the never-inserted state (Theorem 1); it leaves the storage
policy open (App. "Serving measurements" compares a contiguous and an
index-mapped layout). The policy mirrored here is the one the library
implements for its block-paged pool:

* one table per sequence, entries ``(block_idx, slot)`` kept sorted by
  ``block_idx``; ``block_idx`` is unique within a sequence;
* one FIFO of free slots, initially a given order (ascending by default);
  an append takes the slot at the front, a delete puts its slot at the back,
  releasing a sequence puts its slots at the back in ascending block order;
* a failing operation leaves every structure unchanged. Checks run in this
  order: sequence id, block index sign, duplicate / absent block, table
  capacity, pool capacity;
* sharing (exact reuse of a cached block by another table, Sec. 2 "Exact
  composition"): a table entry may name a slot another entry already holds;
  every slot counts its references, and a slot returns to the back of the
  FIFO when its last reference is deleted or released. Without rotary
  phases a block is reused at its own index only (moving it would need a
  re-encode); with position-free rows (the RoPE composite) at any index.
  Share checks: both sequence ids, both indices' signs, the source entry,
  the index rule, a duplicate destination, the destination table's
  capacity.

Error numbers are the ABI's (they are part of the interface contract).
"""
from __future__ import annotations

import bisect
from collections import deque

OK = 0
ERR_INVALID_ARG = -1
ERR_NO_SUCH_SEQ = -3
ERR_DUPLICATE_BLOCK = -4
ERR_NO_SUCH_BLOCK = -5
ERR_POOL_FULL = -6
ERR_TABLE_FULL = -7


class CacheMirror:
    def __init__(self, capacity: int, max_seqs: int, max_blocks_per_seq: int, free_order=None):
        self.capacity = int(capacity)
        self.max_seqs = int(max_seqs)
        self.max_blocks = int(max_blocks_per_seq)
        order = list(range(self.capacity)) if free_order is None else [int(s) for s in free_order]
        if sorted(order) != list(range(self.capacity)):
            raise ValueError("free_order must be a permutation of 0..capacity-1")
        self.fifo = deque(order)
        self.idx = [[] for _ in range(self.max_seqs)]    # sorted block indices
        self.slot = [[] for _ in range(self.max_seqs)]   # slots, same order
        self.refs = [0] * self.capacity                  # table entries naming each slot

    def _seq_ok(self, seq: int) -> bool:
        return 0 <= seq < self.max_seqs

    def append(self, seq: int, block_idx: int):
        """Returns (rc, slot)."""
        if not self._seq_ok(seq):
            return ERR_NO_SUCH_SEQ, -1
        if block_idx < 0:
            return ERR_INVALID_ARG, -1
        ix = self.idx[seq]
        k = bisect.bisect_left(ix, block_idx)
        if k < len(ix) and ix[k] == block_idx:
            return ERR_DUPLICATE_BLOCK, -1
        if len(ix) >= self.max_blocks:
            return ERR_TABLE_FULL, -1
        if not self.fifo:
            return ERR_POOL_FULL, -1
        s = self.fifo.popleft()
        ix.insert(k, block_idx)
        self.slot[seq].insert(k, s)
        self.refs[s] = 1
        return OK, s

    def share(self, src_seq: int, src_idx: int, dst_seq: int, dst_idx: int, any_index: bool = False):
        """Returns (rc, slot): dst_seq's table gains (dst_idx, the slot of src_idx)."""
        if not self._seq_ok(src_seq) or not self._seq_ok(dst_seq):
            return ERR_NO_SUCH_SEQ, -1
        if src_idx < 0 or dst_idx < 0:
            return ERR_INVALID_ARG, -1
        sx = self.idx[src_seq]
        k = bisect.bisect_left(sx, src_idx)
        if k >= len(sx) or sx[k] != src_idx:
            return ERR_NO_SUCH_BLOCK, -1
        if not any_index and dst_idx != src_idx:
            return ERR_INVALID_ARG, -1
        s = self.slot[src_seq][k]
        dx = self.idx[dst_seq]
        j = bisect.bisect_left(dx, dst_idx)
        if j < len(dx) and dx[j] == dst_idx:
            return ERR_DUPLICATE_BLOCK, -1
        if len(dx) >= self.max_blocks:
            return ERR_TABLE_FULL, -1
        dx.insert(j, dst_idx)
        self.slot[dst_seq].insert(j, s)
        self.refs[s] += 1
        return OK, s

    def _drop(self, s: int):
        self.refs[s] -= 1
        if self.refs[s] == 0:
            self.fifo.append(s)

    def delete(self, seq: int, block_idx: int) -> int:
        if not self._seq_ok(seq):
            return ERR_NO_SUCH_SEQ
        if block_idx < 0:
            return ERR_INVALID_ARG
        ix = self.idx[seq]
        k = bisect.bisect_left(ix, block_idx)
        if k >= len(ix) or ix[k] != block_idx:
            return ERR_NO_SUCH_BLOCK
        s = self.slot[seq][k]
        del ix[k]
        del self.slot[seq][k]
        self._drop(s)
        return OK

    def release(self, seq: int) -> int:
        if not self._seq_ok(seq):
            return ERR_NO_SUCH_SEQ
        for s in self.slot[seq]:
            self._drop(s)
        self.idx[seq] = []
        self.slot[seq] = []
        return OK

    def table(self, seq: int):
        return list(self.idx[seq]), list(self.slot[seq])

    def prefix_len(self, seq: int, q_idx: int) -> int:
        """Number of table entries with block index < q_idx."""
        return bisect.bisect_left(self.idx[seq], q_idx)

    def free_list(self):
        return list(self.fifo)

    def live_slots(self):
        return [s for sl in self.slot for s in sl]
