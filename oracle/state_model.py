"""Plain-Python model of the residency state machine (test infrastructure).

Per (layer, logical block): RESIDENT, SWAPPED, DROPPED, INFLIGHT or EMPTY,
following the eviction/restore rules of the ABI: token ranges round outward
to 16-token blocks (the paper evicts at chunk granularity, Sec. 4.2/6.2);
COPY swaps resident blocks; DROP frees a contiguous token range across all
layers for recompute, and may take swapped blocks too (their host copies are
discarded: the eviction policy can move a unit from the copy path to the
recompute path, Algorithm 1); restore moves every swapped block to INFLIGHT; a
completed prefill makes in-flight and recomputed blocks RESIDENT and appends
the prompt.  Physical block numbers are not modelled (any valid, distinct
assignment is correct); the tests check them for validity only.

Pinned by tests/test_oracle_state_pins.py: literal tables and status codes
worked out by hand from the rules above (outward rounding, one contiguous
all-layer DROP range, double eviction, prefill over dropped or swapped
blocks, recompute range, truncation inside a dropped range, DROP over
swapped blocks).
"""
from __future__ import annotations

RESIDENT, SWAPPED, DROPPED, INFLIGHT, EMPTY = 0, 1, 2, 3, 4
OK, INVALID, RANGE, STATE = 0, 1, 2, 3


class StateModel:
    def __init__(self, n_layers: int, max_ctx: int):
        self.L = n_layers
        self.nblk = -(-max_ctx // 16)
        self.max_ctx = max_ctx
        self.st = [[EMPTY] * self.nblk for _ in range(n_layers)]
        self.n_ctx = 0
        self.drop = None  # (t0, t1)
        self.pending = False
        self.inflight = False

    def _nb(self):
        return -(-self.n_ctx // 16)

    def append(self, n):
        if self.n_ctx + n > self.max_ctx:
            return RANGE
        if self.drop and not self.pending:
            return STATE
        if any(s == SWAPPED for row in self.st for s in row[: self._nb()]):
            return STATE
        for l in range(self.L):
            for b in range(self.nblk):
                if self.st[l][b] == INFLIGHT or (self.st[l][b] == DROPPED and self.pending):
                    self.st[l][b] = RESIDENT
            for b in range(self._nb(), -(-(self.n_ctx + n) // 16)):
                self.st[l][b] = RESIDENT
        self.n_ctx += n
        self.drop, self.pending, self.inflight = None, False, False
        return OK

    def evict(self, l0, l1, t0, t1, mode):
        if mode not in (0, 1):
            return INVALID
        if l0 < 0 or l1 > self.L or l0 >= l1:
            return RANGE
        if t0 < 0 or t1 > self.n_ctx or t0 >= t1:
            return RANGE
        if self.inflight or self.pending:
            return STATE
        b0, b1 = t0 // 16, -(-t1 // 16)
        allowed = (RESIDENT, SWAPPED) if mode == 1 else (RESIDENT,)
        if any(self.st[l][b] not in allowed for l in range(l0, l1) for b in range(b0, b1)):
            return STATE
        if mode == 1:
            if l0 != 0 or l1 != self.L:
                return INVALID
            d0, d1 = b0 * 16, min(b1 * 16, self.n_ctx)
            if self.drop and not (d1 == self.drop[0] or d0 == self.drop[1]):
                return INVALID
            for l in range(self.L):
                for b in range(b0, b1):
                    self.st[l][b] = DROPPED
            self.drop = (min(d0, self.drop[0]), max(d1, self.drop[1])) if self.drop else (d0, d1)
            return OK
        for l in range(l0, l1):
            for b in range(b0, b1):
                self.st[l][b] = SWAPPED
        return OK

    def evict_blocks(self, pairs):
        if self.inflight or self.pending:
            return STATE
        nb = self._nb()
        if any(l < 0 or l >= self.L or b < 0 or b >= nb for l, b in pairs):
            return RANGE
        if any(self.st[l][b] != RESIDENT for l, b in pairs):
            return STATE
        if len(set(pairs)) != len(pairs):
            return INVALID
        for l, b in pairs:
            self.st[l][b] = SWAPPED
        return OK

    def recompute_tail(self, p, n):
        if not self.drop:
            return STATE
        if (p, p + n) != self.drop:
            return RANGE
        self.pending = True
        return OK

    def restore(self):
        if self.inflight:
            return STATE
        any_ = False
        for row in self.st:
            for b in range(self._nb()):
                if row[b] == SWAPPED:
                    row[b] = INFLIGHT
                    any_ = True
        self.inflight = any_
        return OK

    def truncate(self, n):
        if n < 0 or n > self.n_ctx:
            return RANGE
        if self.inflight or self.pending:
            return STATE
        for row in self.st:
            for b in range(-(-n // 16), self._nb()):
                row[b] = EMPTY
        self.n_ctx = n
        if self.drop:
            d0, d1 = self.drop[0], min(self.drop[1], n)
            self.drop = (d0, d1) if d1 > d0 else None
        return OK
