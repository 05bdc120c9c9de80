"""Plain model of the lazy paged KV allocator (Sec. 5.4, "Lazy KV Cache
Allocation": a request gets cache blocks only when it needs them).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Policy modelled (the library documents the same policy in its header):

* The pool has ``num_pages`` pages.  Pages are handed out in "pop order":
  0, 1, 2, ... after creation, or ``order[0], order[1], ...`` after
  ``set_page_order(order)`` (allowed only while no page is in use).
* A sequence id is the lowest id not in use.
* Reserving n tokens for a sequence of length s walks positions s .. s+n-1 and
  takes the next page in pop order exactly when a position is the first slot
  of a page (position % P == 0); the page becomes logical page position // P.
  All or nothing: if the pool cannot supply every page, nothing changes and
  ``OutOfPages`` is raised.  Exceeding the page-table row is a ValueError.
* A decode step reserves one token for each sequence of the batch, in batch
  order, all or nothing.
* Freeing a sequence puts its pages back at the front of the pop order, in
  the sequence's logical page order (its logical page 0 is handed out next).
"""
from __future__ import annotations


class OutOfPages(Exception):
    pass


class PagePoolModel:
    def __init__(self, num_pages: int, page_size: int, max_seqs: int, max_pages_per_seq: int):
        self.P = page_size
        self.num_pages = num_pages
        self.max_seqs = max_seqs
        self.max_pages = max_pages_per_seq
        self.free = list(range(num_pages))      # pop order: free[0] goes next
        self.lens: dict[int, int] = {}
        self.pages: dict[int, list[int]] = {}

    # -- pool -------------------------------------------------------------
    def set_page_order(self, order):
        if any(self.pages.values()):
            raise ValueError("pages in use")
        order = [int(x) for x in order]
        if sorted(order) != list(range(self.num_pages)):
            raise ValueError("not a permutation of the pool")
        self.free = order

    def pages_in_use(self) -> int:
        return sum(len(p) for p in self.pages.values())

    # -- sequences ----------------------------------------------------------
    def seq_create(self) -> int:
        for i in range(self.max_seqs):
            if i not in self.lens:
                self.lens[i] = 0
                self.pages[i] = []
                return i
        raise OutOfPages("no free sequence slot")

    def _pages_needed(self, seq: int, n: int) -> int:
        s = self.lens[seq]
        return sum(1 for pos in range(s, s + n) if pos % self.P == 0)

    def seq_reserve(self, seq: int, n: int):
        if seq not in self.lens or n < 0:
            raise ValueError("bad sequence or count")
        s = self.lens[seq]
        if (s + n + self.P - 1) // self.P > self.max_pages:
            raise ValueError("page-table row too short")
        if self._pages_needed(seq, n) > len(self.free):
            raise OutOfPages("pool exhausted")
        for pos in range(s, s + n):
            if pos % self.P == 0:
                self.pages[seq].append(self.free.pop(0))
        self.lens[seq] = s + n

    def seq_free(self, seq: int):
        if seq not in self.lens:
            raise ValueError("bad sequence")
        self.free = list(self.pages[seq]) + self.free
        del self.lens[seq]
        del self.pages[seq]

    def begin_step(self, seq_ids):
        seq_ids = [int(s) for s in seq_ids]
        if len(set(seq_ids)) != len(seq_ids) or any(s not in self.lens for s in seq_ids):
            raise ValueError("batch must hold distinct live sequences")
        for s in seq_ids:
            if (self.lens[s] + 1 + self.P - 1) // self.P > self.max_pages:
                raise ValueError("page-table row too short")
        need = sum(1 for s in seq_ids if self.lens[s] % self.P == 0)
        if need > len(self.free):
            raise OutOfPages("pool exhausted")
        for s in seq_ids:
            self.seq_reserve(s, 1)

    def page_table_row(self, seq: int, width: int | None = None):
        width = self.max_pages if width is None else width
        row = list(self.pages[seq])
        return row + [-1] * (width - len(row))
