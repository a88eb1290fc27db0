"""Paged-layout contract of the library, restated as plain lists.

The paper keeps no page structure of its own (Sec. 3.3 speaks only of resident
positions); the library stores K/V in fixed-size pages, and this module states
where every retained position must sit, so page tables can be compared bit for
bit.  The contract:

* A global pool of page ids ``0 .. n_pages-1``; an allocation always takes the
  lowest free id.
* Each session owns two regions.  ``hist``: a page list filled densely from
  slot 0 (``n_hist`` positions).  ``live``: a page list whose first
  ``live_head`` slots are consumed, followed by ``n_live`` positions.
* Logical retained index ``i < n_hist`` lives in ``hist[i // ps]`` slot
  ``i % ps``; otherwise ``j = live_head + i - n_hist`` lives in
  ``live[j // ps]`` slot ``j % ps``.
* Append writes at the live tail.  Pages are allocated in the call's session
  order, then token order.
* Evict, for a call over several sessions: let ``u*`` be the last unit this
  call evicted in a session and ``end`` the number of live positions whose unit
  is ``<= u*`` (a prefix of the live region, since units never decrease along
  positions).  First, for every session in call order, the survivors among
  those ``end`` positions move, in order, to the hist tail (hist pages
  allocated as needed).  Then, for every session, the live head advances by
  ``end`` and fully consumed live pages are freed.
* Retained logical order is therefore ascending position.
"""
from __future__ import annotations

import heapq


class PagePool:
    def __init__(self, n_pages: int):
        self.n_pages = n_pages
        self._free = list(range(n_pages))
        heapq.heapify(self._free)
        self._in_use = set()

    def free_count(self) -> int:
        return len(self._free)

    def alloc(self) -> int:
        if not self._free:
            raise MemoryError("page pool exhausted")
        pid = heapq.heappop(self._free)
        self._in_use.add(pid)
        return pid

    def release(self, pid: int) -> None:
        self._in_use.remove(pid)
        heapq.heappush(self._free, pid)


class SessionLayout:
    def __init__(self, page_size: int):
        self.ps = page_size
        self.hist_pages: list[int] = []
        self.hist_pos: list[int] = []      # positions stored in hist, in order
        self.live_pages: list[int] = []
        self.live_head = 0
        self.live_pos: list[int] = []      # positions stored in live, in order

    @property
    def n_hist(self) -> int:
        return len(self.hist_pos)

    @property
    def n_live(self) -> int:
        return len(self.live_pos)

    def pages_for_append(self, n_tokens: int) -> int:
        tail = self.live_head + self.n_live
        have = len(self.live_pages) * self.ps
        need = tail + n_tokens - have
        return max(0, -(-need // self.ps))

    def append(self, positions, pool: PagePool) -> None:
        for p in positions:
            tail = self.live_head + self.n_live
            if tail == len(self.live_pages) * self.ps:
                self.live_pages.append(pool.alloc())
            self.live_pos.append(p)

    def move_survivors(self, end: int, survivors: list[int], pool: PagePool) -> None:
        """First phase of an evict: survivors of the first ``end`` live positions join hist."""
        assert all(p in self.live_pos[:end] for p in survivors)
        for p in survivors:
            if self.n_hist == len(self.hist_pages) * self.ps:
                self.hist_pages.append(pool.alloc())
            self.hist_pos.append(p)

    def consume_live(self, end: int, pool: PagePool) -> None:
        """Second phase of an evict: drop ``end`` live positions, free whole pages."""
        consumed = self.live_head + end
        n_free = consumed // self.ps
        for pid in self.live_pages[:n_free]:
            pool.release(pid)
        self.live_pages = self.live_pages[n_free:]
        self.live_head = consumed - n_free * self.ps
        self.live_pos = self.live_pos[end:]

    def slot_of_logical(self, i: int) -> tuple[int, int]:
        if i < self.n_hist:
            return self.hist_pages[i // self.ps], i % self.ps
        j = self.live_head + i - self.n_hist
        return self.live_pages[j // self.ps], j % self.ps

    def retained_positions(self) -> list[int]:
        return self.hist_pos + self.live_pos
