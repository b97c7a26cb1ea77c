"""The paged tensor store, written plainly on the CPU (oracle).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU baseline / reference arm, never by the product path.

What the store computes, and where the paper fixes it:

* Plain definition. A map id -> bytes: ``put`` stores bytes under a new id,
  ``get`` returns them (optionally cast fp32 -> bf16), ``free`` forgets them.
  Intermediate tensors are written once and read by their consumers, never
  updated (§5.3, "Backend-as-a-Service Paradigm": immutability), and are
  reclaimed once no consumer needs them (same paragraph) -- here by an explicit
  ``free`` or after a declared number of consumers (reading 9). A producer writes its output into the local store and a consumer
  later pulls it into its own buffer (§5.2, "Efficient and flexible data
  fetching").
* Capacity. The paper manages its arena with a buddy allocator (§5.2); the
  store uses fixed pages of P bytes instead (reading 1 below), so an object of
  n bytes takes ceil(n / P) pages and the pages in use are the sum of that
  over the live objects.
* Eviction. Cached weights are elastic: under pressure the least recently
  used model's weights go first, layer by layer in reverse layer order, until
  the demand is met (§5.3, "How does it work?"; §1: weights are evictable).
* Compaction has no counterpart in the paper; it answers the fixed-size
  arena problem (§5.3, "Can NVSHMEM region be elastic?") by handing a
  contiguous tail of the pool back.

Readings where the paper is silent:

1. Pages: fixed P-byte pages; an object's pages need not be contiguous; the
   unused tail of its last page is never read.
2. Placement: a LIFO stack of free page numbers, initially ordered so that page
   0 pops first. A put pops its pages one at a time, objects in descriptor
   order; a free pushes an object's pages back in page-list order.
3. Zero-byte objects are allowed: no pages, their get returns nothing.
4. Ids: 1, 2, 3, ... in descriptor order across calls, never reused.
5. Atomicity: a put either stores every object or changes nothing (NOSPACE /
   INVALID). A get validates every id first; if any fails, the call returns
   the first failing status in descriptor order and touches nothing. A
   repeated id inside one get is allowed; inside one free it is INVALID.
6. LRU: recency per ``group`` (a model or an adapter set), kept by a counter
   that every put and successful get advances once per object, in descriptor
   order. Victims come from the least recently used group first; within a
   group the highest ``order`` (layer) first, ties to the highest id.
   Eviction runs only inside a put, object by object, until the free pages
   cover the put's demand. Groups named by the put itself are not victims,
   nor are objects put with evictable = 0. If evicting every allowed object
   would still not make room, the put returns NOSPACE and evicts nothing.
   A get of an evicted id returns EVICTED; a free of an evicted id drops it.
7. Compaction to ``limit`` pages: NOSPACE if more pages are in use; live pages
   numbered >= limit, in ascending order, move one by one to the lowest free
   page below limit; only the valid bytes of a page are copied. Afterwards
   the capacity is ``limit`` and the free stack holds the free pages below it,
   pushed in descending order (the lowest pops first). A larger limit later
   grows the store back.
8. A put descriptor without data reserves pages and copies nothing; the
   object's bytes are undefined (the allocation half of a pull, §5.2).
9. Reclaim by consumer count (§5.3: tensors are reclaimed once no downstream
   function needs them): an object put with k > 0 consumers is freed after
   its k-th successful get item; a get frees the objects it brought to zero
   at its end, in the order of the items that brought them there.
10. Extent placement (``policy = 1``, an alternative to reading 2 that keeps
    objects contiguous so they can be used in place, §5.3 "pointer
    rebinding"): the free pages form a set; an object of k pages takes the
    lowest-numbered run of k consecutive free pages, or, if there is none,
    the k lowest-numbered free pages. ``free_stack`` then lists the free
    pages in ascending order (after a compaction too).
11. Pull between stores (§5.2): see :meth:`OracleStore.pull`.
"""
from __future__ import annotations

import bisect
from dataclasses import dataclass, field

import numpy as np

from .cast import cast_bytes_f32_to_bf16

OK, INVALID, NOSPACE, NOT_FOUND, EVICTED = 0, 1, 2, 3, 4


def pages_for(nbytes: int, page_bytes: int) -> int:
    """Pages an object of ``nbytes`` takes: ceil(nbytes / page_bytes)."""
    return -(-int(nbytes) // int(page_bytes))


@dataclass
class PutItem:
    nbytes: int
    data: np.ndarray | None = None   # uint8 bytes; None reserves pages (reading 8)
    dtype_tag: int = 0
    group: int = 0
    order: int = 0
    evictable: bool = False
    consumers: int = 0


@dataclass
class _Object:
    nbytes: int
    dtype_tag: int
    group: int
    order: int
    evictable: bool
    pages: list = field(default_factory=list)
    data: np.ndarray | None = None
    consumers_left: int = 0


class OracleStore:
    """The store on the CPU. ``keep_bytes`` keeps each object's bytes (the
    definitional map); ``paged_pool`` also keeps an explicit pool byte array,
    writes objects into their pages and reads gets back from the pages (the
    brute-force paged model, for tiny pools)."""

    def __init__(self, pool_bytes: int, page_bytes: int, keep_bytes: bool = True, paged_pool: bool = False,
                 policy: int = 0):
        if page_bytes <= 0 or pool_bytes < 0 or policy not in (0, 1):
            raise ValueError("bad store geometry or policy")
        self.policy = policy
        self.page_bytes = int(page_bytes)
        self.total_pages = int(pool_bytes) // self.page_bytes
        self.limit_pages = self.total_pages
        self.keep_bytes = keep_bytes
        self.pool = np.zeros(self.total_pages * self.page_bytes, np.uint8) if paged_pool else None
        # reading 2: a stack whose end is the top (page 0 pops first);
        # reading 10: the free pages in ascending order
        self.free_stack = list(range(self.total_pages - 1, -1, -1)) if policy == 0 else list(range(self.total_pages))
        self.objects: dict[int, _Object] = {}
        self.evicted: set[int] = set()
        self.next_id = 1
        self.clock = 0
        self.group_last: dict[int, int] = {}
        self.last_evictions: list[int] = []
        self.stats = dict(bytes_put=0, bytes_got=0, gets=0, misses=0, evictions=0,
                          pages_moved=0, bytes_moved=0, puts=0, reclaimed=0)

    # -- accounting ---------------------------------------------------------
    def used_pages(self) -> int:
        return sum(pages_for(o.nbytes, self.page_bytes) for o in self.objects.values())

    def free_pages(self) -> int:
        return len(self.free_stack)

    def pages_of(self, oid: int) -> list[int]:
        return list(self.objects[oid].pages)

    def _touch(self, group: int) -> None:
        self.clock += 1
        self.group_last[group] = self.clock

    def _release(self, oid: int) -> None:
        for p in self.objects[oid].pages:
            if self.policy == 0:
                self.free_stack.append(p)
            else:
                bisect.insort(self.free_stack, p)
        del self.objects[oid]

    def _take_pages(self, k: int) -> list[int]:
        if self.policy == 0:
            return [self.free_stack.pop() for _ in range(k)]
        if k == 0:
            return []
        free = self.free_stack                  # ascending
        run = None
        for i in range(len(free) - k + 1):      # the lowest run of k consecutive pages
            if free[i + k - 1] - free[i] == k - 1:
                run = free[i:i + k]
                break
        if run is None:
            run = free[:k]                      # else the k lowest pages
        for p in run:
            free.remove(p)
        return run

    # -- put ----------------------------------------------------------------
    def _victims(self, demand: int, pinned: set) -> list[int] | None:
        """Eviction order (reading 6), or None if the demand cannot be met."""
        have = len(self.free_stack)
        if have >= demand:
            return []
        candidates = [oid for oid, o in self.objects.items() if o.evictable and o.group not in pinned]
        if have + sum(pages_for(self.objects[c].nbytes, self.page_bytes) for c in candidates) < demand:
            return None
        candidates.sort(key=lambda oid: (self.group_last[self.objects[oid].group],
                                         -self.objects[oid].order, -oid))
        out = []
        for oid in candidates:
            if have >= demand:
                break
            out.append(oid)
            have += pages_for(self.objects[oid].nbytes, self.page_bytes)
        return out

    def put_batch(self, items: list[PutItem]):
        """Returns (status, ids)."""
        self.last_evictions = []
        for it in items:
            if int(it.nbytes) < 0:
                return INVALID, []
            if it.data is not None and np.asarray(it.data).nbytes != int(it.nbytes):
                return INVALID, []
        demand = sum(pages_for(it.nbytes, self.page_bytes) for it in items)
        victims = self._victims(demand, {int(it.group) for it in items})
        if victims is None:
            return NOSPACE, []
        for oid in victims:
            self._release(oid)
            self.evicted.add(oid)
        self.last_evictions = victims
        self.stats["evictions"] += len(victims)
        ids = []
        for it in items:
            n = int(it.nbytes)
            pages = self._take_pages(pages_for(n, self.page_bytes))
            data = None
            if it.data is not None:
                data = np.ascontiguousarray(it.data).view(np.uint8).reshape(-1).copy()
                if self.pool is not None:
                    for j, p in enumerate(pages):
                        chunk = data[j * self.page_bytes:(j + 1) * self.page_bytes]
                        self.pool[p * self.page_bytes:p * self.page_bytes + chunk.size] = chunk
            oid = self.next_id
            self.next_id += 1
            self.objects[oid] = _Object(n, int(it.dtype_tag), int(it.group), int(it.order), bool(it.evictable),
                                        pages, data if self.keep_bytes else None, int(it.consumers))
            self._touch(int(it.group))
            self.stats["bytes_put"] += n
            self.stats["puts"] += 1
            ids.append(oid)
        return OK, ids

    # -- get ----------------------------------------------------------------
    def _read(self, o: _Object) -> np.ndarray | None:
        if self.pool is not None:
            out = np.empty(o.nbytes, np.uint8)
            for j, p in enumerate(o.pages):
                ln = min(self.page_bytes, o.nbytes - j * self.page_bytes)
                out[j * self.page_bytes:j * self.page_bytes + ln] = self.pool[p * self.page_bytes:p * self.page_bytes + ln]
            return out
        return None if o.data is None else o.data.copy()

    def get_batch(self, ids, casts=None):
        """Returns (status, per_item statuses, outputs); outputs[i] is the
        object's bytes (bf16 bytes when cast) or None for reserved objects."""
        casts = [0] * len(ids) if casts is None else list(casts)
        per = []
        for oid, c in zip(ids, casts):
            oid = int(oid)
            if c not in (0, 1):
                per.append(INVALID)
            elif oid in self.objects:
                per.append(INVALID if (c == 1 and self.objects[oid].nbytes % 4) else OK)
            elif oid in self.evicted:
                per.append(EVICTED)
            else:
                per.append(NOT_FOUND)
        self.stats["misses"] += sum(1 for s in per if s == EVICTED)
        bad = [s for s in per if s != OK]
        if bad:
            return bad[0], per, []
        outs = []
        consumed = []
        for oid, c in zip(ids, casts):
            o = self.objects[int(oid)]
            self._touch(o.group)
            raw = self._read(o)
            if raw is not None and c == 1:
                raw = cast_bytes_f32_to_bf16(raw)
            outs.append(raw)
            self.stats["bytes_got"] += o.nbytes
            self.stats["gets"] += 1
            if o.consumers_left > 0:
                o.consumers_left -= 1
                if o.consumers_left == 0:
                    consumed.append(int(oid))
        for oid in consumed:          # reading 9: no consumer needs them any more
            self._release(oid)
            self.stats["reclaimed"] += 1
        return OK, per, outs

    # -- pull (§5.2) ----------------------------------------------------------
    def pull(self, src: "OracleStore", ids, consumers: int = 0):
        """The consumer (self) allocates room in its own store and pulls the
        producer's (src) objects into it (§5.2). Reading 11: every id is
        checked first (statuses as a get's); the new objects are put like
        intermediates (evictable = 0, group 0, order 0, the source's dtype
        tag, ``consumers``); if they do not fit, NOSPACE and nothing happens;
        otherwise the sources are read like a get (recency stamped, one
        consumer counted). Returns (status, per-item statuses, new ids)."""
        if self.page_bytes != src.page_bytes:
            return INVALID, [], []
        per = []
        for oid in ids:
            oid = int(oid)
            per.append(OK if oid in src.objects else EVICTED if oid in src.evicted else NOT_FOUND)
        bad = [x for x in per if x != OK]
        if bad:
            src.stats["misses"] += sum(1 for x in per if x == EVICTED)
            return bad[0], per, []
        items = []
        for oid in ids:
            o = src.objects[int(oid)]
            data = src._read(o)
            items.append(PutItem(o.nbytes, data, o.dtype_tag, 0, 0, False, int(consumers)))
        st, new_ids = self.put_batch(items)
        if st != OK:
            return st, per, []
        src.get_batch(ids)
        return OK, per, new_ids

    # -- free ---------------------------------------------------------------
    def free(self, ids) -> int:
        ids = [int(i) for i in ids]
        if len(set(ids)) != len(ids):
            return INVALID
        for oid in ids:
            if oid not in self.objects and oid not in self.evicted:
                return NOT_FOUND
        for oid in ids:
            if oid in self.objects:
                self._release(oid)
            else:
                self.evicted.discard(oid)
        return OK

    # -- compact ------------------------------------------------------------
    def owners(self) -> dict[int, tuple[int, int]]:
        """page -> (object id, index of the page in the object's page list)."""
        own = {}
        for oid, o in self.objects.items():
            for j, p in enumerate(o.pages):
                own[p] = (oid, j)
        return own

    def compact(self, limit_bytes: int):
        """Returns (status, moves); moves are (src page, dst page, valid bytes)."""
        limit_bytes = int(limit_bytes)
        if limit_bytes < 0 or limit_bytes % self.page_bytes:
            return INVALID, []
        limit = limit_bytes // self.page_bytes
        if limit > self.total_pages:
            return INVALID, []
        if self.used_pages() > limit:
            return NOSPACE, []
        own = self.owners()
        tail_live = sorted(p for p in own if p >= limit)
        head_free = [p for p in range(limit) if p not in own]
        moves = []
        for src, dst in zip(tail_live, head_free):
            oid, j = own[src]
            o = self.objects[oid]
            valid = min(self.page_bytes, o.nbytes - j * self.page_bytes)
            o.pages[j] = dst
            if self.pool is not None:
                P = self.page_bytes
                self.pool[dst * P:dst * P + valid] = self.pool[src * P:src * P + valid]
            moves.append((src, dst, valid))
        own = self.owners()
        self.free_stack = [p for p in range(limit - 1, -1, -1) if p not in own]
        if self.policy == 1:
            self.free_stack.reverse()
        self.limit_pages = limit
        self.stats["pages_moved"] += len(moves)
        self.stats["bytes_moved"] += sum(m[2] for m in moves)
        return OK, moves

    # -- stats --------------------------------------------------------------
    def summary(self) -> dict:
        s = dict(self.stats)
        s.update(used_pages=self.used_pages(), free_pages=self.free_pages(), limit_pages=self.limit_pages,
                 total_pages=self.total_pages, live_objects=len(self.objects))
        return s
