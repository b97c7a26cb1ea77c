"""Pins of the oracle store (CPU only).

The store's results are fixed by identities and invariants the paper's
statement of the problem gives (written once, read back unchanged, reclaimed
when freed; §5.2, §5.3) and by the readings of its silent points listed in
the oracle's header. Each check here is computed independently of the
oracle's own bookkeeping:

* get(put(x)) == x, with the bytes read back from an explicit pool array
  through the page lists (brute force) and compared with the input;
* no two live objects share a page, every page is below the capacity, and the
  free stack is exactly the complement of the used pages;
* pages in use == sum of ceil(n / P), with ceil counted by a loop;
* compaction keeps every object's bytes, leaves every page below the limit,
  moves exactly the live pages at or above the limit, into the lowest free
  pages, and copies exactly the valid bytes;
* hand-derived traces for placement (LIFO) and for LRU victims in reverse
  layer order (§5.3, "How does it work?").

Planted mistakes in the oracle must fail these checks.
"""
import itertools

import numpy as np
import pytest

import oracle.store as ostore
from oracle import EVICTED, INVALID, NOSPACE, NOT_FOUND, OK, OracleStore, PutItem


def ceil_pages_by_counting(n, P):
    k = 0
    while k * P < n:
        k += 1
    return k


def check_invariants(s: OracleStore, inputs: dict):
    """inputs: id -> the bytes that were put (None for reserved objects)."""
    P = s.page_bytes
    seen = {}
    for oid, o in s.objects.items():
        assert len(o.pages) == ceil_pages_by_counting(o.nbytes, P)
        for p in o.pages:
            assert 0 <= p < s.limit_pages, "page outside the capacity"
            assert p not in seen, f"page {p} shared by {seen.get(p)} and {oid}"
            seen[p] = oid
    used = sum(ceil_pages_by_counting(o.nbytes, P) for o in s.objects.values())
    assert s.used_pages() == used
    assert len(s.free_stack) == len(set(s.free_stack))
    assert set(s.free_stack) | set(seen) == set(range(s.limit_pages))
    assert not (set(s.free_stack) & set(seen))
    assert set(s.objects) == set(inputs)
    # brute force read through the page lists of the explicit pool
    if s.pool is not None:
        for oid, want in inputs.items():
            if want is None:
                continue
            o = s.objects[oid]
            got = np.concatenate([s.pool[p * P:p * P + min(P, o.nbytes - j * P)] for j, p in enumerate(o.pages)]) \
                if o.pages else np.zeros(0, np.uint8)
            assert np.array_equal(got, want)


def random_ops(seed, P, total_pages, n_ops, max_pages=3, check=True):
    g = np.random.default_rng(seed)
    s = OracleStore(total_pages * P, P, paged_pool=True)
    inputs = {}
    for _ in range(n_ops):
        r = g.random()
        if r < 0.45:
            k = int(g.integers(1, 4))
            items = []
            for _ in range(k):
                n = int(g.integers(0, max_pages * P + 1))
                data = None if g.random() < 0.1 else g.integers(0, 256, n, dtype=np.uint8)
                items.append(PutItem(n, data, group=int(g.integers(0, 3)), order=int(g.integers(0, 4)),
                                     evictable=bool(g.random() < 0.5),
                                     consumers=int(g.integers(0, 3)) if g.random() < 0.3 else 0))
            free_before = s.free_pages()
            evictable_pages = sum(ceil_pages_by_counting(o.nbytes, P) for o in s.objects.values()
                                  if o.evictable and o.group not in {it.group for it in items})
            demand = sum(ceil_pages_by_counting(it.nbytes, P) for it in items)
            snap = (dict((k2, list(v.pages)) for k2, v in s.objects.items()), list(s.free_stack), s.next_id)
            st, ids = s.put_batch(items)
            if demand > free_before + evictable_pages:
                assert st == NOSPACE
                assert snap == (dict((k2, list(v.pages)) for k2, v in s.objects.items()), list(s.free_stack),
                                s.next_id), "a failed put changed the store"
            else:
                assert st == OK
                for v in s.last_evictions:
                    inputs.pop(v)
                for oid, it in zip(ids, items):
                    inputs[oid] = None if it.data is None else it.data.copy()
        elif r < 0.7 and inputs:
            ids = list(g.choice(list(inputs), size=min(len(inputs), int(g.integers(1, 4))), replace=False))
            st, per, outs = s.get_batch(ids)
            assert st == OK
            for oid, out in zip(ids, outs):
                if inputs[int(oid)] is not None:
                    assert np.array_equal(out, inputs[int(oid)])
            for oid in ids:                      # consumed to zero: reclaimed
                if int(oid) not in s.objects:
                    inputs.pop(int(oid), None)
        elif r < 0.9 and inputs:
            ids = list(g.choice(list(inputs), size=min(len(inputs), int(g.integers(1, 3))), replace=False))
            assert s.free(ids) == OK
            for oid in ids:
                inputs.pop(int(oid))
        else:
            limit = int(g.integers(0, total_pages + 1))
            own_before = {p: (oid, j) for oid, o in s.objects.items() for j, p in enumerate(o.pages)}
            used = len(own_before)
            st, moves = s.compact(limit * P)
            if used > limit:
                assert st == NOSPACE and moves == []
            else:
                assert st == OK
                tail = sorted(p for p in own_before if p >= limit)
                assert [m[0] for m in moves] == tail
                free_head = [p for p in range(limit) if p not in own_before]
                assert [m[1] for m in moves] == free_head[:len(tail)]
                for src, dst, valid in moves:
                    oid, j = own_before[src]
                    n = s.objects[oid].nbytes
                    assert valid == min(P, n - j * P)
                    assert s.objects[oid].pages[j] == dst
                # the free stack pops the lowest page first
                assert s.free_stack == sorted(s.free_stack, reverse=True)
        if check:
            check_invariants(s, inputs)
    return s, inputs


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("P", [64, 256, 4096])
def test_random_sequences_tiny_pools(seed, P):
    random_ops(seed, P, total_pages=8 + seed * 4, n_ops=120)


def test_exhaustive_two_op_sequences():
    """Every pair of (put size, free/compact choice) on a 4-page pool of 64 B
    pages: brute force over a small op alphabet."""
    P = 64
    sizes = [0, 1, 63, 64, 65, 128, 191, 256]
    for a, b, c in itertools.product(sizes, sizes, range(5)):
        s = OracleStore(4 * P, P, paged_pool=True)
        inputs = {}
        for n in (a, b):
            data = np.arange(n, dtype=np.uint8) ^ (n & 0xFF)
            st, ids = s.put_batch([PutItem(n, data)])
            if st == OK:
                inputs[ids[0]] = data
            else:
                assert st == NOSPACE
                assert sum(ceil_pages_by_counting(len(v), P) for v in inputs.values()) + \
                    ceil_pages_by_counting(n, P) > 4
        check_invariants(s, inputs)
        if inputs:
            first = min(inputs)
            assert s.free([first]) == OK
            inputs.pop(first)
        st, _ = s.compact(c * P)
        assert st == (OK if s.used_pages() <= c else NOSPACE)
        check_invariants(s, inputs)


def test_lifo_placement_hand_trace():
    """Pages worked out by hand from readings 2 and 7 (1 KiB pages, 8 pages)."""
    P = 1024
    s = OracleStore(8 * P, P, paged_pool=True)
    _, (a,) = s.put_batch([PutItem(2500, np.full(2500, 1, np.uint8))])
    assert s.pages_of(a) == [0, 1, 2]
    _, (b,) = s.put_batch([PutItem(1024, np.full(1024, 2, np.uint8))])
    assert s.pages_of(b) == [3]
    assert s.free([a]) == OK
    assert s.free_stack == [7, 6, 5, 4, 0, 1, 2]
    _, (c,) = s.put_batch([PutItem(2048, np.full(2048, 3, np.uint8))])
    assert s.pages_of(c) == [2, 1]
    d_bytes = np.arange(3000, dtype=np.uint8)
    _, (d,) = s.put_batch([PutItem(3000, d_bytes)])
    assert s.pages_of(d) == [0, 4, 5]
    assert s.compact(4 * P) == (NOSPACE, [])
    assert s.free([b]) == OK
    st, moves = s.compact(5 * P)
    assert st == OK and moves == [(5, 3, 3000 - 2048)]
    assert s.pages_of(d) == [0, 4, 3] and s.free_stack == []
    assert s.put_batch([PutItem(1, np.zeros(1, np.uint8))])[0] == NOSPACE
    st, moves = s.compact(8 * P)
    assert st == OK and moves == [] and s.free_stack == [7, 6, 5]
    _, (e,) = s.put_batch([PutItem(1, np.zeros(1, np.uint8))])
    assert s.pages_of(e) == [5]
    _, _, (out,) = s.get_batch([d])
    assert np.array_equal(out, d_bytes)
    assert s.stats["pages_moved"] == 1 and s.stats["bytes_moved"] == 952


def test_lru_reverse_layer_hand_trace():
    """Victims worked out by hand from §5.3 (LRU model first, last layers
    first) and reading 6 (1 KiB pages, 6 pages)."""
    P = 1024
    s = OracleStore(6 * P, P)
    st, w1 = s.put_batch([PutItem(P, np.zeros(P, np.uint8), group=1, order=k, evictable=True) for k in range(3)])
    assert st == OK and w1 == [1, 2, 3]
    st, w2 = s.put_batch([PutItem(P, np.zeros(P, np.uint8), group=2, order=k, evictable=True) for k in range(2)])
    assert w2 == [4, 5] and [s.pages_of(i)[0] for i in w1 + w2] == [0, 1, 2, 3, 4]
    assert s.get_batch([1])[0] == OK            # model 1 is now the most recent
    st, (x,) = s.put_batch([PutItem(3 * P, np.zeros(3 * P, np.uint8), group=3)])
    assert st == OK and s.last_evictions == [5, 4]   # model 2 first, layer 1 before layer 0
    assert s.pages_of(x) == [3, 4, 5]
    st, per, _ = s.get_batch([4, 99, 1])
    assert st == EVICTED and per == [EVICTED, NOT_FOUND, OK]
    st, (y,) = s.put_batch([PutItem(P, np.zeros(P, np.uint8), group=2, order=0, evictable=True)])
    assert st == OK and s.last_evictions == [3]      # layer 2 of model 1, now the only evictable model
    assert s.pages_of(y) == [2]
    before = sorted(s.objects)
    st, _ = s.put_batch([PutItem(4 * P, np.zeros(4 * P, np.uint8), group=4)])
    assert st == NOSPACE and s.last_evictions == [] and sorted(s.objects) == before
    # ties inside a group go to the highest id
    s2 = OracleStore(2 * P, P)
    s2.put_batch([PutItem(P, np.zeros(P, np.uint8), group=5, order=1, evictable=True) for _ in range(2)])
    st, _ = s2.put_batch([PutItem(P, np.zeros(P, np.uint8), group=6)])
    assert st == OK and s2.last_evictions == [2]
    # a put's own groups are never victims, even when they are the least recent
    s3 = OracleStore(3 * P, P)
    s3.put_batch([PutItem(P, None, group=7, evictable=True)])
    _, (b3, c3) = s3.put_batch([PutItem(P, None, group=8, order=k, evictable=True) for k in range(2)])
    st, _ = s3.put_batch([PutItem(P, None, group=7, order=1, evictable=True)])
    assert st == OK and s3.last_evictions == [c3]    # model 8's last layer, not model 7's
    # freeing an evicted id drops it; its get is then NOT_FOUND
    assert s.free([4]) == OK and s.get_batch([4])[0] == NOT_FOUND


def test_error_paths_change_nothing():
    P = 256
    s = OracleStore(4 * P, P)
    st, ids = s.put_batch([PutItem(10, np.zeros(10, np.uint8)), PutItem(300, np.zeros(300, np.uint8))])
    assert st == OK and ids == [1, 2]
    assert s.put_batch([PutItem(5, np.zeros(4, np.uint8))])[0] == INVALID
    assert s.free([1, 1]) == INVALID and 1 in s.objects
    assert s.free([1, 77]) == NOT_FOUND and 1 in s.objects
    assert s.get_batch([2], casts=[1])[0] == OK          # 300 % 4 == 0
    assert s.get_batch([1], casts=[1])[0] == INVALID     # 10 % 4 != 0
    assert s.get_batch([1], casts=[2])[0] == INVALID
    assert s.compact(100)[0] == INVALID                  # not a page multiple
    assert s.compact(5 * P)[0] == INVALID                # beyond the pool
    st, per, outs = s.get_batch([1, 1, 2])               # repeats are allowed
    assert st == OK and len(outs) == 3
    assert s.next_id == 3


def test_zero_byte_and_reserved_objects():
    s = OracleStore(4 * 64, 64, paged_pool=True)
    st, (z, r) = s.put_batch([PutItem(0, np.zeros(0, np.uint8)), PutItem(100, None)])
    assert st == OK and s.pages_of(z) == [] and len(s.pages_of(r)) == 2
    st, _, outs = s.get_batch([z])
    assert st == OK and outs[0].size == 0
    check_invariants(s, {z: np.zeros(0, np.uint8), r: None})


def test_cast_on_get_matches_cast_module():
    s = OracleStore(1 << 20, 4096)
    x = np.random.default_rng(0).standard_normal(3000).astype(np.float32)
    _, (i,) = s.put_batch([PutItem(x.nbytes, x.view(np.uint8))])
    _, _, (out,) = s.get_batch([i], casts=[1])
    import torch
    assert np.array_equal(out.view(np.uint16), torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16))


# -- planted mistakes -------------------------------------------------------------

def _expect_failure(fn):
    try:
        fn()
    except AssertionError:
        return True
    return False


def test_planted_floor_pages(monkeypatch):
    monkeypatch.setattr(ostore, "pages_for", lambda n, P: int(n) // int(P))
    assert _expect_failure(lambda: random_ops(1, 64, 12, 60))


def test_planted_reversed_free_push(monkeypatch):
    def release(self, oid):
        for p in reversed(self.objects[oid].pages):
            self.free_stack.append(p)
        del self.objects[oid]
    monkeypatch.setattr(OracleStore, "_release", release)
    assert _expect_failure(test_lifo_placement_hand_trace)


def test_planted_victims_lowest_layer_first(monkeypatch):
    orig = OracleStore._victims

    def victims(self, demand, pinned):
        v = orig(self, demand, pinned)
        if not v:
            return v
        cands = sorted((o for o in self.objects if self.objects[o].evictable and self.objects[o].group not in pinned),
                       key=lambda o: (self.group_last[self.objects[o].group], self.objects[o].order, o))
        return cands[:len(v)]
    monkeypatch.setattr(OracleStore, "_victims", victims)
    assert _expect_failure(test_lru_reverse_layer_hand_trace)


def test_planted_compaction_to_highest_free(monkeypatch):
    orig = OracleStore.compact

    def compact(self, limit_bytes):
        # moves to the highest free pages instead of the lowest
        limit = int(limit_bytes) // self.page_bytes
        if int(limit_bytes) % self.page_bytes or limit > self.total_pages or self.used_pages() > limit:
            return orig(self, limit_bytes)
        own = self.owners()
        tail = sorted(p for p in own if p >= limit)
        head = [p for p in range(limit - 1, -1, -1) if p not in own]
        moves = []
        for src, dst in zip(tail, head):
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
        self.limit_pages = limit
        return OK, moves
    monkeypatch.setattr(OracleStore, "compact", compact)
    assert _expect_failure(test_lifo_placement_hand_trace)
    assert _expect_failure(lambda: [random_ops(sd, 64, 16, 150) for sd in range(6)])


def test_planted_compaction_drops_bytes(monkeypatch):
    orig = OracleStore.compact

    def compact(self, limit_bytes):
        st, moves = orig(self, limit_bytes)
        if self.pool is not None:
            for src, dst, valid in moves:   # forget the last byte of each moved page
                self.pool[dst * self.page_bytes + valid - 1] ^= 0xFF
        return st, moves
    monkeypatch.setattr(OracleStore, "compact", compact)
    assert _expect_failure(lambda: [random_ops(sd, 64, 16, 150) for sd in range(6)])


def test_reclaim_by_consumer_count_hand_trace():
    """Reading 9 (§5.3: reclaimed when no downstream consumer needs it)."""
    P = 256
    s = OracleStore(8 * P, P, paged_pool=True)
    a, b, c = (np.full(300, v, np.uint8) for v in (1, 2, 3))
    st, (ia, ib, ic) = s.put_batch([PutItem(300, a, consumers=2), PutItem(300, b, consumers=1),
                                    PutItem(300, c)])
    assert st == OK and s.pages_of(ia) == [0, 1] and s.pages_of(ib) == [2, 3]
    st, _, outs = s.get_batch([ia, ib])
    assert st == OK and np.array_equal(outs[1], b)
    assert ib not in s.objects and s.free_stack[-2:] == [2, 3] and s.stats["reclaimed"] == 1
    st, _, outs = s.get_batch([ia, ia])          # the last consumer may read twice in its batch
    assert st == OK and np.array_equal(outs[0], a) and np.array_equal(outs[1], a)
    assert ia not in s.objects and s.stats["reclaimed"] == 2
    assert s.get_batch([ia])[0] == NOT_FOUND
    st, _, (oc,) = s.get_batch([ic])
    assert st == OK and ic in s.objects          # consumers = 0: only an explicit free
    assert s.get_batch([ic, 999])[0] == NOT_FOUND and ic in s.objects  # a failed get consumes nothing
    check_invariants(s, {ic: c})


def test_planted_reclaim_before_last_consumer(monkeypatch):
    orig = OracleStore.get_batch

    def get_batch(self, ids, casts=None):
        st, per, outs = orig(self, ids, casts)
        for oid in list(self.objects):         # frees one consumer too early
            if self.objects[oid].consumers_left == 1:
                self._release(oid)
        return st, per, outs
    monkeypatch.setattr(OracleStore, "get_batch", get_batch)
    assert _expect_failure(test_reclaim_by_consumer_count_hand_trace)


def test_extent_policy_hand_trace():
    """Reading 10 (first fit over runs of free pages), worked out by hand
    (1 KiB pages, 8 pages)."""
    P = 1024
    s = OracleStore(8 * P, P, paged_pool=True, policy=1)
    _, (a,) = s.put_batch([PutItem(3 * P, np.full(3 * P, 1, np.uint8))])
    _, (b,) = s.put_batch([PutItem(2 * P, np.full(2 * P, 2, np.uint8))])
    assert s.pages_of(a) == [0, 1, 2] and s.pages_of(b) == [3, 4]
    assert s.free([a]) == OK and s.free_stack == [0, 1, 2, 5, 6, 7]
    _, (c,) = s.put_batch([PutItem(4 * P, np.full(4 * P, 3, np.uint8))])
    assert s.pages_of(c) == [0, 1, 2, 5]       # no run of 4: the 4 lowest pages
    _, (d,) = s.put_batch([PutItem(P, np.full(P, 4, np.uint8))])
    assert s.pages_of(d) == [6]
    assert s.free([b]) == OK and s.free_stack == [3, 4, 7]
    _, (e,) = s.put_batch([PutItem(2 * P, np.full(2 * P, 5, np.uint8))])
    assert s.pages_of(e) == [3, 4]             # the run, not the lowest pages 3 and 7
    assert s.free([c, d, e]) == OK and s.free_stack == list(range(8))
    _, (x, y, z) = s.put_batch([PutItem(5 * P, None), PutItem(P, None), PutItem(2 * P, None)])
    assert s.pages_of(x) == [0, 1, 2, 3, 4] and s.pages_of(y) == [5] and s.pages_of(z) == [6, 7]
    assert s.free([x, z]) == OK                # free runs: 0-4 and 6-7
    _, (f,) = s.put_batch([PutItem(2 * P, np.full(2 * P, 6, np.uint8))])
    assert s.pages_of(f) == [0, 1]             # first fit, not best fit (which would take 6, 7)
    st, moves = s.compact(4 * P)               # live: f = 0, 1 and y = 5 -> y moves to 2
    assert st == OK and moves == [(5, 2, P)] and s.free_stack == [3]


def test_extent_policy_takes_the_lowest_fitting_run():
    """Brute force: every allocation takes the lowest run of free pages long
    enough for it, when one exists (runs computed independently here)."""
    g = np.random.default_rng(3)
    for seed in range(20):
        P = 64
        total = 24
        s = OracleStore(total * P, P, policy=1)
        live = []
        for _ in range(80):
            if live and g.random() < 0.45:
                oid = live.pop(int(g.integers(0, len(live))))
                assert s.free([oid]) == OK
                continue
            k = int(g.integers(1, 6))
            free = sorted(s.free_stack)
            fits = [free[i] for i in range(len(free) - k + 1) if free[i + k - 1] - free[i] == k - 1]
            st, ids = s.put_batch([PutItem(k * P, None)])
            if st != OK:
                assert len(free) < k
                continue
            live.append(ids[0])
            got = s.pages_of(ids[0])
            if fits:
                assert got == list(range(fits[0], fits[0] + k))
            else:
                assert got == free[:k]
            check_invariants(s, {i: None for i in live})


def test_planted_best_fit_is_caught(monkeypatch):
    def take(self, k):
        if self.policy == 0 or k == 0:
            return [self.free_stack.pop() for _ in range(k)]
        free = self.free_stack
        runs, i = [], 0
        while i < len(free):
            j = i
            while j + 1 < len(free) and free[j + 1] == free[j] + 1:
                j += 1
            runs.append((free[i], j - i + 1))
            i = j + 1
        ok = sorted([r for r in runs if r[1] >= k], key=lambda r: (r[1], r[0]))
        run = list(range(ok[0][0], ok[0][0] + k)) if ok else free[:k]
        for p in run:
            free.remove(p)
        return run
    monkeypatch.setattr(OracleStore, "_take_pages", take)
    assert _expect_failure(test_extent_policy_hand_trace)


def test_pull_hand_trace():
    """Reading 11 (§5.2): the consumer's store allocates and copies; the
    producer's object is read like a get."""
    P = 256
    prod = OracleStore(8 * P, P, paged_pool=True)
    cons = OracleStore(4 * P, P, paged_pool=True)
    a = np.arange(600, dtype=np.uint8)
    _, (ia,) = prod.put_batch([PutItem(600, a, dtype_tag=3, group=7, consumers=1)])
    st, per, (ic,) = cons.pull(prod, [ia], consumers=2)
    assert st == OK and per == [OK] and cons.pages_of(ic) == [0, 1, 2]
    o = cons.objects[ic]
    assert (o.dtype_tag, o.group, o.evictable, o.consumers_left) == (3, 0, False, 2)
    assert ia not in prod.objects and prod.stats["reclaimed"] == 1   # its one consumer was the pull
    _, _, (out,) = cons.get_batch([ic])
    assert np.array_equal(out, a)
    st, per, _ = cons.pull(prod, [ia])
    assert st == NOT_FOUND and per == [NOT_FOUND]
    _, (ib,) = prod.put_batch([PutItem(600, a)])
    assert cons.pull(prod, [ib])[0] == NOSPACE and ib in prod.objects  # 3 + 3 pages > 4: nothing happens
    assert prod.objects[ib].consumers_left == 0
    assert cons.pull(OracleStore(4 * 128, 128), [1])[0] == INVALID        # page sizes differ


def _mutant_most_recent_group_first(monkeypatch):
    def victims(self, demand, pinned):
        have = len(self.free_stack)
        if have >= demand:
            return []
        cands = [o for o in self.objects if self.objects[o].evictable and self.objects[o].group not in pinned]
        if have + sum(ostore.pages_for(self.objects[c].nbytes, self.page_bytes) for c in cands) < demand:
            return None
        cands.sort(key=lambda o: (-self.group_last[self.objects[o].group], -self.objects[o].order, -o))
        out = []
        for o in cands:
            if have >= demand:
                break
            out.append(o)
            have += ostore.pages_for(self.objects[o].nbytes, self.page_bytes)
        return out
    monkeypatch.setattr(OracleStore, "_victims", victims)


def _mutant_ties_to_lowest_id(monkeypatch):
    orig = OracleStore._victims

    def victims(self, demand, pinned):
        v = orig(self, demand, pinned)
        if not v:
            return v
        cands = sorted((o for o in self.objects if self.objects[o].evictable and self.objects[o].group not in pinned),
                       key=lambda o: (self.group_last[self.objects[o].group], -self.objects[o].order, o))
        return cands[:len(v)]
    monkeypatch.setattr(OracleStore, "_victims", victims)


def _mutant_put_groups_not_pinned(monkeypatch):
    orig = OracleStore._victims
    monkeypatch.setattr(OracleStore, "_victims", lambda self, demand, pinned: orig(self, demand, set()))


def _mutant_non_evictable_are_victims(monkeypatch):
    orig = OracleStore._victims

    def victims(self, demand, pinned):
        flags = {o: self.objects[o].evictable for o in self.objects}
        for o in self.objects.values():
            o.evictable = True
        try:
            return orig(self, demand, pinned)
        finally:
            for o, f in flags.items():
                if o in self.objects:
                    self.objects[o].evictable = f
    monkeypatch.setattr(OracleStore, "_victims", victims)


def _mutant_nospace_evicts_anyway(monkeypatch):
    orig = OracleStore.put_batch

    def put_batch(self, items):
        st, ids = orig(self, items)
        if st == NOSPACE:
            pinned = {int(it.group) for it in items}
            for o in [o for o in self.objects if self.objects[o].evictable and self.objects[o].group not in pinned]:
                self._release(o)
                self.evicted.add(o)
        return st, ids
    monkeypatch.setattr(OracleStore, "put_batch", put_batch)


def _mutant_get_does_not_touch(monkeypatch):
    orig = OracleStore.get_batch

    def get_batch(self, ids, casts=None):
        saved = (self.clock, dict(self.group_last))
        out = orig(self, ids, casts)
        self.clock, self.group_last = saved[0], saved[1]
        return out
    monkeypatch.setattr(OracleStore, "get_batch", get_batch)


def _mutant_evicts_whole_groups(monkeypatch):
    orig = OracleStore._victims

    def victims(self, demand, pinned):
        v = orig(self, demand, pinned)
        if not v:
            return v
        groups = {self.objects[o].group for o in v}
        extra = sorted((o for o in self.objects if self.objects[o].evictable and self.objects[o].group in groups
                        and o not in v), key=lambda o: (-self.objects[o].order, -o))
        return v + extra
    monkeypatch.setattr(OracleStore, "_victims", victims)


@pytest.mark.parametrize("mutant", [_mutant_most_recent_group_first, _mutant_ties_to_lowest_id,
                                    _mutant_put_groups_not_pinned, _mutant_non_evictable_are_victims,
                                    _mutant_nospace_evicts_anyway, _mutant_get_does_not_touch,
                                    _mutant_evicts_whole_groups])
def test_planted_lru_mistakes_fail_the_hand_trace(monkeypatch, mutant):
    """Each plausible misreading of the victim rule (reading 6; §5.3, "How
    does it work?") planted in the oracle fails the hand-derived trace."""
    mutant(monkeypatch)
    assert _expect_failure(test_lru_reverse_layer_hand_trace)
