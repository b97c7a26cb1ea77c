"""Eviction replays of the adapter-cache workload (test helper).

The workload (512 LoRA sets of 836 bf16 objects behind a 16 GiB pool of
256 KiB pages; 10,000 calls, each a get of a window of 256 objects of one
Zipf(1.1)-popular set) follows one harness rule, the same one the benchmark's
adapter workload follows: before a call's get, the objects of its set that
are not resident -- never loaded, or evicted since their put -- are put
again, only those, in object order, with group = set, order = block and
evictable = 1. The put's victims (least recently used set first, its highest
block first, §5.3 "How does it work?") become missing objects of their own
sets.

``Replay`` applies that rule to any backend with put / last-evictions / get:
the oracle's paged model, the library's host control core alone, or (through
the benchmark's harness) the GPU store. Every decision it takes is recorded,
so two replays can be compared call by call.
"""
from __future__ import annotations

import numpy as np

import workloads as W


class AdapterShapes:
    """The seeded draws of the adapter workload: per-set ranks, per-rank
    object sizes and blocks, and every call's set and window start."""

    def __init__(self, seed: int = 0, n_sets: int = 512, n_calls: int = 10_000, window: int = 256):
        C_ = W.ADAPTERS
        self.window = window
        self.ranks = W.lora_ranks(seed, n_sets)
        objs = {r: W.lora_objects(int(r)) for r in set(int(x) for x in self.ranks)}
        self.sizes = {r: np.array([n for _, n in o], np.int64) for r, o in objs.items()}
        self.blocks = {r: np.array([b for b, _ in o], np.int64) for r, o in objs.items()}
        self.sets, self.starts = W.adapter_calls(seed, n_calls, n_sets, 836, window, C_["zipf_s"])


class OracleBackend:
    """The oracle's paged model, metadata only."""

    def __init__(self, pool_bytes: int, page_bytes: int):
        from oracle import OracleStore

        self.ora = OracleStore(pool_bytes, page_bytes, keep_bytes=False)

    def put(self, nbytes, group: int, order):
        from oracle import OK, PutItem

        st, ids = self.ora.put_batch([PutItem(int(n), None, W.DTYPE_BF16, group, int(b), True)
                                      for n, b in zip(nbytes, order)])
        assert st == OK, st
        return [int(i) for i in ids]

    def last_evictions(self):
        return [int(v) for v in self.ora.last_evictions]

    def get(self, ids):
        from oracle import OK

        st, _, _ = self.ora.get_batch([int(i) for i in ids])
        assert st == OK, st

    def free_pages(self):
        return list(self.ora.free_stack)

    def pages(self, oid: int):
        return list(self.ora.objects[int(oid)].pages)


class CtlBackend:
    """The library's host control core (t2i_ctl_*), without device memory."""

    def __init__(self, pool_bytes: int, page_bytes: int):
        from paper_2607_26566_gb300 import Ctl

        self.ctl = Ctl(pool_bytes // page_bytes, page_bytes, 0)

    def put(self, nbytes, group: int, order):
        from paper_2607_26566_gb300 import put_descs

        n = len(nbytes)
        d = put_descs(np.zeros(n, np.uint64), nbytes=nbytes, dtype_tag=W.DTYPE_BF16, group=group,
                      order=order, evictable=1)
        st, ids = self.ctl.put(d)
        assert st == 0, self.ctl.last_error()
        return [int(i) for i in ids]

    def last_evictions(self):
        return self.ctl.last_evictions()

    def get(self, ids):
        from paper_2607_26566_gb300 import get_descs

        st, _ = self.ctl.get(get_descs(np.asarray(ids, np.uint64)))
        assert st == 0, self.ctl.last_error()

    def free_pages(self):
        return self.ctl.free_pages()

    def pages(self, oid: int):
        st, _, pages = self.ctl.object(int(oid))
        assert st == 0
        return pages

    def close(self):
        self.ctl.close()


class Replay:
    """The harness rule applied to one backend. ``call(k)`` returns the
    object indices reloaded before call k's get (empty if none) and the ids
    that reload evicted, in eviction order."""

    def __init__(self, shapes: AdapterShapes, backend):
        self.sh = shapes
        self.b = backend
        self.ids = {}       # set -> ids of its objects (stale where evicted)
        self.missing = {}   # set -> object indices evicted since their put
        self.owner = {}     # live id -> (set, object index)
        self.victims = []   # every eviction, in order
        self.loads = 0

    def _load(self, s: int):
        r = int(self.sh.ranks[s])
        if s not in self.ids:
            js = list(range(len(self.sh.sizes[r])))
            self.ids[s] = [0] * len(js)
        else:
            js = sorted(self.missing.get(s, ()))
            if not js:
                return [], []
        ids = self.b.put(self.sh.sizes[r][js], s, self.sh.blocks[r][js])
        for j, i in zip(js, ids):
            self.ids[s][j] = i
            self.owner[i] = (s, j)
        self.missing[s] = set()
        ev = self.b.last_evictions()
        for v in ev:
            s2, j2 = self.owner.pop(v)
            self.missing.setdefault(s2, set()).add(j2)
        self.victims.extend(ev)
        self.loads += 1
        return js, ev

    def call(self, k: int):
        s, w = int(self.sh.sets[k]), int(self.sh.starts[k])
        js, ev = [], []
        if s not in self.ids or any(w <= j < w + self.sh.window for j in self.missing.get(s, ())):
            js, ev = self._load(s)
        self.b.get(self.ids[s][w:w + self.sh.window])
        return js, ev
