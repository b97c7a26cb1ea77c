"""The host control core (C++, t2i_ctl_*) against the oracle's paged model, on
the CPU: same op traces, same statuses, page lists, free stack, eviction
victims, compaction moves and counters after every op."""
import numpy as np
import pytest

import workloads as W
from oracle import OracleStore, PutItem
from paper_2607_26566_gb300 import Ctl, get_descs, put_descs


def compare(ctl: Ctl, ora: OracleStore):
    assert ctl.free_pages() == ora.free_stack
    s = ctl.stats()
    o = ora.summary()
    for k in ("used_pages", "free_pages", "limit_pages", "total_pages", "live_objects", "evictions",
              "pages_moved", "bytes_moved", "bytes_put", "bytes_got", "misses", "reclaimed"):
        assert s[k] == o[k], k
    for oid, obj in ora.objects.items():
        st, info, pages = ctl.object(oid)
        assert st == 0 and pages == obj.pages and info["nbytes"] == obj.nbytes
        assert info["group"] == obj.group and info["order"] == obj.order and info["evictable"] == int(obj.evictable)
        assert info["consumers_left"] == obj.consumers_left


def run_trace(seed, P, total_pages, n_ops, groups=4, policy=0):
    g = np.random.default_rng(seed)
    ctl = Ctl(total_pages, P, policy)
    ora = OracleStore(total_pages * P, P, keep_bytes=False, policy=policy)
    issued = []
    for _ in range(n_ops):
        r = g.random()
        if r < 0.45:
            k = int(g.integers(1, 5))
            n = g.integers(0, 4 * P + 1, k)
            grp = g.integers(0, groups, k)
            order = g.integers(0, 6, k)
            ev = (g.random(k) < 0.6).astype(np.uint32)
            cons = np.where(g.random(k) < 0.3, g.integers(1, 4, k), 0).astype(np.uint32)
            d = put_descs([0] * k, nbytes=n, group=grp, order=order, evictable=ev, consumers=cons)
            st, ids = ctl.put(d)
            ost, oids = ora.put_batch([PutItem(int(n[i]), None, 0, int(grp[i]), int(order[i]), bool(ev[i]),
                                               int(cons[i])) for i in range(k)])
            assert st == ost
            if st == 0:
                assert list(ids) == oids
                issued += oids
            assert ctl.last_evictions() == ora.last_evictions
        elif r < 0.7 and issued:
            k = int(g.integers(1, 5))
            ids = [int(x) for x in g.choice(issued, size=k)] + ([10_000_000] if g.random() < 0.05 else [])
            casts = [int(c) for c in (g.random(len(ids)) < 0.2)]
            st, per = ctl.get(get_descs(ids, cast=casts))
            ost, oper, _ = ora.get_batch(ids, casts)
            assert st == ost and list(per) == oper
        elif r < 0.9 and issued:
            k = int(g.integers(1, 4))
            ids = [int(x) for x in g.choice(issued, size=min(k, len(issued)), replace=g.random() < 0.9)]
            if g.random() < 0.05:
                ids.append(10_000_000)
            st = ctl.free(ids)
            assert st == ora.free(ids)
        else:
            limit = int(g.integers(0, total_pages + 1)) * P + (int(g.integers(1, P)) if g.random() < 0.05 else 0)
            st, moves = ctl.compact(limit)
            ost, omoves = ora.compact(limit)
            assert st == ost
            assert [tuple(int(x) for x in m) for m in moves] == omoves
        compare(ctl, ora)
    return ctl, ora


@pytest.mark.parametrize("policy", [0, 1])
@pytest.mark.parametrize("seed", range(16))
def test_random_traces_match_oracle(seed, policy):
    run_trace(seed, P=[256, 4096, 65536][seed % 3], total_pages=6 + 3 * seed, n_ops=300, policy=policy)


def test_hand_lru_trace():
    """The victims of the oracle's hand-derived LRU trace (§5.3)."""
    P = 1024
    ctl = Ctl(6, P)
    st, w1 = ctl.put(put_descs([0] * 3, nbytes=P, group=1, order=[0, 1, 2], evictable=1))
    st, w2 = ctl.put(put_descs([0] * 2, nbytes=P, group=2, order=[0, 1], evictable=1))
    assert list(w1) == [1, 2, 3] and list(w2) == [4, 5]
    assert ctl.get(get_descs([1]))[0] == 0
    st, (x,) = ctl.put(put_descs([0], nbytes=3 * P, group=3))
    assert st == 0 and ctl.last_evictions() == [5, 4] and ctl.object(x)[2] == [3, 4, 5]
    st, per = ctl.get(get_descs([4, 99, 1]))
    assert st == 4 and list(per) == [4, 3, 0]
    st, (y,) = ctl.put(put_descs([0], nbytes=P, group=2, evictable=1))
    assert st == 0 and ctl.last_evictions() == [3] and ctl.object(y)[2] == [2]
    st, _ = ctl.put(put_descs([0], nbytes=4 * P, group=4))
    assert st == 2 and ctl.last_evictions() == []


@pytest.mark.parametrize("policy", [0, 1])
def test_compaction_trace_metadata_matches_oracle(policy):
    """The fragmenting trace on a smaller pool: layout and moves."""
    P = 64 * W.KiB
    pages = 2048
    tr = W.compaction_trace(3, pages, P, n_ops=6000, lo=4 * W.KiB, hi=16 * W.MiB)
    ctl = Ctl(pages, P, policy)
    ora = OracleStore(pages * P, P, keep_bytes=False, policy=policy)
    ids = {}
    for op in tr.ops:
        if op[0] == "alloc":
            st, (i,) = ctl.put(put_descs([0], nbytes=op[2]))
            ost, (oi,) = ora.put_batch([PutItem(op[2])])
            assert st == ost == 0 and i == oi
            ids[op[1]] = oi
        else:
            oid = ids.pop(op[1])
            assert ctl.free([oid]) == ora.free([oid]) == 0
    compare(ctl, ora)
    limit = (pages * 3 // 4) * P
    st, moves = ctl.compact(limit)
    ost, omoves = ora.compact(limit)
    assert st == ost == 0 and (policy == 1 or len(omoves) > 50)  # first fit keeps the tail empty
    assert [tuple(int(x) for x in m) for m in moves] == omoves
    compare(ctl, ora)


def test_error_paths():
    ctl = Ctl(4, 256)
    st, ids = ctl.put(put_descs([0, 0], nbytes=[10, 300]))
    assert st == 0 and list(ids) == [1, 2]
    assert ctl.free([1, 1]) == 1
    assert ctl.free([1, 77]) == 3
    assert ctl.get(get_descs([1], cast=1))[0] == 1
    assert ctl.get(get_descs([2], cast=1))[0] == 0
    d = get_descs([2])
    d["reserved"] = 1
    assert ctl.get(d)[0] == 1
    assert ctl.compact(100)[0] == 1
    assert ctl.compact(5 * 256)[0] == 1
    assert ctl.put(put_descs([0], nbytes=5 * 256))[0] == 2
    # a short moves buffer changes nothing
    ctl2 = Ctl(8, 256)
    ctl2.put(put_descs([0] * 8, nbytes=256))
    ctl2.free([1, 2, 3, 4])
    before = ctl2.free_pages()
    st, moves = ctl2.compact(4 * 256, cap=1)   # retried internally with a big enough buffer
    assert st == 0 and len(moves) == 4 and ctl2.free_pages() == [] and before != []
