"""Recovery from failed launches, injected on the host (marked gpu; no GPU
fault is ever raised: the store reports the failure before issuing the
launch). A failed put leaves pages, ids and counters as before; a failed get
counts no consumer; a failed compaction keeps its page tables; a failed pull
changes neither store."""
import numpy as np
import pytest
import torch

from oracle import OracleStore, PutItem
from paper_2607_26566_gb300 import Store, get_descs, put_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)
CUDA = 5


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def store(pool_bytes, page_bytes, **kw):
    return Store(torch.empty(pool_bytes, dtype=torch.uint8, device=DEV), page_bytes, **kw)


def snapshot(st):
    s = st.stats()
    return (st.ctl.free_pages(), s["used_pages"], s["live_objects"], s["puts"], s["bytes_put"], s["gets"],
            s["limit_pages"], s["pages_moved"])


def test_failed_multi_launch_put_is_rolled_back():
    P = 4096
    st = store(4000 * P, P)
    ora = OracleStore(4000 * P, P, keep_bytes=False)
    buf = torch.randint(0, 256, (1500 * P,), dtype=torch.uint8, device=DEV)
    s, first = st.put_batch(put_descs([buf.data_ptr()], nbytes=[3 * P]))
    ora.put_batch([PutItem(3 * P)])
    before = snapshot(st)
    d = put_descs(buf.data_ptr() + P * np.arange(1500), nbytes=np.full(1500, P))
    assert st.inject_launch_failure(2) == 0           # the second of the batch's launches fails
    s, _ = st.put_batch(d)
    assert s == CUDA and "injected" in st.last_error()
    assert snapshot(st) == before
    s, ids = st.put_batch(d)                          # the same batch again: as if the failure never was
    _, oids = ora.put_batch([PutItem(P)] * 1500)
    assert s == 0 and list(ids) == oids
    assert st.ctl.free_pages() == ora.free_stack
    for oid in oids[::101]:
        assert st.ctl.object(oid)[2] == ora.objects[oid].pages


def test_failed_get_counts_no_consumer():
    P = 64 * 1024
    st = store(16 * P, P)
    x = torch.randint(0, 256, (3 * P,), dtype=torch.uint8, device=DEV)
    s, (i,) = st.put_batch(put_descs([x], consumers=1))
    out = torch.zeros_like(x)
    assert st.inject_launch_failure(1) == 0
    assert st.get_batch(get_descs([int(i)], [out]))[0] == CUDA
    assert st.ctl.object(int(i))[1]["consumers_left"] == 1 and st.stats()["gets"] == 0
    assert st.get_batch(get_descs([int(i)], [out]))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, x) and st.stats()["reclaimed"] == 1


def test_failed_compaction_keeps_its_page_tables():
    P = 64 * 1024
    st = store(8 * P, P)
    a = torch.randint(0, 256, (4 * P,), dtype=torch.uint8, device=DEV)
    b = torch.randint(0, 256, (4 * P - 9,), dtype=torch.uint8, device=DEV)
    s, (ia, ib) = st.put_batch(put_descs([a, b]))
    assert st.free([int(ia)]) == 0
    before = snapshot(st)
    pages_b = st.ctl.object(int(ib))[2]
    assert st.inject_launch_failure(1) == 0
    s, moved = st.compact(4 * P)
    assert s == CUDA and moved == 0
    assert snapshot(st) == before and st.ctl.object(int(ib))[2] == pages_b
    out = torch.zeros_like(b)
    assert st.get_batch(get_descs([int(ib)], [out]))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, b)
    s, moved = st.compact(4 * P)                      # and it still works
    assert s == 0 and moved == 4 and max(st.ctl.object(int(ib))[2]) < 4
    assert st.get_batch(get_descs([int(ib)], [out]))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, b)


def test_failed_pull_changes_neither_store():
    P = 64 * 1024
    prod, cons = store(16 * P, P), store(16 * P, P)
    x = torch.randint(0, 256, (5 * P,), dtype=torch.uint8, device=DEV)
    s, (i,) = prod.put_batch(put_descs([x], consumers=1))
    bp, bc = snapshot(prod), snapshot(cons)
    assert cons.inject_launch_failure(1) == 0
    s, _, _ = cons.pull(prod, [int(i)])
    assert s == CUDA
    assert snapshot(prod) == bp and snapshot(cons) == bc
    assert prod.ctl.object(int(i))[1]["consumers_left"] == 1
    s, (j,), _ = cons.pull(prod, [int(i)])
    assert s == 0 and prod.stats()["reclaimed"] == 1
    out = torch.zeros_like(x)
    assert cons.get_batch(get_descs([int(j)], [out]))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, x)


SLEEP_CYCLES_PER_MS = 2.0e6   # torch.cuda._sleep spins ~this many clock cycles per millisecond


def _late(stream, ms):
    """Keeps ``stream`` busy for about ``ms`` (torch's bounded sleep kernel)."""
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(ms * SLEEP_CYCLES_PER_MS))


def test_failed_put_still_orders_the_pages_it_hands_back():
    """A put that fails at its second launch has its first launch enqueued,
    late, on its stream. The pages it hands back go to the next put, on
    another stream, which must wait for that launch: else the late launch
    overwrites the new object's bytes."""
    P = 256
    st = store(8000 * P, P)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    a = torch.randint(0, 256, (8000 * P,), dtype=torch.uint8, device=DEV)
    b = torch.randint(0, 256, (8000 * P,), dtype=torch.uint8, device=DEV)
    # a put and a free first: the pages then pop in descending order, so the
    # object's page list is not one run and takes two launches
    s, (k,) = st.put_batch(put_descs([a]), stream=s1)
    assert s == 0 and st.free([int(k)]) == 0
    torch.cuda.synchronize()
    _late(s1, 30)
    assert st.inject_launch_failure(2) == 0          # 8,000 scattered pages take two launches
    s, _ = st.put_batch(put_descs([a]), stream=s1)
    assert s == CUDA and st.stats()["used_pages"] == 0
    s, (j,) = st.put_batch(put_descs([b]), stream=s2)
    assert s == 0 and st.ctl.object(int(j))[2] == list(range(7999, -1, -1))   # the same pages
    out = torch.zeros_like(b)
    assert st.get_batch(get_descs([int(j)], [out]), stream=s2)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, b), "a launch of the failed put wrote pages handed to a later put"


def test_failed_compaction_still_orders_the_pages_it_wrote():
    """A compaction of 2,000 pages fails at its second launch, the first
    (late on its stream) already enqueued. Its destination pages are free
    again; a put on another stream that takes them must wait for that
    launch. Every object, old and new, keeps its bytes."""
    P = 4096
    st = store(8000 * P, P)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    src = torch.randint(0, 256, (8000 * P,), dtype=torch.uint8, device=DEV)
    new = torch.randint(0, 256, (2000 * P,), dtype=torch.uint8, device=DEV)
    s, ids = st.put_batch(put_descs(src.data_ptr() + P * np.arange(8000), nbytes=np.full(8000, P)))
    assert s == 0
    assert st.free([int(i) for i in ids[0:4000:2]]) == 0      # pages 0, 2, ..., 3998
    torch.cuda.synchronize()
    _late(s1, 30)
    assert st.inject_launch_failure(2) == 0
    s, moved = st.compact(6000 * P, stream=s1)        # 2,000 one-page moves: several launches
    assert s == CUDA and moved == 0
    s, nids = st.put_batch(put_descs(new.data_ptr() + P * np.arange(2000), nbytes=np.full(2000, P)), stream=s2)
    assert s == 0
    assert sorted(p for i in nids for p in st.ctl.object(int(i))[2]) == list(range(0, 4000, 2))
    out = torch.zeros(2000 * P, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs(nids, out.data_ptr() + P * np.arange(2000), dst_bytes=np.full(2000, P)),
                        stream=s2)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, new), "a launch of the failed compaction wrote pages handed to a later put"
    live = [int(i) for i in ids[1:4000:2]] + [int(i) for i in ids[4000:]]
    out = torch.zeros(len(live) * P, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs(live, out.data_ptr() + P * np.arange(len(live)),
                                  dst_bytes=np.full(len(live), P)))[0] == 0
    torch.cuda.synchronize()
    want = torch.cat([src[(2 * k + 1) * P:(2 * k + 2) * P] for k in range(2000)] + [src[4000 * P:]])
    assert torch.equal(out, want)
