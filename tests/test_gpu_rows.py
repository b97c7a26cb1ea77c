"""GPU parity for the weight-restore, adapter-cache and compaction workloads
at the full sizes the benchmark times (marked gpu).

Full-size outputs are compared with what the oracle's get returns for them
(the bytes that were put: pinned host sources, bank windows); the page
layout, the moves and the eviction decisions are compared with the oracle's
paged model replaying the same operations.
"""
import numpy as np
import pytest
import torch

import bench
import workloads as W
from adapter_replay import AdapterShapes, OracleBackend, Replay
from oracle import OK, OracleStore, PutItem

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def test_weight_restore_full_size():
    """22.05 GiB of bf16 weights from pinned host (zero-copy kernel), every
    byte got back; page lists equal the oracle's."""
    wr = bench.WeightRestore(DEV)
    ora = OracleStore(W.WEIGHTS["pool_bytes"], W.WEIGHTS["page_bytes"], keep_bytes=False)
    wr.put_all()
    for b, (total, members) in enumerate(wr.layout):
        st, _ = ora.put_batch([PutItem(wr.specs[i].nbytes, None, W.DTYPE_BF16, 0, b, True) for i, _ in members])
        assert st == OK
    wr.get_all()
    torch.cuda.synchronize()
    assert wr.verify()
    for oid, o in list(ora.objects.items())[::37]:
        assert wr.store.ctl.object(oid)[2] == o.pages
    assert wr.store.ctl.free_pages() == ora.free_stack
    wr.free_all()
    wr.close()


def test_weight_restore_copy_engine():
    """The same restore through the copy engine (one cudaMemcpyAsync per run
    of consecutive pages), on the first 6 blocks."""
    wr = bench.WeightRestore(DEV, h2d_mode=1, n_blocks=6)
    wr.put_all()
    wr.get_all()
    torch.cuda.synchronize()
    assert wr.verify()
    assert wr.store.stats()["h2d_copies"] > 0
    wr.close()


def test_compaction_full_size():
    """64 GiB pool, the 100,000-op trace, compact to 48 GiB: moves and page
    lists equal the oracle's; every survivor's bytes survive."""
    cp = bench.Compaction(DEV)
    cp.build()
    P = cp.P
    ora = OracleStore(cp.pool_bytes, P, keep_bytes=False)
    ids = {}
    for op in cp.trace.ops:
        if op[0] == "alloc":
            st, (i,) = ora.put_batch([PutItem(op[2])])
            ids[op[1]] = i
        else:
            ora.free([ids.pop(op[1])])
    assert ids == cp.ids
    st, moves = ora.compact(cp.limit)
    assert st == OK
    s0 = cp.store.stats()
    st, moved = cp.store.compact(cp.limit)
    assert st == 0 and moved == len(moves) > 3000
    s1 = cp.store.stats()
    assert s1["bytes_moved"] - s0["bytes_moved"] == sum(m[2] for m in moves)
    assert cp.store.ctl.free_pages() == ora.free_stack
    for oid, o in ora.objects.items():
        assert cp.store.ctl.object(oid)[2] == o.pages
        assert all(p < cp.limit // P for p in o.pages)
    assert cp.verify()
    # grow back: nothing moves, the tail is free again
    st, moved = cp.store.compact(cp.pool_bytes)
    assert st == 0 and moved == 0 and ora.compact(cp.pool_bytes)[0] == OK
    assert cp.store.ctl.free_pages() == ora.free_stack
    cp.close()


def _oracle_replay(ad: "bench.Adapters", n_calls: int) -> Replay:
    """The harness's decisions on the same draws, replayed on the oracle's
    paged model (metadata only)."""
    sh = AdapterShapes(n_sets=len(ad.ranks), n_calls=len(ad.sets), window=ad.window)
    assert np.array_equal(sh.sets, ad.sets) and np.array_equal(sh.starts, ad.starts)
    rep = Replay(sh, OracleBackend(ad.pool.numel(), W.ADAPTERS["page_bytes"]))
    for k in range(n_calls):
        rep.call(k)
    return rep


def test_adapters_small_vs_oracle():
    """64 sets behind a 2 GiB pool, 400 calls: the same reloads, the same
    victims in the same order, the same page lists; every got window equals
    its bank bytes."""
    ad = bench.Adapters(DEV, n_sets=64, n_calls=400, pool_bytes=2 << 30)
    sh = AdapterShapes(n_sets=64, n_calls=400)
    oa = Replay(sh, OracleBackend(ad.pool.numel(), W.ADAPTERS["page_bytes"]))
    for k in range(400):
        s, w = ad.call(k)
        oa.call(k)
        assert ad.victims == oa.victims, k
        n = ad.expected(s, w).numel()
        assert torch.equal(ad.dst[:n], ad.expected(s, w)), k
    assert ad.victims and ad.loads > 64          # evictions and partial reloads happened
    assert ad.loads == oa.loads
    for s, ids in oa.ids.items():
        for oid in ids[::50]:
            o = oa.b.ora.objects.get(int(oid))
            if o is not None:
                assert ad.store.ctl.object(int(oid))[2] == o.pages
    assert ad.store.ctl.free_pages() == oa.b.free_pages()
    ad.close()


def test_adapters_full_size_vs_oracle():
    """The full adapter workload (512 sets, 16 GiB pool, 256 KiB pages), all
    10,000 calls of its trace on the GPU store: the store evicts exactly the
    oracle's victims in the oracle's order, reloads as often, and ends with
    the oracle's free-page stack; every got window equals its bank bytes.
    (The CPU tests also compare the control core with the oracle after every
    call of the same trace.)"""
    n = W.ADAPTERS["n_calls"]
    ad = bench.Adapters(DEV, n_calls=n)
    for k in range(n):
        s, w = ad.call(k)
        m = ad.expected(s, w).numel()
        assert torch.equal(ad.dst[:m], ad.expected(s, w)), k
    oa = _oracle_replay(ad, n)
    assert len(ad.victims) == len(oa.victims) > 1_000_000
    assert ad.victims == oa.victims
    assert ad.loads == oa.loads
    assert ad.store.ctl.free_pages() == oa.b.free_pages()
    st = ad.store.stats()
    assert st["evictions"] == len(oa.victims) and st["used_pages"] <= st["limit_pages"]
    ad.close()
