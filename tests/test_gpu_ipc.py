"""A pull across processes on one GPU (marked gpu): a producer process puts
objects into its store and shares the store's pool through CUDA IPC; this
process maps it and pulls the objects into its own store with
t2i_pull_pages (§5.2: the consumer pulls the producer's output into its own
arena). Every pulled byte is compared with the producer's."""
import numpy as np
import pytest
import torch

from paper_2607_26566_gb300 import Store, get_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def test_pull_pages_from_another_process():
    import torch.multiprocessing as tmp

    from tests import ipc_producer

    P = 64 * 1024
    sizes = [5 * P + 3, 100, 2 * P, 17 * P - 9]
    ctx = tmp.get_context("spawn")
    to_parent, from_parent = ctx.Queue(), ctx.Queue()
    child = ctx.Process(target=ipc_producer.run, args=(to_parent, from_parent, sizes, P, 11))
    child.start()
    try:
        s, src_pool, objects, expected = to_parent.get(timeout=300)
        assert s == 0
        st = Store(torch.empty(64 * P, dtype=torch.uint8, device=DEV), P)
        s, ids = st.pull_pages(src_pool, objects, consumers=1)
        assert s == 0, st.last_error()
        outs = [torch.zeros(n, dtype=torch.uint8, device=DEV) for n in sizes]
        assert st.get_batch(get_descs(ids, outs))[0] == 0
        torch.cuda.synchronize()
        for o, e in zip(outs, expected):
            assert torch.equal(o.cpu(), e)
        assert st.stats()["live_objects"] == 0         # one consumer each: reclaimed after the get
        # a page outside the source pool, or a wrong page count: nothing happens
        bad = [(objects[0][0], [10 ** 6] + list(objects[0][1][1:]), 7)]
        assert st.pull_pages(src_pool, bad)[0] == 1
        assert st.pull_pages(src_pool, [(objects[0][0], objects[0][1][:-1], 7)])[0] == 1
        assert st.stats()["used_pages"] == 0
        del src_pool
        from_parent.put("done")
        child.join(timeout=120)
        assert child.exitcode == 0
    finally:
        if child.is_alive():
            child.terminate()
            child.join(timeout=30)
