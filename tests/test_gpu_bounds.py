"""Bounds (marked gpu): the store writes only the bytes it was asked to.
The pool sits between two 1 MiB guard regions of a larger allocation and
every destination between guards; after random puts, gets (with and without
the cast, at every alignment) and a compaction, every guard byte and the
unused tail of every object's last page still hold the guard pattern."""
import numpy as np
import pytest
import torch

from paper_2607_26566_gb300 import Store, get_descs, put_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)
G = 0xCD
GUARD = 1 << 20


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


@pytest.mark.parametrize("P,policy", [(4096, 0), (64 * 1024, 1), (256, 0)])
def test_writes_stay_inside_objects_and_destinations(P, policy):
    rng = np.random.default_rng(P + policy)
    pages = 96
    big = torch.full((GUARD + pages * P + GUARD,), G, dtype=torch.uint8, device=DEV)
    pool = big[GUARD:GUARD + pages * P]
    st = Store(pool, P, alloc_policy=policy)
    sizes = [int(rng.integers(1, 3 * P)) & ~3 for _ in range(24)]
    sizes = [max(4, n) for n in sizes]
    srcs = []
    for n in sizes:
        off = int(rng.integers(0, 16))
        b = torch.randint(0, 256, (n + 32,), dtype=torch.uint8, device=DEV)
        srcs.append(b[off:off + n])
    s, ids = st.put_batch(put_descs(srcs))
    assert s == 0
    torch.cuda.synchronize()
    host_pool = pool.cpu().numpy()

    def check_tails():
        hp = pool.cpu().numpy()
        for i, n in zip(ids, sizes):
            if st.ctl.object(int(i))[0] != 0:
                continue
            pl = st.ctl.object(int(i))[2]
            last = pl[-1]
            used = n - (len(pl) - 1) * P
            assert (hp[last * P + used:(last + 1) * P] == G).all(), "a put wrote past its object"

    check_tails()
    # gets at every alignment into guarded destinations
    for k, (i, n, src) in enumerate(zip(ids, sizes, srcs)):
        cast = k % 3 == 0
        out_n = n // 2 if cast else n
        off = (2 * (k % 8)) if cast else (k % 16)
        dst = torch.full((out_n + 2 * 64,), G, dtype=torch.uint8, device=DEV)
        d0 = 64 + off - (off % 2 if cast else 0)
        s, _ = st.get_batch(get_descs([int(i)], [dst.data_ptr() + d0], dst_bytes=[out_n], cast=int(cast)))
        assert s == 0
        torch.cuda.synchronize()
        h = dst.cpu().numpy()
        assert (h[:d0] == G).all() and (h[d0 + out_n:] == G).all(), "a get wrote outside its destination"
        if not cast:
            assert np.array_equal(h[d0:d0 + n], src.cpu().numpy())
    # free half and compact: the compaction may write only the valid bytes of
    # each moved page at its new place; every other pool byte stays as it was
    gone = [int(i) for i in ids[::2]]
    assert st.free(gone) == 0
    ids = [i for i in ids if int(i) not in gone]
    sizes = [n for k, n in enumerate(sizes) if k % 2 == 1]
    before_pages = {int(i): st.ctl.object(int(i))[2] for i in ids}
    torch.cuda.synchronize()
    snap = pool.cpu().numpy()
    s, moved = st.compact((pages // 2) * P)
    assert s == 0
    torch.cuda.synchronize()
    after = pool.cpu().numpy()
    allowed = np.zeros(after.size, bool)
    n_moved = 0
    for i, n in zip(ids, sizes):
        new_pages = st.ctl.object(int(i))[2]
        for j, (p0, p1) in enumerate(zip(before_pages[int(i)], new_pages)):
            if p0 != p1:
                n_moved += 1
                valid = min(P, n - j * P)
                allowed[p1 * P:p1 * P + valid] = True
                assert np.array_equal(after[p1 * P:p1 * P + valid], snap[p0 * P:p0 * P + valid])
    assert n_moved == moved
    assert np.array_equal(after[~allowed], snap[~allowed]), "the compaction wrote outside the moved bytes"
    hb = big.cpu().numpy()
    assert (hb[:GUARD] == G).all() and (hb[GUARD + pages * P:] == G).all(), "a kernel wrote outside the pool"
