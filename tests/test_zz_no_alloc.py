"""The allocation-free gather (t2i_gather_noalloc), called through the C ABI
and compared with the store's own get (t2i_get_batch) on the same object
(marked gpu). It serves callers that cannot allocate device memory while
they move data, such as a serving process whose free HBM an inference engine
or PyTorch's caching allocator has already reserved. Each case makes two
calls in a row, because every call shares the library's static scratch
counters and the second must not see what the first left behind.

This file is collected last on purpose: a failure here stops a first-failure
run only after every other test has run."""
import ctypes as C

import numpy as np
import pytest
import torch

from paper_2607_26566_gb300 import Store, _lib as L, get_descs, put_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)
INVALID = 1


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def noalloc(pool, P, pages, nbytes, dst_addr, dst_bytes, cast, stream=None):
    """One call of the entry point through the C ABI (no binding logic)."""
    lib = L.load()
    pg = np.ascontiguousarray(pages, dtype=np.uint32)
    s = torch.cuda.current_stream() if stream is None else stream
    return lib.t2i_gather_noalloc(pool.data_ptr(), pool.numel(), P, pg.ctypes.data_as(C.POINTER(C.c_uint32)),
                                  len(pg), nbytes, dst_addr, dst_bytes, cast, 0, s.cuda_stream)


def stored(P, pool_pages, x):
    """A store holding x; returns (store, pool, id, page list)."""
    pool = torch.empty(pool_pages * P, dtype=torch.uint8, device=DEV)
    st = Store(pool, P)
    s, (i,) = st.put_batch(put_descs([x]))
    assert s == 0, st.last_error()
    return st, pool, int(i), st.ctl.object(int(i))[2]


def reference(st, oid, n_out, cast, offset=0):
    """The store's own get of the object into a fresh buffer."""
    ref = torch.zeros(n_out + offset, dtype=torch.uint8, device=DEV)
    s, _ = st.get_batch(get_descs([oid], [ref.data_ptr() + offset], dst_bytes=[n_out], cast=cast))
    assert s == 0, st.last_error()
    return ref


@pytest.mark.parametrize("cast", [0, 1])
def test_two_calls_match_get_batch(cast):
    """fp32 object of 3 MiB + 12 bytes in 64 KiB pages (ragged last page),
    copied or cast; two calls in a row into separate buffers."""
    P = 64 * 1024
    x = torch.randn((3 * (1 << 20) + 12) // 4, dtype=torch.float32, device=DEV).view(torch.uint8)
    st, pool, oid, pages = stored(P, 64, x)
    n_out = x.numel() // 2 if cast else x.numel()
    ref = reference(st, oid, n_out, cast)
    outs = [torch.zeros(n_out, dtype=torch.uint8, device=DEV) for _ in range(2)]
    for o in outs:
        assert noalloc(pool, P, pages, x.numel(), o.data_ptr(), n_out, cast) == 0, L.load().t2i_last_error(None)
    torch.cuda.synchronize()
    for o in outs:
        assert torch.equal(o, ref)


def test_two_calls_multi_launch_unaligned():
    """9,000 pages of 256 B (two launches, two scratch counters) into a
    destination 3 bytes past 16-byte alignment (the any-alignment kernel)."""
    P = 256
    x = torch.randint(0, 256, (9000 * P - 100,), dtype=torch.uint8, device=DEV)
    st, pool, oid, pages = stored(P, 9500, x)
    assert len(pages) == 9000
    ref = reference(st, oid, x.numel(), 0, offset=3)
    for _ in range(2):
        out = torch.zeros_like(ref)
        assert noalloc(pool, P, pages, x.numel(), out.data_ptr() + 3, x.numel(), 0) == 0, \
            L.load().t2i_last_error(None)
        torch.cuda.synchronize()
        assert torch.equal(out, ref) and torch.equal(out[3:], x)


def test_two_calls_large_object_cast():
    """256 MiB of fp32 in 2 MiB pages: ~18 chunks per CTA, cast to bf16."""
    P = 2 << 20
    x = torch.randn(64 << 20, dtype=torch.float32, device=DEV).view(torch.uint8)
    st, pool, oid, pages = stored(P, 130, x)
    n_out = x.numel() // 2
    ref = reference(st, oid, n_out, 1)
    for _ in range(2):
        out = torch.zeros(n_out, dtype=torch.uint8, device=DEV)
        assert noalloc(pool, P, pages, x.numel(), out.data_ptr(), n_out, 1) == 0, L.load().t2i_last_error(None)
        torch.cuda.synchronize()
        assert torch.equal(out, ref)
    assert torch.equal(ref.view(torch.bfloat16), x.view(torch.float32).to(torch.bfloat16))


def test_sizes_beyond_the_maximum_are_rejected():
    """More pages than 64 launches of scratch counters cover, a page list
    that does not match nbytes, and a page outside the pool: INVALID with a
    message, nothing enqueued."""
    P = 256
    pool = torch.empty(1 << 20, dtype=torch.uint8, device=DEV)
    dst = torch.empty(1 << 20, dtype=torch.uint8, device=DEV)
    lib = L.load()
    n = 64 * 7930 + 1
    assert noalloc(pool, P, np.zeros(n, np.uint32), n * P, dst.data_ptr(), dst.numel(), 0) == INVALID
    assert b"maximum" in lib.t2i_last_error(None)
    assert noalloc(pool, P, np.zeros(3, np.uint32), 5 * P, dst.data_ptr(), dst.numel(), 0) == INVALID
    assert noalloc(pool, P, np.array([4096], np.uint32), P, dst.data_ptr(), dst.numel(), 0) == INVALID
    assert b"outside the pool" in lib.t2i_last_error(None)
    torch.cuda.synchronize()
