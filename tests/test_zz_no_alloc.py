"""The allocation-free gather (t2i_gather_noalloc), called through the C ABI
(marked gpu). It serves callers that cannot allocate device memory while
they move data, such as a serving process whose free HBM an inference engine
or PyTorch's caching allocator has already reserved.

Every output is compared with what the oracle fixes for it: the object's own
bytes (get(put(x)) == x), or, with the cast, the oracle's round-to-nearest-
even of those bytes (oracle.cast, written independently of the kernels).
Each case makes two calls in a row, because every call shares the library's
static scratch counters and the second must not see what the first left
behind. The cast inputs are random bit patterns, so NaNs, infinities,
subnormals and exact ties all occur.

This file is collected last on purpose: a failure here stops a first-failure
run only after every other test has run."""
import ctypes as C

import numpy as np
import pytest
import torch

from oracle.cast import f32_bits_to_bf16_bits
from paper_2607_26566_gb300 import Store, _lib as L, get_descs, put_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)
INVALID = 1
GUARD = 64


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


def random_f32_bits(n_floats: int, seed: int) -> torch.Tensor:
    """n_floats random fp32 bit patterns on the device, as bytes."""
    g = np.random.default_rng(seed)
    return torch.from_numpy(g.integers(0, 1 << 32, n_floats, dtype=np.uint64).astype(np.uint32)
                            .view(np.uint8)).to(DEV)


def expected(x: torch.Tensor, cast: int) -> np.ndarray:
    """What the oracle fixes for the output: the bytes, or their RNE cast."""
    raw = x.cpu().numpy()
    return f32_bits_to_bf16_bits(raw.view(np.uint32)).view(np.uint8) if cast else raw


def run_twice(pool, P, pages, x, cast, offset):
    """Two calls in a row, each into a fresh buffer at `offset` bytes past a
    256-byte boundary with guard bytes around it; returns the outputs."""
    n_out = x.numel() // 2 if cast else x.numel()
    outs = []
    for _ in range(2):
        buf = torch.full((n_out + offset + GUARD,), 0xA5, dtype=torch.uint8, device=DEV)
        st = noalloc(pool, P, pages, x.numel(), buf.data_ptr() + offset, n_out, cast)
        assert st == 0, L.load().t2i_last_error(None)
        torch.cuda.synchronize()
        h = buf.cpu().numpy()
        assert (h[:offset] == 0xA5).all() and (h[offset + n_out:] == 0xA5).all(), "wrote outside the destination"
        outs.append(h[offset:offset + n_out])
    return outs


@pytest.mark.parametrize("cast", [0, 1])
def test_two_calls_match_the_oracle(cast):
    """fp32 object of 3 MiB + 12 bytes in 64 KiB pages (ragged last page),
    copied or cast into an aligned destination; the store's own get gives
    the same bytes."""
    P = 64 * 1024
    x = random_f32_bits((3 * (1 << 20) + 12) // 4, seed=1 + cast)
    st, pool, oid, pages = stored(P, 64, x)
    want = expected(x, cast)
    for out in run_twice(pool, P, pages, x, cast, 0):
        assert np.array_equal(out, want)
    ref = torch.empty(want.size, dtype=torch.uint8, device=DEV)
    s, _ = st.get_batch(get_descs([oid], [ref], cast=cast))
    assert s == 0, st.last_error()
    assert np.array_equal(ref.cpu().numpy(), want)


def test_two_calls_multi_launch_unaligned():
    """9,000 pages of 256 B (two launches, two scratch counters) copied into a
    destination 3 bytes past 16-byte alignment (the any-alignment copy)."""
    P = 256
    x = torch.randint(0, 256, (9000 * P - 100,), dtype=torch.uint8, device=DEV)
    st, pool, oid, pages = stored(P, 9500, x)
    assert len(pages) == 9000
    want = expected(x, 0)
    for out in run_twice(pool, P, pages, x, 0, 3):
        assert np.array_equal(out, want)


@pytest.mark.parametrize("offset", [2, 6, 14])
def test_cast_into_2_byte_aligned_destination_two_launches(offset):
    """An fp32 object of 9,000 pages of 256 B with a ragged last page (two
    launches) cast into a destination that is 2-byte but not 16-byte
    aligned (the any-alignment cast)."""
    P = 256
    x = random_f32_bits((9000 * P - 100) // 4, seed=10 + offset)
    st, pool, oid, pages = stored(P, 9500, x)
    assert len(pages) == 9000
    want = expected(x, 1)
    for out in run_twice(pool, P, pages, x, 1, offset):
        assert np.array_equal(out, want)


@pytest.mark.parametrize("offset", [0, 6])
def test_two_calls_large_object_cast(offset):
    """256 MiB of fp32 in 2 MiB pages (~18 chunks per CTA), cast to bf16
    into an aligned destination and one 6 bytes past alignment."""
    P = 2 << 20
    x = random_f32_bits(64 << 20, seed=20 + offset)
    st, pool, oid, pages = stored(P, 130, x)
    want = expected(x, 1)
    for out in run_twice(pool, P, pages, x, 1, offset):
        assert np.array_equal(out, want)


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
