"""Edge cases of the launch packing on the GPU (marked gpu): an object whose
page list is longer than one launch's parameter space, a batch whose
descriptors span several launches, 1 GiB pages, empty and zero-byte batches,
and both unaligned kernels; all compared with the oracle's get."""
import numpy as np
import pytest
import torch

from oracle import OracleStore, PutItem
from oracle.cast import f32_bits_to_bf16_bits
from paper_2607_26566_gb300 import Store, get_descs, put_descs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def store(pool_bytes, page_bytes, **kw):
    return Store(torch.empty(pool_bytes, dtype=torch.uint8, device=DEV), page_bytes, **kw)


def test_object_longer_than_one_launch():
    """8,000 pages of 256 B in descending order (LIFO reuse): the page list
    is split across launches. On a fresh store the same object's pages are
    consecutive and travel as one run, in one launch."""
    P = 256
    st = store(9000 * P, P)
    x = torch.randint(0, 256, (8000 * P - 77,), dtype=torch.uint8, device=DEV)
    s, (i,) = st.put_batch(put_descs([x]))
    assert s == 0 and st.stats()["launches"] == 1 and st.ctl.object(int(i))[2] == list(range(8000))
    out = torch.zeros_like(x)
    assert st.get_batch(get_descs([int(i)], [out]))[0] == 0 and st.stats()["launches"] == 2
    torch.cuda.synchronize()
    assert torch.equal(out, x)
    assert st.free([int(i)]) == 0
    # the freed pages pop back in descending order: no run
    l0 = st.stats()["launches"]
    s, (j,) = st.put_batch(put_descs([x]))
    assert s == 0 and st.ctl.object(int(j))[2] == list(range(7999, -1, -1))
    assert st.stats()["launches"] - l0 >= 2
    out.zero_()
    l0 = st.stats()["launches"]
    assert st.get_batch(get_descs([int(j)], [out]))[0] == 0
    assert st.stats()["launches"] - l0 >= 2
    torch.cuda.synchronize()
    assert torch.equal(out, x)


def test_batch_spanning_several_launches():
    """1,500 objects in one call: descriptors for several launches; every
    object's bytes and every page list as the oracle's."""
    P = 4096
    rng = np.random.default_rng(8)
    st = store(4000 * P, P)
    ora = OracleStore(4000 * P, P)
    sizes = rng.integers(1, 2 * P + 1, 1500)
    buf = torch.randint(0, 256, (int(sizes.sum()) + 16,), dtype=torch.uint8, device=DEV)
    offs = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    s, ids = st.put_batch(put_descs(buf.data_ptr() + offs, nbytes=sizes))
    assert s == 0 and st.stats()["launches"] >= 2
    host = buf.cpu().numpy()
    _, oids = ora.put_batch([PutItem(int(n), host[o:o + n]) for o, n in zip(offs, sizes)])
    assert list(ids) == oids
    out = torch.zeros(int(sizes.sum()) + 64 * 1500, dtype=torch.uint8, device=DEV)
    doffs = np.concatenate([[0], np.cumsum(sizes + 64)[:-1]]) + 3     # unaligned destinations
    assert st.get_batch(get_descs(ids, out.data_ptr() + doffs, dst_bytes=sizes))[0] == 0
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    _, _, want = ora.get_batch(oids)
    for d, n, w in zip(doffs, sizes, want):
        assert np.array_equal(got[d:d + n], w)
    for oid in oids[::97]:
        assert st.ctl.object(oid)[2] == ora.objects[oid].pages


def test_gigabyte_pages():
    P = 1 << 30
    st = store(2 * P, P)
    x = torch.randint(0, 256, (P + P // 2 + 5,), dtype=torch.uint8, device=DEV)
    s, (i,) = st.put_batch(put_descs([x]))
    assert s == 0 and st.ctl.object(int(i))[2] == [0, 1]
    out = torch.empty_like(x)
    assert st.get_batch(get_descs([int(i)], [out]))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, x)
    del x, out


def test_empty_and_zero_byte_batches():
    P = 4096
    st = store(16 * P, P)
    assert st.put_batch(put_descs([]))[0] == 0
    assert st.get_batch(get_descs([]))[0] == 0
    assert st.free([]) == 0
    s, ids = st.put_batch(put_descs([0, 0, 0], nbytes=[0, 0, 0]))
    assert s == 0 and len(ids) == 3 and st.stats()["launches"] == 0
    assert st.get_batch(get_descs(ids, [0, 0, 0], dst_bytes=[0, 0, 0]))[0] == 0
    assert st.stats()["launches"] == 0 and st.stats()["used_pages"] == 0


def test_unaligned_cast_and_copy_kernels():
    """Sources at every 16-byte misalignment (put), destinations at every
    misalignment (copy) and every even one (cast): the any-alignment kernels."""
    P = 8192
    st = store(512 * P, P)
    rng = np.random.default_rng(2)
    f = rng.standard_normal(3 * P // 4 + 13).astype(np.float32)
    for m in range(16):
        raw = torch.zeros(f.nbytes + 32, dtype=torch.uint8, device=DEV)
        raw[m:m + f.nbytes].copy_(torch.from_numpy(f.view(np.uint8)))
        s, (i,) = st.put_batch(put_descs([raw.data_ptr() + m], nbytes=[f.nbytes]))
        assert s == 0
        out = torch.zeros(f.nbytes + 32, dtype=torch.uint8, device=DEV)
        assert st.get_batch(get_descs([int(i)], [out.data_ptr() + (15 - m)], dst_bytes=[f.nbytes]))[0] == 0
        bf = torch.zeros(f.nbytes // 2 + 32, dtype=torch.uint8, device=DEV)
        e = 2 * (m % 8)
        assert st.get_batch(get_descs([int(i)], [bf.data_ptr() + e], dst_bytes=[f.nbytes // 2], cast=1))[0] == 0
        torch.cuda.synchronize()
        assert np.array_equal(out.cpu().numpy()[15 - m:15 - m + f.nbytes], f.view(np.uint8))
        got = bf.cpu().numpy()[e:e + f.nbytes // 2].view(np.uint16)
        assert np.array_equal(got, f32_bits_to_bf16_bits(f.view(np.uint32)))
        assert st.free([int(i)]) == 0


def test_cast_into_two_byte_aligned_destinations():
    """The cast into destinations 2..14 bytes past a 16-byte boundary, for
    objects of 1 to 70 floats (shorter than, equal to and longer than the
    aligning head of up to 7 elements, with and without a tail) and one of
    several 32 KiB pieces, holding every class of value: each output equals
    the oracle's RNE, and the bytes around it stay untouched."""
    P = 4096
    st = store(4096 * P, P)
    rng = np.random.default_rng(17)
    special = np.array([0x7F800000, 0xFF800000, 0x7FC00001, 0xFF812345, 0x00000001, 0x80000001, 0x007FFFFF,
                        0x3F808000, 0x3F818000, 0x7F7FFFFF, 0x00000000, 0x80000000], np.uint32)
    counts = list(range(1, 18)) + [23, 24, 25, 31, 32, 33, 70, 3 * 8192 + 5]
    fs = []
    for k, nf in enumerate(counts):
        bits = rng.integers(0, 1 << 32, nf, dtype=np.uint64).astype(np.uint32)
        bits[: min(nf, len(special))] = np.roll(special, k)[: min(nf, len(special))]
        fs.append(bits)
    srcs = [torch.from_numpy(b.view(np.uint8).copy()).to(DEV) for b in fs]
    s, ids = st.put_batch(put_descs(srcs))
    assert s == 0, st.last_error()
    for e in range(2, 16, 2):
        outs = [torch.full((b.size * 2 + 64,), 0xA5, dtype=torch.uint8, device=DEV) for b in fs]
        s, per = st.get_batch(get_descs([int(i) for i in ids], [o.data_ptr() + 16 + e for o in outs],
                                        dst_bytes=[b.size * 2 for b in fs], cast=1))
        assert s == 0 and list(per) == [0] * len(fs), st.last_error()
        torch.cuda.synchronize()
        for b, o in zip(fs, outs):
            h = o.cpu().numpy()
            lo, hi = 16 + e, 16 + e + 2 * b.size
            assert np.array_equal(h[lo:hi].view(np.uint16), f32_bits_to_bf16_bits(b)), (e, b.size)
            assert (h[:lo] == 0xA5).all() and (h[hi:] == 0xA5).all(), (e, b.size)


def test_object_larger_than_64_gib():
    """An object of 65 GiB + a ragged tail in 1 GiB pages: its launch byte
    space is split into segments of at most 64 GiB, so 32-bit granule
    offsets never wrap. Every GiB of the get is compared with the put."""
    G = 1 << 30
    if torch.cuda.get_device_properties(0).total_memory < 180 * G:
        pytest.skip("needs a GPU with room for two 66 GiB buffers")
    n = 65 * G + 12345
    st = store(66 * G, G)
    g = torch.Generator(device=DEV)
    g.manual_seed(65)
    pat = torch.randint(0, 256, (G,), dtype=torch.uint8, device=DEV, generator=g)
    x = torch.empty(n, dtype=torch.uint8, device=DEV)
    for i in range(66):
        lo, hi = i * G, min((i + 1) * G, n)
        x[lo:hi] = pat[:hi - lo] ^ (i % 251)
    s, (oid,) = st.put_batch(put_descs([x]))
    assert s == 0
    x.zero_()
    assert st.get_batch(get_descs([int(oid)], [x]))[0] == 0
    torch.cuda.synchronize()
    for i in range(66):
        lo, hi = i * G, min((i + 1) * G, n)
        assert torch.equal(x[lo:hi], pat[:hi - lo] ^ (i % 251)), i
    del x


def test_large_unaligned_launches_take_chunks():
    """A 704 MiB object put from a source 3 bytes past alignment and got into
    destinations 5 bytes (copy) and 2 bytes (cast) past it: launches large
    enough for chunks from the work counter (at least 1 MiB per resident
    CTA of the any-alignment kernels, 4 per SM), in those kernels."""
    P = 2 << 20
    n = 704 << 20
    st = store(360 * P, P)
    g = torch.Generator(device=DEV)
    g.manual_seed(400)
    f = torch.randn(n // 4, generator=g, device=DEV)
    src = torch.zeros(n + 16, dtype=torch.uint8, device=DEV)
    src[3:3 + n] = f.view(torch.uint8)
    s, (i,) = st.put_batch(put_descs([src.data_ptr() + 3], nbytes=[n]))
    assert s == 0
    out = torch.zeros(n + 16, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs([int(i)], [out.data_ptr() + 5], dst_bytes=[n]))[0] == 0
    bf = torch.zeros(n // 2 + 16, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs([int(i)], [bf.data_ptr() + 2], dst_bytes=[n // 2], cast=1))[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out[5:5 + n], f.view(torch.uint8))
    assert torch.equal(bf[2:2 + n // 2].view(torch.bfloat16), f.to(torch.bfloat16))
    assert out[:5].sum() == 0 and out[5 + n:].sum() == 0


@pytest.mark.parametrize("P", [256, 1024, 4096, 16384])
def test_small_page_rounds(P):
    """Objects spanning many pages smaller than a copy round: rounds that
    cover several pages in put, get, get with a cast in the same launch, and
    the any-alignment kernels (a source 3 bytes past alignment); every byte
    against the oracle's get."""
    rng = np.random.default_rng(P)
    n_pages = (6 << 20) // P
    st = store(n_pages * P, P)
    ora = OracleStore(n_pages * P, P)
    sizes = [(1 << 20) + 48, 256 * 1024 - 32, (512 << 10) + 4 * 7]
    datas = [rng.integers(0, 256, n, dtype=np.uint8) for n in sizes]
    datas[2] = rng.standard_normal(sizes[2] // 4).astype(np.float32).view(np.uint8)
    srcs = [torch.from_numpy(d).to(DEV) for d in datas]
    raw = torch.zeros(sizes[0] + 16, dtype=torch.uint8, device=DEV)
    raw[3:3 + sizes[0]] = srcs[0]
    s, ids = st.put_batch(put_descs([raw.data_ptr() + 3, srcs[1], srcs[2]], nbytes=sizes))
    assert s == 0
    _, oids = ora.put_batch([PutItem(n, d) for n, d in zip(sizes, datas)])
    assert list(ids) == oids
    outs = [torch.zeros(sizes[0], dtype=torch.uint8, device=DEV), torch.zeros(sizes[1], dtype=torch.uint8, device=DEV),
            torch.zeros(sizes[2] // 2, dtype=torch.uint8, device=DEV)]
    assert st.get_batch(get_descs(ids, outs, dst_bytes=[sizes[0], sizes[1], sizes[2] // 2], cast=[0, 0, 1]))[0] == 0
    plain = [torch.zeros(n, dtype=torch.uint8, device=DEV) for n in sizes]
    assert st.get_batch(get_descs(ids, plain))[0] == 0
    torch.cuda.synchronize()
    _, _, want = ora.get_batch(oids, [0, 0, 1])
    for o, w in zip(outs, want):
        assert np.array_equal(o.cpu().numpy(), w)
    for o, d in zip(plain, datas):
        assert np.array_equal(o.cpu().numpy(), d)
