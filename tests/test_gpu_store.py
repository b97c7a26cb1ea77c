"""GPU parity: the CUDA store against the oracle, bit for bit (marked gpu).

Small cases compare every byte of every get with the oracle (the definitional
map plus the oracle's RNE) and the page lists with the oracle's paged model;
they span several 16 KiB units per page, ragged tails, zero-byte objects,
misaligned user pointers, pinned-host sources and destinations, evictions and
compactions.
"""
import numpy as np
import pytest
import torch

import workloads as W
from oracle import OracleStore, PutItem
from oracle.cast import cast_bytes_f32_to_bf16, f32_bits_to_bf16_bits
from paper_2607_26566_gb300 import Store, get_descs, put_descs

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _built(lib):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield


def dev_bytes(a: np.ndarray, offset: int = 0) -> torch.Tensor:
    """A device uint8 view of ``a`` starting ``offset`` bytes into a fresh allocation."""
    a = np.ascontiguousarray(a).view(np.uint8).reshape(-1)
    buf = torch.empty(a.size + offset + 16, dtype=torch.uint8, device=DEV)
    v = buf[offset:offset + a.size]
    v.copy_(torch.from_numpy(a))
    return v


def dev_empty(n: int, offset: int = 0) -> torch.Tensor:
    buf = torch.full((n + offset + 16,), 0xA5, dtype=torch.uint8, device=DEV)
    return buf[offset:offset + n]


def host(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy()


def make_store(pool_bytes, page_bytes, **kw):
    pool = torch.empty(pool_bytes, dtype=torch.uint8, device=DEV)
    return Store(pool, page_bytes, **kw)


def compare_meta(st: Store, ora: OracleStore):
    assert st.ctl.free_pages() == ora.free_stack
    for oid, o in ora.objects.items():
        assert st.ctl.object(oid)[2] == o.pages


def check_all_gets(st: Store, ora: OracleStore, rng, with_cast=True):
    """Get every live object (random alignment, random cast where allowed)
    and compare with the oracle's get."""
    ids = [oid for oid, o in ora.objects.items() if o.data is not None]
    if not ids:
        return
    casts = [int(with_cast and ora.objects[i].nbytes % 4 == 0 and rng.random() < 0.3) for i in ids]
    offs = [int(rng.integers(0, 16)) if rng.random() < 0.3 else 0 for _ in ids]
    offs = [o & ~1 if c else o for o, c in zip(offs, casts)]
    dsts = [dev_empty(ora.objects[i].nbytes // (2 if c else 1), o) for i, c, o in zip(ids, casts, offs)]
    s, per = st.get_batch(get_descs(ids, dsts, cast=casts))
    assert s == 0, st.last_error()
    ost, _, outs = ora.get_batch(ids, casts)
    assert ost == 0
    torch.cuda.synchronize()
    for i, d, want in zip(ids, dsts, outs):
        assert np.array_equal(host(d), want), f"object {i}"


def test_tiny_config_bit_exact():
    """64 MiB pool, 64 KiB pages: put 32, get all, free every third, put 8 more, get all."""
    C = W.TINY
    first, more = W.tiny_objects(0)
    st = make_store(C["pool_bytes"], C["page_bytes"])
    ora = OracleStore(C["pool_bytes"], C["page_bytes"])
    srcs = [dev_bytes(x) for x in first]
    s, ids = st.put_batch(put_descs(srcs))
    assert s == 0, st.last_error()
    ost, oids = ora.put_batch([PutItem(x.size, x) for x in first])
    assert list(ids) == oids
    rng = np.random.default_rng(0)
    check_all_gets(st, ora, rng, with_cast=False)
    gone = [oids[i] for i in W.tiny_freed_indices()]
    assert st.free(gone) == 0 and ora.free(gone) == 0
    srcs2 = [dev_bytes(x) for x in more]
    s, ids2 = st.put_batch(put_descs(srcs2))
    assert s == 0
    ora.put_batch([PutItem(x.size, x) for x in more])
    compare_meta(st, ora)
    check_all_gets(st, ora, rng, with_cast=False)
    assert st.stats()["live_objects"] == 30


@pytest.mark.parametrize("seed,P,pages,policy", [(0, 256, 64, 0), (1, 4096, 48, 0), (2, 64 * 1024, 24, 0),
                                                 (3, 2 * 1024 * 1024, 6, 0), (4, 32 * 1024, 40, 0), (5, 1024, 200, 0),
                                                 (6, 256, 64, 1), (7, 4096, 48, 1), (8, 64 * 1024, 24, 1)])
def test_random_ops_vs_oracle(seed, P, pages, policy):
    """Random puts (evictions included), gets, frees and compactions: every
    status, id, eviction, page list and byte equal to the oracle's, under
    both placement policies."""
    rng = np.random.default_rng(seed)
    st = make_store(pages * P, P, alloc_policy=policy)
    ora = OracleStore(pages * P, P, policy=policy)
    keep = []
    for step in range(60):
        r = rng.random()
        if r < 0.45:
            k = int(rng.integers(1, 6))
            items, descs_src = [], []
            for _ in range(k):
                n = int(rng.integers(0, 3 * P + 1)) if rng.random() < 0.8 else int(rng.integers(0, 64))
                n -= n % 4 if rng.random() < 0.5 else 0
                data = rng.integers(0, 256, n, dtype=np.uint8)
                off = int(rng.integers(0, 16)) if rng.random() < 0.3 else 0
                t = dev_bytes(data, off)
                keep.append(t)
                items.append(PutItem(n, data, group=int(rng.integers(0, 3)), order=int(rng.integers(0, 5)),
                                     evictable=bool(rng.random() < 0.5)))
                descs_src.append(t)
            d = put_descs(descs_src, group=[it.group for it in items], order=[it.order for it in items],
                          evictable=[int(it.evictable) for it in items])
            s, ids = st.put_batch(d)
            ost, oids = ora.put_batch(items)
            assert s == ost, st.last_error()
            if s == 0:
                assert list(ids) == oids
                assert st.ctl.last_evictions() == ora.last_evictions
        elif r < 0.65:
            check_all_gets(st, ora, rng)
        elif r < 0.85 and ora.objects:
            ids = [int(x) for x in rng.choice(list(ora.objects), size=min(2, len(ora.objects)), replace=False)]
            assert st.free(ids) == ora.free(ids) == 0
        else:
            limit = int(rng.integers(0, pages + 1)) * P
            s, moved = st.compact(limit)
            ost, moves = ora.compact(limit)
            assert s == ost
            if s == 0:
                assert moved == len(moves)
        compare_meta(st, ora)
    check_all_gets(st, ora, rng)
    torch.cuda.synchronize()


def test_cast_structured_patterns():
    """Every rounding case of every exponent through the fused cast."""
    from tests.test_oracle_cast import structured_patterns

    u = structured_patterns(7).astype(np.uint32)
    st = make_store(64 << 20, 2 << 20)
    src = dev_bytes(u.view(np.uint8))
    s, (i,) = st.put_batch(put_descs([src]))
    assert s == 0
    out = torch.empty(u.size, dtype=torch.int16, device=DEV)
    s, _ = st.get_batch(get_descs([int(i)], [out], cast=1))
    assert s == 0, st.last_error()
    got = host(out).view(np.uint16)
    assert np.array_equal(got, f32_bits_to_bf16_bits(u))


def test_cast_exhaustive_2_32():
    """All 2^32 fp32 bit patterns, in chunks of 2^26, against the oracle's RNE."""
    chunk = 1 << 26
    st = make_store(2 << 30, 2 << 20)
    out = torch.empty(chunk, dtype=torch.int16, device=DEV)
    base = torch.arange(chunk, dtype=torch.int64, device=DEV)
    for c in range((1 << 32) // chunk):
        pat = base + c * chunk                      # the fp32 bit patterns of this chunk
        bits = torch.where(pat >= 2**31, pat - 2**32, pat).to(torch.int32)
        s, (i,) = st.put_batch(put_descs([bits]))
        assert s == 0
        s, _ = st.get_batch(get_descs([int(i)], [out], cast=1))
        assert s == 0
        got = host(out).view(np.uint16)
        want = f32_bits_to_bf16_bits(np.arange(c * chunk, (c + 1) * chunk, dtype=np.uint64).astype(np.uint32))
        assert np.array_equal(got, want), f"chunk {c}"
        assert st.free([int(i)]) == 0


def test_handoff_small_vs_oracle():
    """The handoff workload at reduced tensor sizes, every byte vs the oracle."""
    specs = W.handoff_specs(2, text_len=40, text_dim=96, pooled_dim=24, lat_c=4, lat_hw=24, img_hw=40)
    P = 16 * 1024
    st = make_store(1024 * P, P)
    ora = OracleStore(1024 * P, P)
    ci = W.handoff_cast_index()
    all_ids = []
    for r in range(12):
        arrs = W.handoff_request(5, r, specs)
        srcs = [dev_bytes(a) for a in arrs]
        s, ids = st.put_batch(put_descs(srcs, dtype_tag=[sp.dtype_tag for sp in specs]))
        assert s == 0
        ost, oids = ora.put_batch([PutItem(a.nbytes, a.view(np.uint8).reshape(-1), sp.dtype_tag)
                                   for a, sp in zip(arrs, specs)])
        assert list(ids) == oids
        all_ids.append(oids)
    compare_meta(st, ora)
    for oids in all_ids:
        casts = [1 if j == ci else 0 for j in range(len(specs))]
        dsts = [dev_empty(ora.objects[i].nbytes // (2 if c else 1)) for i, c in zip(oids, casts)]
        s, _ = st.get_batch(get_descs(oids, dsts, cast=casts))
        assert s == 0
        _, _, outs = ora.get_batch(oids, casts)
        for d, w in zip(dsts, outs):
            assert np.array_equal(host(d), w)
        assert st.free(oids) == ora.free(oids) == 0
    assert st.stats()["used_pages"] == 0


@pytest.mark.parametrize("B", [1, 4, 8])
def test_handoff_full_size(B):
    """8 GiB pool, 2 MiB pages, 64 requests in flight, the launch shape the
    benchmark times. Every non-cast get must equal its input byte for byte
    (get(put(x)) == x), and every request's cast latents must equal the
    oracle's RNE of its input."""
    C = W.HANDOFF
    specs = W.handoff_specs(B)
    st = make_store(C["pool_bytes"], C["page_bytes"])
    ora = OracleStore(C["pool_bytes"], C["page_bytes"], keep_bytes=False)
    ci = W.handoff_cast_index()
    reqs, ids_all = [], []
    for r in range(C["requests"]):
        ts = W.handoff_request_torch(0, r, specs, DEV)
        s, ids = st.put_batch(put_descs(ts, nbytes=[sp.nbytes for sp in specs]))
        assert s == 0, st.last_error()
        ost, oids = ora.put_batch([PutItem(sp.nbytes, None) for sp in specs])
        assert list(ids) == oids
        reqs.append(ts)
        ids_all.append(oids)
    compare_meta(st, ora)
    for r, (ts, oids) in enumerate(zip(reqs, ids_all)):
        outs = [torch.empty_like(t) if j != ci else torch.empty(t.shape, dtype=torch.bfloat16, device=DEV)
                for j, t in enumerate(ts)]
        casts = [1 if j == ci else 0 for j in range(len(specs))]
        s, _ = st.get_batch(get_descs(oids, outs, dst_bytes=[sp.nbytes // (2 if c else 1)
                                                             for sp, c in zip(specs, casts)], cast=casts))
        assert s == 0, st.last_error()
        for j, (t, o) in enumerate(zip(ts, outs)):
            if j != ci:
                assert torch.equal(t.view(torch.uint8).reshape(-1), o.view(torch.uint8).reshape(-1)), (r, j)
        lat = ts[ci].reshape(-1).view(torch.int32).cpu().numpy().view(np.uint32)
        got = outs[ci].reshape(-1).view(torch.int16).cpu().numpy().view(np.uint16)
        assert np.array_equal(got, f32_bits_to_bf16_bits(lat)), r
    for oids in ids_all:
        assert st.free(oids) == 0
    assert st.stats()["used_pages"] == 0


@pytest.mark.parametrize("h2d_mode", [0, 1])
def test_host_sources_and_destinations(h2d_mode):
    """Puts from pinned and pageable host memory, gets into pinned host memory."""
    rng = np.random.default_rng(9)
    P = 64 * 1024
    st = make_store(256 * P, P, h2d_mode=h2d_mode)
    ora = OracleStore(256 * P, P)
    datas = [rng.integers(0, 256, int(n), dtype=np.uint8) for n in (1, 100, P, 3 * P + 17, 5 * P, 12345)]
    pinned = [torch.from_numpy(d).pin_memory() for d in datas[:4]]
    pageable = [np.ascontiguousarray(d) for d in datas[4:]]
    s, ids = st.put_batch(put_descs(pinned + pageable, src_is_host=1))
    assert s == 0, st.last_error()
    ora.put_batch([PutItem(d.size, d) for d in datas])
    outs = [torch.empty(d.size, dtype=torch.uint8).pin_memory() for d in datas]
    s, _ = st.get_batch(get_descs([int(i) for i in ids], outs))
    assert s == 0, st.last_error()
    torch.cuda.synchronize()
    for o, d in zip(outs, datas):
        assert np.array_equal(o.numpy(), d)
    stats = st.stats()
    assert stats["h2d_copies"] > 0                 # pageable sources always take the copy engine
    assert stats["launches"] >= (2 if h2d_mode == 0 else 1)


@pytest.mark.parametrize("h2d_mode", [0, 1])
def test_copy_engine_gets_into_host(h2d_mode):
    """d2h_mode = 1: gets into pinned host memory take the copy engine (one
    copy per run of consecutive pages, any alignment), items with the cast
    and device destinations stay in the kernel, all in one call."""
    rng = np.random.default_rng(11)
    P = 64 * 1024
    st = make_store(256 * P, P, h2d_mode=h2d_mode, d2h_mode=1)
    ora = OracleStore(256 * P, P)
    # fragment the free stack so that page lists break into several runs
    s, filler = st.put_batch(put_descs([0] * 6, nbytes=[7 * P] * 6))
    assert s == 0 and st.free([int(x) for x in filler[::2]]) == 0
    ora.put_batch([PutItem(7 * P) for _ in range(6)])
    ora.free([1, 3, 5])
    sizes = (1, 100, P, 3 * P + 17, 9 * P + 5, 12345)
    datas = [rng.integers(0, 256, n, dtype=np.uint8) for n in sizes]
    f = rng.standard_normal(3 * P // 4 + 3).astype(np.float32)
    f[:4] = [np.inf, -np.inf, np.nan, -0.0]
    datas.append(f.view(np.uint8))
    srcs = [torch.from_numpy(d).to(DEV) for d in datas]
    s, ids = st.put_batch(put_descs(srcs))
    assert s == 0, st.last_error()
    _, oids = ora.put_batch([PutItem(d.size, d) for d in datas])
    assert [int(i) for i in ids] == oids
    compare_meta(st, ora)
    big = torch.zeros(sum(sizes) + 64, dtype=torch.uint8).pin_memory()
    offs = np.cumsum([3] + [n + 5 for n in sizes[:-1]])           # odd offsets: unaligned host pointers
    host_outs = [big[int(o):int(o) + n] for o, n in zip(offs, sizes)]
    cast_out = torch.empty(f.size, dtype=torch.bfloat16).pin_memory()
    dev_out = torch.empty(sizes[3], dtype=torch.uint8, device=DEV)
    gd = get_descs([int(i) for i in ids[:6]] + [int(ids[6]), int(ids[3])], host_outs + [cast_out, dev_out],
                   cast=[0] * 6 + [1, 0])
    launches0, d2h0 = st.stats()["launches"], st.stats()["d2h_copies"]
    s, per = st.get_batch(gd)
    assert s == 0 and list(per) == [0] * 8, st.last_error()
    torch.cuda.synchronize()
    for o, d in zip(host_outs, datas):
        assert np.array_equal(o.numpy(), d)
    assert np.array_equal(cast_out.view(torch.int16).numpy().view(np.uint16),
                          f32_bits_to_bf16_bits(f.view(np.uint32)))
    assert np.array_equal(dev_out.cpu().numpy(), datas[3])
    stats = st.stats()
    assert stats["launches"] - launches0 == 1          # the cast and the device destination
    runs = sum(1 + sum(1 for a, b in zip(ps, ps[1:]) if b != a + 1)
               for ps in (ora.pages_of(i) for i in oids[:6]))
    assert stats["d2h_copies"] - d2h0 == runs and runs > 6
    # pageable destinations stay refused: nothing is enqueued or written
    pageable = np.full(sizes[2], 7, np.uint8)
    s, per = st.get_batch(get_descs([int(ids[2])], [pageable]))
    assert s == 1 and list(per) == [1] and (pageable == 7).all()
    assert st.stats()["d2h_copies"] == stats["d2h_copies"]


def test_copy_engine_get_orders_before_page_reuse():
    """A copy-engine get on one stream, then a put on another stream that
    reuses the pages: the put waits for the copy (write after read)."""
    P = 2 << 20
    st = make_store(64 * P, P, d2h_mode=1)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    a = torch.randint(0, 256, (64 * P,), dtype=torch.uint8, device=DEV)
    b = torch.randint(0, 256, (64 * P,), dtype=torch.uint8, device=DEV)
    host = torch.empty(64 * P, dtype=torch.uint8).pin_memory()
    want = a.cpu()
    torch.cuda.synchronize()
    for _ in range(3):
        s, (i,) = st.put_batch(put_descs([a]), stream=s1)
        assert s == 0
        s, _ = st.get_batch(get_descs([int(i)], [host]), stream=s2)
        assert s == 0
        assert st.free([int(i)]) == 0
        s, (j,) = st.put_batch(put_descs([b]), stream=s3)     # the same pages
        assert s == 0
        torch.cuda.synchronize()
        assert torch.equal(host, want)
        assert st.free([int(j)]) == 0
    assert st.stats()["d2h_copies"] >= 3


def test_streams_are_ordered():
    """Put on one stream, get on another, free, re-put on a third: the store
    orders its own work across streams."""
    P = 2 << 20
    st = make_store(8 * P, P)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    a = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    b = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    out = torch.empty_like(a)
    for _ in range(5):
        s, (i,) = st.put_batch(put_descs([a]), stream=s1)
        assert s == 0
        s, _ = st.get_batch(get_descs([int(i)], [out]), stream=s2)
        assert s == 0
        assert st.free([int(i)]) == 0
        s, (j,) = st.put_batch(put_descs([b]), stream=s3)  # reuses the same pages
        assert s == 0
        assert st.free([int(j)]) == 0
        torch.cuda.synchronize()
        assert torch.equal(out, a)


def test_error_paths_never_reach_the_gpu():
    P = 64 * 1024
    st = make_store(16 * P, P)
    x = torch.zeros(1000, dtype=torch.uint8, device=DEV)
    s, (i,) = st.put_batch(put_descs([x]))
    assert s == 0
    pageable = np.zeros(1000, np.uint8)
    assert st.put_batch(put_descs([pageable]))[0] == 1                  # host memory as a device source
    assert st.put_batch(put_descs([x], nbytes=[10**8]))[0] == 1        # runs past the allocation
    assert st.put_batch(put_descs([12345], nbytes=[10]))[0] == 1       # unknown pointer
    assert st.put_batch(put_descs([st.pool], nbytes=[100]))[0] == 1    # source inside the pool
    small = torch.empty(10, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs([int(i)], [small]))[0] == 1          # destination too small
    assert st.get_batch(get_descs([int(i)], [st.pool], dst_bytes=[1000]))[0] == 1  # into the pool
    assert st.get_batch(get_descs([int(i)], [pageable]))[0] == 1       # pageable destination
    assert st.get_batch(get_descs([999], [x]))[0] == 3
    assert st.put_batch(put_descs([0], nbytes=[17 * P]))[0] == 2
    odd = torch.empty(1001, dtype=torch.uint8, device=DEV)
    assert st.get_batch(get_descs([int(i)], [odd[1:]], cast=1))[0] == 1  # cast into an odd address
    torch.cuda.synchronize()
    assert st.stats()["live_objects"] == 1 and st.stats()["used_pages"] == 1


def test_error_paths_through_the_cpython_entry_points():
    """The same refusals through the CPython entry points (prepared batches'
    path): bad sources and destinations come back INVALID from the library
    before any launch, unknown ids NOT_FOUND, and the store is unchanged."""
    P = 64 * 1024
    st = make_store(16 * P, P)
    assert st._fast is not None, "the CPython entry points were not built"
    stream = int(torch.cuda.current_stream().cuda_stream)
    x = torch.zeros(1000, dtype=torch.uint8, device=DEV)
    pp = st.prepare_put(put_descs([x]))
    s, ids = st.put_prepared(pp)
    assert s == 0
    good = int(ids[0])
    bad_puts = [put_descs([x], nbytes=[10**8]), put_descs([12345], nbytes=[10]),
                put_descs([st.pool], nbytes=[100])]
    out = np.zeros(1, np.uint64)
    for d in bad_puts:
        assert st._fast.put_batch(st._hi, d.ctypes.data, 1, out.ctypes.data, stream) == 1
    small = torch.empty(10, dtype=torch.uint8, device=DEV)
    pg = st.prepare_get(get_descs([0], [small]))
    assert st.get_prepared(pg, np.array([good], np.uint64)) == 1          # destination too small
    assert list(pg.descs["id"]) == [good]
    pg2 = st.prepare_get(get_descs([0], [x]))
    assert st.get_prepared(pg2, np.array([999], np.uint64)) == 3          # unknown id
    assert list(pg2.out) == [3]
    torch.cuda.synchronize()
    assert st.stats()["live_objects"] == 1 and st.stats()["used_pages"] == 1
    assert st.stats()["gets"] == 0


def test_compaction_moves_bytes_vs_oracle():
    """A fragmented store compacted to a smaller limit and grown back: every
    byte vs the oracle, page lists vs the oracle's paged model."""
    P = 256 * 1024
    pages = 512
    tr = W.compaction_trace(11, pages, P, n_ops=4000, lo=4 * W.KiB, hi=24 * W.MiB)
    st = make_store(pages * P, P)
    ora = OracleStore(pages * P, P)
    ids = {}
    survivors = set(tr.survivors)
    keep = []
    for op in tr.ops:
        if op[0] == "alloc":
            k, n = op[1], op[2]
            if k in survivors:
                data = W.object_bytes(11, k, n)
                t = dev_bytes(data)
                keep.append(t)
                s, (i,) = st.put_batch(put_descs([t]))
                _, (oi,) = ora.put_batch([PutItem(n, data)])
            else:
                s, (i,) = st.put_batch(put_descs([0], nbytes=[n]))
                _, (oi,) = ora.put_batch([PutItem(n, None)])
            assert s == 0 and i == oi
            ids[k] = oi
        else:
            oid = ids.pop(op[1])
            assert st.free([oid]) == ora.free([oid]) == 0
    compare_meta(st, ora)
    limit = (pages // 2 + 16) * P
    s, moved = st.compact(limit)
    ost, moves = ora.compact(limit)
    assert s == ost == 0 and moved == len(moves) > 20
    compare_meta(st, ora)
    rng = np.random.default_rng(0)
    check_all_gets(st, ora, rng)
    s, moved = st.compact(pages * P)
    assert s == 0 and moved == 0 and ora.compact(pages * P)[0] == 0
    compare_meta(st, ora)


def test_consumer_reclaim_and_deferred_get():
    """An object put with 2 consumers is freed after its second get; a get
    issued with a producer's event waits for it on the GPU (the producer runs
    on a stream the store never saw, so only the event orders them)."""
    P = 64 * 1024
    st = make_store(64 * P, P)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    x = torch.randint(0, 256, (5 * P + 3,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    s, (i,) = st.put_batch(put_descs([x], consumers=2), stream=s1)
    assert s == 0 and st.ctl.object(int(i))[1]["consumers_left"] == 2
    with torch.cuda.stream(s3):
        torch.cuda._sleep(int(2.0e9 * 0.03))     # a 30 ms producer
    ev = torch.cuda.Event()
    ev.record(s3)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    out = torch.empty_like(x)
    t0.record(s2)
    s, _ = st.get_batch(get_descs([int(i)], [out]), stream=s2, wait_event=ev)
    t1.record(s2)
    assert s == 0
    torch.cuda.synchronize()
    assert t0.elapsed_time(t1) > 10.0, "the get did not wait for the producer's event"
    assert torch.equal(out, x)
    assert st.ctl.object(int(i))[1]["consumers_left"] == 1
    out2 = torch.empty_like(x)
    s, _ = st.get_batch(get_descs([int(i)], [out2]), stream=s2)
    assert s == 0
    torch.cuda.synchronize()
    assert torch.equal(out2, x)
    stats = st.stats()
    assert stats["reclaimed"] == 1 and stats["live_objects"] == 0 and stats["used_pages"] == 0
    assert st.get_batch(get_descs([int(i)], [out]))[0] == 3


SLEEP_CYCLES_PER_MS = 2.0e6   # torch.cuda._sleep spins ~this many clock cycles per millisecond


def _late(stream, ms):
    """Keeps ``stream`` busy for about ``ms`` (torch's bounded sleep kernel)."""
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(ms * SLEEP_CYCLES_PER_MS))


def test_cross_stream_read_after_write():
    """A get on another stream waits for the put that wrote its pages, even
    when that put runs late."""
    P = 64 * 1024
    st = make_store(16 * P, P)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    a = torch.randint(0, 256, (6 * P + 7,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    _late(s1, 30)
    s, (i,) = st.put_batch(put_descs([a]), stream=s1)
    assert s == 0
    out = torch.zeros_like(a)
    s, _ = st.get_batch(get_descs([int(i)], [out]), stream=s2)
    assert s == 0
    torch.cuda.synchronize()
    assert torch.equal(out, a)


def test_cross_stream_write_after_read():
    """A put that reuses the pages of a freed object waits for a late get of
    that object on another stream."""
    P = 64 * 1024
    st = make_store(8 * P, P)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    b = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    c = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    s, (ib,) = st.put_batch(put_descs([b]), stream=s1)
    assert s == 0
    _late(s2, 30)
    out = torch.zeros_like(b)
    s, _ = st.get_batch(get_descs([int(ib)], [out]), stream=s2)   # runs ~30 ms from now
    assert s == 0 and st.free([int(ib)]) == 0
    s, (ic,) = st.put_batch(put_descs([c]), stream=s3)          # the same 8 pages
    assert s == 0 and sorted(st.ctl.object(int(ic))[2]) == list(range(8))
    torch.cuda.synchronize()
    assert torch.equal(out, b), "the put overwrote pages a pending get still had to read"
    out2 = torch.zeros_like(c)
    assert st.get_batch(get_descs([int(ic)], [out2]), stream=s1)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out2, c)


def test_independent_streams_do_not_wait_for_each_other():
    """Puts of independent objects on two streams overlap: the second does not
    wait for the first stream's late work."""
    P = 2 << 20
    st = make_store(64 * P, P)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    x = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    y = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    _late(s1, 60)
    s, (ix,) = st.put_batch(put_descs([x]), stream=s1)
    assert s == 0
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(s2)
    s, (iy,) = st.put_batch(put_descs([y]), stream=s2)
    t1.record(s2)
    assert s == 0
    t1.synchronize()
    assert t0.elapsed_time(t1) < 20.0, "an independent put waited for another stream"
    torch.cuda.synchronize()
    outs = [torch.empty_like(x), torch.empty_like(y)]
    assert st.get_batch(get_descs([int(ix), int(iy)], outs), stream=s2)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(outs[0], x) and torch.equal(outs[1], y)


def test_handoff_spread_over_streams():
    """The handoff at B = 4 with request r on stream r % 4 and no
    synchronisation between steps; steps alternate between two input sets and
    two output sets, and one stream's gets of the first step run late, so a
    put of the second step that reused a page before its last get read it
    would show in the first step's outputs."""
    C = W.HANDOFF
    specs = W.handoff_specs(4)
    n, R, k = len(specs), C["requests"], 4
    st = make_store(C["pool_bytes"], C["page_bytes"])
    streams = [torch.cuda.Stream() for _ in range(k)]
    ins = [[W.handoff_request_torch(seed, r, specs, DEV) for r in range(R)] for seed in (0, 1)]
    outs = [[[torch.empty_like(t) for t in ts] for ts in reqs] for reqs in ins]
    torch.cuda.synchronize()
    for rep in range(2):
        for step in (0, 1):
            ids = []
            for r in range(R):
                s, i = st.put_batch(put_descs(ins[step][r], nbytes=[sp.nbytes for sp in specs]),
                                    stream=streams[r % k])
                assert s == 0, st.last_error()
                ids.append(i)
            if step == 0:
                _late(streams[1], 30)
            for r in range(R):
                s, _ = st.get_batch(get_descs(ids[r], outs[step][r]), stream=streams[r % k])
                assert s == 0, st.last_error()
            assert st.free(np.concatenate(ids)) == 0
        torch.cuda.synchronize()
        for step in (0, 1):
            for r in range(R):
                for j in range(n):
                    assert torch.equal(outs[step][r][j], ins[step][r][j]), (rep, step, r, j)
    assert st.stats()["used_pages"] == 0


@pytest.mark.parametrize("B,binding", [(1, "cpython"), (8, "cpython"), (1, "ctypes")])
def test_bench_step_over_streams(B, binding):
    """The benchmark's own multi-stream step (phase joins included), at the
    headline's size and launch configuration (B = 8, 64 requests, 4 streams)
    and at B = 1, through the CPython entry points and through ctypes (the
    form used where the CPython module was not built): get(put(x)) == x for
    every output, the oracle's cast for sampled requests."""
    import bench

    hw = bench.Handoff(B, W.HANDOFF["requests"], DEV)
    if binding == "ctypes":
        hw.fast = None
    else:
        assert hw.fast is not None, "the CPython entry points were not built"
    streams = [torch.cuda.current_stream()] + [torch.cuda.Stream() for _ in range(3)]
    for _ in range(3):
        hw.step_streams(streams)
    torch.cuda.synchronize()
    hw.verify()
    for r in (0, 17, 63):
        lat = hw.inputs[r][hw.ci].reshape(-1).view(torch.int32).cpu().numpy().view(np.uint32)
        got = hw.outputs[r][hw.ci].view(torch.int16).cpu().numpy().view(np.uint16)
        assert np.array_equal(got, f32_bits_to_bf16_bits(lat)), r
    hw.store.close()


def test_cross_stream_compaction():
    """A compaction on one stream waits for a late put of the pages it moves,
    and a get on a third stream waits for the compaction."""
    P = 64 * 1024
    st = make_store(8 * P, P)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    f = torch.randint(0, 256, (4 * P,), dtype=torch.uint8, device=DEV)
    a = torch.randint(0, 256, (4 * P - 5,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    s, (i_f,) = st.put_batch(put_descs([f]))
    torch.cuda.synchronize()
    _late(s1, 30)
    s, (ia,) = st.put_batch(put_descs([a]), stream=s1)          # pages 4..7, written late
    assert s == 0 and min(st.ctl.object(int(ia))[2]) >= 4
    assert st.free([int(i_f)]) == 0
    s, moved = st.compact(4 * P, stream=s2)
    assert s == 0 and moved == 4
    out = torch.zeros_like(a)
    assert st.get_batch(get_descs([int(ia)], [out]), stream=s3)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, a)


def test_views_in_place():
    """Extent placement keeps objects contiguous; a view reads them in place
    (no copy) and equals what was put."""
    P = 64 * 1024
    st = make_store(64 * P, P, alloc_policy=1)
    xs = [torch.randint(0, 256, (n,), dtype=torch.uint8, device=DEV) for n in (3 * P + 5, P, 10, 7 * P)]
    s, ids = st.put_batch(put_descs(xs))
    assert s == 0
    for i, x in zip(ids, xs):
        s, t = st.tensor_view(int(i))
        assert s == 0 and t.data_ptr() != x.data_ptr() and torch.equal(t, x)
    assert st.stats()["views"] == len(xs)
    # LIFO placement after a free hands pages out in descending order: no view
    st0 = make_store(8 * P, P)
    a = torch.randint(0, 256, (2 * P,), dtype=torch.uint8, device=DEV)
    s, (ia, ib) = st0.put_batch(put_descs([a, a]))
    assert st0.free([int(ia)]) == 0
    s, (ic,) = st0.put_batch(put_descs([a]))
    assert st0.ctl.object(int(ic))[2] == [1, 0]
    assert st0.view(int(ic))[0] == 6                       # NOT_CONTIGUOUS
    assert st0.view(int(ib))[0] == 0 and st0.view(999)[0] == 3


def test_view_is_ordered_after_its_writer_and_before_reuse():
    """A view on one stream waits for a late put on another; a put reusing
    the viewed pages waits for the view stream's late reads."""
    P = 64 * 1024
    st = make_store(8 * P, P, alloc_policy=1)
    s1, s2, s3 = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    x = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    y = torch.randint(0, 256, (8 * P,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    _late(s1, 30)
    s, (ix,) = st.put_batch(put_descs([x]), stream=s1)
    assert s == 0
    s, t = st.tensor_view(int(ix), stream=s2)
    assert s == 0
    _late(s2, 30)
    with torch.cuda.stream(s2):
        z = t.clone()                         # a late reader, in place
    assert st.free([int(ix)]) == 0
    s, (iy,) = st.put_batch(put_descs([y]), stream=s3)   # the same pages
    assert s == 0 and st.ctl.object(int(iy))[2] == list(range(8))
    torch.cuda.synchronize()
    assert torch.equal(z, x)


def test_pull_between_stores_vs_oracle():
    """A consumer's store pulls objects from a producer's store page to page
    (§5.2): statuses, ids, placement and bytes as the oracle's pull."""
    P = 64 * 1024
    rng = np.random.default_rng(21)
    prod, cons = make_store(64 * P, P), make_store(16 * P, P, alloc_policy=1)
    o_prod, o_cons = OracleStore(64 * P, P), OracleStore(16 * P, P, policy=1)
    datas = [rng.integers(0, 256, int(n), dtype=np.uint8) for n in (3 * P + 11, 1000, 5 * P, 17, 2 * P)]
    cons_n = [1, 0, 0, 2, 0]
    s, ids = prod.put_batch(put_descs([dev_bytes(d) for d in datas], dtype_tag=2, consumers=cons_n))
    assert s == 0
    _, oids = o_prod.put_batch([PutItem(d.size, d, 2, 0, 0, False, c) for d, c in zip(datas, cons_n)])
    pick = [int(ids[0]), int(ids[2]), int(ids[3])]
    s, new, per = cons.pull(prod, pick, consumers=1)
    ost, oper, onew = o_cons.pull(o_prod, pick, consumers=1)
    assert s == ost == 0 and list(per) == oper and list(new) == onew
    compare_meta(cons, o_cons)
    compare_meta(prod, o_prod)
    assert prod.stats()["reclaimed"] == o_prod.stats["reclaimed"] == 1   # object 0's only consumer was the pull
    outs = [dev_empty(datas[i].size) for i in (0, 2, 3)]
    assert cons.get_batch(get_descs([int(x) for x in new], outs))[0] == 0
    torch.cuda.synchronize()
    for o, i in zip(outs, (0, 2, 3)):
        assert np.array_equal(host(o), datas[i])
    assert cons.stats()["reclaimed"] == 3                                # consumers = 1 each
    # failures change nothing
    assert cons.pull(prod, [int(ids[0])])[0] == 3                       # reclaimed in the producer
    big = dev_bytes(rng.integers(0, 256, 17 * P, dtype=np.uint8))
    s, (ib,) = prod.put_batch(put_descs([big]))
    assert cons.pull(prod, [int(ib)])[0] == 2 and prod.ctl.object(int(ib))[0] == 0
    assert cons.pull(cons, [int(ib)])[0] == 1
    other = make_store(16 * 4096, 4096)
    assert other.pull(prod, [int(ib)])[0] == 1                          # page sizes differ


def test_pull_waits_for_a_late_producer():
    P = 64 * 1024
    prod, cons = make_store(16 * P, P), make_store(16 * P, P)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    x = torch.randint(0, 256, (9 * P + 3,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    _late(s1, 30)
    s, (ix,) = prod.put_batch(put_descs([x]), stream=s1)
    assert s == 0
    s, (iy,), _ = cons.pull(prod, [int(ix)], stream=s2)
    assert s == 0
    out = torch.zeros_like(x)
    assert cons.get_batch(get_descs([int(iy)], [out]), stream=s2)[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, x)


def test_chunked_launches_on_eight_streams_at_once():
    """Large gets (>= 1 MiB per CTA: chunks from the work counters) on eight
    streams at once, each stream with its own counter; every byte checked,
    twice in a row (each launch leaves its counter at zero)."""
    P = 2 << 20
    n = 600 << 20                                    # 300 pages, 1.3 MiB per CTA of the get grid
    st = make_store(8 * (n // P) * P + 8 * P, P)
    streams = [torch.cuda.Stream() for _ in range(8)]
    xs = [torch.randint(0, 256, (n,), dtype=torch.uint8, device=DEV) for _ in range(8)]
    s, ids = st.put_batch(put_descs(xs))
    assert s == 0
    torch.cuda.synchronize()
    for _ in range(2):
        outs = [torch.zeros_like(x) for x in xs]
        torch.cuda.synchronize()
        for k in range(8):
            assert st.get_batch(get_descs([int(ids[k])], [outs[k]]), stream=streams[k])[0] == 0
        torch.cuda.synchronize()
        for x, o in zip(xs, outs):
            assert torch.equal(x, o)


def test_streams_beyond_the_counter_slots_split_statically():
    """A store has work counters for its first 64 streams; later streams use
    equal static shares. A large get on the 70th stream is still exact."""
    P = 2 << 20
    n = 600 << 20
    st = make_store(n + 8 * P, P)
    x = torch.randint(0, 256, (n,), dtype=torch.uint8, device=DEV)
    s, (i,) = st.put_batch(put_descs([x]))
    assert s == 0
    streams = [torch.cuda.Stream() for _ in range(70)]
    small = torch.zeros(64, dtype=torch.uint8, device=DEV)
    tiny = torch.randint(0, 256, (64,), dtype=torch.uint8, device=DEV)
    torch.cuda.synchronize()
    s, (j,) = st.put_batch(put_descs([tiny]))
    for sm in streams:                                # register 70 streams with the store
        assert st.get_batch(get_descs([int(j)], [small]), stream=sm)[0] == 0
    out = torch.zeros_like(x)
    assert st.get_batch(get_descs([int(i)], [out]), stream=streams[-1])[0] == 0
    torch.cuda.synchronize()
    assert torch.equal(out, x) and torch.equal(small, tiny)


def test_prepared_batches():
    """Prepared put and get batches (descriptors converted once, issued many
    times) move the same bytes as the plain calls, call after call."""
    P = 64 * 1024
    st = make_store(64 * P, P)
    xs = [torch.randint(0, 256, (n,), dtype=torch.uint8, device=DEV) for n in (5 * P + 3, 100, 2 * P)]
    outs = [torch.zeros_like(x) for x in xs]
    pp = st.prepare_put(put_descs(xs))
    pg = st.prepare_get(get_descs(np.zeros(3, np.uint64), outs))
    for k in range(3):
        s, ids = st.put_prepared(pp)
        assert s == 0
        assert st.get_prepared(pg, ids) == 0 and list(pg.out) == [0, 0, 0]
        torch.cuda.synchronize()
        assert all(torch.equal(o, x) for o, x in zip(outs, xs)), k
        assert st.free(ids.copy()) == 0
        for o in outs:
            o.zero_()
    assert st.stats()["used_pages"] == 0


def _cudart():
    """The CUDA runtime library, to allocate managed memory (torch does not)."""
    import ctypes
    import os

    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH") or "/usr/local/cuda"
    for name in ("libcudart.so", "libcudart.so.13", "libcudart.so.12"):
        for path in (os.path.join(home, "lib64", name), name):
            try:
                return ctypes.CDLL(path)
            except OSError:
                pass
    pytest.fail("no CUDA runtime library found to allocate managed memory")


def test_puts_the_kernels_do_not_prefetch():
    """Sources whose bytes the put kernels must not ask L2 for ahead of their
    wait: managed memory (checked as such), and every source of a store
    without pointer checks (the kind of memory is unknown). Every get equals
    the oracle's, and so do the page lists."""
    import ctypes

    rng = np.random.default_rng(21)
    P = 64 * 1024
    datas = [rng.integers(0, 256, int(n), dtype=np.uint8) for n in (1000, 3 * P + 5, 70001, 2 * P, 17)]
    rt = _cudart()
    managed = []
    try:
        for d in datas:
            p = ctypes.c_void_p()
            assert rt.cudaMallocManaged(ctypes.byref(p), ctypes.c_size_t(d.size), 1) == 0
            ctypes.memmove(p, d.ctypes.data, d.size)  # managed memory is host-accessible
            managed.append(p.value)
        for check in (1, 0):
            st = make_store(64 * P, P, check_pointers=check)
            ora = OracleStore(64 * P, P)
            srcs = np.array(managed, np.uint64) if check else [dev_bytes(d, 3 * k) for k, d in enumerate(datas)]
            s, ids = st.put_batch(put_descs(srcs, nbytes=[d.size for d in datas]))
            assert s == 0, st.last_error()
            ost, oids = ora.put_batch([PutItem(d.size, d) for d in datas])
            assert ost == 0 and list(ids) == oids
            compare_meta(st, ora)
            outs = [dev_empty(d.size, k) for k, d in enumerate(datas)]
            s, _ = st.get_batch(get_descs(oids, outs))
            assert s == 0, st.last_error()
            torch.cuda.synchronize()
            for o, d in zip(outs, datas):
                assert np.array_equal(host(o), d)
            st.close()
    finally:
        torch.cuda.synchronize()
        for p in managed:
            rt.cudaFree(ctypes.c_void_p(p))
