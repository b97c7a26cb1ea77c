"""Python binding of the paged tensor store: argument marshalling only.

Every call goes straight to the C ABI of libt2istore.so (include/t2istore.h)
with the same name; every byte is moved by the library's CUDA kernels (or,
for host sources on request, the copy engine). Descriptor batches are numpy
structured arrays with the C layout, so large batches cost one array build,
not a Python loop per object.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from . import _lib as L

PUT_DTYPE = np.dtype([("src", "<u8"), ("nbytes", "<u8"), ("src_is_host", "<u4"), ("dtype_tag", "<u4"),
                      ("group", "<u8"), ("order", "<u4"), ("evictable", "<u4"), ("consumers", "<u4"),
                      ("reserved", "<u4")])
GET_DTYPE = np.dtype([("id", "<u8"), ("dst", "<u8"), ("dst_bytes", "<u8"), ("cast", "<u4"), ("reserved", "<u4")])
MOVE_DTYPE = np.dtype([("src_page", "<u4"), ("dst_page", "<u4"), ("valid_bytes", "<u8")])
assert PUT_DTYPE.itemsize == C.sizeof(L.PutDesc) and GET_DTYPE.itemsize == C.sizeof(L.GetDesc)
assert MOVE_DTYPE.itemsize == C.sizeof(L.Move)


class T2IError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{L.STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def _ptr(x) -> int:
    """Address of a tensor / array / int. A buffer's bytes travel as one
    range, so tensors and arrays must be contiguous (a strided view would
    copy the wrong bytes, or overwrite its neighbours on a get)."""
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if hasattr(x, "is_contiguous") and not x.is_contiguous():
            raise ValueError("a tensor buffer must be contiguous (call .contiguous() first)")
        return int(x.data_ptr())
    if isinstance(x, np.ndarray):
        if not x.flags.c_contiguous:
            raise ValueError("an array buffer must be C-contiguous")
        return int(x.ctypes.data)
    raise TypeError(f"cannot take the address of {type(x)}")


def _nbytes(x) -> int:
    if hasattr(x, "untyped_storage") and hasattr(x, "element_size"):
        return int(x.numel() * x.element_size())
    return int(x.nbytes)


def _stream(stream) -> int:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _addrs(xs):
    if isinstance(xs, np.ndarray) and xs.dtype.kind in "iu":
        return xs
    return [_ptr(x) for x in xs]


def put_descs(srcs, nbytes=None, src_is_host=0, dtype_tag=0, group=0, order=0, evictable=0,
              consumers=0) -> np.ndarray:
    """A put descriptor array. ``srcs``: tensors / arrays / addresses (an
    integer numpy array of addresses is taken as is; 0 or None reserves
    pages); scalars broadcast."""
    n = len(srcs)
    d = np.zeros(n, PUT_DTYPE)
    d["src"] = _addrs(srcs)
    d["nbytes"] = [_nbytes(s) for s in srcs] if nbytes is None else nbytes
    d["src_is_host"] = src_is_host
    d["dtype_tag"] = dtype_tag
    d["group"] = group
    d["order"] = order
    d["evictable"] = evictable
    d["consumers"] = consumers
    return d


def get_descs(ids, dsts=None, dst_bytes=None, cast=0) -> np.ndarray:
    """A get descriptor array; ``dsts``: tensors / arrays / addresses."""
    n = len(ids)
    d = np.zeros(n, GET_DTYPE)
    d["id"] = ids
    if dsts is not None:
        d["dst"] = _addrs(dsts)
        d["dst_bytes"] = [_nbytes(x) for x in dsts] if dst_bytes is None else dst_bytes
    elif dst_bytes is not None:
        d["dst_bytes"] = dst_bytes
    d["cast"] = cast
    return d


def _as(arr: np.ndarray, ctype, dtype):
    if arr.dtype != dtype or not arr.flags.c_contiguous:
        raise TypeError("descriptor array has the wrong layout")
    return arr.ctypes.data_as(C.POINTER(ctype))


def _addr(arr: np.ndarray, dtype) -> int:
    """Address of a descriptor array with the C layout (for the calls that
    take plain addresses)."""
    if arr.dtype != dtype or not arr.flags.c_contiguous:
        raise TypeError("descriptor array has the wrong layout")
    return arr.ctypes.data


class Ctl:
    """The host control core alone (t2i_ctl_*): page allocator, directory,
    LRU and compaction planner without device memory."""

    def __init__(self, total_pages: int = 0, page_bytes: int = 0, alloc_policy: int = 0, _borrowed=None,
                 _owner=None):
        self._lib = L.load()
        self._owner = _owner
        if _borrowed is not None:
            self._h = C.c_void_p(_borrowed)
            self._owned = False
            return
        h = C.c_void_p()
        st = self._lib.t2i_ctl_create(total_pages, page_bytes, alloc_policy, C.byref(h))
        if st != L.OK:
            raise T2IError(st, self._lib.t2i_ctl_last_error(None).decode())
        self._h = h
        self._owned = True

    def close(self):
        if getattr(self, "_owned", False) and self._h:
            self._lib.t2i_ctl_destroy(self._h)
            self._h = C.c_void_p()

    __del__ = close

    def last_error(self) -> str:
        return self._lib.t2i_ctl_last_error(self._h).decode()

    def put(self, descs: np.ndarray):
        ids = np.zeros(len(descs), np.uint64)
        st = self._lib.t2i_ctl_put(self._h, _as(descs, L.PutDesc, PUT_DTYPE), len(descs),
                                   ids.ctypes.data_as(C.POINTER(C.c_uint64)))
        return st, ids

    def get(self, descs: np.ndarray):
        per = np.zeros(len(descs), np.int32)
        st = self._lib.t2i_ctl_get(self._h, _as(descs, L.GetDesc, GET_DTYPE), len(descs),
                                   per.ctypes.data_as(C.POINTER(C.c_int32)))
        return st, per

    def free(self, ids) -> int:
        ids = np.ascontiguousarray(ids, np.uint64)
        return self._lib.t2i_ctl_free(self._h, ids.ctypes.data_as(C.POINTER(C.c_uint64)), len(ids))

    def compact(self, limit_bytes: int, cap: int | None = None):
        n = C.c_uint64(0)
        if cap is None:
            cap = 1 << 16
        moves = np.zeros(cap, MOVE_DTYPE)
        st = self._lib.t2i_ctl_compact(self._h, limit_bytes, _as(moves, L.Move, MOVE_DTYPE), cap, C.byref(n))
        if st == L.ERR_INVALID and n.value > cap:
            return self.compact(limit_bytes, cap=int(n.value))
        return st, moves[:n.value].copy() if st == L.OK else moves[:0]

    def object(self, oid: int):
        """(status, info dict, page list)."""
        info = L.ObjectInfo()
        st = self._lib.t2i_ctl_object(self._h, oid, C.byref(info), None, 0)
        if st != L.OK:
            return st, None, None
        pages = np.zeros(max(1, info.n_pages), np.uint32)
        self._lib.t2i_ctl_object(self._h, oid, C.byref(info), pages.ctypes.data_as(C.POINTER(C.c_uint32)),
                                 info.n_pages)
        d = {n: int(getattr(info, n)) for n, _ in L.ObjectInfo._fields_}
        return st, d, pages[:info.n_pages].tolist()

    def free_pages(self) -> list:
        n = C.c_uint64(0)
        self._lib.t2i_ctl_free_pages(self._h, None, 0, C.byref(n))
        out = np.zeros(max(1, n.value), np.uint32)
        self._lib.t2i_ctl_free_pages(self._h, out.ctypes.data_as(C.POINTER(C.c_uint32)), n.value, C.byref(n))
        return out[:n.value].tolist()

    def last_evictions(self) -> list:
        n = C.c_uint64(0)
        self._lib.t2i_ctl_last_evictions(self._h, None, 0, C.byref(n))
        out = np.zeros(max(1, n.value), np.uint64)
        self._lib.t2i_ctl_last_evictions(self._h, out.ctypes.data_as(C.POINTER(C.c_uint64)), n.value, C.byref(n))
        return [int(x) for x in out[:n.value]]

    def stats(self) -> dict:
        s = L.Stats()
        st = self._lib.t2i_ctl_stats(self._h, C.byref(s))
        if st != L.OK:
            raise T2IError(st, "stats")
        return s.as_dict()


class Store:
    """A store over a device pool (``t2i_store_create``). ``pool`` is a CUDA
    tensor (kept alive by the store object) or an address with ``pool_bytes``.

    Calls are asynchronous like ``cudaMemcpyAsync``: a put source must keep
    its bytes, and a get destination its memory, until the call's stream has
    run the call. The binding does not hold the tensors named in descriptor
    arrays. A tensor used on a stream other than the one it was allocated on
    needs ``tensor.record_stream(stream)`` before it is dropped, as for any
    cross-stream use under PyTorch's caching allocator."""

    def __init__(self, pool, page_bytes: int, pool_bytes: int | None = None, device: int | None = None,
                 h2d_mode: int = 0, check_pointers: int = 1, alloc_policy: int = 0, d2h_mode: int = 0):
        self._lib = L.load()
        self.pool = pool
        if pool_bytes is None:
            pool_bytes = _nbytes(pool)
        if device is None:
            device = int(pool.device.index) if hasattr(pool, "device") else 0
        self.device = device
        self.page_bytes = int(page_bytes)
        self.pool_bytes = int(pool_bytes)
        cfg = L.StoreConfig(pool_bytes, page_bytes, h2d_mode, check_pointers, alloc_policy, d2h_mode)
        h = C.c_void_p()
        st = self._lib.t2i_store_create(C.c_void_p(_ptr(pool)), C.byref(cfg), device, C.byref(h))
        if st != L.OK:
            raise T2IError(st, self._lib.t2i_last_error(None).decode())
        self._h = h
        self._hi = int(h.value)  # the handle as an integer, for the CPython entry points
        self._fast = L.pycall()
        self.ctl = Ctl(_borrowed=self._lib.t2i_store_ctl(h), _owner=self)

    def close(self):
        if getattr(self, "_h", None):
            self._lib.t2i_store_destroy(self._h)
            self._h = None
            self._hi = 0

    __del__ = close

    def last_error(self) -> str:
        return self._lib.t2i_last_error(self._h).decode()

    def put_batch(self, descs: np.ndarray, stream=None):
        """(status, ids) -- t2i_put_batch."""
        ids = np.zeros(len(descs), np.uint64)
        st = self._lib.t2i_put_batch(self._h, _addr(descs, PUT_DTYPE), len(descs), ids.ctypes.data, _stream(stream))
        return st, ids

    # -- prepared batches: descriptors whose buffers stay the same from call
    #    to call (a serving loop's staging tensors) are checked and converted
    #    once; each call then passes cached addresses only
    class Prepared:
        __slots__ = ("descs", "n", "addr", "out", "out_addr")

        def __init__(self, descs: np.ndarray, dtype, out_dtype):
            self.descs = descs
            self.n = len(descs)
            self.addr = _addr(descs, dtype)
            self.out = np.zeros(self.n, out_dtype)
            self.out_addr = self.out.ctypes.data

    def prepare_put(self, descs: np.ndarray) -> "Store.Prepared":
        """A put batch for :meth:`put_prepared` (the array is kept, not copied)."""
        return Store.Prepared(descs, PUT_DTYPE, np.uint64)

    def put_prepared(self, p: "Store.Prepared", stream=None):
        """(status, ids) -- t2i_put_batch on a prepared batch. ``ids`` is the
        batch's own array, overwritten by the next call."""
        if self._fast is not None:
            return self._fast.put_batch(self._hi, p.addr, p.n, p.out_addr, _stream(stream)), p.out
        return self._lib.t2i_put_batch(self._h, p.addr, p.n, p.out_addr, _stream(stream)), p.out

    def prepare_get(self, descs: np.ndarray) -> "Store.Prepared":
        """A get batch for :meth:`get_prepared` (the array is kept, not copied)."""
        return Store.Prepared(descs, GET_DTYPE, np.int32)

    def get_prepared(self, p: "Store.Prepared", ids=None, stream=None) -> int:
        """t2i_get_batch on a prepared batch, after setting its ids to ``ids``
        (if given: a uint64 array of at least ``p.n`` ids, e.g. the ids a
        prepared put returned); per-item statuses land in ``p.out``."""
        if self._fast is not None and (ids is None or (isinstance(ids, np.ndarray) and ids.dtype == np.uint64
                                                       and ids.flags.c_contiguous and len(ids) >= p.n)):
            if ids is None:
                return self._fast.get_batch(self._hi, p.addr, p.n, p.out_addr, _stream(stream))
            return self._fast.get_batch_ids(self._hi, p.addr, p.n, ids.ctypes.data, p.out_addr, _stream(stream))
        if ids is not None:
            p.descs["id"] = ids
        return self._lib.t2i_get_batch(self._h, p.addr, p.n, p.out_addr, _stream(stream))

    def get_batch(self, descs: np.ndarray, stream=None, per_item: bool = True, wait_event=None):
        """(status, per-item statuses) -- t2i_get_batch, or t2i_get_batch_after
        when ``wait_event`` (a torch.cuda.Event or a cudaEvent_t address) is given."""
        per = np.zeros(len(descs), np.int32) if per_item else None
        per_p = per.ctypes.data if per_item else None
        if wait_event is None:
            st = self._lib.t2i_get_batch(self._h, _addr(descs, GET_DTYPE), len(descs), per_p, _stream(stream))
        else:
            ev = wait_event if isinstance(wait_event, int) else int(wait_event.cuda_event)
            if not ev:
                raise ValueError("wait_event has never been recorded")
            st = self._lib.t2i_get_batch_after(self._h, _addr(descs, GET_DTYPE), len(descs), per_p,
                                               _stream(stream), ev)
        return st, per

    def free(self, ids) -> int:
        ids = np.ascontiguousarray(ids, np.uint64)
        return self._lib.t2i_free(self._h, ids.ctypes.data, len(ids))

    def pull_pages(self, src_pool, objects, src_pool_bytes: int | None = None, consumers: int = 0, stream=None):
        """(status, new ids) -- t2i_pull_pages: pulls objects laid out in pages
        of another pool (e.g. a producer store's pool shared from another
        process). ``objects``: (nbytes, page list, dtype_tag) triples."""
        objs = (L.PagedObject * max(1, len(objects)))()
        keep = []
        for i, (nbytes, pages, tag) in enumerate(objects):
            pg = np.ascontiguousarray(pages, np.uint32)
            keep.append(pg)
            objs[i] = L.PagedObject(int(nbytes), pg.ctypes.data if len(pg) else None, len(pg), int(tag))
        out = np.zeros(len(objects), np.uint64)
        nb = src_pool_bytes if src_pool_bytes is not None else _nbytes(src_pool)
        st = self._lib.t2i_pull_pages(self._h, _ptr(src_pool), int(nb), C.addressof(objs), len(objects), consumers,
                                      out.ctypes.data, _stream(stream))
        return st, out

    def pull(self, src: "Store", ids, consumers: int = 0, stream=None):
        """(status, new ids, per-item statuses) -- t2i_pull: this store (the
        consumer) pulls ``ids`` from the producer's store ``src``."""
        ids = np.ascontiguousarray(ids, np.uint64)
        out = np.zeros(len(ids), np.uint64)
        per = np.zeros(len(ids), np.int32)
        st = self._lib.t2i_pull(self._h, src._h, ids.ctypes.data, len(ids), consumers, out.ctypes.data, per.ctypes.data,
                                _stream(stream))
        return st, out, per

    def view(self, oid: int, stream=None):
        """(status, device address, nbytes) -- t2i_view."""
        ptr = C.c_void_p()
        n = C.c_uint64()
        st = self._lib.t2i_view(self._h, oid, _stream(stream), C.byref(ptr), C.byref(n))
        return st, int(ptr.value or 0), int(n.value)

    def tensor_view(self, oid: int, dtype=None, shape=None, stream=None):
        """The object as a tensor over the pool, without a copy (the pool must
        be a torch tensor): status, tensor (None on failure)."""
        st, ptr, n = self.view(oid, stream)
        if st != L.OK:
            return st, None
        off = ptr - int(self.pool.data_ptr()) if n else 0
        t = self.pool.view(-1)[off:off + n]
        if dtype is not None:
            t = t.view(dtype)
        if shape is not None:
            t = t.view(shape)
        return st, t

    def put_layers(self, descs: np.ndarray, layer_off, first: int = 0, stream=None, events=None):
        """(status, ids) -- t2i_put_layers. ``layer_off``: n_layers + 1 offsets
        into ``descs``; ``events``: one torch.cuda.Event (or cudaEvent_t) per
        layer, or None."""
        off = np.ascontiguousarray(layer_off, np.uint32)
        n_layers = len(off) - 1
        ids = np.zeros(len(descs), np.uint64)
        ev_arr = None
        if events is not None:
            handles = []
            for e in events:
                if not isinstance(e, int) and not e.cuda_event:
                    e.record(stream if stream is not None and not isinstance(stream, int) else None)  # creates it
                handles.append(e if isinstance(e, int) else int(e.cuda_event))
            ev_arr = (C.c_void_p * n_layers)(*handles)
        st = self._lib.t2i_put_layers(self._h, _as(descs, L.PutDesc, PUT_DTYPE),
                                      off.ctypes.data_as(C.POINTER(C.c_uint32)), n_layers, first,
                                      ids.ctypes.data_as(C.POINTER(C.c_uint64)), _stream(stream), ev_arr)
        return st, ids

    def compact(self, limit_bytes: int, stream=None):
        """(status, pages moved) -- t2i_compact."""
        n = C.c_uint64(0)
        st = self._lib.t2i_compact(self._h, limit_bytes, _stream(stream), C.byref(n))
        return st, int(n.value)

    def inject_launch_failure(self, countdown: int) -> int:
        """t2i_inject_launch_failure (testing)."""
        return self._lib.t2i_inject_launch_failure(self._h, countdown)

    def stats(self) -> dict:
        s = L.Stats()
        st = self._lib.t2i_store_stats(self._h, C.byref(s))
        if st != L.OK:
            raise T2IError(st, "stats")
        return s.as_dict()

    def check(self, st: int):
        if st != L.OK:
            raise T2IError(st, self.last_error())


# ---------------------------------------------------------------- prefix caching (§5.1)
def gather_noalloc(pool, page_bytes: int, pages, nbytes: int, dst, dst_bytes: int | None = None, cast: int = 0,
                   stream=None, device: int | None = None, pool_bytes: int | None = None) -> int:
    """t2i_gather_noalloc: one object's pages (``pages``, indices into
    ``pool``) gathered into ``dst`` with no store and no allocation, for
    callers that cannot allocate device memory. Returns the status; every
    call shares the library's static scratch counters, so calls that overlap
    on the GPU race."""
    lib = L.load()
    pg = np.ascontiguousarray(pages, dtype=np.uint32)
    if device is None:
        device = int(pool.device.index) if hasattr(pool, "device") else 0
    return lib.t2i_gather_noalloc(_ptr(pool), int(pool_bytes if pool_bytes is not None else _nbytes(pool)),
                                  int(page_bytes), pg.ctypes.data_as(C.POINTER(C.c_uint32)), len(pg), int(nbytes),
                                  _ptr(dst), int(dst_bytes if dst_bytes is not None else _nbytes(dst)), int(cast),
                                  int(device), _stream(stream))


def _dbl(x):
    a = np.ascontiguousarray(x, np.float64)
    return a, a.ctypes.data_as(C.POINTER(C.c_double))


def e2e_latency(n_layers: int, n_cached: int, t_load: float, t_comp: float) -> float:
    """Eq. (1) -- t2i_e2e_latency."""
    lib = L.load()
    out = C.c_double()
    st = lib.t2i_e2e_latency(n_layers, n_cached, t_load, t_comp, C.byref(out))
    if st != L.OK:
        raise T2IError(st, lib.t2i_last_error(None).decode())
    return out.value


def prefix_layers(n_layers: int, t_load: float, t_comp: float) -> int:
    """Eq. (2) -- t2i_prefix_layers."""
    lib = L.load()
    out = C.c_uint32()
    st = lib.t2i_prefix_layers(n_layers, t_load, t_comp, C.byref(out))
    if st != L.OK:
        raise T2IError(st, lib.t2i_last_error(None).decode())
    return int(out.value)


def pipeline_latency(t_load, t_comp, n_cached: int) -> float:
    """t2i_pipeline_latency for per-layer times."""
    lib = L.load()
    a, pa = _dbl(t_load)
    b, pb = _dbl(t_comp)
    out = C.c_double()
    st = lib.t2i_pipeline_latency(pa, pb, len(b), n_cached, C.byref(out))
    if st != L.OK:
        raise T2IError(st, lib.t2i_last_error(None).decode())
    return out.value


def prefix_layers_pipeline(t_load, t_comp) -> int:
    """t2i_prefix_layers_pipeline for per-layer times."""
    lib = L.load()
    a, pa = _dbl(t_load)
    b, pb = _dbl(t_comp)
    out = C.c_uint32()
    st = lib.t2i_prefix_layers_pipeline(pa, pb, len(b), C.byref(out))
    if st != L.OK:
        raise T2IError(st, lib.t2i_last_error(None).decode())
    return int(out.value)
