"""The C-ABI library loads and exports every call include/t2istore.h declares,
with the struct layouts the header gives (CPU only: no compute calls)."""
import ctypes as C
import os
import re
import subprocess

import pytest

from paper_2607_26566_gb300 import _lib as L

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include"))) if f.endswith(".h")]


def declared_functions():
    names = []
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_ ]*?\**\s*\**(t2i_[a-z0-9_]+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_store_calls():
    names = declared_functions()
    for required in ("t2i_store_create", "t2i_put_batch", "t2i_get_batch", "t2i_free", "t2i_compact"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert names
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(L.PROTOTYPES), "binding prototypes and header disagree"


def test_only_t2i_symbols_are_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", L.LIB_PATH], capture_output=True, text=True).stdout
    syms = [line.split()[-1] for line in out.splitlines() if line.strip()]
    assert syms and all(s.startswith("t2i_") for s in syms), [s for s in syms if not s.startswith("t2i_")][:5]


def test_struct_layouts_match_the_header(tmp_path):
    prog = tmp_path / "sizes.c"
    prog.write_text("""
#include <stdio.h>
#include <stddef.h>
#include "t2istore.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu\\n", sizeof(t2i_store_config), sizeof(t2i_put_desc), sizeof(t2i_get_desc),
         sizeof(t2i_move), sizeof(t2i_stats), sizeof(t2i_object_info));
  printf("%zu %zu %zu\\n", offsetof(t2i_put_desc, group), offsetof(t2i_get_desc, cast), offsetof(t2i_move, valid_bytes));
  printf("%zu %zu\\n", sizeof(t2i_paged_object), offsetof(t2i_paged_object, n_pages));
  return 0;
}
""")
    exe = tmp_path / "sizes"
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I" + os.path.join(ROOT, "include"), str(prog), "-o", str(exe)],
                   check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    got = [int(x) for x in out]
    want = [C.sizeof(L.StoreConfig), C.sizeof(L.PutDesc), C.sizeof(L.GetDesc), C.sizeof(L.Move), C.sizeof(L.Stats),
            C.sizeof(L.ObjectInfo), L.PutDesc.group.offset, L.GetDesc.cast.offset, L.Move.valid_bytes.offset,
            C.sizeof(L.PagedObject), L.PagedObject.n_pages.offset]
    assert got == want


def test_store_create_without_a_gpu_fails_cleanly(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    cfg = L.StoreConfig(1 << 20, 1 << 16, 0, 1)
    h = C.c_void_p()
    st = lib.t2i_store_create(C.c_void_p(1 << 20), C.byref(cfg), 0, C.byref(h))
    assert st in (L.ERR_CUDA, L.ERR_INVALID) and not h.value
    assert lib.t2i_last_error(None)


def test_strided_buffers_are_refused():
    """A buffer travels as one byte range: strided tensors and arrays are
    refused before any descriptor is built."""
    import numpy as np
    import torch

    from paper_2607_26566_gb300 import get_descs, put_descs
    t = torch.zeros(8, 6)
    with pytest.raises(ValueError):
        put_descs([t[:, :3]])
    with pytest.raises(ValueError):
        get_descs([1], [t.t()])
    with pytest.raises(ValueError):
        put_descs([np.zeros((4, 4), np.float32)[:, 1]])
    d = put_descs([t[2:5], np.zeros(16, np.uint8)[4:]])   # contiguous slices are fine
    assert list(d["nbytes"]) == [3 * 6 * 4, 12]


def test_store_create_refuses_bad_flags(lib):
    """Flags are checked before the device is touched (no GPU needed)."""
    for fields in ({"d2h_mode": 2}, {"h2d_mode": 2}, {"alloc_policy": 2}, {"check_pointers": 2}):
        cfg = L.StoreConfig(1 << 20, 1 << 16, 0, 1, 0, 0)
        for k, v in fields.items():
            setattr(cfg, k, v)
        h = C.c_void_p()
        st = lib.t2i_store_create(C.c_void_p(1 << 21), C.byref(cfg), 0, C.byref(h))
        assert st == L.ERR_INVALID and not h.value, fields
        assert b"bad flag" in lib.t2i_last_error(None)


C_DRIVER = r"""
#include <stdio.h>
#include <string.h>
#include "t2istore.h"

static t2i_put_desc pd(uint64_t nbytes, uint64_t group, uint32_t order, uint32_t evictable) {
    t2i_put_desc d;
    memset(&d, 0, sizeof d);
    d.nbytes = nbytes;
    d.group = group;
    d.order = order;
    d.evictable = evictable;
    return d;
}
static void show_pages(const t2i_ctl* c, t2i_id id) {
    t2i_object_info info;
    uint32_t pg[16];
    t2i_ctl_object(c, id, &info, pg, 16);
    printf("pages %llu:", (unsigned long long)id);
    for (uint32_t i = 0; i < info.n_pages; ++i) printf(" %u", pg[i]);
    printf("\n");
}
static void show_evictions(const t2i_ctl* c) {
    t2i_id ev[16];
    uint64_t n = 0;
    t2i_ctl_last_evictions(c, ev, 16, &n);
    printf("evicted:");
    for (uint64_t i = 0; i < n; ++i) printf(" %llu", (unsigned long long)ev[i]);
    printf("\n");
}
int main(void) {
    const uint64_t P = 1024;
    t2i_ctl* c = NULL;
    if (t2i_ctl_create(6, P, 0, &c) != T2I_OK) return 1;
    t2i_put_desc w1[3] = {pd(P, 1, 0, 1), pd(P, 1, 1, 1), pd(P, 1, 2, 1)};
    t2i_put_desc w2[2] = {pd(P, 2, 0, 1), pd(P, 2, 1, 1)};
    t2i_id ids[4];
    printf("put %d\n", t2i_ctl_put(c, w1, 3, ids));
    printf("put %d\n", t2i_ctl_put(c, w2, 2, ids));
    t2i_get_desc g;
    memset(&g, 0, sizeof g);
    g.id = 1;
    printf("get %d\n", t2i_ctl_get(c, &g, 1, NULL));
    t2i_put_desc x = pd(3 * P, 3, 0, 0);
    printf("put %d\n", t2i_ctl_put(c, &x, 1, ids));
    show_evictions(c);
    show_pages(c, ids[0]);
    t2i_get_desc g3[3];
    memset(g3, 0, sizeof g3);
    g3[0].id = 4;
    g3[1].id = 99;
    g3[2].id = 1;
    t2i_status per[3];
    const t2i_status gs = t2i_ctl_get(c, g3, 3, per);
    printf("get %d per %d %d %d\n", gs, per[0], per[1], per[2]);
    t2i_put_desc y = pd(P, 2, 0, 1);
    printf("put %d\n", t2i_ctl_put(c, &y, 1, ids));
    show_evictions(c);
    show_pages(c, ids[0]);
    t2i_put_desc big = pd(4 * P, 4, 0, 0);
    printf("put %d\n", t2i_ctl_put(c, &big, 1, ids));
    show_evictions(c);
    t2i_stats s;
    t2i_ctl_stats(c, &s);
    printf("used %llu free %llu evictions %llu\n", (unsigned long long)s.used_pages, (unsigned long long)s.free_pages,
           (unsigned long long)s.evictions);
    t2i_ctl_destroy(c);
    return 0;
}
"""

C_DRIVER_WANT = """put 0
put 0
get 0
put 0
evicted: 5 4
pages 6: 3 4 5
get 4 per 4 3 0
put 0
evicted: 3
pages 7: 2
put 2
evicted:
used 6 free 0 evictions 3
"""


def test_control_core_from_c_follows_the_hand_trace(lib, tmp_path):
    """A plain C program linked against the library drives the host control
    core through the C ABI: the LRU victims and pages worked out by hand from
    §5.3 and the readings of the LRU and placement rules (the same trace the
    oracle is pinned by)."""
    src = tmp_path / "drive.c"
    src.write_text(C_DRIVER)
    exe = tmp_path / "drive"
    lib_dir = os.path.dirname(L.LIB_PATH)
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I" + os.path.join(ROOT, "include"), str(src), "-o",
                    str(exe), "-L" + lib_dir, "-l:libt2istore.so", "-Wl,-rpath," + lib_dir], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    assert out == C_DRIVER_WANT


def test_cpython_binding_marshals_only(lib):
    """The CPython entry points pass their integer arguments to the same C-ABI
    calls: a null store handle comes back INVALID from the library, the ids
    given to get_batch_ids land in the descriptors' id fields first, and bad
    argument lists raise before any call."""
    import numpy as np

    from paper_2607_26566_gb300 import build as b
    from paper_2607_26566_gb300.store import GET_DTYPE

    fast = L.pycall()
    if fast is None:
        assert not b._have_python_h()
        pytest.skip("built without Python.h: the ctypes binding serves every call")
    assert fast.put_batch(0, 0, 0, 0, 0) == L.ERR_INVALID
    assert fast.get_batch(0, 0, 0, 0, 0) == L.ERR_INVALID
    assert fast.free(0, 0, 0) == L.ERR_INVALID
    descs = np.zeros(3, GET_DTYPE)
    ids = np.array([7, 9, 11], np.uint64)
    assert fast.get_batch_ids(0, descs.ctypes.data, 3, ids.ctypes.data, 0, 0) == L.ERR_INVALID
    assert list(descs["id"]) == [7, 9, 11]
    with pytest.raises(TypeError):
        fast.put_batch(0, 0, 0, 0)
    with pytest.raises(ValueError):
        fast.get_batch_ids(0, 0, 2, 0, 0, 0)
    with pytest.raises(OverflowError):
        fast.get_batch(0, 0, 1 << 40, 0, 0)


def test_c_driver_builds_against_the_header_and_library(lib):
    """cdriver/handoff_step.c, the handoff workload driven from C through the
    C ABI, compiles and links against include/t2istore.h and the library (it
    runs in the GPU tests and the benchmark)."""
    from paper_2607_26566_gb300 import build as b

    exe = b.build_cdriver()
    assert os.access(exe, os.X_OK)
