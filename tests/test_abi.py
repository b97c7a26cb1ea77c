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
