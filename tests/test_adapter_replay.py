"""The adapter-cache workload's eviction decisions at full size, on the CPU.

512 LoRA sets behind a 16 GiB pool of 256 KiB pages, all 10,000 Zipf(1.1)
calls of 256-object gets, with the harness's reload-only-the-missing rule:
the library's host control core (t2i_ctl_*) and the oracle's paged model take
the same decisions at every call -- the same objects reloaded, the same
victims in the same order (least recently used set first, its highest block
first, ties to the highest id: §5.3 "How does it work?" and reading 6), the
same free-page stack after every reload, and the same page list for every
live object at checkpoints. The GPU store runs the same control core; its
victims on this trace are compared with the oracle's in the GPU tests.
"""
import numpy as np

import workloads as W
from adapter_replay import AdapterShapes, CtlBackend, OracleBackend, Replay


def _free_pages_np(ctl):
    """The control core's free-page stack as a numpy array (bottom to top)."""
    import ctypes as C

    n = C.c_uint64(0)
    ctl._lib.t2i_ctl_free_pages(ctl._h, None, 0, C.byref(n))
    out = np.zeros(max(1, n.value), np.uint32)
    ctl._lib.t2i_ctl_free_pages(ctl._h, out.ctypes.data_as(C.POINTER(C.c_uint32)), n.value, C.byref(n))
    return out[:n.value]


def _all_pages_equal(core: Replay, ora: Replay):
    live = list(ora.b.ora.objects)
    assert core.b.ctl.stats()["live_objects"] == len(live)
    for oid in live:
        assert core.b.pages(oid) == ora.b.pages(oid), oid


def test_full_adapter_trace_control_core_matches_oracle(lib):
    sh = AdapterShapes()
    pool, P = W.ADAPTERS["pool_bytes"], W.ADAPTERS["page_bytes"]
    ora = Replay(sh, OracleBackend(pool, P))
    core = Replay(sh, CtlBackend(pool, P))
    n_calls = len(sh.sets)
    assert n_calls == W.ADAPTERS["n_calls"] == 10_000
    for k in range(n_calls):
        js_o, ev_o = ora.call(k)
        js_c, ev_c = core.call(k)
        assert js_c == js_o, k                  # the same objects reloaded
        assert ev_c == ev_o, k                  # the same victims, in order
        if js_o:
            assert np.array_equal(_free_pages_np(core.b.ctl), np.asarray(ora.b.free_pages(), np.uint32)), k
            s = int(sh.sets[k])
            for j in (js_o[0], js_o[len(js_o) // 2], js_o[-1]):
                assert core.b.pages(core.ids[s][j]) == ora.b.pages(ora.ids[s][j]), (k, j)
        if k % 2500 == 2499:
            _all_pages_equal(core, ora)
    # the workload exercises what it is meant to: many partial reloads, most
    # of the pool turned over by eviction
    assert ora.loads == core.loads > 3000
    assert len(ora.victims) == len(core.victims) > 1_000_000
    partial = sum(1 for s, m in ora.missing.items() if 0 < len(m) < len(ora.ids[s]))
    assert partial > 0
    st = core.b.ctl.stats()
    assert st["evictions"] == ora.b.ora.stats["evictions"] == len(ora.victims)
    assert st["used_pages"] == ora.b.ora.used_pages()
    core.b.close()
