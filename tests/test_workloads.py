"""The synthetic workloads have the sizes the five store configurations state."""
import numpy as np

import workloads as W
from oracle import OracleStore, PutItem


def test_tiny_objects():
    first, more = W.tiny_objects(0)
    assert len(first) == 32 and len(more) == 8
    sizes = [x.size for x in first + more]
    assert min(sizes) >= 1024 and max(sizes) < 2 * W.MiB
    assert W.tiny_freed_indices() == [2, 5, 8, 11, 14, 17, 20, 23, 26, 29]
    a, _ = W.tiny_objects(0)
    assert all(np.array_equal(x, y) for x, y in zip(first, a))


def test_handoff_sizes():
    for B, pages in ((1, 7), (4, 23), (8, 45)):
        specs = W.handoff_specs(B)
        assert [s.nbytes for s in specs] == [B * 4 * W.MiB, B * 1536, B * W.MiB, B * 6 * W.MiB]
        assert sum(-(-s.nbytes // (2 * W.MiB)) for s in specs) == pages
    specs = W.handoff_specs(1, text_len=8, text_dim=16, pooled_dim=8, lat_c=2, lat_hw=4, img_hw=8)
    arrs = W.handoff_request(0, 3, specs)
    assert [a.nbytes for a in arrs] == [s.nbytes for s in specs]
    assert arrs[0].dtype == np.uint16 and arrs[2].dtype == np.float32 and arrs[3].dtype == np.float16


def test_dit_weights():
    specs = W.dit_weight_specs()
    assert len(specs) == 1140
    assert sum(s.numel for s in specs) == 11_837_283_328
    layout = W.block_layout(specs)
    assert len(layout) == 57
    for total, members in layout:
        for i, off in members:
            assert off % 256 == 0 and off + specs[i].nbytes <= total


def test_lora_sets():
    proj = W.lora_projections()
    assert len(proj) == 418
    objs = W.lora_objects(8)
    assert len(objs) == 836
    assert sum(n for _, n in objs) == 8 * 8_171_520
    assert abs(sum(n for _, n in W.lora_objects(64)) / W.MiB - 498.75) < 0.01
    ranks = W.lora_ranks(0)
    assert set(np.unique(ranks)) <= {8, 16, 32, 64}
    sets, starts = W.adapter_calls(0, n_calls=20000)
    assert sets.min() >= 0 and sets.max() < 512 and starts.min() >= 0 and starts.max() <= 580
    # the 48 most popular sets take about 72% of the calls under Zipf(1.1)
    top = np.bincount(sets, minlength=512)
    assert 0.68 < np.sort(top)[::-1][:48].sum() / 20000 < 0.76


def test_compaction_trace_small():
    P = 64 * W.KiB
    tr = W.compaction_trace(1, 512, P, n_ops=3000, lo=4 * W.KiB, hi=8 * W.MiB)
    s = OracleStore(512 * P, P, keep_bytes=False)
    ids = {}
    for op in tr.ops:
        if op[0] == "alloc":
            st, (i,) = s.put_batch([PutItem(op[2])])
            assert st == 0
            ids[op[1]] = i
        else:
            assert s.free([ids.pop(op[1])]) == 0
    assert sorted(ids) == tr.survivors
    assert s.used_pages() <= 256
