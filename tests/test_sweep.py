"""The tuning-sweep tool's reading of a bench line (CPU only; the sweep itself
runs bench.py on a GPU)."""
from paper_2607_26566_gb300.sweep import summary


def test_summary_takes_the_compared_figures():
    line = {"value": 7100.0,
            "roofline": {"kernel": "scatter_put_kernel", "achieved": 7090.0,
                         "other_kernel": {"name": "gather_get_kernel", "achieved": 7130.0},
                         "one_stream": {"step_gbs": 6570.0, "put_achieved": 6560.0, "get_achieved": 6590.0}},
            "sweep": {"B1": 6600.0, "B1_one_stream": 4000.0, "B4": 7080.0},
            "rows": {"adapters": {"hit_gbs": 6700.0}, "unaligned": {"cast_dst+2_gbs": 6500.0, "bit_exact": True}}}
    s = summary(line)
    assert s == {"headline": 7100.0, "put_4s": 7090.0, "get_4s": 7130.0, "step_1s": 6570.0, "put_1s": 6560.0,
                 "get_1s": 6590.0, "B1": 6600.0, "B1_one_stream": 4000.0, "B4": 7080.0, "adapter_hits": 6700.0,
                 "cast_dst+2_gbs": 6500.0}
    # a get-dominated line and a rows-only line
    line["roofline"]["kernel"] = "gather_get_kernel"
    line["roofline"]["other_kernel"]["name"] = "scatter_put_kernel"
    assert summary(line)["get_4s"] == 7090.0 and summary(line)["put_4s"] == 7130.0
    assert summary({"rows": {"compaction": {"gbs": 7000.0, "call_gbs": 6800.0}}}) == {
        "compaction": 7000.0, "compaction_call": 6800.0}
