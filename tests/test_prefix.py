"""The library's prefix-caching arithmetic (t2i_e2e_latency, t2i_prefix_layers,
t2i_pipeline_latency, t2i_prefix_layers_pipeline) against the oracle, on CPU."""
import numpy as np
import pytest

import oracle.prefix as op
from paper_2607_26566_gb300 import (T2IError, e2e_latency, pipeline_latency, prefix_layers,
                                    prefix_layers_pipeline)
from tests.test_oracle_prefix import golden_rows


def test_golden(lib):
    for L, tl, tc, le, t_at, t_below in golden_rows():
        assert prefix_layers(L, tl, tc) == le
        assert e2e_latency(L, le, tl, tc) == pytest.approx(t_at, abs=1e-12)
        assert e2e_latency(L, le - 1, tl, tc) == pytest.approx(t_below, abs=1e-12)


def test_uniform_vs_oracle(lib):
    g = np.random.default_rng(4)
    for _ in range(2000):
        L = int(g.integers(0, 120))
        tc = float(g.uniform(0.0, 3.0))
        tl = float(g.uniform(0.01, 30.0))
        assert prefix_layers(L, tl, tc) == op.prefix_layers_eq2(L, tl, tc)
        le = int(g.integers(0, L + 1))
        assert e2e_latency(L, le, tl, tc) == op.e2e_latency_eq1(L, le, tl, tc)


def test_nonuniform_vs_oracle(lib):
    g = np.random.default_rng(5)
    for _ in range(300):
        L = int(g.integers(1, 60))
        loads = g.uniform(0.0, 5.0, L)
        comps = g.uniform(0.0, 2.0, L)
        for le in (0, L // 3, L):
            assert pipeline_latency(loads, comps, le) == op.pipeline_latency(list(loads), list(comps), le)
        assert prefix_layers_pipeline(loads, comps) == op.prefix_layers_search(list(loads), list(comps))


def test_invalid_arguments(lib):
    with pytest.raises(T2IError):
        e2e_latency(4, 5, 1.0, 1.0)
    with pytest.raises(T2IError):
        prefix_layers(4, 0.0, 1.0)
    with pytest.raises(T2IError):
        pipeline_latency([1.0, float("nan")], [1.0, 1.0], 0)
