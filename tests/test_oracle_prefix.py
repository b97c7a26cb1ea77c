"""Pins of the oracle's prefix-caching equations (§5.1, Eq. 1 and Eq. 2).

Eq. (1) is pinned by the layer-by-layer schedule it summarises (a different
computation: a simulation, not the closed form) and Eq. (2) by searching all
prefixes for the smallest one that hides loading; both by hand-evaluated
values in tests/golden/prefix_layers.txt. Planted mistakes must fail them.
"""
import os

import numpy as np
import pytest

import oracle.prefix as op

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "prefix_layers.txt")


def golden_rows():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            L, tl, tc, le, t1, t0 = line.split()
            rows.append((int(L), float(tl), float(tc), int(le), float(t1), float(t0)))
    return rows


def check_golden(eq1, eq2):
    for L, tl, tc, le, t_at, t_below in golden_rows():
        if eq2(L, tl, tc) != le:
            return False
        if abs(eq1(L, le, tl, tc) - t_at) > 1e-9 or abs(eq1(L, le - 1, tl, tc) - t_below) > 1e-9:
            return False
    return True


def check_against_schedule(eq1, eq2, n=400, seed=0):
    g = np.random.default_rng(seed)
    for _ in range(n):
        L = int(g.integers(1, 80))
        tc = float(g.uniform(0.1, 2.0))
        tl = tc * float(g.uniform(1.0, 15.0))          # T_load >= T_comp, the equations' domain
        loads, comps = [tl] * L, [tc] * L
        for L_e in {0, L // 2, L, int(g.integers(0, L + 1))}:
            if abs(op.pipeline_latency(loads, comps, L_e) - eq1(L, L_e, tl, tc)) > 1e-9 * L * tl:
                return False
        if op.prefix_layers_search(loads, comps) != eq2(L, tl, tc):
            return False
    return True


def test_golden_values():
    assert check_golden(op.e2e_latency_eq1, op.prefix_layers_eq2)


def test_eq1_is_the_schedule_and_eq2_its_minimal_prefix():
    assert check_against_schedule(op.e2e_latency_eq1, op.prefix_layers_eq2)


def test_schedule_special_cases():
    # everything cached: pure compute; nothing cached, one layer: load then compute
    assert op.pipeline_latency([5.0] * 3, [1.0] * 3, 3) == 3.0
    assert op.pipeline_latency([5.0], [1.0], 0) == 6.0
    # compute slower than loading: one cached layer is not needed once loads keep up
    assert op.pipeline_latency([1.0] * 4, [2.0] * 4, 0) == 9.0     # 1 + 4 * 2
    assert op.prefix_layers_eq2(10, 1.0, 2.0) == 0                # clamped
    # non-uniform: a big first layer, small later ones
    loads, comps = [10.0, 1.0, 1.0, 1.0], [1.0, 1.0, 1.0, 1.0]
    assert op.prefix_layers_search(loads, comps) == 1


def _eq2_floor(L, tl, tc):
    return min(max(int(np.floor((L * (tl - tc) + tc) / tl)), 0), L)


def _eq2_no_tcomp(L, tl, tc):
    return min(max(int(np.ceil(L * (tl - tc) / tl)), 0), L)


def _eq1_no_tcomp(L, L_e, tl, tc):
    return max(L * tc, (L - L_e) * tl)


@pytest.mark.parametrize("eq1,eq2", [(op.e2e_latency_eq1, _eq2_floor), (op.e2e_latency_eq1, _eq2_no_tcomp),
                                     (_eq1_no_tcomp, op.prefix_layers_eq2)])
def test_planted_mistakes_are_caught(eq1, eq2):
    assert not (check_golden(eq1, eq2) and check_against_schedule(eq1, eq2))
