"""First-layer prefix caching (§5.1, Eq. 1 and Eq. 2) and its pipeline (oracle).

TEST INFRASTRUCTURE ONLY: imported by ``tests/`` and ``bench.py``, never by
the product path.

A model of L layers keeps its first L_e layers in GPU memory; the others are
loaded from host memory one after another while inference runs. Loading one
layer takes T_load, computing one takes T_comp.

* Eq. (1), the paper's end-to-end latency for uniform layers with
  T_load >> T_comp:  T_e2e(L_e) = max(L * T_comp, (L - L_e) * T_load + T_comp).
* Eq. (2), the smallest prefix that hides loading completely:
  L_e' = ceil((L * (T_load - T_comp) + T_comp) / T_load), here clamped to
  [0, L] (a negative value means nothing has to be cached; the paper states
  the formula for T_load >> T_comp).
* The pipeline the equations summarise, written as a step-by-step schedule
  (used to pin Eq. 1 and for the non-uniform extension the paper mentions
  without giving): layer l's load starts when layer l-1's load ends (cached
  layers need none), its computation starts when its load and layer l-1's
  computation have both ended. The end of the last computation is the
  latency. The smallest prefix for non-uniform layers is the smallest L_e
  whose latency equals the sum of the computations (nothing exposed).
"""
from __future__ import annotations

import math


def e2e_latency_eq1(L: int, L_e: int, t_load: float, t_comp: float) -> float:
    """Eq. (1)."""
    return max(L * t_comp, (L - L_e) * t_load + t_comp)


def prefix_layers_eq2(L: int, t_load: float, t_comp: float) -> int:
    """Eq. (2), clamped to [0, L]."""
    v = math.ceil((L * (t_load - t_comp) + t_comp) / t_load)
    return min(max(v, 0), L)


def pipeline_latency(t_load: list, t_comp: list, L_e: int) -> float:
    """The schedule above, simulated layer by layer."""
    load_end = 0.0       # when the last issued load finished
    comp_end = 0.0
    for l in range(len(t_comp)):
        if l < L_e:
            ready = 0.0                      # cached: available at once
        else:
            load_end = load_end + t_load[l]  # loads run one after another from t = 0
            ready = load_end
        start = max(comp_end, ready)
        comp_end = start + t_comp[l]
    return comp_end


def prefix_layers_search(t_load: list, t_comp: list, rel_tol: float = 1e-12) -> int:
    """Smallest L_e whose pipeline latency equals sum(t_comp), by trying them all."""
    total = sum(t_comp)
    for L_e in range(len(t_comp) + 1):
        if pipeline_latency(t_load, t_comp, L_e) <= total * (1 + rel_tol):
            return L_e
    return len(t_comp)
