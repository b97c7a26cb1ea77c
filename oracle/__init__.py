"""CPU oracle of the paged tensor store.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its CPU-baseline leg and ``--impl reference``) may import it.
The product path (``paper_2607_26566_gb300``) never imports, calls or links
anything here, and nothing here imports the product: the two share only the
seeded input generators in ``workloads/``.

* :mod:`oracle.store` -- the store as a map id -> bytes plus the paged model
  (free-page stack, page lists, LRU, compaction) that fixes its metadata.
* :mod:`oracle.cast`  -- fp32 -> bf16 round-to-nearest-even on bit patterns.
"""
from .cast import cast_bytes_f32_to_bf16, f32_bits_to_bf16_bits  # noqa: F401
from .store import (EVICTED, INVALID, NOSPACE, NOT_FOUND, OK, OracleStore, PutItem,  # noqa: F401
                    pages_for)
