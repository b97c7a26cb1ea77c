"""GB300-native paged tensor store: the GPU-resident data plane of a
serverless text-to-image system (arxiv 2607.26566, §5).

The library is ``libt2istore.so`` (C ABI in ``include/t2istore.h``), built
in-tree by :mod:`paper_2607_26566_gb300.build`. This package is its thin
Python binding; importing :class:`Store` or :class:`Ctl` loads the library and
fails loudly if it has not been built.
"""
from .store import (GET_DTYPE, MOVE_DTYPE, PUT_DTYPE, Ctl, Store, T2IError, e2e_latency, gather_noalloc,  # noqa: F401
                    get_descs, pipeline_latency, prefix_layers, prefix_layers_pipeline, put_descs)
