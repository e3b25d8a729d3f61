"""GB300 (sm_103a) evaluator of the Wasserstein-DRO KV-reservation cost grid.

The computation lives in the CUDA library built from ``csrc/`` (C ABI in
``include/kvdro.h``); ``kvdro`` is its Python binding.  ``bcd`` runs the block-coordinate
descent of Alg. 1 on the host around the library's worst-case cost curves.
"""

from . import kvdro  # noqa: F401
from .kvdro import (  # noqa: F401
    KVDRO_FP32,
    KVDRO_ENVELOPE,
    KVDRO_EXACT,
    KVDRO_FP64,
    KvdroError,
    kvdro_create,
    kvdro_destroy,
    kvdro_eval_dual,
    kvdro_eval_grid,
    kvdro_eval_grid_noalloc,
    kvdro_last_error,
    kvdro_last_grid_ms,
    kvdro_load_samples,
    kvdro_quantiles,
    kvdro_sorted_samples,
    kvdro_sync,
)
