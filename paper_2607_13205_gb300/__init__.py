"""GB300-native (sm_103a) hot path of role-conditional KV-cache eviction
(arXiv 2607.13205): SnapKV / H2O attention-mass scores, role-conditional
per-bucket top-k and K/V gather-compaction, in librolekv (C ABI,
include/rolekv.h) with a thin ctypes binding (``rolekv``)."""

from . import rolekv  # noqa: F401
from .rolekv import (Batch, h2o_score, kept_count, kv_compact, role_alloc_select,  # noqa: F401
                     rolekv_compress, select_params, snapkv_score, workspace, workspace_size)
