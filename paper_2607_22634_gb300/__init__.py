"""PRESTO tree draft-and-verify step on one GB300 (sm_103a).

The computation lives in libpresto.so (hand-written CUDA, C ABI in
include/presto.h; libpresto_checks.so, loaded under PRESTO_CHECKS=1, is the same code
with device-side bounds checks); this package holds its build script, a ctypes binding with the
same entry-point names, and `DraftVerifyStep`, which keeps one round's buffers
resident and replays the round's calls (optionally as one CUDA graph).
"""

from ._lib import (  # noqa: F401
    BUILD_CHECKS,
    DEV_STATUS_BITS,
    SEARCH_BEAM,
    SEARCH_BEST_FIRST,
    SEARCH_EAGER,
    Ngram3Table,
    PrestoError,
    dev_status_names,
    lib_path,
    load,
    pack_trigram_keys,
    presto_accept,
    presto_attn_launches,
    presto_attn_workspace,
    presto_build_flags,
    presto_build_workspace,
    presto_score_build_tree,
    presto_score_build_tree_noalloc,
    presto_selftest_wait_timeout,
    presto_topk,
    presto_topk_entropy,
    presto_topk_slots,
    presto_topk_workspace,
    presto_tree_attention,
    presto_tree_mask,
)
from .step import DraftVerifyStep, StagedRounds  # noqa: F401
