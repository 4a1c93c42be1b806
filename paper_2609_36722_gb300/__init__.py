"""GB300-native artifact-KV read path of Attuner (query-side adaptation over a
frozen, independently cached artifact KV store).

The compute runs in libattuner.so (hand-written CUDA for sm_103a); this
package is its ctypes binding.  Build with ``python -m
paper_2609_36722_gb300.build``.
"""

from .attuner import (  # noqa: F401
    AttunerError,
    Context,
    Plan,
    EXPORTS,
    OPT_PREFILL_KERNEL,
    OPT_SPLIT_BLOCKS,
    OPT_WAIT_LIMIT,
    OPT_QPROJ_SPLIT_K,
    OPT_SPLIT_MERGE,
    OPT_SYNC_CHECK,
    OPT_QPROJ_ROWS,
    OPT_SHARE_READS,
    OPT_TEST_STUCK_WAIT,
    lib,
    load_library,
)
