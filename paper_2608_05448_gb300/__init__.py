"""DBLast draft+verify step on one GB300 (sm_103a), behind a C ABI.

The computation runs in libdblast.so (CUDA kernels for sm_103a); this package
is its ctypes binding and build script.  Importing it loads the library and
raises if it cannot be built or loaded: there is no CPU fallback.
"""
from .binding import (DBLastError, Head, Workspace, alloc_draft_out,  # noqa: F401
                      alloc_verify_out, dblast_al_objective, dblast_device_status,
                      dblast_draft_and_verify, dblast_draft_block,
                      dblast_set_checks, dblast_set_wait_limit, dblast_stats_get,
                      dblast_stats_reset, dblast_target_determinism,
                      dblast_verify_block, lib)

lib()
