"""GB300 (sm_103a) prefill-only KV selection after MM-ShiftKV.

The computation lives in libmmshift.so (CUDA kernels behind the C ABI of
include/mmshift.h); ``_lib`` is its ctypes binding with the same entry-point
names, ``selector.KVSelector`` a torch-facing convenience, ``synth`` the seeded
synthetic workloads. Importing the package does not load the library; the first
call does, and fails loudly if the library cannot be built or loaded.
"""
from . import synth  # noqa: F401
from ._lib import (MMShiftError, Params, Shape, Debug, check, default_params,  # noqa: F401
                   load_library, make_debug, make_shape, mmshift_build_proxies, mmshift_gather,
                   mmshift_output_rows, mmshift_poll_status, mmshift_proxy_mass,
                   mmshift_scores_topk, mmshift_scores_topk_noalloc, mmshift_select, mmshift_topk,
                   mmshift_workspace_size, mmshift_prefill_stats, mmshift_prefill_stats_workspace_size,
                   mmshift_build_proxies_from_stats, mmshift_select_with_stats,
                   mmshift_hidden_stats_workspace_size, mmshift_hidden_stats,
                   mmshift_hidden_proxies_workspace_size, mmshift_build_hidden_proxies,
                   mmshift_coverage_workspace_size, mmshift_coverage,
                   mmshift_select_head_budgets, mmshift_topk_head_budgets)
