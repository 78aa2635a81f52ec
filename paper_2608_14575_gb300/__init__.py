"""GB300 (sm_103a) batched, SLO-aware route scoring for HW-Router.

The compute path is the CUDA library libhwr (C ABI in include/hwr.h); this
package holds its sources (csrc/), its build script and a thin ctypes binding.
"""
from ._hwr import (HwrError, Router, load, lib_path, HWR_SEQUENTIAL,
                   HWR_DEVICE_PTRS, HWR_ASYNC, HWR_SCORE_CONVEX, HWR_PATH_SIMT,
                   HWR_PATH_TENSOR, HWR_PROFILE, HWR_F32, HWR_BF16, KERNELS,
                   hwr_create, hwr_update_snapshot, hwr_get_snapshot,
                   hwr_route_batch, hwr_route_batch_slo, hwr_slo_spec, hwr_route_batch_multi,
                   hwr_score_batch,
                   hwr_route_batch_noalloc, HWR_NOALLOC_MAX_Q,
                   hwr_synchronize, hwr_destroy,
                   hwr_status_string, hwr_last_error, hwr_get_stats)
from .build import build
