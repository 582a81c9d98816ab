"""GB300-native batched evaluation of physical execution plans.

The product is the CUDA library ``libwf.so`` (C ABI in ``include/wf.h``);
``wf`` is its ctypes binding.  Build with ``paper_2609_03335_gb300.build.build()``.
"""
from .wf import (DevicePlans, Results, Ctx, WfError, evaluate, load_library, wf_ctx_create,
                 wf_ctx_destroy, wf_ctx_status, wf_eval_plans, wf_forecast_readiness, wf_last_error,
                 wf_problem_check, wf_strerror, wf_topk)

__all__ = ["DevicePlans", "Results", "Ctx", "WfError", "evaluate", "load_library", "wf_ctx_create",
           "wf_ctx_destroy", "wf_ctx_status", "wf_eval_plans", "wf_forecast_readiness",
           "wf_last_error", "wf_problem_check", "wf_strerror", "wf_topk"]
