"""GB300 (sm_103a) parameter-space hot path of 1.5-SPSA: probe generation,
fused perturb, probe-space preconditioner and fused K-probe update, behind the
C ABI of include/zo.h. The shared library is loaded on first use; a missing
library raises (there is no fallback).
"""
from .zo import (ZO_ERR_ALIGN, ZO_ERR_ARG, ZO_ERR_CUDA, ZO_ERR_DTYPE, ZO_ERR_NONFINITE, ZO_ERR_TOO_MANY_PROBES,
                 ZO_ERR_WORKSPACE, ZO_MAX_PROBES, ZO_OK, ZO_PRECOND_ONE_SIDED, ZO_PRECOND_RELATIVE_CURVATURE,
                 ZO_QUADRATIC_LOSS_STATIC_MAX_N, ParamList, QuadraticLoss, QuadraticPass, ZoError, get_packing, packing, perturb,
                 perturb2, perturb_pair, perturb_quadratic_loss, perturb_quadratic_loss_workspace_size, precondition,
                 probe_bytes, probe_signs, quadratic_loss, quadratic_loss_static, quadratic_loss_workspace_size,
                 set_packing, status_string, update, update_sequential, version)
from . import replicas

__all__ = ["replicas", "ParamList", "QuadraticLoss", "QuadraticPass", "ZoError", "perturb_quadratic_loss",
           "perturb_quadratic_loss_workspace_size", "set_packing", "get_packing", "packing", "perturb", "perturb2", "perturb_pair",
           "precondition", "update", "update_sequential", "probe_bytes", "probe_signs", "quadratic_loss",
           "quadratic_loss_static", "quadratic_loss_workspace_size", "status_string", "version", "ZO_OK",
           "ZO_ERR_ARG", "ZO_ERR_DTYPE", "ZO_ERR_ALIGN", "ZO_ERR_NONFINITE", "ZO_ERR_CUDA", "ZO_ERR_TOO_MANY_PROBES",
           "ZO_ERR_WORKSPACE", "ZO_MAX_PROBES", "ZO_QUADRATIC_LOSS_STATIC_MAX_N", "ZO_PRECOND_ONE_SIDED",
           "ZO_PRECOND_RELATIVE_CURVATURE"]
