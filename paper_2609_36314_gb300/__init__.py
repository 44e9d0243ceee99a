"""GB300-native (sm_103a) Frac selective fractional state-space scan (arXiv 2609.36314).

The scan runs in hand-written CUDA kernels behind the C ABI of include/frac.h
(libfrac.so, built in-tree); this package only marshals torch tensors to it.
"""
from .api import (bwd_workspace_size, conv1d_bwd, conv1d_fwd, conv1d_step, decode_step,
                  fwd_workspace_size, gated_rmsnorm_bwd, gated_rmsnorm_fwd, make_dims,
                  param_prep_bwd, param_prep_fwd, prep_config, scan_bwd, scan_fwd)
from ._lib import FracError

__all__ = ["scan_fwd", "scan_bwd", "decode_step", "fwd_workspace_size", "bwd_workspace_size",
           "make_dims", "param_prep_fwd", "param_prep_bwd", "prep_config", "conv1d_fwd",
           "conv1d_bwd", "conv1d_step", "gated_rmsnorm_fwd", "gated_rmsnorm_bwd", "FracError"]
