"""GB300-native (sm_103a) Higher-order Linear Attention.

The compute lives in the CUDA library ``libhla.so`` (C ABI in include/hla.h);
``paper_2510_27258_gb300.hla`` is its Python binding.  Build the library with
``paper_2510_27258_gb300.build.build()``.
"""
from .hla import (HLAError, alloc_workspace, hla2_forward, hla2_forward_path, hla2_state_floats, hla2_step, hla2_workspace_bytes,
                  hla3_forward, hla3_state_floats, hla3_workspace_bytes, hla_poll_error, hla_status_string)

__all__ = ["HLAError", "alloc_workspace", "hla2_forward", "hla2_forward_path", "hla2_state_floats", "hla2_step", "hla2_workspace_bytes",
           "hla3_forward", "hla3_state_floats", "hla3_workspace_bytes", "hla_poll_error", "hla_status_string"]
