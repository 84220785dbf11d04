"""GradLev token scans on GB300 (sm_103a).

The token-parallel hot path of GradLev (Token-Parallel Test-Time Training via
Costate Prediction): the forward exclusive prefix scan (Sec. 3 step 2, Eq. 3)
and the costate transpose scan (Sec. 3 step 3, Eq. 4) of a fast-weight
linear map, with optional activation fusion for the two-layer MLP of
Appendix A, both scans of a map in one pass with the consistency term of Eq. 5
(fused_scan), the token-by-token deployment calls (decode_read /
decode_write), document resets for packed sequences (document_gates, or
doc_start= on the scans), the anti-causal suffix read behind the step-size
gradients (suffix_scan / eta_grad), and the derivatives with respect to the
per-token gates eta_t and alpha_t through the decayed suffix read (gate_grads).  Every step runs in the CUDA library
``libgradlev.so`` (see ``include/gradlev.h``); this package only marshals torch
tensors into that C ABI.  There is no CPU fallback: without the library or a GB300 every call
raises.
"""
from ._binding import (ACT_GELU_ERF, ACT_GELU_TANH, ACT_NONE, ACT_TANH, GradLevError,
                       costate_scan, decode_read, decode_workspace_bytes, decode_write,
                       document_gates,
                       device_supported, eta_grad, forward_scan, fused_scan, gate_grads,
                       library_path,
                       load_library,
                       mlp_costate, mlp_forward, suffix_scan, workspace_bytes, workspace_status)

__all__ = ["forward_scan", "costate_scan", "fused_scan", "document_gates", "mlp_forward", "mlp_costate",
           "decode_read", "decode_write", "decode_workspace_bytes", "suffix_scan", "eta_grad",
           "gate_grads",
           "workspace_bytes",
           "workspace_status", "device_supported", "load_library", "library_path", "GradLevError",
           "ACT_NONE", "ACT_GELU_TANH", "ACT_GELU_ERF", "ACT_TANH"]
