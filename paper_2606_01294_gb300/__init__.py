"""GB300-native Curvature-Conditioned Query (arxiv 2606.01294) kernels.

The hot path -- CCQ-GLA / CCQ-Gated-DeltaNet chunkwise forward and the CCQ
decode step -- runs in libccq.so (hand-written sm_103a CUDA, C ABI in
include/ccq.h).  This package is its thin binding; it needs a CUDA device.
"""
from .ccq import (  # noqa: F401
    CCQError,
    CCQState,
    GDN,
    GLA,
    decode_step,
    device_status,
    gdn_fwd,
    gla_fwd,
    load_library,
)
