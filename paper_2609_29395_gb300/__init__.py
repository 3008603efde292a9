"""GB300-native GCPSL (Global Clustered Parallel Split Learning) training step.

The compute path is libgcpsl.so (hand-written sm_103a CUDA behind the C ABI
of include/gcpsl.h); `binding` marshals arguments to it.  `synth`,
`clustering` and `configs` build the host-side inputs (data, client split,
fixed cluster map of Algorithm 1, initial parameters).
"""
from . import binding, clustering, configs, synth  # noqa: F401
from .binding import Context, GcpslError, gcpsl_num_params, load  # noqa: F401
