"""GB300 (sm_103a) hot path of Scale-QLoRA's scale-only training step.

The compute lives in libscaleqlora.so (C ABI in include/scaleqlora.h); this
package holds its ctypes binding (`_lib`), the nvcc build (`build`) and the
seeded synthetic-workload generator (`synth`).
"""
from ._lib import BLOCK, MXFP4, NVFP4, GroupedWeight, Handle, QuantWeight, SQError, load  # noqa: F401
