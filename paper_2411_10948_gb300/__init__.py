"""GB300-native ShiftQuant (arXiv 2411.10948): quantized training GEMMs on sm_103a.

The compute path is libshiftquant.so (hand-written CUDA behind the C ABI declared in
include/shiftquant.h).  `native` binds it one-to-one; `layer` strings the calls of one
quantized linear layer together; `workloads` generates the seeded synthetic inputs.
Importing this package does not load the CUDA library; the first native call does.
"""
__all__ = ["native", "layer", "workloads", "build"]
