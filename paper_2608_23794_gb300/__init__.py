"""MoCE (Mixture of Channel Experts) layer forward for NVIDIA GB300 (sm_103a).

Modules:
  moce       Python binding of the C ABI in include/moce.h (torch tensors in, CUDA kernels run)
  build      nvcc build of libmoce.so
  synth      seeded synthetic layers (inputs only)
  costmodel  the paper's MAC / storage / byte accounting
"""
