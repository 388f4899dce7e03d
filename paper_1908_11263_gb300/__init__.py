"""GB300-native quantized HWC convolution (PULP-NN, arXiv 1908.11263).

The compute path lives in the CUDA library libqnn.so (csrc/); `qnn` is its thin
Python binding.  `inputs` draws the seeded synthetic workloads.
"""
__version__ = "0.1.0"
