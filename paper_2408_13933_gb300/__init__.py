"""GB300-native integer-only quantized linear layer (MobileQuant, arXiv 2408.13933).

Submodules:
  mq     -- ctypes binding of the C-ABI library libmq.so (the CUDA path).
  synth  -- seeded synthetic inputs (no layer arithmetic).
  build  -- in-tree build of libmq.so with nvcc for sm_103a.

Importing the package loads nothing; ``from paper_2408_13933_gb300 import mq``
loads the CUDA library and fails loudly if it is missing.
"""
