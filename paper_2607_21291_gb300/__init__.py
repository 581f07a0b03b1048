"""GB300-native depth-sparse forward of AdaDSF (Adaptive Depth Sparse Framework).

Submodules:
  adadsf  ctypes binding of the C ABI (include/adadsf.h) -> libadadsf.so
  synth   seeded synthetic inputs and backbone shapes
  build   nvcc build of libadadsf.so for sm_103a
"""
