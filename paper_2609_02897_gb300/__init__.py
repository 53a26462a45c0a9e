"""GB300-native tree verification for margin-based lossy speculative decoding.

Submodules
  asd    ctypes binding of the C-ABI library libasd (loads it on import and
         raises if it has not been built)
  synth  seeded synthetic workloads (inputs only)
  build  compiles libasd for sm_103a with nvcc
"""
