"""RippleKV serving hot path on GB300 (sm_103a).

Submodules:
  ripple  -- ctypes binding of the C-ABI library libripple.so (the product path)
  synth   -- seeded synthetic inputs (no step of the method)
  serving -- per-layer decode loop between the caller's projections, in a CUDA graph
  build   -- in-tree build of libripple.so with nvcc/gcc

Nothing is imported eagerly, so that importing the package never loads CUDA.
"""
