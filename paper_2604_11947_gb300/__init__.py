"""ResBM boundary bottleneck on GB300 (sm_103a): the residual encoder-decoder bottleneck at a
pipeline-stage boundary, its identity path, and its backward pass, as hand-written CUDA
kernels behind a C ABI (libresbm.so, include/resbm.h).

Submodules:
  resbm  -- the Python binding of the C ABI (same function names; argument marshalling only)
  synth  -- seeded synthetic inputs shared by tests and benchmarks
  build  -- compiles libresbm.so for sm_103a
"""
