"""GB300-native hot path of Multimodal Speculative Decoding (MSD, arXiv 2505.14260).

One greedy draft-then-verify decode step of a LLaVA-style decoder, written as
hand-written sm_103a CUDA kernels behind the C ABI declared in include/msd.h.

Submodules:
  synth  seeded synthetic workloads (weights, prompts); holds none of the
         method's arithmetic and is shared by the tests, the bench and the oracle
         harness.
  msd    thin ctypes binding of the C ABI (argument marshalling only).
  build  compiles the CUDA library in-tree for sm_103a.
"""
