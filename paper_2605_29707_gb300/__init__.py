"""GB300-native (sm_103a) Domino draft-side block step.

The work happens in libdomino.so (hand-written CUDA: tcgen05 tensor-core GEMMs with TMA, a
cooperative GRU kernel and a best-first tree kernel) behind the C ABI of include/domino.h.
`binding` mirrors that ABI with ctypes; `step.DraftStep` owns device buffers for one shape;
`inputs` draws the seeded synthetic workloads.  Nothing here falls back to a CPU path.
"""
__all__ = ["binding", "step", "inputs", "build"]
