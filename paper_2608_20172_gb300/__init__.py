"""GB300-native FlashRelation: the exact causal Self-Exchange / Multi-Head Relation
operator (arxiv 2608.20172) as hand-written sm_103a CUDA kernels behind a C ABI.

The compute path is ``librelation.so`` (see ``include/relation.h``); this package
holds its build step (``build``), a thin ctypes binding (``binding``) and the seeded
synthetic workloads (``workloads``).  Importing the package does not load the CUDA
library; ``binding.load()`` does, and fails loudly when it is missing.
"""
__all__ = ["build", "binding", "workloads"]
