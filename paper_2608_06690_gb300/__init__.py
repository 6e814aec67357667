"""GB300-native policy-masked private-expert MoE layer (arXiv 2608.06690).

``paper_2608_06690_gb300.pmpe`` is the ctypes binding over ``libpmpe.so``
(the C-ABI declared in ``include/pmpe.h``); it is imported on first use so
that the seeded input generator (``inputs``) and the workload registry
(``configs``) load without the CUDA library.
"""
__all__ = ["inputs", "configs", "pmpe"]
