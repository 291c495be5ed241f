"""GB300-native (sm_103a) DBRX-style Mixture-of-Experts layer.

The layer of arxiv 2506.23635 (Sec. 2.1, Table 1): a router with softmax and
top-k selection, a token-to-expert dispatch, a SiLU-GLU expert FFN over the
selected experts, and a weighted combine.  Every step is a hand-written CUDA
kernel behind the C ABI declared in ``include/moe.h``; ``paper_2506_23635_gb300.moe``
is the Python binding.  Submodules are imported lazily so that the input
generators can be used without loading the CUDA library.
"""
__all__ = ["inputs", "moe", "perf_model", "expert_parallel"]
