"""GB300-native Delta Attention prefill (arXiv 2505.11254).

The compute path is the CUDA library ``libdeltaattn.so`` (sm_103a kernels
behind a C ABI, declared in ``include/delta_attn.h``); ``binding`` is its thin
ctypes binding.  ``inputs`` draws the seeded synthetic workloads and ``flops``
does the work accounting.  Importing this package does not load the CUDA
library; ``binding.load()`` does, and fails loudly when it is missing.
"""
__all__ = ["binding", "inputs", "flops"]
