"""GB300 (sm_103a) implementation of the multi-byte-prediction decode step of a byte-level
hierarchical LM with a Latent-Causal-Attention head. The work happens in ``liblca.so``
(CUDA, C ABI in ``include/lca.h``); ``lca`` is its ctypes binding and ``build`` compiles it."""
