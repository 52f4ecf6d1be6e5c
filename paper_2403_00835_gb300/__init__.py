"""GB300-native (sm_103a) Jacobi decoding of LLaMA-style decoders, the
computation that Consistency LLMs (arXiv 2403.00835) accelerate.

The compute path is the CUDA library behind include/cllm.h; ``cllm`` is its
Python binding and ``synthetic`` the seeded input generators."""
