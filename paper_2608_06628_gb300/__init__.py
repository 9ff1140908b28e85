"""Block-hybrid attention for blockwise dLLM decoding on GB300 (sm_103a).

Section 3.1 of "Retrofitting Linear Attention into Diffusion Language
Models": exact softmax inside the active block, a fixed-size Hedgehog
linear-attention state over committed blocks, and a gated shared normaliser.
The compute runs in the CUDA library libhybrid.so (C ABI in include/hybrid.h);
``hybrid`` is its Python binding, ``state_pool`` allocates states and
``workloads`` draws seeded synthetic inputs.
"""
from . import hybrid, state_pool, workloads  # noqa: F401
from .hybrid import *  # noqa: F401,F403
