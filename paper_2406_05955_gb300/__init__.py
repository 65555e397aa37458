"""GB300-native activation-sparse dReLU FFN (Turbo Sparse, arXiv 2406.05955).

``binding`` wraps the C ABI of libtsffn (include/ts_ffn.h); ``workload`` draws
the seeded synthetic inputs; ``build`` compiles the sm_103a library in-tree.
"""
from .binding import (Ffn, Graph, Moe, Predictor, TsError, lib, moe_stack_forward,  # noqa: F401
                      stack_forward, stack_forward_predicted)
