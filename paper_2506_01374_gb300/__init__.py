"""GB300-native schedule-parameterised tensor programs (arXiv 2506.01374).

The data-parallel hot path of the paper's compilation method: executing and
device-timing the schedule variants that a Monte Carlo tree search (Sec. 3.2)
measures, for GEMM with a fused epilogue, a SwiGLU MLP block, causal GQA
attention, implicit-GEMM conv2d and an MoE layer. The kernels live in
``librc.so`` (C ABI in ``include/rc.h``); ``rc`` is its Python binding.
"""
from . import rc  # noqa: F401  (the binding loads librc.so lazily, on first use)

__all__ = ["rc"]
