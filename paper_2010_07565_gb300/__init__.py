"""GB300-native Bi-GCN binarized graph-convolution layer forward.

The compute path is a C-ABI CUDA library (``libbigcn.so``, declared in
``include/bigcn.h``); :mod:`.binding` marshals torch device tensors into it
under the same function names. :mod:`.inputs` draws the seeded synthetic
workloads, and :mod:`.cost_model` restates the paper's analytic size and
operation counts (Sec. 5). Importing the package loads nothing native: the
library is loaded on first use of the binding, which fails loudly if it has
not been built.
"""

__all__ = ["binding", "inputs", "cost_model"]
