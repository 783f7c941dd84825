"""GB300-native implementation of BAG's cached DiT sampling path (budget-aware gating).

The compute path lives in libbag.so (hand-written sm_103a CUDA behind the C ABI of
include/bag.h); `bag` is its Python binding.
"""

from . import configs, synth  # noqa: F401
