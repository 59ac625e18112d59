"""GB300-native budget-routed decode (BUDDY, arXiv 2606.09514).

The compute path is libbuddy.so (CUDA kernels for sm_103a behind the C ABI in
include/buddy.h); `binding` marshals arguments to it.  There is no CPU path.
"""
from .binding import (Context, KVCache, BuddyError, load_library, pack_layer,  # noqa: F401
                      buddy_budget_to_k)
