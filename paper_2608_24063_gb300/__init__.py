"""GB300-native (sm_103a) PruneKV visual-KV compression pass of VisCache.

``viscache`` is the Python binding of the C-ABI library ``_lib/libviscache.so``
(see ``include/viscache.h``); ``synth`` draws the seeded synthetic inputs.
"""
from . import synth  # noqa: F401

__all__ = ["synth", "viscache"]
