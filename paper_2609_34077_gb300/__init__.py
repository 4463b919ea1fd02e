"""mcft: GB300-native masked MoE layer forward with a per-layer expert cache.

The compute path is the CUDA library ``libmcft.so`` (C ABI declared in ``include/mcft.h``); this
package only marshals arguments to it. ``inputs`` draws the seeded synthetic inputs.
"""
