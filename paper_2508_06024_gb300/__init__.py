"""GB300-native EC²MoE MoE-layer forward (arXiv 2508.06024).

The compute path lives in ``libec2moe.so`` (hand-written CUDA for sm_103a
behind the C ABI declared in ``include/ec2moe.h``); ``ec2moe`` is its thin
ctypes binding.  Importing this package does not load the library.
"""
