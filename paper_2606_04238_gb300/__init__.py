"""W4/W2-GateUp decode MLP for GB300 (sm_103a).

``wq`` is the Python binding of libwq.so (include/wq.h); ``synth`` draws the
seeded synthetic inputs; ``_build`` compiles the CUDA library in-tree.
"""
__all__ = ["wq", "synth"]
