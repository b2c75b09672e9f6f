"""TransX serving hot path on GB300 (sm_103a).

``build`` compiles libtxs.so in-tree, ``txs`` is the ctypes binding of its C ABI
(include/txs.h) and ``workload`` draws the seeded synthetic inputs.  The binding
is imported lazily so that the input generator works without a GPU.
"""
__all__ = ["build", "txs", "workload"]
