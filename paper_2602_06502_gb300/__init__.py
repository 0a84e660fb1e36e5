"""GB300 (sm_103a) implementation of DualMap's batched request-routing path
(arxiv 2602.06502): prompt hashing, dual consistent-hash rings, cache-index
probes, SLO-aware choice, LRU commit, hotspot rebalancing, ring add/remove.

The compute lives in libdualmap.so (hand-written CUDA behind the C ABI in
include/dualmap.h); `dualmap` is its ctypes binding and `scheduler` a thin
wrapper holding torch device buffers.
"""
