"""GB300-native (sm_103a) MPCache decode path: static eviction, hierarchical
clustering, hierarchical cluster selection with cross-layer index sharing and
sparse decode attention, behind the C ABI declared in include/mpcache.h.

Importing the package loads nothing; ``paper_2501_06807_gb300.mpcache`` loads
the CUDA library on first use and raises if it is missing.
"""
