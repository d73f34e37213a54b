"""GB300-native TPP-SD sampler (arxiv 2507.09252): C-ABI CUDA library + binding.

The product path is libtppsd.so (built from csrc/ for sm_103a) called through
paper_2507_09252_gb300.tppsd.  There is no CPU fallback.
"""
