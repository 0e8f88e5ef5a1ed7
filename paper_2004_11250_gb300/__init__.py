"""GB300-native pattern- and connectivity-pruned 3x3 convolution.

``paper_2004_11250_gb300.ppconv`` is the Python binding of the C-ABI library
(``include/ppconv.h``); importing it loads the compiled CUDA library and fails
loudly when it is missing.  ``paper_2004_11250_gb300.synth`` draws the seeded
synthetic workloads.  This package file itself loads nothing.
"""
