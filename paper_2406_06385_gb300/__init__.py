"""GB300-native LR-QAT linear layer (arXiv 2406.06385).

The CUDA library (``_lib/liblrqat.so``) is loaded lazily by
``paper_2406_06385_gb300.lrqat``; importing this package does not touch CUDA.
"""
