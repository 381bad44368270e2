"""GB300-native FP8 / NVFP4 quantized linear layer (libqlin + thin binding).

The CUDA library is loaded lazily by :mod:`paper_2609_21849_gb300.qlin`.
"""
