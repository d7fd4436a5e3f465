"""GB300-native fused temporal scan for spiking neural networks (arXiv 2211.10725).

The compute lives in libsnn.so (CUDA, sm_103a) behind the C ABI of
include/snn.h; ``paper_2211_10725_gb300.snn`` is its ctypes binding and
``paper_2211_10725_gb300.workloads`` draws seeded synthetic inputs.
"""
__all__ = ["snn", "workloads", "build_lib"]
