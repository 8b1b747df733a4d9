"""GB300-native GraceKV prefill-time KV-cache compression pass.

The compression pass (curvature-guided segmentation, prototype trees, global
greedy allocation, ragged gather) runs in hand-written sm_103a CUDA kernels
behind the C ABI of include/gracekv.h; ``paper_2608_07001_gb300.gracekv`` is
the Python binding and ``paper_2608_07001_gb300.synth`` the seeded input
generator.
"""
